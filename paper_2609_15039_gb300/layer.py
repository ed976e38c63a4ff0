"""One decoder layer's outsourced linears, run through the C ABI.

Sec. 5.2: the inputs of Q, K and V are the same, so one mask serves all
three (three corrections); Gate and Up likewise share one mask (two
corrections); O (and Down, which the paper keeps in the TEE but this
workload includes) get one each.  Per input group the step is

    a2+a3  spl_noise_mask                 X~ = X + eta, eta kept for a4
    a4     spl_precompute_noise_product   C_p = eta W_p^T   for each projection p
    a5+a6  spl_masked_linear_unmask       Y_p = X~ W_p^T - C_p

with the noise scale b = Delta / eps from Thms. 1-3 (a1), evaluated once per
layer by ``sensitivities``.  This module only sequences library calls.
"""

from dataclasses import dataclass, field

import torch

from . import spl



@dataclass
class ProjectionWeights:
    name: str
    group: str
    K: int
    N: int
    W: torch.Tensor
    W_hi: torch.Tensor = None
    W_lo: torch.Tensor = None


@dataclass
class MaskedLayer:
    """Device-resident weights of one layer plus the per-group noise scales."""

    model: object
    projections: list
    deltas: dict = field(default_factory=dict)
    workspace: torch.Tensor = None
    M_max: int = 0

    @classmethod
    def from_weights(cls, model, weights, split=True, device="cuda"):
        """weights: {name: [N, K] fp32 tensor}.  Splits each for TF32X3 when split=True."""
        projs = []
        for name, K, N, g in model.projections():
            W = weights[name].to(device=device, dtype=torch.float32).contiguous()
            pw = ProjectionWeights(name, g, K, N, W)
            if split:
                pw.W_hi = torch.empty_like(W)
                pw.W_lo = torch.empty_like(W)
                spl.spl_split_tf32(pw.W_hi, pw.W_lo, W)
            projs.append(pw)
        return cls(model, projs)

    def proj(self, name):
        return next(p for p in self.projections if p.name == name)

    def sensitivities(self, alpha=None, beta=None, power_iters=100):
        """a1: Delta per input group (Thm. 1 for qkv/gateup, Thm. 2 for o, Thm. 3 for down)."""
        d = self.model.d_model
        a = torch.ones(d) if alpha is None else torch.as_tensor(alpha, dtype=torch.float32)
        d_ln = spl.spl_delta_layernorm(a)
        wv = spl.spl_spectral_norm(self.proj("v").W, iters=power_iters)
        wup = spl.spl_spectral_norm(self.proj("up").W, iters=power_iters)
        wgate = spl.spl_spectral_norm(self.proj("gate").W, iters=power_iters)
        self.deltas = {
            "qkv": d_ln,
            "gateup": d_ln,
            "o": spl.spl_delta_attention(a, wv),
            "down": spl.spl_delta_activation(a, beta, self.model.d_ff, wup, wgate),
        }
        self.norms = {"v": wv, "up": wup, "gate": wgate}
        return self.deltas

    def ensure_workspace(self, M, path="auto"):
        need = max(spl.spl_linear_workspace_bytes(M, p.K, p.N, path) for p in self.projections)
        if self.workspace is None or self.workspace.numel() < need:
            self.workspace = spl.workspace(need, self.projections[0].W.device)
        self.M_max = max(self.M_max, M)
        return self.workspace

    def step(self, inputs, eps, mech, seed, outputs=None, scratch=None, path="auto", stream=None, timer=None):
        """Run every group of the layer once.

        inputs:  {group: X [M, K] device tensor}
        outputs: {name: Y [M, N]} (allocated if None); scratch holds X~, eta, C.
        Philox stream ids: one per group (0..3) under ``seed``, so no two groups
        (and no two layers, if seeds differ) share a counter.  ``timer`` (if
        given) is called as timer("begin"|"end", kind) around each product call.
        """
        ws = self.ensure_workspace(max(x.shape[0] for x in inputs.values()), path)
        outputs = {} if outputs is None else outputs
        scratch = {} if scratch is None else scratch
        for gi, (g, K, names) in enumerate(self.model.input_groups()):
            X = inputs[g]
            M = X.shape[0]
            xt = scratch.get(("xt", g))
            if xt is None or xt.shape != X.shape:
                xt = scratch[("xt", g)] = torch.empty_like(X)
                scratch[("eta", g)] = torch.empty_like(X)
            eta = scratch[("eta", g)]
            spl.spl_noise_mask(xt, eta, X, self.deltas[g], eps, mech, seed, stream_id=gi, stream=stream)
            for name in names:
                p = self.proj(name)
                C = scratch.get(("c", name))
                if C is None or C.shape[0] != M:
                    C = scratch[("c", name)] = torch.empty((M, p.N), device=X.device)
                Y = outputs.get(name)
                if Y is None or Y.shape[0] != M:
                    Y = outputs[name] = torch.empty((M, p.N), device=X.device)
                if timer:
                    timer("begin", "precompute")
                spl.spl_precompute_noise_product(C, eta, p.W, p.W_hi, p.W_lo, path=path, workspace=ws, stream=stream)
                if timer:
                    timer("end", "precompute")
                    timer("begin", "masked_linear_unmask")
                spl.spl_masked_linear_unmask(Y, xt, p.W, C, p.W_hi, p.W_lo, path=path, workspace=ws, stream=stream)
                if timer:
                    timer("end", "masked_linear_unmask")
        return outputs, scratch

    def flops(self, M):
        """Algorithmic flops of one step: the masked product and the correction, 2 M K N each."""
        return sum(2 * 2 * M * p.K * p.N for p in self.projections)
