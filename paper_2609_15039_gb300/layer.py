"""One decoder layer's outsourced linears, run through the C ABI.

Sec. 5.2 of the paper keeps a noise bank: masks and their corrections are
precomputed, one mask serves every projection that shares an input (Q, K, V
share one; Gate and Up share one; O and Down one each), and each entry is
consumed once.  This module keeps that structure, GB300 style:

* weights that share an input are stored as one matrix (Q|K|V is [5120, d],
  Gate|Up is [2 d_ff, d] for Llama), so one product call serves the group and
  its output columns are the individual projections;
* the bank holds only corrections.  ``refill`` draws D masks per group in
  one pass (a2) and computes their corrections C = eta W^T as one product of
  D*M rows (a4, "precomputed in a batch"), each output summed in the same
  order as the online product of M rows, so the rounding errors of the two
  products cancel in the unmask;
* an ``online`` step regenerates its mask from the same Philox counters
  (seed, group stream, block offset of draw d) instead of reading it back,
  masks the input (a3) and runs the masked product with the unmask fused
  into its epilogue, Y = X~ W^T - C_d (a5 + a6);
* ``capture`` records the steps of one bank cycle as CUDA graphs (draw 0
  with the refill): the Philox block offset of each group then lives on the
  device and the last graph moves it to the next cycle, so the same graphs
  replay cycle after cycle with fresh noise and no host work per kernel.

The noise scale Delta per group comes from Thms. 1-3 (a1, ``sensitivities``).
This module only sequences library calls; all arithmetic is in libspl.
"""

from dataclasses import dataclass, field

import torch

from . import spl


@dataclass
class GroupWeights:
    name: str            # qkv | o | gateup | down
    K: int
    names: list          # projections in column order
    widths: list         # output width of each projection
    W: torch.Tensor      # [sum(widths), K]
    wt: spl.Weight = None  # W with the splits the tensor-core paths read

    @property
    def N(self):
        return self.W.shape[0]

    def columns(self, name):
        i = self.names.index(name)
        off = sum(self.widths[:i])
        return off, off + self.widths[i]


@dataclass
class MaskedLayer:
    """Device-resident fused weights of one layer, its noise scales and its correction bank."""

    model: object
    groups: list
    deltas: dict = field(default_factory=dict)
    workspace: torch.Tensor = None
    bank: dict = field(default_factory=dict)
    draws: int = 0
    M: int = 0
    paths: dict = field(default_factory=dict)   # per group, from calibrate(); "auto" if not calibrated
    calibration: dict = field(default_factory=dict)
    rng_base: torch.Tensor = None               # [groups] int64 on the device: Philox block offset of the cycle
    fp64: set = field(default_factory=set)      # groups computed in binary64 (Sec. 5.5; normally {"down"})

    @classmethod
    def from_weights(cls, model, weights, split=True, device="cuda"):
        """weights: {projection: [N, K] fp32}.  Concatenates per input group; splits for TF32X3 and FP16X3."""
        groups = []
        for g, K, names in model.input_groups():
            parts = [weights[n].to(device=device, dtype=torch.float32) for n in names]
            W = torch.cat(parts, dim=0).contiguous() if len(parts) > 1 else parts[0].contiguous()
            gw = GroupWeights(g, K, list(names), [p.shape[0] for p in parts], W)
            gw.wt = spl.Weight.prepare(W) if split else spl.Weight(W)
            groups.append(gw)
        return cls(model, groups)

    def group(self, name):
        return next(g for g in self.groups if g.name == name)

    def weight(self, proj):
        """The [N, K] block of one projection (a view into its group's matrix)."""
        for g in self.groups:
            if proj in g.names:
                a, b = g.columns(proj)
                return g.W[a:b]
        raise KeyError(proj)

    def sensitivities(self, alpha=None, beta=None, power_iters=1000):
        """a1: Delta per input group (Thm. 1 for qkv/gateup, Thm. 2 for o, Thm. 3 for down).

        ||W||_2 comes from power iteration, which approaches it from below;
        enough iterations make the shortfall negligible next to the noise scale.
        """
        d = self.model.d_model
        a = torch.ones(d) if alpha is None else torch.as_tensor(alpha, dtype=torch.float32)
        d_ln = spl.spl_delta_layernorm(a)
        norms = {p: spl.spl_spectral_norm(self.weight(p).contiguous(), iters=power_iters) for p in ("v", "up", "gate")}
        self.deltas = {
            "qkv": d_ln,
            "gateup": d_ln,
            "o": spl.spl_delta_attention(a, norms["v"]),
            "down": spl.spl_delta_activation(a, beta, self.model.d_ff, norms["up"], norms["gate"]),
        }
        self.norms = norms
        return self.deltas

    def calibrate(self, inputs, eps, mech, seed, rows=128):
        """a8: choose FP16X3, TF32X3 or FP32 per group from the bound on a masked sample (spl_choose_path).

        The sample is the first ``rows`` rows of each group's input with a fresh mask drawn
        under a stream id no online step uses.
        """
        for gi, g in enumerate(self.groups):
            X = inputs[g.name][:rows].contiguous()
            eta = torch.empty_like(X)
            spl.spl_noise(eta, self.deltas[g.name], eps, mech, seed, stream_id=1000 + gi)
            name, stats = spl.spl_choose_path(X, eta, g.wt)
            self.paths[g.name] = name
            self.calibration[g.name] = {"path": name, "rows": X.shape[0], **stats}
        return self.paths

    def path_of(self, g, path, rows):
        """The calibrated path for products of more than 8 rows under AUTO (the range where AUTO
        weighs the tensor-core path); smaller products keep AUTO's streaming decode kernel."""
        if path == "auto" and rows > 8:
            return self.paths.get(g.name, path)
        return path

    # ------------------------------------------------------------------ bank
    def workspace_bytes(self, M, draws, path="auto"):
        """Workspace for products of M rows and a bank refill of draws x M rows, every group."""
        need = 0
        for g in self.groups:
            need = max(need, spl.spl_linear_workspace_bytes(M, g.K, g.N, path),
                       spl.spl_precompute_matched_workspace_bytes(draws * M, g.K, g.N, M, path))
            if g.name in self.fp64:
                need = max(need, spl.spl_f64_workspace_bytes(M, g.K, g.N),
                           spl.spl_f64_workspace_bytes(draws * M, g.K, g.N))
        return need

    def allocate(self, M, draws, path="auto", workspace=None, stored_noise=False):
        """Buffers for M tokens and a bank of ``draws`` corrections per group.  ``workspace`` may be
        shared with other layers whose calls run on the same stream.  stored_noise: the FP16X3
        groups keep the bank's fp32 noise, and each online step masks with its rows (spl_mask_split)
        instead of drawing them again -- the same X~ bit for bit, the paper's precomputed noise.  Off
        by default: on GB300 writing and reading the fp32 noise costs more than drawing it again
        (Llama layer at 128 tokens: 267-268 against 271 TFLOP/s), since the split kernel that draws
        it runs while the next product's CTAs start."""
        dev = self.groups[0].W.device
        need = self.workspace_bytes(M, draws, path)
        if workspace is not None:
            assert workspace.numel() >= need, "shared workspace too small"
            self.workspace = workspace
        elif self.workspace is None or self.workspace.numel() < need:
            self.workspace = spl.workspace(need, dev)
        self.M, self.draws = M, draws
        self.stored_noise = bool(stored_noise)
        self.rng_base = torch.zeros(len(self.groups), dtype=torch.int64, device=dev)
        self.bank = {}
        for g in self.groups:
            wide = torch.float64 if g.name in self.fp64 else torch.float32  # binary64 mask and correction
            self.bank[g.name] = {
                "eta": torch.empty((draws * M, g.K), device=dev),  # the draws being precomputed (kept with stored noise)
                "C": torch.empty((draws * M, g.N), device=dev, dtype=wide),
                "xt": torch.empty((M, g.K), device=dev, dtype=wide),
                "Y": torch.empty((M, g.N), device=dev),
            }
            if self._fused_split(g, path, M):  # the fp16 splits of X~ and of the bank's noise
                b = self.bank[g.name]
                b["xs"] = spl.Weight(None, f16_hi=torch.empty((M, g.K), dtype=torch.int16, device=dev),
                                     f16_lo=torch.empty((M, g.K), dtype=torch.int16, device=dev),
                                     f16_exp=torch.empty(M, dtype=torch.int32, device=dev))
                b["es"] = spl.Weight(None, f16_hi=torch.empty((draws * M, g.K), dtype=torch.int16, device=dev),
                                     f16_lo=torch.empty((draws * M, g.K), dtype=torch.int16, device=dev),
                                     f16_exp=torch.empty(draws * M, dtype=torch.int32, device=dev))

    # ------------------------------------------------------------------ stacked schedule
    def allocate_stacked(self, M, draws, path="auto", workspace=None, out=None):
        """Buffers of the stacked schedule: step d of a bank cycle multiplies, in one product of 2M rows
        (spl_masked_linear_unmask_precompute), the M rows of X~ for draw d of this cycle and the M noise
        rows of draw d of the next cycle, so every step carries its share of the bank and the products
        run in the launch shape of 2M rows.  Per group: the left operand [2M, K] (its fp16 split when
        the product runs FP16X3, else fp32) and out[p][d] [2M, N] for parities p = 0, 1: a cycle of
        parity p reads its corrections from out[p][d][M:] and writes [Y; the next cycle's corrections]
        into out[1 - p][d].  A correction and the masked row that later meets it sit in products of
        the same shape, which sum every row in the same order, so their roundings cancel.  When the
        2M rows run on the FP32 decode kernel and fit its fused form (2M <= 4: decode), the noise
        draw, the mask and the product of a step are one launch (spl_noise_mask_linear_unmask_precompute)
        and the left operand is the fp32 X~ it writes.  ``out(name)``, if given, supplies a group's
        out[p][d] (contiguous [2M, N] tensors, e.g. views of a buffer pooled over layers)."""
        dev = self.groups[0].W.device
        need = max(spl.spl_linear_workspace_bytes(2 * M, g.K, g.N, self.path_of(g, path, 2 * M)) for g in self.groups)
        if workspace is not None:
            assert workspace.numel() >= need, "shared workspace too small"
            self.workspace = workspace
        elif self.workspace is None or self.workspace.numel() < need:
            self.workspace = spl.workspace(need, dev)
        self.M, self.draws = M, draws
        self.rng_base = torch.zeros(len(self.groups), dtype=torch.int64, device=dev)
        self.stacked = {}
        for g in self.groups:
            if g.name in self.fp64:
                raise ValueError("stacked schedule: the binary64 group keeps the separate bank")
            fused = self._fused_split(g, path, 2 * M)
            if fused and M % 4:
                raise ValueError("stacked schedule on FP16X3: M % 4 == 0 (the split's row exponents of each "
                                 "half are 16-byte aligned)")
            fused_mask = self._fused_mask(g, path, 2 * M)
            a = (spl.Weight(None, f16_hi=torch.empty((2 * M, g.K), dtype=torch.int16, device=dev),
                            f16_lo=torch.empty((2 * M, g.K), dtype=torch.int16, device=dev),
                            f16_exp=torch.empty(2 * M, dtype=torch.int32, device=dev))
                 if fused else spl.Weight(torch.empty((2 * M, g.K), device=dev)))
            if out is not None:
                bufs = out(g.name)
                assert all(b.shape == (2 * M, g.N) and b.is_contiguous() for row in bufs for b in row)
            else:
                bufs = [[torch.zeros((2 * M, g.N), device=dev) for _ in range(draws)] for _ in range(2)]
            resolved = spl.PATH_NAMES[spl.spl_resolve_path(2 * M, g.K, g.N, self.path_of(g, path, 2 * M))]
            self.stacked[g.name] = {"a": a, "out": bufs, "fused": fused, "fused_mask": fused_mask, "path": resolved}

    def stacked_step(self, inputs, eps, mech, seed, d, parity, cycle=0, path="auto", stream=None, timer=None,
                     device_base=False):
        """Step d of a cycle of parity ``parity`` in the stacked schedule (see allocate_stacked): the mask
        of draw d of this cycle, the noise of draw d of the next cycle, and their product with W in one
        call whose first M rows are unmasked with this cycle's correction.  The arithmetic path of each
        group is the one resolved when the buffers were allocated.  Returns {group: Y [M, N]}."""
        out = {}
        for gi, g in enumerate(self.groups):
            self._stacked_prepare(gi, g, inputs, eps, mech, seed, d, cycle, device_base, stream)
            out[g.name] = self._stacked_product(gi, g, inputs, eps, mech, seed, d, parity, cycle, device_base,
                                                stream, timer)
        return out

    def _stacked_prepare(self, gi, g, inputs, eps, mech, seed, d, cycle, device_base, stream):
        """The left operand of group g for step d where the product takes it ready-made (the noise of
        both halves, the mask and, on FP16X3, the split, in one launch there); nothing where the
        product draws it itself (the one-launch decode form)."""
        M, D = self.M, self.draws
        st = self.stacked[g.name]
        if st["fused_mask"]:
            return
        a = st["a"]
        off, off_dev = self._offset(gi, g, cycle, d, device_base)
        off_next = off + D * (M * g.K // 4)  # draw d of the next cycle
        delta = self.deltas[g.name]
        if st["fused"]:  # both halves of the left operand in one launch
            spl.spl_noise_mask_split_stacked(a.f16_hi, a.f16_lo, a.f16_exp, inputs[g.name], delta, eps, mech, seed,
                                             M, off_next - off, stream_id=gi, offset=off, stream=stream,
                                             offset_dev=off_dev)
        else:
            spl.spl_noise_mask(a.w[:M], None, inputs[g.name], delta, eps, mech, seed, stream_id=gi, offset=off,
                               stream=stream, offset_dev=off_dev)
            spl.spl_noise(a.w[M:], delta, eps, mech, seed, stream_id=gi, offset=off_next, stream=stream,
                          offset_dev=off_dev)

    def _stacked_product(self, gi, g, inputs, eps, mech, seed, d, parity, cycle, device_base, stream, timer):
        """The product call of group g for step d (after _stacked_prepare); returns Y [M, N]."""
        M, D = self.M, self.draws
        st = self.stacked[g.name]
        a = st["a"]
        res = st["out"][1 - parity][d]
        if timer:
            timer("begin", "masked_linear_unmask", g.name)
        if st["fused_mask"]:  # noise, mask and product of both halves in one decode launch
            off, off_dev = self._offset(gi, g, cycle, d, device_base)
            off_next = off + D * (M * g.K // 4)
            spl.spl_noise_mask_linear_unmask_precompute(
                res, a.w, inputs[g.name], g.wt, st["out"][parity][d][M:], self.deltas[g.name], eps, mech, seed, M,
                off_next - off, stream_id=gi, offset=off, path=st["path"], workspace=self.workspace,
                stream=stream, offset_dev=off_dev)
        else:
            spl.spl_masked_linear_unmask_precompute(res, a, g.wt, st["out"][parity][d][M:], M, path=st["path"],
                                                    workspace=self.workspace, stream=stream)
        if timer:
            timer("end", "masked_linear_unmask", g.name)
        return res[:M]

    def enable_overlap(self):
        """A second correction buffer per group (and noise buffer, for stored noise), so that a bank
        cycle can run its online steps on one while the next cycle's are filled into the other
        (capture_overlapped)."""
        for g in self.groups:
            b = self.bank[g.name]
            if "Cs" not in b:
                b["Cs"] = [b["C"], torch.empty_like(b["C"])]
                # the fp32 noise is read again only with stored noise; otherwise one buffer serves
                b["etas"] = [b["eta"], torch.empty_like(b["eta"]) if self.stored_noise else b["eta"]]

    def _C(self, g, parity):
        b = self.bank[g.name]
        return b["Cs"][parity] if "Cs" in b else b["C"]

    def _eta(self, g, parity):
        b = self.bank[g.name]
        return b["etas"][parity] if "etas" in b else b["eta"]

    def _fused_split(self, g, path, M):
        """True when the online product of group g runs FP16X3: then the mask kernel also writes the
        fp16 split of X~ and the product skips its own split pass."""
        if g.name in self.fp64 or g.wt is None or g.wt.f16_hi is None or g.K % 8 or g.K > 16384:
            return False
        return spl.spl_resolve_path(M, g.K, g.N, self.path_of(g, path, M)) == spl.SPL_PATH_FP16X3

    def _fused_mask(self, g, path, M):
        """True when the online product of group g is the FP32 decode kernel at 2 <= M <= 4 rows: then
        one launch draws the noise, masks and multiplies (spl_noise_mask_linear_unmask).  At one row
        the two-launch form is faster on GB300 (Llama shapes: 76 against 79 us per layer): there the
        product's blocks load their first W lines while the small mask kernel runs, whereas the
        fused blocks can only start on W after drawing their noise."""
        if g.name in self.fp64 or not 2 <= M <= 4:
            return False
        return spl.spl_resolve_path(M, g.K, g.N, self.path_of(g, path, M)) == spl.SPL_PATH_FP32

    def block_offset(self, g, cycle, d):
        """First Philox block of draw d of bank cycle ``cycle`` for group g."""
        per_draw = self.M * g.K // 4  # K % 4 == 0, so a draw is a whole number of blocks
        return (cycle * self.draws + d) * per_draw

    def _offset(self, gi, g, cycle, d, device_base):
        """(host offset, device offset tensor or None) of draw d of cycle ``cycle``."""
        if device_base:  # the cycle's base is on the device (set_cycle / the last captured graph)
            return d * (self.M * g.K // 4), self.rng_base[gi:gi + 1]
        return self.block_offset(g, cycle, d), None

    def set_cycle(self, cycle):
        """Put the device-side Philox bases at bank cycle ``cycle`` (for captured graphs)."""
        base = torch.tensor([self.block_offset(g, cycle, 0) for g in self.groups], dtype=torch.int64)
        self.rng_base.copy_(base)

    def refill(self, eps, mech, seed, cycle, path="auto", stream=None, timer=None, device_base=False,
               parallel=False, parity=0, ahead=0, workspace=None):
        """a2 + a4: draw ``draws`` masks per group and precompute their corrections in one product.

        parallel: the FP16X3 groups' corrections that need no workspace (the noise comes split and
        the tensor-core kernel reduces on chip: spl_split_workspace_bytes is 0) run side by side on
        streams of their own, so the tiles of one fill the SMs another leaves idle; the others (the
        swapped kernel of few rows, which sums partial tiles through the workspace) run in order on
        the current stream.  The current stream waits for all of them.
        parity: the correction buffer to fill (see enable_overlap); ahead: the draws of cycle
        ``cycle + ahead`` (with device_base: that many cycles past the device-side base).
        workspace: the workspace of the corrections that take one (default: the layer's), e.g. a
        second one while online steps run beside them."""
        main = torch.cuda.current_stream() if stream is None else stream
        ws = self.workspace if workspace is None else workspace
        forks = []
        for gi, g in enumerate(self.groups):
            b = self.bank[g.name]
            off, off_dev = self._offset(gi, g, cycle + (0 if device_base else ahead), 0, device_base)
            if device_base:
                off += ahead * self.draws * (self.M * g.K // 4)
            C = self._C(g, parity)
            es = b.get("es") if self._fused_split(g, path, self.M) else None
            if es is not None:  # the FP16X3 correction reads only the split: the noise is split as drawn
                side = main
                if parallel and spl.spl_split_workspace_bytes(self.draws * self.M, g.K, g.N, self.M, "fp16x3") == 0:
                    side = self._side_stream(gi)
                    side.wait_stream(main)
                    forks.append(side)
                with torch.cuda.stream(side):
                    # with stored noise, the fp32 draws are kept for the online steps' masks
                    keep = self._eta(g, parity) if self.stored_noise else None
                    spl.spl_noise_mask_split(keep, es.f16_hi, es.f16_lo, es.f16_exp, None, self.deltas[g.name], eps,
                                             mech, seed, stream_id=gi, offset=off, stream=side, offset_dev=off_dev)
                    if timer:
                        timer("begin", "precompute", g.name)
                    spl.spl_precompute_noise_product_matched_split(C, es, g.wt, self.M,
                                                                   path=self.path_of(g, path, self.M),
                                                                   workspace=ws, stream=side)
                    if timer:
                        timer("end", "precompute", g.name)
                continue
            spl.spl_noise(b["eta"], self.deltas[g.name], eps, mech, seed, stream_id=gi, offset=off, stream=stream,
                          offset_dev=off_dev)
            if timer:
                timer("begin", "precompute", g.name)
            if g.name in self.fp64:
                spl.spl_precompute_noise_product_f64(C, b["eta"], g.W, workspace=ws, stream=stream)
            else:
                # summed in the order the online product of M rows uses, so their rounding cancels
                spl.spl_precompute_noise_product_matched(C, b["eta"], g.wt, self.M,
                                                         path=self.path_of(g, path, self.M), workspace=ws,
                                                         stream=stream)
            if timer:
                timer("end", "precompute", g.name)
        for side in forks:
            main.wait_stream(side)

    def _side_stream(self, gi):
        """A stream of this layer for group gi's correction (created once)."""
        if not hasattr(self, "_sides"):
            self._sides = {}
        if gi not in self._sides:
            self._sides[gi] = torch.cuda.Stream()
        return self._sides[gi]

    def online(self, inputs, eps, mech, seed, cycle, d, path="auto", stream=None, timer=None, device_base=False,
               group_hooks=None, parity=0):
        """a3 + a5 + a6 for draw d: regenerate eta_d, mask, masked product with fused unmask.

        inputs: {group: X [M, K]}.  Returns {group: Y [M, N_group]} (views of the layer's buffers).
        group_hooks: (before(gi, name), after(gi, name)) called around each group's calls (e.g. to
        wait for its input copy and to start copying its result out).
        """
        M = self.M
        out = {}
        for gi, g in enumerate(self.groups):
            if group_hooks:
                group_hooks[0](gi, g.name)
            self._online_group(gi, g, inputs, eps, mech, seed, cycle, d, path, stream, timer, device_base, out, parity)
            if group_hooks:
                group_hooks[1](gi, g.name)
        return out

    def _online_group(self, gi, g, inputs, eps, mech, seed, cycle, d, path, stream, timer, device_base, out, parity):
        M = self.M
        b = self.bank[g.name]
        Cd = self._C(g, parity)[d * M:(d + 1) * M]
        off, off_dev = self._offset(gi, g, cycle, d, device_base)
        fp64 = g.name in self.fp64
        xs = b.get("xs") if self._fused_split(g, path, M) else None
        if self._fused_mask(g, path, M):
            if timer:
                timer("begin", "masked_linear_unmask", g.name)
            spl.spl_noise_mask_linear_unmask(b["Y"], b["xt"], inputs[g.name], g.wt, Cd,
                                             self.deltas[g.name], eps, mech, seed, stream_id=gi, offset=off,
                                             path=self.path_of(g, path, M), workspace=self.workspace,
                                             stream=stream, offset_dev=off_dev)
            if timer:
                timer("end", "masked_linear_unmask", g.name)
            out[g.name] = b["Y"]
            return
        if fp64:
            spl.spl_noise_mask_f64(b["xt"], inputs[g.name], self.deltas[g.name], eps, mech, seed, stream_id=gi,
                                   offset=off, stream=stream, offset_dev=off_dev)
        elif xs is not None and self.stored_noise:  # the noise drawn with the bank: its rows for draw d
            spl.spl_mask_split(None, xs.f16_hi, xs.f16_lo, xs.f16_exp, inputs[g.name],
                               self._eta(g, parity)[d * M:(d + 1) * M], stream=stream)
        elif xs is not None:  # the FP16X3 product reads only the split: X~ itself is not written
            spl.spl_noise_mask_split(None, xs.f16_hi, xs.f16_lo, xs.f16_exp, inputs[g.name], self.deltas[g.name],
                                     eps, mech, seed, stream_id=gi, offset=off, stream=stream, offset_dev=off_dev)
        else:
            spl.spl_noise_mask(b["xt"], None, inputs[g.name], self.deltas[g.name], eps, mech, seed, stream_id=gi,
                               offset=off, stream=stream, offset_dev=off_dev)
        if timer:
            timer("begin", "masked_linear_unmask", g.name)
        if fp64:
            spl.spl_masked_linear_unmask_f64(b["Y"], b["xt"], g.W, Cd,
                                             workspace=self.workspace, stream=stream)
        elif xs is not None:
            spl.spl_masked_linear_unmask_split(b["Y"], xs, g.wt, Cd,
                                               path=self.path_of(g, path, M), workspace=self.workspace,
                                               stream=stream)
        else:
            spl.spl_masked_linear_unmask(b["Y"], b["xt"], g.wt, Cd,
                                         path=self.path_of(g, path, M), workspace=self.workspace, stream=stream)
        if timer:
            timer("end", "masked_linear_unmask", g.name)
        out[g.name] = b["Y"]

    def capture(self, inputs, eps, mech, seed, path="auto", timer=None, before=None, after=None, group_hooks=None):
        """CUDA graphs of the ``draws`` steps of one bank cycle: graph d runs online step d (graph 0
        refills the bank first); the last graph moves every group's Philox base on by one cycle.
        Replay graphs[s % draws] for step s after set_cycle(s // draws) -- the graphs read their
        offsets on the device, so they replay cycle after cycle.  ``before(d)`` / ``after(d)`` run
        inside the capture around the step (host-to-device input copies, device-to-host result
        copies), ``group_hooks`` around each group's calls (see online).  ``inputs`` may be a list
        of input dicts: graph d then reads inputs[d % len(inputs)].  Every library call must have run
        once before (warm-up), so nothing is set up during capture.  Returns the graphs and the
        number of library kernels in each."""
        graphs, launches = [], []
        for d in range(self.draws):
            graph = torch.cuda.CUDAGraph()
            n0 = spl.spl_launch_count()
            with torch.cuda.graph(graph):
                if before:
                    before(d)
                if d == 0:
                    self.refill(eps, mech, seed, 0, path=path, timer=timer, device_base=True, parallel=timer is None)
                inp = inputs[d % len(inputs)] if isinstance(inputs, (list, tuple)) else inputs
                self.online(inp, eps, mech, seed, 0, d, path=path, timer=timer, device_base=True,
                            group_hooks=group_hooks)
                if after:
                    after(d)
                if d == self.draws - 1:
                    for gi, g in enumerate(self.groups):
                        spl.spl_rng_advance(self.rng_base[gi:gi + 1], self.draws * (self.M * g.K // 4))
            graphs.append(graph)
            launches.append(spl.spl_launch_count() - n0)
        return graphs, launches

    def capture_overlapped(self, inputs, eps, mech, seed, path="auto", before=None, after=None, group_hooks=None):
        """Two CUDA graphs, each a whole bank cycle: graph p runs the ``draws`` online steps on
        correction buffer p while, on streams of lower priority, the next cycle's corrections are
        computed into buffer 1 - p, filling the SMs and the bandwidth the online products leave
        idle; the graph ends when both are done and moves the Philox bases on by one cycle.  Replay
        graphs[c % 2] for cycle c after set_cycle(c) and a refill of buffer c % 2 for cycle c.
        ``before(d)`` / ``after(d)`` / ``group_hooks`` as in capture; ``inputs`` may be a list
        (step d reads inputs[d % len(inputs)]).  Returns the graphs and their kernel counts."""
        # the two sides must not share the workspace: the corrections take a workspace of their own
        if not all(self._fused_split(g, path, self.M) for g in self.groups):
            raise ValueError("capture_overlapped needs every group on FP16X3 with the fused split")
        self.enable_overlap()
        if not hasattr(self, "_bank_ws"):
            self._bank_ws = spl.workspace(self.workspace_bytes(self.M, self.draws), self.groups[0].W.device)
        lo, hi = torch.cuda.Stream.priority_range()
        if not hasattr(self, "_bank_stream"):
            self._bank_stream = torch.cuda.Stream(priority=lo)
            self._online_stream = torch.cuda.Stream(priority=hi)
        graphs, launches = [], []
        for parity in range(2):
            graph = torch.cuda.CUDAGraph()
            n0 = spl.spl_launch_count()
            with torch.cuda.graph(graph, stream=self._online_stream):
                main = torch.cuda.current_stream()
                self._bank_stream.wait_stream(main)
                with torch.cuda.stream(self._bank_stream):
                    self.refill(eps, mech, seed, 0, path=path, device_base=True, parallel=True, parity=1 - parity,
                                ahead=1, workspace=self._bank_ws)
                for d in range(self.draws):
                    if before:
                        before(d)
                    inp = inputs[d % len(inputs)] if isinstance(inputs, (list, tuple)) else inputs
                    self.online(inp, eps, mech, seed, 0, d, path=path, device_base=True, group_hooks=group_hooks,
                                parity=parity)
                    if after:
                        after(d)
                main.wait_stream(self._bank_stream)
                for gi, g in enumerate(self.groups):
                    spl.spl_rng_advance(self.rng_base[gi:gi + 1], self.draws * (self.M * g.K // 4))
            graphs.append(graph)
            launches.append(spl.spl_launch_count() - n0)
        return graphs, launches

    def bound_check(self, inputs, outs, eps, mech, seed, cycle, d):
        """The paper's bound on the GPU over every output of an online step (per group).  For a
        binary64 group the errors are measured the same way against the binary32 bound (its mask
        is passed rounded to fp32, which moves S_xt by at most 2^-24 relative)."""
        res = {}
        for gi, g in enumerate(self.groups):
            eta = torch.empty((self.M, g.K), device=g.W.device)
            off = self.block_offset(g, cycle, d)
            spl.spl_noise(eta, self.deltas[g.name], eps, mech, seed, stream_id=gi, offset=off)
            if g.name in self.fp64:
                xt = self.bank[g.name]["xt"].float().contiguous()
            else:  # the step's X~, drawn again (online steps that feed the split do not keep it)
                xt = torch.empty_like(eta)
                spl.spl_noise_mask(xt, None, inputs[g.name], self.deltas[g.name], eps, mech, seed, stream_id=gi,
                                   offset=off)
            res[g.name] = spl.spl_bound_check(outs[g.name], inputs[g.name], xt, eta, g.W)
        return res

    def flops_per_step(self):
        """Algorithmic flops per online step: the masked product plus its share of the batched correction."""
        return sum(2 * 2 * self.M * g.K * g.N for g in self.groups)


class MaskedStack:
    """The linear layers of a decoder stack, each a MaskedLayer with its own weights, noise scales,
    Philox seed and correction bank, run in order on one stream with one shared workspace."""

    def __init__(self, layers, seeds):
        self.layers, self.seeds = layers, seeds
        self.out_pool = None  # stacked schedule built by build(): {group: [2, draws, layers, 2M, N]}

    @classmethod
    def build(cls, model, n_layers, M, draws, base_seed, device="cuda", split=True, power_iters=1000, path="auto",
              stacked=False):
        """Seeded synthetic weights per layer (workloads.layer_seed), Delta per layer (Thms. 1-3).
        stacked: buffers of the stacked schedule (MaskedLayer.allocate_stacked) instead of a bank."""
        from . import workloads as wl
        layers = []
        for li in range(n_layers):
            weights = {name: wl.weight(N, K, seed=wl.layer_seed(base_seed, li, pi), device=device)
                       for pi, (name, K, N, _g) in enumerate(model.projections())}
            layer = MaskedLayer.from_weights(model, weights, split=split, device=device)
            del weights
            layer.sensitivities(power_iters=power_iters)
            layers.append(layer)
        pool = None
        if stacked:
            need = max(spl.spl_linear_workspace_bytes(2 * M, g.K, g.N, path) for l in layers for g in l.groups)
            ws = spl.workspace(need, device)
            # each group's outputs pooled over the layers, [parity, draw, layer, 2M, N]: the Y rows of one
            # step of every layer then sit at one pitch (StackIO moves them with one copy per group)
            pool = {g.name: torch.zeros((2, draws, n_layers, 2 * M, g.N), device=device) for g in layers[0].groups}
            for li, layer in enumerate(layers):
                layer.allocate_stacked(M, draws, path, workspace=ws,
                                       out=lambda name, li=li: [[pool[name][p, d, li] for d in range(draws)]
                                                                for p in range(2)])
        else:
            need = max(l.workspace_bytes(M, draws, path) for l in layers)
            ws = spl.workspace(need, device)
            for layer in layers:
                layer.allocate(M, draws, path, workspace=ws)
        stack = cls(layers, [wl.layer_seed(base_seed, li, 99) for li in range(n_layers)])
        stack.out_pool = pool
        return stack

    @property
    def draws(self):
        return self.layers[0].draws

    def inputs(self, base_seed, device="cuda"):
        """Seeded synthetic activations per layer and group (the enclave-side ops between the
        linears -- attention, norms, activation -- are not part of this path)."""
        from . import workloads as wl
        return [{g: wl.activations(layer.M, K, seed=wl.layer_seed(base_seed, li, 50 + gi), device=device)
                 for gi, (g, K, _n) in enumerate(layer.model.input_groups())} for li, layer in enumerate(self.layers)]

    def step(self, inputs, eps, mech, s, path="auto", refill=True):
        """Eager step s (draw s % draws of bank cycle s // draws) through every layer."""
        cycle, d = divmod(s, self.draws)
        for layer, x, seed in zip(self.layers, inputs, self.seeds):
            if d == 0 and refill:
                layer.refill(eps, mech, seed, cycle, path=path)
            layer.online(x, eps, mech, seed, cycle, d, path=path)

    def set_cycle(self, cycle):
        for layer in self.layers:
            layer.set_cycle(cycle)

    def capture(self, inputs, eps, mech, path="auto", refill=True, timer=None):
        """CUDA graphs of one bank cycle for the whole stack (see MaskedLayer.capture); graph 0
        refills every layer's bank first unless ``refill`` is False.  ``timer(d, li, phase, kind,
        group)``, when given, is called around every library call of the online steps (e.g. to put
        CUDA events into the graphs)."""
        graphs, launches = [], []
        D = self.draws
        for d in range(D):
            graph = torch.cuda.CUDAGraph()
            n0 = spl.spl_launch_count()
            with torch.cuda.graph(graph):
                for li, (layer, x, seed) in enumerate(zip(self.layers, inputs, self.seeds)):
                    if d == 0 and refill:
                        layer.refill(eps, mech, seed, 0, path=path, device_base=True, parallel=True)
                    t = (lambda phase, kind, group, _d=d, _li=li: timer(_d, _li, phase, kind, group)) if timer else None
                    layer.online(x, eps, mech, seed, 0, d, path=path, device_base=True, timer=t)
                if d == D - 1:
                    for layer in self.layers:
                        for gi, g in enumerate(layer.groups):
                            spl.spl_rng_advance(layer.rng_base[gi:gi + 1], D * (layer.M * g.K // 4))
            graphs.append(graph)
            launches.append(spl.spl_launch_count() - n0)
        return graphs, launches

    def capture_overlapped(self, inputs, eps, mech, bank_workspace, path="auto", after=None):
        """Two CUDA graphs, each a whole bank cycle of the stack: graph p runs the ``draws`` steps
        through every layer on correction buffers p while, on a stream of lower priority, the next
        cycle's corrections of every layer are computed into buffers 1 - p, with a workspace of their
        own (``bank_workspace``, at least max(layer.workspace_bytes(M, draws))).  The graph ends when
        both are done and moves every Philox base on by one cycle.  Replay graphs[c % 2] for cycle
        c after set_cycle(c) and a refill of buffers c % 2 for cycle c (start_overlapped).
        ``after(d)`` is called after step d's launches (e.g. to copy its results inside the graph).
        Returns the graphs and their kernel counts."""
        lo, hi = torch.cuda.Stream.priority_range()
        if not hasattr(self, "_bank_stream"):
            self._bank_stream = torch.cuda.Stream(priority=lo)
            self._online_stream = torch.cuda.Stream(priority=hi)
        for layer in self.layers:
            layer.enable_overlap()
        D = self.draws
        graphs, launches = [], []
        for parity in range(2):
            graph = torch.cuda.CUDAGraph()
            n0 = spl.spl_launch_count()
            with torch.cuda.graph(graph, stream=self._online_stream):
                main = torch.cuda.current_stream()
                self._bank_stream.wait_stream(main)
                with torch.cuda.stream(self._bank_stream):
                    for layer, seed in zip(self.layers, self.seeds):
                        layer.refill(eps, mech, seed, 0, path=path, device_base=True, parity=1 - parity, ahead=1,
                                     workspace=bank_workspace)
                for d in range(D):
                    for layer, x, seed in zip(self.layers, inputs, self.seeds):
                        layer.online(x, eps, mech, seed, 0, d, path=path, device_base=True, parity=parity)
                    if after:
                        after(d)
                main.wait_stream(self._bank_stream)
                for layer in self.layers:
                    for gi, g in enumerate(layer.groups):
                        spl.spl_rng_advance(layer.rng_base[gi:gi + 1], D * (layer.M * g.K // 4))
            graphs.append(graph)
            launches.append(spl.spl_launch_count() - n0)
        return graphs, launches

    def bank_slice(self, d):
        """Layers whose next-cycle corrections step d of a cycle computes (capture_steps): the
        layers split as evenly as whole layers allow over the ``draws`` steps."""
        L, D = len(self.layers), self.draws
        return range(d * L // D, (d + 1) * L // D)

    def capture_steps(self, inputs, eps, mech, bank_workspace, path="auto", timer=None):
        """CUDA graphs of single steps, each carrying its share of the next bank cycle: graphs[p][d]
        runs step d of a cycle through every layer on correction buffers p while, on a stream of
        lower priority, the layers of bank_slice(d) compute their next-cycle corrections into buffers
        1 - p (with ``bank_workspace``, at least max(layer.workspace_bytes(M, draws))); the graph ends
        when both are done, and graph d = draws - 1 moves every Philox base on by one cycle.  After
        start_overlapped(c), replay graphs[(s // draws) % 2][s % draws] for steps s = c draws, c
        draws + 1, ... -- any number of them: every step holds its online pass and an equal share of
        the refill, so a run of any length times the whole method.  ``timer(d, li, phase, kind,
        group)`` as in capture.  Returns the graphs and their kernel counts."""
        lo, hi = torch.cuda.Stream.priority_range()
        if not hasattr(self, "_bank_stream"):
            self._bank_stream = torch.cuda.Stream(priority=lo)
            self._online_stream = torch.cuda.Stream(priority=hi)
        for layer in self.layers:
            layer.enable_overlap()
        D = self.draws
        graphs, launches = [[], []], [[], []]
        for parity in range(2):
            for d in range(D):
                graph = torch.cuda.CUDAGraph()
                n0 = spl.spl_launch_count()
                with torch.cuda.graph(graph, stream=self._online_stream):
                    main = torch.cuda.current_stream()
                    self._bank_stream.wait_stream(main)
                    with torch.cuda.stream(self._bank_stream):
                        for li in self.bank_slice(d):
                            self.layers[li].refill(eps, mech, self.seeds[li], 0, path=path, device_base=True,
                                                   parity=1 - parity, ahead=1, workspace=bank_workspace)
                    for li, (layer, x, seed) in enumerate(zip(self.layers, inputs, self.seeds)):
                        t = (lambda phase, kind, group, _d=d, _li=li: timer(_d, _li, phase, kind, group)) \
                            if timer else None
                        layer.online(x, eps, mech, seed, 0, d, path=path, device_base=True, parity=parity, timer=t)
                    main.wait_stream(self._bank_stream)
                    if d == D - 1:
                        for layer in self.layers:
                            for gi, g in enumerate(layer.groups):
                                spl.spl_rng_advance(layer.rng_base[gi:gi + 1], D * (layer.M * g.K // 4))
                graphs[parity].append(graph)
                launches[parity].append(spl.spl_launch_count() - n0)
        return graphs, launches

    def capture_stacked(self, inputs, eps, mech, path="auto", timer=None):
        """CUDA graphs of the stacked schedule (MaskedLayer.allocate_stacked): graphs[p][d] runs step d of
        a cycle of parity p through every layer -- each product also computing the next cycle's
        correction of draw d -- and graph d = draws - 1 moves every Philox base on by one cycle.  After
        start_stacked(c), replay graphs[(s // draws) % 2][s % draws] for steps s = c draws, ...: any
        number of them, each one step of the method with its share of the bank.  ``timer(d, li, phase,
        kind, group)`` as in capture.  ``inputs``: the per-layer input dicts, or n sets of them with n
        dividing draws (step d then reads inputs[d % n], so step s reads set s % n).  Host transfers go
        beside the replays (StackIO).  Returns the graphs and their kernel counts."""
        sets = isinstance(inputs, (list, tuple)) and len(inputs) > 0 and isinstance(inputs[0], (list, tuple))
        D = self.draws
        if sets and D % len(inputs):
            raise ValueError("capture_stacked: the number of input sets must divide draws")
        graphs, launches = [[], []], [[], []]
        for parity in range(2):
            for d in range(D):
                graph = torch.cuda.CUDAGraph()
                n0 = spl.spl_launch_count()
                step_inputs = inputs[d % len(inputs)] if sets else inputs
                with torch.cuda.graph(graph):
                    for li, (layer, x, seed) in enumerate(zip(self.layers, step_inputs, self.seeds)):
                        t = (lambda phase, kind, group, _d=d, _li=li: timer(_d, _li, phase, kind, group)) \
                            if timer else None
                        layer.stacked_step(x, eps, mech, seed, d, parity, timer=t, device_base=True)
                    if d == D - 1:
                        for layer in self.layers:
                            for gi, g in enumerate(layer.groups):
                                spl.spl_rng_advance(layer.rng_base[gi:gi + 1], D * (layer.M * g.K // 4))
                graphs[parity].append(graph)
                launches[parity].append(spl.spl_launch_count() - n0)
        return graphs, launches

    def step_outputs(self, parity, d):
        """The outputs of step d of a cycle of parity ``parity`` (stacked schedule): per layer {group: Y}."""
        return [{g.name: layer.stacked[g.name]["out"][1 - parity][d][:layer.M] for g in layer.groups}
                for layer in self.layers]

    def previous_step(self, parity, d):
        """(parity, draw) of the step before step d of a cycle of parity ``parity``."""
        return (parity, d - 1) if d > 0 else (1 - parity, self.draws - 1)

    def replay_stacked(self, graphs, s):
        """Step s of the stacked schedule: replays graphs[(s // draws) % 2][s % draws] (capture_stacked).
        Host transfers beside the replays: StackIO."""
        D = self.draws
        graphs[(s // D) % 2][s % D].replay()

    def start_stacked(self, cycle, graphs):
        """Before replaying the stacked graphs from cycle ``cycle``: run cycle ``cycle - 1``'s graphs once
        (their outputs are discarded; their corrections, for cycle ``cycle``, are kept), leaving the
        device-side Philox bases at ``cycle``."""
        if cycle < 1:
            raise ValueError("start_stacked: the cycle before must exist")
        self.set_cycle(cycle - 1)
        for g in graphs[(cycle - 1) % 2]:
            g.replay()

    def refill_all(self, eps, mech, path="auto", parity=0, ahead=0, workspace=None):
        """Every layer's bank for the cycle at the device-side bases (+ ``ahead`` cycles), into
        correction buffers ``parity``, on the current stream."""
        for layer, seed in zip(self.layers, self.seeds):
            layer.refill(eps, mech, seed, 0, path=path, device_base=True, parity=parity, ahead=ahead,
                         workspace=workspace)

    def start_overlapped(self, cycle, eps, mech, path="auto"):
        """Before replaying the overlapped graphs from bank cycle ``cycle``: the device-side Philox
        bases at ``cycle`` and that cycle's corrections in buffers cycle % 2."""
        self.set_cycle(cycle)
        for layer, seed in zip(self.layers, self.seeds):
            layer.refill(eps, mech, seed, 0, path=path, device_base=True, parity=cycle % 2)

    def flops_per_step(self):
        return sum(l.flops_per_step() for l in self.layers)


def split_outputs(layer, outs):
    """{projection: [M, N_p] view} from the per-group outputs."""
    res = {}
    for g in layer.groups:
        for p in g.names:
            a, b = g.columns(p)
            res[p] = outs[g.name][:, a:b]
    return res


class StackIO:
    """Host transfers of the stacked schedule beside its graph replays, few and large.

    Each input group of every layer sits in one page-locked host buffer ``host_in[group]`` and in
    ``sets`` device sets ([layers, M, K]; step s reads set s % sets, as capture_stacked does with the
    sets from ``layer_inputs()``), and the Y rows of one step of every layer lie at one pitch in the
    stack's pooled output buffer (MaskedStack.build), so a step moves each group in with one copy
    and out with one strided copy (spl_copy_2d): a handful of host calls per step, which lets the
    host run far ahead of the device.  Inputs go in on one stream and outputs out on another, the
    two directions of the host link at once.  Inputs go in up to sets - 1 steps ahead (never past
    ``stop``) and step s waits only for its own; its outputs go to host slot s % ring once it is
    done, and only have to be out before step s + 2 draws rewrites the same device buffer, so a copy
    that stalls holds the steps up only once it has fallen that far behind.

    Measured on GB300 (28-layer Llama stack, 1.0 GB in and 1.6 GB out per step): a step's inputs
    take 4.8 ms and its outputs 8.2 ms, beside the 14.5-15 ms of compute.  On some boxes the host
    side stalls now and then (one direction's copies 50-250 ms at a time, the host thread too): the
    earlier schedule -- a copy per layer and group, inputs then outputs on one stream that each step
    waited for, the host a step or two ahead -- put every stall on the step time (20.4 ms per step
    on average); here the host is hundreds of steps ahead and a stall holds the steps up only once
    the copies have fallen sets - 1 steps (inputs) or 2 draws steps (outputs) behind, but a timed
    run still ends only when its last outputs are on the host.  ``streams=1`` puts both directions
    on one copy stream."""

    def __init__(self, stack, host_in, ring=2, sets=None, streams=2):
        if stack.out_pool is None:
            raise ValueError("StackIO: a stack built with stacked=True (pooled outputs)")
        if streams not in (1, 2):
            raise ValueError("StackIO: one copy stream or one per direction")
        D = stack.draws
        if sets is None:  # the most sets up to 8 that divide the draws
            sets = max([n for n in range(2, min(D, 8) + 1) if D % n == 0], default=0)
        if sets < 2 or D % sets:
            raise ValueError("StackIO: at least two input sets, a divisor of draws")
        self.stack, self.sets = stack, sets
        L, M = len(stack.layers), stack.layers[0].M
        dev = stack.layers[0].groups[0].W.device
        self.host_in = host_in
        for g, x in host_in.items():
            if not x.is_pinned() or x.shape[:2] != (L, M):
                raise ValueError("StackIO: host_in[group] is page-locked [layers, M, K]")
        self.dev_in = [{g: torch.zeros(x.shape, device=dev) for g, x in host_in.items()} for _ in range(sets)]
        self.host_out = [{g: torch.empty((L, M, p.shape[-1])).pin_memory() for g, p in stack.out_pool.items()}
                         for _ in range(ring)]
        self.h2d = torch.cuda.Stream()
        self.d2h = self.h2d if streams == 1 else torch.cuda.Stream()
        self._in, self._done, self._out = {}, {}, {}

    def layer_inputs(self):
        """The device sets as capture_stacked takes them: per set, per layer {group: [M, K] view}."""
        L = len(self.stack.layers)
        return [[{g: x[li] for g, x in dset.items()} for li in range(L)] for dset in self.dev_in]

    def bytes_per_step(self):
        """(bytes in, bytes out) per step."""
        return (sum(x.numel() * x.element_size() for x in self.host_in.values()),
                sum(y.numel() * y.element_size() for y in self.host_out[0].values()))

    @staticmethod
    def _event(stream):
        e = torch.cuda.Event()
        e.record(stream)
        return e

    def _prefetch(self, s):
        done = self._done.pop(s - self.sets, None)  # set s % sets was last read by step s - sets
        if done is not None:
            self.h2d.wait_event(done)
        dst = self.dev_in[s % self.sets]
        with torch.cuda.stream(self.h2d):
            for g, x in self.host_in.items():
                dst[g].copy_(x, non_blocking=True)
        self._in[s] = self._event(self.h2d)

    def step(self, graphs, s, stop=None):
        """Step s with graphs from capture_stacked(layer_inputs(), ...): the inputs of steps s to
        s + sets - 1 in (those not already there, none from step ``stop`` on), the replay, then this
        step's outputs out to host slot s % ring."""
        D, M = self.stack.draws, self.stack.layers[0].M
        if stop is not None and s >= stop:
            raise ValueError("StackIO.step: s is past stop")
        main = torch.cuda.current_stream()
        if not self._in and not self._done:  # first step: the sets may still be read by earlier work
            self.h2d.wait_stream(main)
        hi = s + self.sets if stop is None else min(s + self.sets, stop)
        for t in range(s, hi):  # set t % sets was last read by step t - sets < s
            if t not in self._in:
                self._prefetch(t)
        main.wait_event(self._in.pop(s))
        out_back = self._out.pop(s - 2 * D, None)  # the last copy out of the device buffer step s rewrites
        if out_back is not None:
            main.wait_event(out_back)
        p, d = (s // D) % 2, s % D
        graphs[p][d].replay()
        done = self._event(main)
        self._done[s] = done
        self.d2h.wait_event(done)
        dst = self.host_out[s % len(self.host_out)]
        with torch.cuda.stream(self.d2h):
            for g, y in dst.items():
                src = self.stack.out_pool[g][1 - p, d]  # [layers, 2M, N]: rows [0, M) of each layer are Y
                row = M * src.shape[-1] * src.element_size()
                spl.spl_copy_2d(y, src, src.shape[0], row, row, 2 * row, stream=self.d2h)
        self._out[s] = self._event(self.d2h)

    def outputs(self, s):
        """Host slot of step s ({group: [layers, M, N]}) and the event after which it holds step s's
        outputs (until step s + ring is copied out into the same slot)."""
        return self.host_out[s % len(self.host_out)], self._out.get(s)

    def finish(self):
        """The current stream waits until every output issued so far is on the host."""
        torch.cuda.current_stream().wait_stream(self.d2h)
