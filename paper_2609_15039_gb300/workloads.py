"""Seeded synthetic inputs and the model shapes of the paper's workloads.

This module holds no arithmetic of the masked-linear method.  It only
draws the inputs that both the CUDA path and the CPU oracle consume:

* activations: rows ~ N(0, 1), then either RMS-normalised (the input of a
  projection follows RMSNorm, Sec. 2.2.2; ||x||_2 = sqrt(K)) or clipped to
  unit l2 norm (x * min(1, 1/||x||), which makes max ||x - y|| = 2);
* weights: i.i.d. N(0, 0.02^2), stored [N_out, K_in] like nn.Linear.

Trained Llama/Qwen weights and the Dolly/Pile prompts are not available;
these stand in for them with the shapes of Sec. 5.4 ("Inference Models").
"""

from dataclasses import dataclass

import torch

WEIGHT_STD = 0.02


@dataclass(frozen=True)
class ModelShape:
    """Linear-layer dimensions of a decoder-only model (Sec. 5.4)."""

    name: str
    layers: int
    d_model: int
    d_ff: int
    q_out: int
    kv_out: int
    vocab: int

    def projections(self):
        """(name, K_in, N_out, input group) for the seven linears of one layer.

        Q/K/V share one masked input and Gate/Up share another (Sec. 5.2).
        """
        d = self.d_model
        return [
            ("q", d, self.q_out, "qkv"),
            ("k", d, self.kv_out, "qkv"),
            ("v", d, self.kv_out, "qkv"),
            ("o", self.q_out, d, "o"),
            ("gate", d, self.d_ff, "gateup"),
            ("up", d, self.d_ff, "gateup"),
            ("down", self.d_ff, d, "down"),
        ]

    def input_groups(self):
        """(group, K_in, [projection names]) in the order a layer consumes them."""
        groups = {}
        for name, k, _n, g in self.projections():
            groups.setdefault(g, (k, []))[1].append(name)
        return [(g, k, names) for g, (k, names) in groups.items()]

    def weights_per_layer(self):
        return sum(k * n for _name, k, n, _g in self.projections())

    def flops_per_token_layer(self):
        return 2 * self.weights_per_layer()


# Llama-3.2-3B: 28 layers, hidden 3072, MLP 8192, 24 Q heads / 8 KV heads
# (Q and O over 3072, K and V to 1024), vocabulary 128256 (Sec. 5.4).
LLAMA_3_2_3B = ModelShape("llama-3.2-3b", 28, 3072, 8192, 3072, 1024, 128256)
# Qwen3-4B: 36 layers, hidden 2560, MLP 9728, Q to 4096, K/V to 1024,
# O 4096 -> 2560, vocabulary 151936 (Sec. 5.4).
QWEN3_4B = ModelShape("qwen3-4b", 36, 2560, 9728, 4096, 1024, 151936)


def _generator(seed, device):
    g = torch.Generator(device=device)
    g.manual_seed(int(seed) % (2 ** 63))
    return g


def activations(M, K, seed, norm="rms", device="cpu"):
    """[M, K] fp32 activations: N(0,1) rows, RMS-normalised ("rms") or unit-clipped ("unit")."""
    g = _generator(seed, device)
    x = torch.randn((M, K), generator=g, device=device, dtype=torch.float32)
    if M == 0 or K == 0:
        return x
    if norm == "rms":
        x = x * torch.rsqrt(torch.mean(x.double() * x.double(), dim=1, keepdim=True)).float()
    elif norm == "unit":
        nrm = torch.linalg.vector_norm(x.double(), dim=1, keepdim=True)
        x = (x.double() * torch.clamp(1.0 / nrm, max=1.0)).float()
    elif norm != "none":
        raise ValueError(norm)
    return x.contiguous()


def weight(N, K, seed, std=WEIGHT_STD, device="cpu"):
    """[N, K] fp32 weight with i.i.d. N(0, std^2) entries."""
    g = _generator(seed, device)
    w = torch.randn((N, K), generator=g, device=device, dtype=torch.float32)
    return (w * std).contiguous()


def layer_seed(base, layer, proj_index):
    """Distinct seeds per (layer, projection) for the weights of a synthetic stack."""
    return int(base) * 1_000_003 + layer * 101 + proj_index


# The five workloads the build is measured on (synthetic stand-ins).
CONFIGS = {
    "single": dict(  # one masked linear: X 16x256 unit-norm rows, W 256->512, Laplace, Delta = 2
        M=16, K=256, N=512, norm="unit", mech="laplace", sensitivity=2.0, eps=(1.0, float("inf")), seed=0),
    "llama_layer": dict(  # one Llama-3.2-3B layer, 128 prompt tokens
        model=LLAMA_3_2_3B, M=128, eps=(0.5, 1.0, 4.0), mech="gaussian"),
    "llama_stack": dict(  # 28 Llama layers, prefill 512 + 256 decode steps at M = 1
        model=LLAMA_3_2_3B, M=512, decode_steps=256, eps=(1.0,), mech="laplace", draws=8),
    "qwen_stack": dict(  # 36 Qwen3-4B layers, prefill 2048
        model=QWEN3_4B, M=2048, eps=(0.1, 1.0, 10.0), mech="gaussian"),
    "qwen_sweep": dict(  # Qwen3-4B shapes, M sweep, and the mask alone at 10^9 elements
        model=QWEN3_4B, Ms=(1, 4, 16, 64, 256, 1024), eps=(1.0,), mech="gaussian", mask_elems=10 ** 9),
}
