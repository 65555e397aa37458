"""Seeded synthetic inputs for the sparse dReLU FFN: weights, tokens, routers, predictor lists.

This module draws inputs only; it holds none of the method's arithmetic. The
CUDA path and the CPU oracle both consume what it returns.

Recipe (shapes and activation rates of the paper's Mistral / Mixtral FFNs,
Sec. 5 and Sec. 6.2; the real checkpoints and activations are not available):

* Every matrix is neuron-major ``[m][d]``.
* ``W_gate``, ``W_up`` entries ~ N(0, 1/d); the last input column (index d-1) of
  both holds one shared per-neuron offset ``b_j ~ N(mu, sigma_b^2)``.
* ``W_down`` entries ~ N(0, 1/m).
* Token activations have the bias channel ``x[d-1] = 1`` and unit-variance
  entries elsewhere, so the pre-activations of neuron j are
  ``g_j = z_g + b_j``, ``u_j = z_u + b_j`` with ``z ~ N(0, ~1)``. The fraction of
  gate-active neurons is ``Phi(mu / sqrt(1 + sigma_b^2))`` and of both-active
  neurons ``E_b[Phi(b)^2]``; ``MU_FOR_ACTIVATION`` solves the latter for mu.
  The spread of ``b_j`` makes some neurons hot and others cold.
* bf16 tensors are rounded to nearest-even from the fp32 draw.
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import torch

# offset mean mu for a target both-active fraction at sigma_b = 0.5
MU_FOR_ACTIVATION = {0.05: -0.999, 0.10: -0.662, 0.20: -0.250, 0.25: -0.092, 0.50: 0.550}
# offset for the "every neuron active" case: g, u = N(0,1) + 10 > 0
ALL_ACTIVE_OFFSET = 10.0
SIGMA_B = 0.5


@dataclass
class FfnLayer:
    """One dReLU FFN's weights (``[m][d]`` each) and the offsets written into column d-1."""
    w_gate: torch.Tensor
    w_up: torch.Tensor
    w_down: torch.Tensor
    offsets: torch.Tensor  # fp32 [m], before rounding to the weight dtype

    @property
    def d(self) -> int:
        return int(self.w_gate.shape[1])

    @property
    def m(self) -> int:
        return int(self.w_gate.shape[0])


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=torch.device(device))
    g.manual_seed(int(seed))
    return g


def mu_for(activation: float) -> float | None:
    """Offset mean for a target both-active fraction; None means every neuron active."""
    if activation >= 1.0:
        return None
    return MU_FOR_ACTIVATION[round(float(activation), 2)]


def ffn_layer(d: int, m: int, *, activation: float = 0.10, mu: float | None = None,
              sigma_b: float = SIGMA_B, dtype=torch.bfloat16, seed: int = 0,
              device="cpu") -> FfnLayer:
    """Draw one FFN layer. ``mu`` overrides ``activation``; ``activation >= 1`` gives all-active."""
    g = _gen(seed, device)
    if mu is None:
        mu = mu_for(activation)
    wg = torch.randn(m, d, generator=g, device=device) / math.sqrt(d)
    wu = torch.randn(m, d, generator=g, device=device) / math.sqrt(d)
    if mu is None:
        b = torch.full((m,), ALL_ACTIVE_OFFSET, device=device)
    else:
        b = mu + sigma_b * torch.randn(m, generator=g, device=device)
    wg[:, d - 1] = b
    wu[:, d - 1] = b
    wd = torch.randn(m, d, generator=g, device=device) / math.sqrt(m)
    return FfnLayer(wg.to(dtype).contiguous(), wu.to(dtype).contiguous(),
                    wd.to(dtype).contiguous(), b.float())


# ---------------------------------------------------------------------------
# INT4 weight storage (the weight-only 4-bit rows of the paper's INT4 models,
# Tables 7-9): per neuron row of d weights, d/2 bytes of 4-bit codes followed
# by d/32 IEEE binary16 scales (little-endian), one per group of 32
# consecutive elements. A stored weight is scale * (code - 8). Within a
# group's 16 code bytes, read as four little-endian 32-bit words, element
# e = 8s + 2t + h (s, t in 0..3, h in 0..1) sits in word t at nibble s + 4h
# (bits 4(s+4h) .. 4(s+4h)+3).
# ---------------------------------------------------------------------------
INT4_GROUP = 32


def int4_row_bytes(d: int) -> int:
    return d // 2 + (d // INT4_GROUP) * 2


def quantize_int4(w: torch.Tensor) -> torch.Tensor:
    """Round ``[m][d]`` weights to INT4 rows (uint8 ``[m][d/2 + d/16]``).

    Per group of 32: scale = max|w| / 7 rounded to binary16 (1 where the group
    is all zero), code = clamp(round(w / scale), -8, 7) + 8.
    """
    m, d = w.shape
    if d % INT4_GROUP:
        raise ValueError("d must be a multiple of 32 for INT4 rows")
    wf = w.detach().float().reshape(m, d // INT4_GROUP, INT4_GROUP)
    scale = (wf.abs().amax(-1) / 7.0).to(torch.float16)
    scale = torch.where(scale == 0, torch.ones_like(scale), scale)
    q = torch.clamp(torch.round(wf / scale.float().unsqueeze(-1)), -8, 7).to(torch.int64) + 8  # [m][G][32]
    # element e = 8s + 2t + h -> word t, nibble s + 4h
    q = q.reshape(m, d // INT4_GROUP, 4, 4, 2)          # [m][G][s][t][h]
    shifts = 4 * (torch.arange(4, device=w.device).view(4, 1, 1) +
                  4 * torch.arange(2, device=w.device).view(1, 1, 2))  # [s][1][h]
    words = (q << shifts).sum(dim=(2, 4))               # [m][G][t], disjoint nibbles
    codes = torch.stack([(words >> (8 * b)) & 0xFF for b in range(4)], dim=-1).to(torch.uint8)
    codes = codes.reshape(m, d // 2)
    scales = scale.contiguous().view(torch.uint8).reshape(m, (d // INT4_GROUP) * 2)
    return torch.cat([codes, scales], dim=1).contiguous()


@dataclass
class FfnLayerInt4:
    """One dReLU FFN's INT4 rows (uint8 ``[m][d/2 + d/16]`` each) and the offsets they were drawn with."""
    w_gate: torch.Tensor
    w_up: torch.Tensor
    w_down: torch.Tensor
    offsets: torch.Tensor
    d: int

    @property
    def m(self) -> int:
        return int(self.w_gate.shape[0])


def ffn_layer_int4(d: int, m: int, *, activation: float = 0.10, mu: float | None = None,
                   sigma_b: float = SIGMA_B, seed: int = 0, device="cpu") -> FfnLayerInt4:
    """Draw a layer as ``ffn_layer`` does (fp32), then store it as INT4 rows."""
    L = ffn_layer(d, m, activation=activation, mu=mu, sigma_b=sigma_b, dtype=torch.float32, seed=seed,
                  device=device)
    return FfnLayerInt4(quantize_int4(L.w_gate), quantize_int4(L.w_up), quantize_int4(L.w_down),
                        L.offsets, d)


@dataclass
class Predictor:
    w1: torch.Tensor  # [r][d]
    w2: torch.Tensor  # [m][r]


def predictor_weights(d: int, r: int, m: int, offsets: torch.Tensor, *, dtype=torch.bfloat16, seed: int = 0,
                      device="cpu") -> Predictor:
    """Synthetic weights of the rank-r activation predictor (a two-layer ReLU
    MLP): W1 ~ N(0, 1/d) with its last row picking the bias channel x[d-1] = 1
    (so that hidden unit is constantly 1), W2 ~ N(0, 1/r) with its last column
    holding the layer's per-neuron offsets b_j, which favours the layer's hot
    neurons. Trained weights do not exist here; these only have the shapes."""
    g = _gen(seed, device)
    w1 = torch.randn(r, d, generator=g, device=device) / math.sqrt(d)
    w1[r - 1] = 0.0
    w1[r - 1, d - 1] = 1.0
    w2 = torch.randn(m, r, generator=g, device=device) / math.sqrt(r)
    w2[:, r - 1] = offsets.to(device=device, dtype=torch.float32)
    return Predictor(w1.to(dtype).contiguous(), w2.to(dtype).contiguous())


def tokens(B: int, d: int, *, dtype=torch.bfloat16, seed: int = 0, device="cpu") -> torch.Tensor:
    """Token activations ``[B][d]``: N(0,1) entries with the bias channel ``x[:, d-1] = 1``."""
    x = torch.randn(B, d, generator=_gen(seed, device), device=device)
    x[:, d - 1] = 1.0
    return x.to(dtype).contiguous()


def residual(B: int, d: int, *, seed: int = 0, device="cpu") -> torch.Tensor:
    """Initial residual stream ``h_0 [B][d]`` (fp32, N(0,1)) of the synthetic layer stack."""
    return torch.randn(B, d, generator=_gen(seed, device), device=device).contiguous()


def router(E: int, d: int, *, dtype=torch.bfloat16, seed: int = 0, device="cpu") -> torch.Tensor:
    """Router matrix ``W_r [E][d]`` with N(0, 1/d) entries."""
    w = torch.randn(E, d, generator=_gen(seed, device), device=device) / math.sqrt(d)
    return w.to(dtype).contiguous()


def predictor_list(offsets: torch.Tensor, k: int, *, zipf_s: float = 1.1, seed: int = 0) -> torch.Tensor:
    """A predictor's neuron list: k distinct neurons, sorted ascending, int32.

    Neurons are ranked by offset, hottest (largest ``b_j``) first; k ranks are
    drawn without replacement with Zipf weights ``(r+1)^-s``, so the list
    favours hot neurons the way a trained predictor would.
    """
    b = offsets.detach().float().cpu()
    m = b.numel()
    k = max(0, min(int(k), m))
    if k == 0:
        return torch.zeros(0, dtype=torch.int32)
    order = torch.argsort(b, descending=True, stable=True)
    weights = (torch.arange(m, dtype=torch.float64) + 1.0).pow(-zipf_s)
    ranks = torch.multinomial(weights, k, replacement=False, generator=_gen(seed, "cpu"))
    rows = order[ranks]
    return torch.sort(rows).values.to(torch.int32).contiguous()


# ---------------------------------------------------------------------------
# The five workloads (shapes of the paper's Mistral-7B / Mixtral-47B FFNs)
# ---------------------------------------------------------------------------
MISTRAL_D, MISTRAL_M = 4096, 14336
N_LAYERS = 32

WORKLOADS = {
    "drelu-ffn-fp32-d512-m1408": dict(
        d=512, m=1408, dtype="f32", batch=1, n_tokens=16, layers=1, mu=-0.7, seed=0,
        desc="single dReLU FFN, fp32, 16 decode tokens one at a time"),
    "mistral7b-ffn-stack-bf16-b1-act10": dict(
        d=MISTRAL_D, m=MISTRAL_M, dtype="bf16", batch=1, layers=N_LAYERS, activation=0.10, seed=1000,
        desc="32-layer Mistral-shaped FFN stack, ~10% combined activation, batch 1"),
    "mistral7b-ffn-stack-bf16-sweep": dict(
        d=MISTRAL_D, m=MISTRAL_M, dtype="bf16", batches=(1, 4, 16, 64),
        activations=(0.05, 0.10, 0.25, 0.50, 1.0), layers=N_LAYERS, seed=2000,
        desc="batch x activation sweep on the Mistral-shaped stack, next to dense cuBLAS"),
    "mixtral47b-moe-stack-bf16-top2": dict(
        d=MISTRAL_D, m=MISTRAL_M, dtype="bf16", experts=8, top_k=2, batches=(1, 8), layers=N_LAYERS,
        activation=0.20, seed=3000,
        desc="32-layer Mixtral-shaped MoE, 8 experts, top-2, ~20% combined activation per expert"),
    "mistral7b-ffn-stack-int4-b1-act10": dict(
        d=MISTRAL_D, m=MISTRAL_M, dtype="int4", batch=1, layers=N_LAYERS, activation=0.10, seed=1000,
        desc="the batch-1 Mistral-shaped stack with INT4 rows (4-bit codes, binary16 scale per 32)"),
    "mixtral47b-moe-stack-int4-top2": dict(
        d=MISTRAL_D, m=MISTRAL_M, dtype="int4", experts=8, top_k=2, batches=(1,), layers=N_LAYERS,
        activation=0.20, seed=3000,
        desc="the Mixtral-shaped MoE stack with INT4 experts (the paper's Mixtral-47B-INT4 setting)"),
    "mistral7b-ffn-topk5-b1": dict(
        d=MISTRAL_D, m=MISTRAL_M, dtype="bf16", batch=1, layers=N_LAYERS, activation=0.10, keep=717,
        seed=1000,
        desc="top-k magnitude mask (Eq. 3-4) keeping 717 of 14336 neurons (5%) per token, 32 layers at ~10% dReLU activity"),
    "mistral7b-ffn-stack-bf16-predictor": dict(
        d=MISTRAL_D, m=MISTRAL_M, dtype="bf16", batch=1, layers=N_LAYERS, activation=0.10,
        list_len=1434, zipf_s=1.1, seed=1000,
        desc="predictor-driven mode: per-layer sorted lists of 1434 neurons (Zipf 1.1 over hotness)"),
    "mistral7b-ffn-stack-bf16-b1-prednet": dict(
        d=MISTRAL_D, m=MISTRAL_M, dtype="bf16", batch=1, layers=N_LAYERS, activation=0.10, rank=512, k=1434,
        seed=1000,
        desc="per-layer predictor network (two-layer ReLU MLP, rank 512) choosing 1434 neurons (10%) "
             "for the FFN's predictor mode, 32 layers, batch 1"),
}


def torch_dtype(name: str):
    return {"bf16": torch.bfloat16, "f32": torch.float32}[name]


def layer_seed(base: int, layer: int, expert: int = 0) -> int:
    """Seed of layer ``layer`` (and expert ``expert``) of a workload with base seed ``base``."""
    return int(base) + 1009 * int(layer) + 17 * int(expert)
