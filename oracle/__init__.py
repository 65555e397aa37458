"""fp64 CPU oracle for the dReLU activation-sparse FFN (Turbo Sparse, arXiv 2406.05955).

TEST INFRASTRUCTURE ONLY: only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package. It shares no code with
the CUDA library and never imports it.

The arithmetic lives in ``ts_oracle.c`` (plain C, double precision, fixed
ascending summation order, built with ``-ffp-contract=off``). This module builds
it, marshals numpy arrays into it, and composes the two multi-call forms the
paper describes in prose:

* MoE (Sec. 4, Sec. 6.2): ``y_t = sum_k w_{t,k} * FFN_{e_{t,k}}(x_t)`` over the
  top-k experts the router picks for token t.
* The synthetic layer stack: ``x_l = rmsnorm(h_l)``, ``h_{l+1} = h_l + FFN_l(x_l)``
  (glue with no counterpart in the paper; see ``ts_oracle_rmsnorm``).

Array conventions: weights and activations are numpy ``float32`` (fp32 data) or
``uint16`` (bf16 bit patterns); every matrix is neuron-major ``[m][d]``.
Results are float64 numpy arrays.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "ts_oracle.c")
_LIB = os.path.join(_HERE, "_build", "libtsoracle.so")
_lock = threading.Lock()
_lib = None

F32, BF16, INT4 = 0, 1, 2
INT4_GROUP = 32  # weights per binary16 scale in an INT4 row
RMS_EPS = 1e-5


def build(force: bool = False) -> str:
    """Compile ts_oracle.c into oracle/_build/libtsoracle.so (gcc, OpenMP)."""
    if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC):
        return _LIB
    os.makedirs(os.path.dirname(_LIB), exist_ok=True)
    tmp = _LIB + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fopenmp",
           "-fPIC", "-shared", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P = ctypes.c_void_p
            I = ctypes.c_int
            lib.ts_oracle_ffn.argtypes = [I, I, I, I, P, P, P, P, P, I, P, P, P, P, P, I]
            lib.ts_oracle_ffn.restype = I
            lib.ts_oracle_ffn_w.argtypes = [I, I, I, I, P, I, P, P, P, P, I, P, P, P, P, P, I]
            lib.ts_oracle_ffn_w.restype = I
            lib.ts_oracle_ffn_topk.argtypes = [I, I, I, I, P, I, P, P, P, I, P, P, P, P, I]
            lib.ts_oracle_ffn_topk.restype = I
            lib.ts_oracle_predict.argtypes = [I, I, I, I, I, P, P, P, I, P, P]
            lib.ts_oracle_predict.restype = I
            lib.ts_oracle_router.argtypes = [I, I, I, I, P, P, I, P, P, P]
            lib.ts_oracle_router.restype = I
            lib.ts_oracle_rmsnorm.argtypes = [I, I, P, ctypes.c_double, I, P]
            lib.ts_oracle_rmsnorm.restype = I
            lib.ts_oracle_max_threads.argtypes = []
            lib.ts_oracle_max_threads.restype = I
            _lib = lib
    return _lib


def max_threads() -> int:
    """Threads an oracle call uses when ``threads`` is not given."""
    return int(_load().ts_oracle_max_threads())


def as_array(t) -> np.ndarray:
    """A torch tensor or numpy array as the oracle's storage: float32, bf16 bits
    (uint16), or INT4 rows (uint8, ``[m][d/2 + d/16]``)."""
    if isinstance(t, np.ndarray):
        if t.dtype not in (np.float32, np.uint16, np.uint8):
            raise TypeError(f"oracle arrays are float32, uint16 (bf16 bits) or uint8 (INT4 rows), got {t.dtype}")
        return np.ascontiguousarray(t)
    import torch  # plain torch CPU ops, only to read a tensor's stored bits

    t = t.detach().to("cpu").contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    if t.dtype == torch.float32:
        return t.numpy()
    if t.dtype == torch.uint8:
        return t.numpy()
    raise TypeError(f"oracle tensors are float32, bfloat16 or uint8 (INT4 rows), got {t.dtype}")


def _dtype_of(a: np.ndarray) -> int:
    if a.dtype == np.uint8:
        return INT4
    return BF16 if a.dtype == np.uint16 else F32


def int4_row_bytes(d: int) -> int:
    """Bytes of one INT4 row of d weights: d/2 code bytes and d/32 binary16 scales."""
    return d // 2 + (d // INT4_GROUP) * 2


def _ptr(a: np.ndarray | None):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def ffn(x, w_gate, w_up, w_down, rows=None, threads: int = 0) -> dict:
    """Dense dReLU FFN of Eq. 1 + Eq. 2 for a batch of tokens.

    ``x`` is ``[B][d]`` (or ``[d]``), fp32 or bf16; the weights ``[m][d]`` in the
    activations' storage type, or all three INT4 rows (uint8 ``[m][d/2 + d/16]``,
    the weight-only 4-bit storage of the paper's INT4 rows) with bf16 or fp32
    activations.
    ``rows`` (optional, sorted unique int32) restricts the sum to the listed
    neurons (Sec. 7 predictor mode). Returns float64 ``y [B][d]``, ``g``, ``u``
    ``[B][m]`` and uint8 ``gate_mask`` / ``both_mask`` ``[B][m]``.
    """
    x, w_gate, w_up, w_down = (as_array(a) for a in (x, w_gate, w_up, w_down))
    if x.ndim == 1:
        x = x[None, :]
    B, d = x.shape
    m = w_gate.shape[0]
    dt = _dtype_of(x)
    if dt == INT4:
        raise ValueError("activations are fp32 or bf16")
    wdt = _dtype_of(w_gate)
    for w in (w_gate, w_up, w_down):
        if wdt == INT4:
            if d % INT4_GROUP != 0 or w.shape != (m, int4_row_bytes(d)) or _dtype_of(w) != INT4:
                raise ValueError("INT4 weights must be [m][d/2 + d/16] uint8, d a multiple of 32")
        elif w.shape != (m, d) or _dtype_of(w) != dt:
            raise ValueError("weights must be [m][d] in the activations' storage type")
    r = None
    n_rows = 0
    if rows is not None:
        r = np.ascontiguousarray(np.asarray(rows, dtype=np.int32))
        n_rows = int(r.size)
    g = np.zeros((B, m), np.float64)
    u = np.zeros((B, m), np.float64)
    gm = np.zeros((B, m), np.uint8)
    bm = np.zeros((B, m), np.uint8)
    y = np.zeros((B, d), np.float64)
    rc = _load().ts_oracle_ffn_w(d, m, B, dt, _ptr(x), wdt, _ptr(w_gate), _ptr(w_up), _ptr(w_down),
                                 _ptr(r), n_rows, _ptr(g), _ptr(u), _ptr(gm), _ptr(bm), _ptr(y),
                                 int(threads))
    if rc != 0:
        raise ValueError("ts_oracle_ffn rejected its arguments (bad shape or row list)")
    return {"y": y, "g": g, "u": u, "gate_mask": gm, "both_mask": bm}


def ffn_topk(x, w_gate, w_up, w_down, keep: int, threads: int = 0) -> dict:
    """FFN with the top-k magnitude mask of Eq. 3 and Eq. 4: per token only the
    ``keep`` neurons with the largest |Combined| (lower index first on a tie)
    enter ``(Combined * Mask) W_down``. Same storage rules as ``ffn`` (no row
    list). Returns float64 ``y [B][d]``, ``g``, ``u``, ``c`` ``[B][m]`` and uint8
    ``sel [B][m]`` (the kept neurons)."""
    x, w_gate, w_up, w_down = (as_array(a) for a in (x, w_gate, w_up, w_down))
    if x.ndim == 1:
        x = x[None, :]
    B, d = x.shape
    m = w_gate.shape[0]
    dt, wdt = _dtype_of(x), _dtype_of(w_gate)
    if dt == INT4:
        raise ValueError("activations are fp32 or bf16")
    for w in (w_gate, w_up, w_down):
        if wdt == INT4:
            if d % INT4_GROUP != 0 or w.shape != (m, int4_row_bytes(d)) or _dtype_of(w) != INT4:
                raise ValueError("INT4 weights must be [m][d/2 + d/16] uint8, d a multiple of 32")
        elif w.shape != (m, d) or _dtype_of(w) != dt:
            raise ValueError("weights must be [m][d] in the activations' storage type")
    g = np.zeros((B, m), np.float64)
    u = np.zeros((B, m), np.float64)
    sel = np.zeros((B, m), np.uint8)
    y = np.zeros((B, d), np.float64)
    rc = _load().ts_oracle_ffn_topk(d, m, B, dt, _ptr(x), wdt, _ptr(w_gate), _ptr(w_up), _ptr(w_down),
                                    int(keep), _ptr(g), _ptr(u), _ptr(sel), _ptr(y), int(threads))
    if rc != 0:
        raise ValueError("ts_oracle_ffn_topk rejected its arguments")
    return {"y": y, "g": g, "u": u, "c": np.maximum(g, 0) * np.maximum(u, 0), "sel": sel}


def predict(x, w1, w2, K: int) -> dict:
    """Activation predictor (a two-layer ReLU MLP, the reading of Sec. 7's
    predictor): ``s = W2 max(0, W1 x)`` per token; the list is the K neurons
    with the largest max-over-tokens score (lower index first on a tie), in
    ascending order. Returns float64 ``scores [B][m]`` and int32 ``list [K]``."""
    x, w1, w2 = (as_array(a) for a in (x, w1, w2))
    if x.ndim == 1:
        x = x[None, :]
    B, d = x.shape
    r = w1.shape[0]
    m = w2.shape[0]
    dt = _dtype_of(x)
    if dt == INT4 or w1.shape != (r, d) or w2.shape != (m, r) or _dtype_of(w1) != dt or _dtype_of(w2) != dt:
        raise ValueError("predictor weights are W1 [r][d] and W2 [m][r] in the activations' storage type")
    scores = np.zeros((B, m), np.float64)
    lst = np.zeros(max(K, 1), np.int32)
    rc = _load().ts_oracle_predict(d, r, m, B, dt, _ptr(x), _ptr(w1), _ptr(w2), int(K), _ptr(scores), _ptr(lst))
    if rc != 0:
        raise ValueError("ts_oracle_predict rejected its arguments")
    return {"scores": scores, "list": lst[:K]}


def router(x, w_r, top_k: int = 2) -> dict:
    """Top-k router: logits ``[B][E]``, chosen experts ``sel [B][k]`` and softmax weights ``w``."""
    x, w_r = as_array(x), as_array(w_r)
    if x.ndim == 1:
        x = x[None, :]
    B, d = x.shape
    E = w_r.shape[0]
    if w_r.shape != (E, d) or _dtype_of(w_r) != _dtype_of(x):
        raise ValueError("router weights must be [E][d] in the activations' storage type")
    logits = np.zeros((B, E), np.float64)
    sel = np.zeros((B, top_k), np.int32)
    w = np.zeros((B, top_k), np.float64)
    rc = _load().ts_oracle_router(d, E, B, _dtype_of(x), _ptr(x), _ptr(w_r), int(top_k),
                                  _ptr(logits), _ptr(sel), _ptr(w))
    if rc != 0:
        raise ValueError("ts_oracle_router rejected its arguments")
    return {"logits": logits, "sel": sel, "w": w}


def moe(x, w_r, experts, top_k: int = 2, threads: int = 0, sel=None, w=None) -> dict:
    """Top-k MoE layer: ``y_t = sum_k w_{t,k} FFN_{e_{t,k}}(x_t)``, each expert a dReLU FFN.

    ``experts`` is a sequence of ``(w_gate, w_up, w_down)``. ``sel``/``w`` override the
    router's choice (used to compare outputs under a given selection when two
    logits tie). Returns ``y [B][d]``, the routing, and per-expert FFN results
    ``expert_out[e] = {token: ffn-result-for-that-token}``.
    """
    x = as_array(x)
    if x.ndim == 1:
        x = x[None, :]
    B, d = x.shape
    rt = router(x, w_r, top_k)
    if sel is None:
        sel, w = rt["sel"], rt["w"]
    sel = np.asarray(sel, np.int32)
    w = np.asarray(w, np.float64)
    y = np.zeros((B, d), np.float64)
    expert_out: dict[int, dict[int, dict]] = {}
    for e in sorted(set(int(v) for v in sel.ravel())):
        toks = [t for t in range(B) if e in sel[t]]
        wg, wu, wd = experts[e]
        res = ffn(x[toks], wg, wu, wd, threads=threads)
        expert_out[e] = {t: {k: res[k][n] for k in res} for n, t in enumerate(toks)}
    for t in range(B):
        for k in range(sel.shape[1]):
            y[t] += w[t, k] * expert_out[int(sel[t, k])][t]["y"]
    return {"y": y, "logits": rt["logits"], "sel": sel, "w": w, "expert_out": expert_out}


def rmsnorm(h, out_dtype: int = BF16, eps: float = RMS_EPS) -> np.ndarray:
    """Stack glue: ``round(h / sqrt(mean(h^2) + eps))`` with the bias channel ``x[d-1] = 1``."""
    h = np.ascontiguousarray(np.asarray(h, np.float32))
    if h.ndim == 1:
        h = h[None, :]
    B, d = h.shape
    out = np.zeros((B, d), np.uint16 if out_dtype == BF16 else np.float32)
    rc = _load().ts_oracle_rmsnorm(d, B, _ptr(h), float(eps), int(out_dtype), _ptr(out))
    if rc != 0:
        raise ValueError("ts_oracle_rmsnorm rejected its arguments")
    return out


def bf16_bits_to_f64(a: np.ndarray) -> np.ndarray:
    """Exact value of bf16 bit patterns (the upper half of a binary32)."""
    return (np.asarray(a, np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def values(a: np.ndarray) -> np.ndarray:
    """Exact float64 values of an oracle storage array (float32 or bf16 bits)."""
    a = as_array(a)
    return bf16_bits_to_f64(a) if a.dtype == np.uint16 else a.astype(np.float64)


def stack(h0, layers, threads: int = 0, record: bool = True) -> dict:
    """The synthetic pre-norm residual stack: ``x_l = rmsnorm(h_l)``, ``h_{l+1} = h_l + FFN_l(x_l)``.

    ``h0`` is float32 ``[B][d]``; ``layers`` a sequence of ``(w_gate, w_up, w_down)``.
    The residual is stored in float32 between layers (the exact fp64 sum is
    rounded once per layer). Returns the final ``h`` and, if ``record``, per layer
    ``x`` (storage bits), ``y`` (float64) and the masks.
    """
    h = np.ascontiguousarray(np.asarray(h0, np.float32))
    if h.ndim == 1:
        h = h[None, :]
    per_layer = []
    for wg, wu, wd in layers:
        wg = as_array(wg)
        x = rmsnorm(h, BF16 if _dtype_of(wg) == INT4 else _dtype_of(wg))  # INT4 rows take bf16 activations
        res = ffn(x, wg, wu, wd, threads=threads)
        h_next = (h.astype(np.float64) + res["y"]).astype(np.float32)
        if record:
            per_layer.append({"h_in": h, "x": x, "y": res["y"], "gate_mask": res["gate_mask"],
                              "both_mask": res["both_mask"]})
        h = h_next
    return {"h": h, "layers": per_layer}
