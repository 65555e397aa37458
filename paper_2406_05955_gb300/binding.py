"""ctypes binding of libtsffn (include/ts_ffn.h): argument marshalling only.

Every step of the sparse FFN runs in the library's CUDA kernels; this module
turns torch tensors into device pointers and streams, keeps borrowed weights
alive, and raises ``TsError`` on a non-OK status. It never computes anything
itself and has no fallback: if the library is not built, it raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

import numpy as np
import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
# TS_FFN_DEBUG=1 in the environment loads the debug build instead (the same
# kernels with every gathered row index range-checked into the status word).
_DEBUG = os.environ.get("TS_FFN_DEBUG", "") == "1"
LIB_PATH = os.path.join(_HERE, "_build", "debug", "libtsffn_debug.so") if _DEBUG else \
    os.path.join(_HERE, "_build", "libtsffn.so")

TS_OK, TS_ERR_INVALID_ARG, TS_ERR_CUDA, TS_ERR_OOM, TS_ERR_BAD_INDEX, TS_ERR_TIMEOUT, \
    TS_ERR_UNSUPPORTED, TS_ERR_SCRATCH = range(8)
TS_F32, TS_BF16, TS_INT4 = 0, 1, 2

_lock = threading.Lock()
_lib = None

P = ctypes.c_void_p
I = ctypes.c_int
PP = ctypes.POINTER(ctypes.c_void_p)
IP = ctypes.POINTER(ctypes.c_int)

# name -> (restype, argtypes), mirroring include/ts_ffn.h
SIGNATURES = {
    "ts_status_str": (ctypes.c_char_p, [I]),
    "ts_version": (I, []),
    "ts_ffn_create": (I, [PP, I, I, I, P, P, P, I]),
    "ts_ffn_destroy": (None, [P]),
    "ts_ffn_forward": (I, [P, P, I, P, P, P, I]),
    "ts_ffn_forward_topk": (I, [P, P, I, P, P, I]),
    "ts_ffn_gate_up": (I, [P, P, I, P, P, I]),
    "ts_ffn_down": (I, [P, I, P, P]),
    "ts_stack_forward": (I, [P, I, P, I, P, P, P]),
    "ts_ffn_get_active": (I, [P, P, I, P, IP, P, IP]),
    "ts_ffn_get_error": (I, [P, P]),
    "ts_ffn_check_scratch": (I, [P, P]),
    "ts_ffn_poke_guard": (I, [P, I]),
    "ts_ffn_set_test_stall": (I, [P, I]),
    "ts_ffn_forward_noalloc": (I, [I, I, I, P, P, P, P, I, P, P, P, I]),
    "ts_moe_create": (I, [PP, I, I, I, I, P, P, I]),
    "ts_moe_destroy": (None, [P]),
    "ts_moe_forward": (I, [P, P, I, P, P]),
    "ts_moe_stack_forward": (I, [P, I, P, I, P]),
    "ts_moe_get_routing": (I, [P, P, P, P]),
    "ts_moe_get_active": (I, [P, P, I, I, P, IP, P, IP]),
    "ts_moe_get_error": (I, [P, P]),
    "ts_moe_check_scratch": (I, [P, P]),
    "ts_graph_capture_stack": (I, [PP, P, I, P, I, P, P]),
    "ts_graph_capture_stack_fused": (I, [PP, P, I, P, I, P, P]),
    "ts_graph_capture_moe_stack": (I, [PP, P, I, P, I]),
    "ts_predictor_create": (I, [PP, I, I, I, I, P, P, I]),
    "ts_predictor_destroy": (None, [P]),
    "ts_predictor_check_scratch": (I, [P, P]),
    "ts_predict": (I, [P, P, I, I, P, P, P]),
    "ts_stack_forward_predicted": (I, [P, P, I, P, I, P, P, P]),
    "ts_graph_capture_stack_predicted": (I, [PP, P, P, I, P, I, P, P]),
    "ts_graph_launch": (I, [P, P]),
    "ts_graph_destroy": (None, [P]),
}


class TsError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {status_str(status)}")


def lib() -> ctypes.CDLL:
    """The loaded libtsffn; raises if it has not been built (no fallback exists)."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise ImportError(f"libtsffn is not built ({LIB_PATH} missing); "
                                  "run __graft_entry__.build() or python -m paper_2406_05955_gb300.build")
            L = ctypes.CDLL(LIB_PATH)
            for name, (res, args) in SIGNATURES.items():
                fn = getattr(L, name)
                fn.restype = res
                fn.argtypes = args
            _lib = L
    return _lib


def status_str(s: int) -> str:
    return lib().ts_status_str(int(s)).decode()


def _check(s: int, what: str) -> None:
    if s != TS_OK:
        raise TsError(s, what)


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return TS_BF16
    if t.dtype == torch.float32:
        return TS_F32
    raise TypeError(f"weights and activations must be bfloat16 or float32, got {t.dtype}")


def _dev(t: torch.Tensor, what: str) -> torch.Tensor:
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{what} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{what} must be contiguous")
    return t


def _stream(stream) -> int:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream
    return int(stream)


_EMPTY_LISTS: dict = {}


def _list(active_idx):
    """(device pointer, length) of a predictor list; None means detected mode.

    An empty CUDA tensor has a null data pointer, which the C ABI reads as "no
    list", so an empty list is passed as a valid one-element buffer of length 0.
    """
    if active_idx is None:
        return None, 0
    _dev(active_idx, "active_idx")
    if active_idx.dtype != torch.int32:
        raise TypeError("active_idx must be int32")
    n = int(active_idx.numel())
    if n == 0:
        dev = active_idx.device
        if dev not in _EMPTY_LISTS:
            _EMPTY_LISTS[dev] = torch.zeros(1, dtype=torch.int32, device=dev)
        return _EMPTY_LISTS[dev].data_ptr(), 0
    return active_idx.data_ptr(), n


class Ffn:
    """One dReLU FFN layer (or MoE expert) over borrowed device weights: ``[m][d]``
    bf16 / fp32, or INT4 rows (uint8 ``[m][9d/16]``, with bf16 activations)."""

    def __init__(self, w_gate: torch.Tensor, w_up: torch.Tensor, w_down: torch.Tensor,
                 max_batch: int = 1):
        for t, n in ((w_gate, "w_gate"), (w_up, "w_up"), (w_down, "w_down")):
            _dev(t, n)
        if not (w_gate.dtype == w_up.dtype == w_down.dtype):
            raise TypeError("weights must share one dtype")
        m, cols = w_gate.shape
        if w_gate.dtype == torch.uint8:
            d = cols * 16 // 9
            if d % 256 or d // 2 + d // 16 != cols:
                raise ValueError("INT4 rows must be [m][9d/16] bytes with d a multiple of 256")
            self.wcode, self.dtype = TS_INT4, torch.bfloat16
        else:
            d = cols
            self.wcode, self.dtype = _dtype_code(w_gate), w_gate.dtype
        if w_up.shape != (m, cols) or w_down.shape != (m, cols):
            raise ValueError("w_gate, w_up, w_down must have one shape")
        self.d, self.m, self.max_batch = int(d), int(m), int(max_batch)
        self._keep = (w_gate, w_up, w_down)
        h = ctypes.c_void_p()
        _check(lib().ts_ffn_create(ctypes.byref(h), self.d, self.m, self.wcode,
                                   w_gate.data_ptr(), w_up.data_ptr(), w_down.data_ptr(),
                                   self.max_batch), "ts_ffn_create")
        self._h = h

    @property
    def handle(self) -> ctypes.c_void_p:
        if self._h is None:
            raise RuntimeError("handle is closed")
        return self._h

    def _x(self, x: torch.Tensor) -> torch.Tensor:
        _dev(x, "x")
        if x.dtype != self.dtype or x.dim() != 2 or x.shape[1] != self.d:
            raise ValueError(f"x must be [batch][{self.d}] {self.dtype}")
        return x

    def forward(self, x, y=None, active_idx=None, stream=None) -> torch.Tensor:
        x = self._x(x)
        if y is None:
            y = torch.empty(x.shape[0], self.d, dtype=torch.float32, device=x.device)
        _dev(y, "y")
        ptr, n = _list(active_idx)
        _check(lib().ts_ffn_forward(self.handle, x.data_ptr(), x.shape[0], y.data_ptr(),
                                    _stream(stream), ptr, n), "ts_ffn_forward")
        return y

    __call__ = forward

    def forward_topk(self, x, keep: int, y=None, stream=None) -> torch.Tensor:
        """``ts_ffn_forward_topk``: the top-k magnitude mask of Eq. 3-4."""
        x = self._x(x)
        if y is None:
            y = torch.empty(x.shape[0], self.d, dtype=torch.float32, device=x.device)
        _dev(y, "y")
        _check(lib().ts_ffn_forward_topk(self.handle, x.data_ptr(), x.shape[0], y.data_ptr(),
                                         _stream(stream), int(keep)), "ts_ffn_forward_topk")
        return y

    def gate_up(self, x, active_idx=None, stream=None) -> None:
        x = self._x(x)
        ptr, n = _list(active_idx)
        _check(lib().ts_ffn_gate_up(self.handle, x.data_ptr(), x.shape[0], _stream(stream), ptr, n),
               "ts_ffn_gate_up")

    def down(self, batch: int, y=None, stream=None, device=None) -> torch.Tensor:
        if y is None:
            y = torch.empty(batch, self.d, dtype=torch.float32,
                            device=device or self._keep[0].device)
        _dev(y, "y")
        _check(lib().ts_ffn_down(self.handle, int(batch), y.data_ptr(), _stream(stream)), "ts_ffn_down")
        return y

    def get_active(self, token: int = -1, stream=None):
        """Active sets of the last forward: (gate-active ids, both-active ids), int32 numpy."""
        g = np.zeros(self.m, np.int32)
        b = np.zeros(self.m, np.int32)
        ng, nb = ctypes.c_int(), ctypes.c_int()
        _check(lib().ts_ffn_get_active(self.handle, _stream(stream), int(token),
                                       g.ctypes.data_as(P), ctypes.byref(ng),
                                       b.ctypes.data_as(P), ctypes.byref(nb)), "ts_ffn_get_active")
        return g[: ng.value].copy(), b[: nb.value].copy()

    def get_error(self, stream=None) -> int:
        return int(lib().ts_ffn_get_error(self.handle, _stream(stream)))

    def check_scratch(self, stream=None) -> int:
        """Status of the scratch guard zones: TS_OK, or TS_ERR_SCRATCH if one was overwritten."""
        return int(lib().ts_ffn_check_scratch(self.handle, _stream(stream)))

    def poke_guard(self, i: int) -> None:
        """Test hook: overwrite one byte of scratch guard zone ``i`` from the host."""
        _check(lib().ts_ffn_poke_guard(self.handle, int(i)), "ts_ffn_poke_guard")

    def set_test_stall(self, on: bool) -> None:
        """Failure-detection test hook: the next forwards' bounded waits run out."""
        _check(lib().ts_ffn_set_test_stall(self.handle, int(bool(on))), "ts_ffn_set_test_stall")

    def close(self) -> None:
        if getattr(self, "_h", None) is not None:
            lib().ts_ffn_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def ffn_forward_noalloc(w_gate, w_up, w_down, x, y, active_idx=None, stream=None) -> torch.Tensor:
    """``ts_ffn_forward_noalloc``: one FFN forward into the caller's ``y`` with
    the library's static scratch (no handle, no device allocation)."""
    for t, n in ((w_gate, "w_gate"), (w_up, "w_up"), (w_down, "w_down"), (x, "x"), (y, "y")):
        _dev(t, n)
    m, d = w_gate.shape
    if w_up.shape != (m, d) or w_down.shape != (m, d):
        raise ValueError("w_gate, w_up, w_down must all be [m][d]")
    if not (w_gate.dtype == w_up.dtype == w_down.dtype == x.dtype):
        raise TypeError("weights and x must share one dtype")
    if x.dim() != 2 or x.shape[1] != d or y.dtype != torch.float32 or tuple(y.shape) != tuple(x.shape):
        raise ValueError(f"x must be [batch][{d}] and y [batch][{d}] float32")
    ptr, n = _list(active_idx)
    _check(lib().ts_ffn_forward_noalloc(int(d), int(m), _dtype_code(w_gate), w_gate.data_ptr(),
                                        w_up.data_ptr(), w_down.data_ptr(), x.data_ptr(), x.shape[0],
                                        y.data_ptr(), _stream(stream), ptr, n), "ts_ffn_forward_noalloc")
    return y


def _addr(arr):
    return None if arr is None else ctypes.cast(arr, ctypes.c_void_p)


def _handles(objs) -> ctypes.Array:
    arr = (ctypes.c_void_p * len(objs))()
    for i, o in enumerate(objs):
        arr[i] = o.handle.value
    return arr


def _lists(active_idx, n_layers):
    if active_idx is None:
        return None, None, []
    if len(active_idx) != n_layers:
        raise ValueError("one active_idx entry per layer")
    ptrs = (ctypes.c_void_p * n_layers)()
    ns = (ctypes.c_int * n_layers)()
    keep = []
    for i, a in enumerate(active_idx):
        p, n = _list(a)
        ptrs[i] = p
        ns[i] = n
        keep.append(a)
    return ptrs, ns, keep


def stack_forward(layers, h: torch.Tensor, active_idx=None, stream=None) -> torch.Tensor:
    """In-place pre-norm residual stack over ``layers`` on fp32 ``h [batch][d]``."""
    _dev(h, "h")
    if h.dtype != torch.float32:
        raise TypeError("h must be float32")
    arr = _handles(layers)
    ptrs, ns, _keep = _lists(active_idx, len(layers))
    _check(lib().ts_stack_forward(_addr(arr), len(layers), h.data_ptr(), h.shape[0], _stream(stream),
                                  _addr(ptrs), _addr(ns)), "ts_stack_forward")
    return h


class Predictor:
    """Activation predictor of one FFN layer over borrowed ``w1 [r][d]`` and
    ``w2 [m][r]`` (bf16 or fp32): ``ts_predict`` gives the K neurons with the
    largest max-over-tokens score of ``w2 relu(w1 x)``, ascending."""

    def __init__(self, w1: torch.Tensor, w2: torch.Tensor, max_batch: int = 1):
        _dev(w1, "w1")
        _dev(w2, "w2")
        if w1.dtype != w2.dtype:
            raise TypeError("w1 and w2 must share one dtype")
        self.r, self.d = int(w1.shape[0]), int(w1.shape[1])
        self.m = int(w2.shape[0])
        if w2.dim() != 2 or w2.shape[1] != self.r:
            raise ValueError("w2 must be [m][r] with r = w1.shape[0]")
        self.dtype, self.max_batch = w1.dtype, int(max_batch)
        self._keep = (w1, w2)
        h = ctypes.c_void_p()
        _check(lib().ts_predictor_create(ctypes.byref(h), self.d, self.r, self.m, _dtype_code(w1),
                                         w1.data_ptr(), w2.data_ptr(), self.max_batch), "ts_predictor_create")
        self._h = h

    @property
    def handle(self) -> ctypes.c_void_p:
        if self._h is None:
            raise RuntimeError("handle is closed")
        return self._h

    def predict(self, x, K: int, out=None, scores=None, stream=None) -> torch.Tensor:
        """The predicted list (int32 [K], ascending); ``scores`` (fp32
        [batch][m]), when given, receives every neuron's score."""
        _dev(x, "x")
        if x.dtype != self.dtype or x.dim() != 2 or x.shape[1] != self.d:
            raise ValueError(f"x must be [batch][{self.d}] {self.dtype}")
        if out is None:
            out = torch.empty(max(int(K), 1), dtype=torch.int32, device=x.device)
        _dev(out, "out")
        if out.dtype != torch.int32 or out.numel() < K:
            raise ValueError("out must be int32 with at least K entries")
        sp = None
        if scores is not None:
            _dev(scores, "scores")
            if scores.dtype != torch.float32 or tuple(scores.shape) != (x.shape[0], self.m):
                raise ValueError(f"scores must be [batch][{self.m}] float32")
            sp = scores.data_ptr()
        _check(lib().ts_predict(self.handle, x.data_ptr(), x.shape[0], int(K), out.data_ptr(), sp,
                                _stream(stream)), "ts_predict")
        return out[: int(K)]

    def check_scratch(self, stream=None) -> int:
        """Status of the scratch guard zones (as Ffn.check_scratch)."""
        return int(lib().ts_predictor_check_scratch(self.handle, _stream(stream)))

    def close(self) -> None:
        if getattr(self, "_h", None) is not None:
            lib().ts_predictor_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def _predicted_args(layers, preds, K, lists):
    n = len(layers)
    if len(preds) != n or len(K) != n or len(lists) != n:
        raise ValueError("one predictor, K and list buffer per layer")
    ks = (ctypes.c_int * n)(*[int(k) for k in K])
    ptrs = (ctypes.c_void_p * n)()
    for i, (buf, k) in enumerate(zip(lists, K)):
        _dev(buf, "lists[i]")
        if buf.dtype != torch.int32 or buf.numel() < max(int(k), 1):
            raise ValueError("each list buffer must be int32 with at least max(K, 1) entries")
        ptrs[i] = buf.data_ptr()
    return _handles(layers), _handles(preds), ks, ptrs


def stack_forward_predicted(layers, preds, h: torch.Tensor, K, lists, stream=None) -> torch.Tensor:
    """``ts_stack_forward_predicted``: each layer predicts its list from
    rmsnorm(h) into ``lists[l]`` and runs the FFN over it; ``h`` in place."""
    _dev(h, "h")
    if h.dtype != torch.float32:
        raise TypeError("h must be float32")
    la, pa, ks, ptrs = _predicted_args(layers, preds, K, lists)
    _check(lib().ts_stack_forward_predicted(_addr(la), _addr(pa), len(layers), h.data_ptr(), h.shape[0],
                                            _addr(ks), _addr(ptrs), _stream(stream)),
           "ts_stack_forward_predicted")
    return h


class Moe:
    """Top-k MoE layer over ``Ffn`` experts and a borrowed router ``w_router [E][d]``."""

    def __init__(self, w_router: torch.Tensor, experts, top_k: int = 2, max_batch: int = 1):
        _dev(w_router, "w_router")
        self.E, self.d = int(w_router.shape[0]), int(w_router.shape[1])
        self.top_k, self.max_batch = int(top_k), int(max_batch)
        self.dtype = w_router.dtype
        self.experts = list(experts)
        self._keep = (w_router,)
        arr = _handles(self.experts)
        h = ctypes.c_void_p()
        _check(lib().ts_moe_create(ctypes.byref(h), self.d, self.E, self.top_k, self.experts[0].wcode,
                                   w_router.data_ptr(), _addr(arr), self.max_batch), "ts_moe_create")
        self._h = h
        self.m = self.experts[0].m

    @property
    def handle(self) -> ctypes.c_void_p:
        if self._h is None:
            raise RuntimeError("handle is closed")
        return self._h

    def forward(self, x, y=None, stream=None) -> torch.Tensor:
        _dev(x, "x")
        if x.dtype != self.dtype or x.dim() != 2 or x.shape[1] != self.d:
            raise ValueError(f"x must be [batch][{self.d}] {self.dtype}")
        if y is None:
            y = torch.empty(x.shape[0], self.d, dtype=torch.float32, device=x.device)
        _dev(y, "y")
        _check(lib().ts_moe_forward(self.handle, x.data_ptr(), x.shape[0], y.data_ptr(), _stream(stream)),
               "ts_moe_forward")
        return y

    __call__ = forward

    def get_routing(self, batch: int, stream=None):
        sel = np.zeros((batch, self.top_k), np.int32)
        w = np.zeros((batch, self.top_k), np.float32)
        _check(lib().ts_moe_get_routing(self.handle, _stream(stream), sel.ctypes.data_as(P),
                                        w.ctypes.data_as(P)), "ts_moe_get_routing")
        return sel, w

    def get_active(self, expert: int, token: int = -1, stream=None):
        g = np.zeros(self.m, np.int32)
        b = np.zeros(self.m, np.int32)
        ng, nb = ctypes.c_int(), ctypes.c_int()
        _check(lib().ts_moe_get_active(self.handle, _stream(stream), int(expert), int(token),
                                       g.ctypes.data_as(P), ctypes.byref(ng),
                                       b.ctypes.data_as(P), ctypes.byref(nb)), "ts_moe_get_active")
        return g[: ng.value].copy(), b[: nb.value].copy()

    def get_error(self, stream=None) -> int:
        return int(lib().ts_moe_get_error(self.handle, _stream(stream)))

    def check_scratch(self, stream=None) -> int:
        """Status of the scratch guard zones (as Ffn.check_scratch)."""
        return int(lib().ts_moe_check_scratch(self.handle, _stream(stream)))

    def close(self) -> None:
        if getattr(self, "_h", None) is not None:
            lib().ts_moe_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def moe_stack_forward(layers, h: torch.Tensor, stream=None) -> torch.Tensor:
    _dev(h, "h")
    arr = _handles(layers)
    _check(lib().ts_moe_stack_forward(_addr(arr), len(layers), h.data_ptr(), h.shape[0], _stream(stream)),
           "ts_moe_stack_forward")
    return h


class Graph:
    """A multi-layer forward captured once (``ts_graph_capture_*``) and replayed."""

    def __init__(self, handle: ctypes.c_void_p, keep):
        self._h = handle
        self._keep = keep

    @classmethod
    def stack(cls, layers, h: torch.Tensor, active_idx=None) -> "Graph":
        _dev(h, "h")
        arr = _handles(layers)
        ptrs, ns, keep = _lists(active_idx, len(layers))
        g = ctypes.c_void_p()
        _check(lib().ts_graph_capture_stack(ctypes.byref(g), _addr(arr), len(layers), h.data_ptr(),
                                            h.shape[0], _addr(ptrs), _addr(ns)), "ts_graph_capture_stack")
        return cls(g, (list(layers), h, keep))

    @classmethod
    def stack_fused(cls, layers, h: torch.Tensor, active_idx=None) -> "Graph":
        """The stack as one persistent launch (ts_graph_capture_stack_fused);
        raises TsError(TS_ERR_UNSUPPORTED) where it does not apply."""
        _dev(h, "h")
        arr = _handles(layers)
        ptrs, ns, keep = _lists(active_idx, len(layers))
        g = ctypes.c_void_p()
        _check(lib().ts_graph_capture_stack_fused(ctypes.byref(g), _addr(arr), len(layers), h.data_ptr(),
                                                  h.shape[0], _addr(ptrs), _addr(ns)),
               "ts_graph_capture_stack_fused")
        return cls(g, (list(layers), h, keep))

    @classmethod
    def stack_predicted(cls, layers, preds, h: torch.Tensor, K, lists) -> "Graph":
        _dev(h, "h")
        la, pa, ks, ptrs = _predicted_args(layers, preds, K, lists)
        g = ctypes.c_void_p()
        _check(lib().ts_graph_capture_stack_predicted(ctypes.byref(g), _addr(la), _addr(pa), len(layers),
                                                      h.data_ptr(), h.shape[0], _addr(ks), _addr(ptrs)),
               "ts_graph_capture_stack_predicted")
        return cls(g, (list(layers), list(preds), h, ks, ptrs, list(lists)))

    @classmethod
    def moe_stack(cls, layers, h: torch.Tensor) -> "Graph":
        _dev(h, "h")
        arr = _handles(layers)
        g = ctypes.c_void_p()
        _check(lib().ts_graph_capture_moe_stack(ctypes.byref(g), _addr(arr), len(layers), h.data_ptr(),
                                                h.shape[0]), "ts_graph_capture_moe_stack")
        return cls(g, (list(layers), h))

    def launch(self, stream=None) -> None:
        _check(lib().ts_graph_launch(self._h, _stream(stream)), "ts_graph_launch")

    def close(self) -> None:
        if getattr(self, "_h", None) is not None:
            lib().ts_graph_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
