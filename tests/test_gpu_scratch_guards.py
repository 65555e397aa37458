"""Scratch guard zones (a debugging aid around the method's kernels, not part
of the paper): after forwards over the edge shapes of every kernel family,
every guard zone behind every scratch block of the handles must still hold its
fill, so no kernel wrote past the end of its partial sums, bitmaps, c values or
status word. A byte overwritten from the host must make the check fire."""
import pytest
import torch

from paper_2406_05955_gb300 import binding
from paper_2406_05955_gb300 import workload as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ts():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    import paper_2406_05955_gb300 as ts

    ts.lib()
    return ts


def _ffn(ts, L, max_batch):
    dev = torch.device("cuda")
    return ts.Ffn(L.w_gate.to(dev), L.w_up.to(dev), L.w_down.to(dev), max_batch=max_batch)


@pytest.mark.parametrize("d,m,B,act,dtype", [
    (4096, 14336, 1, 0.10, torch.bfloat16),   # batch-1 rows kernel, per-CTA partials
    (4096, 14336, 2, 1.0, torch.bfloat16),    # every row active: the longest partial lists
    (256, 1001, 3, 0.25, torch.bfloat16),     # ragged chunks, a pass of 2 then 1
    (512, 2048, 8, 0.5, torch.bfloat16),      # 8-token tensor-core pass
    (1024, 2048, 64, 0.10, torch.bfloat16),   # wide tcgen05 path
    (512, 1408, 5, 0.10, torch.float32),      # fp32 rows
])
def test_guards_after_forward(ts, d, m, B, act, dtype):
    L = wl.ffn_layer(d, m, activation=act, dtype=dtype, seed=9100 + m + B)
    f = _ffn(ts, L, B)
    x = wl.tokens(B, d, dtype=dtype, seed=9101).cuda()
    for b in sorted({1, B}):
        f.forward(x[:b])
    assert f.get_error() == binding.TS_OK
    assert f.check_scratch() == binding.TS_OK


@pytest.mark.parametrize("list_len", [1, 700, 14336])
def test_guards_after_predictor_list(ts, list_len):
    d, m = 4096, 14336
    L = wl.ffn_layer(d, m, activation=0.10, dtype=torch.bfloat16, seed=9110)
    f = _ffn(ts, L, 2)
    idx = wl.predictor_list(L.offsets, list_len, seed=9111).cuda()
    f.forward(wl.tokens(2, d, seed=9112).cuda(), active_idx=idx)
    assert f.get_error() == binding.TS_OK
    assert f.check_scratch() == binding.TS_OK


def test_guards_after_int4(ts):
    d, m = 4096, 14336
    L = wl.ffn_layer_int4(d, m, activation=0.10, seed=9120)
    f = _ffn(ts, L, 2)
    f.forward(wl.tokens(2, d, seed=9121).cuda())
    assert f.check_scratch() == binding.TS_OK


@pytest.mark.parametrize("B", [1, 8])
def test_guards_after_moe(ts, B):
    d, m, E = 512, 1024, 8
    dev = torch.device("cuda")
    ex = [_ffn(ts, wl.ffn_layer(d, m, activation=0.2, dtype=torch.bfloat16, seed=wl.layer_seed(9130, 0, e)), B)
          for e in range(E)]
    moe = ts.Moe(wl.router(E, d, seed=9131).to(dev), ex, top_k=2, max_batch=B)
    moe.forward(wl.tokens(B, d, seed=9132).to(dev))
    assert moe.get_error() == binding.TS_OK
    assert moe.check_scratch() == binding.TS_OK


def test_guards_after_predict(ts):
    d, r, m, B = 1024, 256, 3584, 2
    L = wl.ffn_layer(d, m, activation=0.10, dtype=torch.bfloat16, seed=9140)
    P = wl.predictor_weights(d, r, m, L.offsets, seed=9141)
    pred = ts.Predictor(P.w1.cuda(), P.w2.cuda(), max_batch=B)
    pred.predict(wl.tokens(B, d, seed=9142).cuda(), 358)
    assert pred.check_scratch() == binding.TS_OK


def test_poked_guard_is_caught(ts):
    d, m = 256, 1001
    L = wl.ffn_layer(d, m, activation=0.25, dtype=torch.bfloat16, seed=9150)
    f = _ffn(ts, L, 2)
    x = wl.tokens(2, d, seed=9151).cuda()
    y0 = f.forward(x).clone()
    assert f.check_scratch() == binding.TS_OK
    f.poke_guard(0)
    assert f.check_scratch() == binding.TS_ERR_SCRATCH
    with pytest.raises(ts.TsError):
        f.poke_guard(10_000)
    # the guard is outside every block: the handle still computes the same output
    assert torch.equal(f.forward(x), y0)
