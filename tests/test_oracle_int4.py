"""Pins for the oracle's INT4 weight storage (the 4-bit weight-only rows of the
paper's INT4 models, Tables 7-9), against things other than the oracle.

Row layout: d/2 bytes of 4-bit codes, then d/32 little-endian IEEE binary16
scales; weight = scale * (code - 8). A group of 32 elements owns 16 code bytes,
read as four little-endian 32-bit words: element e = 8s + 2t + h (s, t in
0..3, h in 0..1) is nibble s + 4h of word t.
Pinned by: a hand-worked FFN whose codes and scales were chosen so every value
is exact; binary16 special cases against numpy's float16 decoding; random
layers against an independent numpy decoding followed by library matmuls; the
all-active case as a plain ReGLU FFN; and mistakes planted in a CPU
restatement of the decoding (the two halves of a word swapped, plain sequential
nibbles, offset 7, a shifted scale group, big-endian scales), which the pins
reject.
"""
import numpy as np
import pytest
import torch

from paper_2406_05955_gb300 import workload as wl

D = 32  # one group per row


def _pack(c: np.ndarray) -> np.ndarray:
    """Code bytes of one row of d codes: per group of 32, word t holds element
    8s + 2t + h at nibble s + 4h; words stored little-endian."""
    out = []
    for g in range(len(c) // 32):
        grp = c[32 * g: 32 * g + 32]
        for t in range(4):
            word = 0
            for s_ in range(4):
                for h in range(2):
                    word |= int(grp[8 * s_ + 2 * t + h]) << (4 * (s_ + 4 * h))
            out += [(word >> (8 * b)) & 0xFF for b in range(4)]
    return np.array(out, np.uint8)


def _unpack(q: np.ndarray, d: int, halves=(0, 1), sequential=False) -> np.ndarray:
    """Codes [rows][d] from the code bytes of each row (the inverse of _pack)."""
    b = q[:, : d // 2].astype(np.int64)
    codes = np.empty((q.shape[0], d), np.int64)
    if sequential:  # a planted mistake: element i in byte i/2, low nibble for even i
        codes[:, 0::2], codes[:, 1::2] = b & 0x0F, b >> 4
        return codes
    words = b.reshape(q.shape[0], d // 32, 4, 4)
    words = words[..., 0] | (words[..., 1] << 8) | (words[..., 2] << 16) | (words[..., 3] << 24)
    for s_ in range(4):
        for t in range(4):
            for h in range(2):
                codes[:, 8 * s_ + 2 * t + h::32] = (words[:, :, t] >> (4 * (s_ + 4 * halves[h]))) & 0xF
    return codes


def _row(codes: dict, scale_bits: int, d: int = D) -> np.ndarray:
    """One INT4 row: codes {element: code} (others 8, i.e. weight 0) and one scale per group."""
    c = np.full(d, 8, np.uint8)
    for i, v in codes.items():
        c[i] = v
    scales = np.full(d // 32, scale_bits, np.uint16).astype("<u2").view(np.uint8)
    return np.concatenate([_pack(c), scales])


def _bf16(v):
    return torch.tensor(np.asarray(v, np.float64), dtype=torch.float32).to(torch.bfloat16)


# hand-worked case (every value exact): x = (1, 2, 0, ...)
#   W_gate rows: 0.5*(1, 0)      -> g0 = 0.5
#                0.25*(-2, 2)    -> g1 = -0.5 + 1 = 0.5
#                1.0*(0, -4)     -> g2 = -8
#   W_up rows:   0.5*(6, 0)      -> u0 = 3
#                2.0*(0, -1)     -> u1 = -4
#                1.0*(7, 0)      -> u2 = 7
#   gate-active {0, 1}, both-active {0}, c = (1.5, 0, 0)
#   W_down row 0: 0.125*(2, 4, 0, ..., -8) -> y = 1.5 * (0.25, 0.5, 0, ..., -1)
H_HALF, H_QUARTER, H_ONE, H_TWO, H_EIGHTH = 0x3800, 0x3400, 0x3C00, 0x4000, 0x3000


def _handworked():
    wg = np.stack([_row({0: 9, 1: 8}, H_HALF), _row({0: 6, 1: 10}, H_QUARTER), _row({1: 4}, H_ONE)])
    wu = np.stack([_row({0: 14}, H_HALF), _row({1: 7}, H_TWO), _row({0: 15}, H_ONE)])
    wd = np.stack([_row({0: 10, 1: 12, 31: 0}, H_EIGHTH), _row({5: 15}, H_ONE), _row({7: 0}, H_ONE)])
    x = np.zeros(D)
    x[0], x[1] = 1.0, 2.0
    y = np.zeros(D)
    y[0], y[1], y[31] = 1.5 * 0.25, 1.5 * 0.5, 1.5 * -1.0
    return x, wg, wu, wd, y


def test_int4_handworked(oracle_mod):
    x, wg, wu, wd, y = _handworked()
    for xs in (_bf16(x[None]), torch.tensor(x[None], dtype=torch.float32)):
        r = oracle_mod.ffn(xs, wg, wu, wd)
        assert np.array_equal(r["g"][0], [0.5, 0.5, -8.0])
        assert np.array_equal(r["u"][0], [3.0, -4.0, 7.0])
        assert list(np.nonzero(r["gate_mask"][0])[0]) == [0, 1]
        assert list(np.nonzero(r["both_mask"][0])[0]) == [0]
        assert np.array_equal(r["y"][0], y)


@pytest.mark.parametrize("bits", [0x0001, 0x03FF, 0x0400, 0x3C00, 0x7BFF, 0xB800, 0x8001, 0x3555])
def test_int4_scale_decoding_matches_numpy_float16(oracle_mod, bits):
    # x = e_0 and code 9 (+1) at element 0: g_0 = scale exactly
    wg = _row({0: 9}, bits)[None]
    wu = _row({0: 9}, 0x3C00)[None]
    wd = _row({}, 0x3C00)[None]
    x = np.zeros((1, D), np.float32)
    x[0, 0] = 1.0
    r = oracle_mod.ffn(x, wg, wu, wd)
    expect = float(np.array([bits], np.uint16).view(np.float16)[0])
    assert r["g"][0, 0] == expect


def _numpy_dequant(q: np.ndarray, d: int) -> np.ndarray:
    """Independent decoding with numpy: nibbles, float16 view, broadcast per group."""
    codes = _unpack(q, d)
    scales = np.ascontiguousarray(q[:, d // 2:]).view("<f2").astype(np.float64)
    return np.repeat(scales, 32, axis=1) * (codes - 8)


@pytest.mark.parametrize("act", [0.10, 1.0])
def test_int4_random_layers_against_numpy(oracle_mod, act):
    d, m, B = 256, 96, 3
    L = wl.ffn_layer_int4(d, m, activation=act, seed=77)
    x = wl.tokens(B, d, seed=78)
    r = oracle_mod.ffn(x, L.w_gate, L.w_up, L.w_down)
    wg, wu, wd = (_numpy_dequant(t.numpy(), d) for t in (L.w_gate, L.w_up, L.w_down))
    xv = x.float().double().numpy()
    g, u = xv @ wg.T, xv @ wu.T
    assert np.allclose(r["g"], g, rtol=1e-12, atol=1e-12)
    assert np.allclose(r["u"], u, rtol=1e-12, atol=1e-12)
    if act >= 1.0:
        assert r["both_mask"].all()
        y = (np.maximum(g, 0) * np.maximum(u, 0)) @ wd  # a plain ReGLU FFN
        assert np.allclose(r["y"], y, rtol=1e-12, atol=1e-12)


def test_quantizer_round_trip_bound():
    w = torch.randn(64, 128, generator=torch.Generator().manual_seed(5)) * 0.1
    w[3] = 0.0  # an all-zero row: scale 1, codes 8
    q = wl.quantize_int4(w)
    assert q.shape == (64, wl.int4_row_bytes(128)) and q.dtype == torch.uint8
    back = _numpy_dequant(q.numpy(), 128)
    scales = np.repeat(np.ascontiguousarray(q.numpy()[:, 64:]).view("<f2").astype(np.float64), 32, axis=1)
    err = np.abs(back - w.double().numpy())
    assert (err <= 0.5 * scales * (1 + 2.0 ** -10) + 1e-12).all()
    assert np.array_equal(back[3], np.zeros(128))


def _planted(q_rows, d, mistake):
    codes = _unpack(q_rows, d, halves=(1, 0) if mistake == "swapped_halves" else (0, 1),
                    sequential=mistake == "sequential")
    sc = np.ascontiguousarray(q_rows[:, d // 2:])
    scales = sc.view(">f2" if mistake == "big_endian_scale" else "<f2").astype(np.float64)
    per = np.repeat(scales, 32, axis=1)
    if mistake == "shifted_group":
        per = np.roll(per, 32, axis=1)
    off = 7 if mistake == "offset_7" else 8
    return per * (codes - off)


@pytest.mark.parametrize("mistake", ["swapped_halves", "sequential", "offset_7", "big_endian_scale",
                                     "shifted_group"])
def test_int4_pins_reject_planted_mistakes(mistake):
    x, wg, wu, wd, y = _handworked()
    # the hand-worked case with a second group, so a shifted group is visible
    d = 64
    x2 = np.concatenate([x, np.zeros(32)])
    pad = lambda rows: np.stack([np.concatenate([r[:16], _row({}, H_ONE)[:16], r[16:], _row({}, 0x4400)[16:]]) for r in rows])
    mats = [_planted(pad(m_), d, mistake) for m_ in (wg, wu, wd)]
    g, u = x2 @ mats[0].T, x2 @ mats[1].T
    yy = (np.maximum(g, 0) * np.maximum(u, 0)) @ mats[2]
    reproduced = np.array_equal(yy[:32], y) and np.array_equal(g, [0.5, 0.5, -8.0])
    assert reproduced == (mistake is None)


def test_int4_planted_mistake_control():
    test_int4_pins_reject_planted_mistakes(None)


def test_header_packing_text_matches_quantize_int4():
    """Pack INT4 rows exactly as the public header describes them and compare
    the bytes with the generator's quantizer (the format the library reads):
    group G's codes are the 16 bytes at 16G, four little-endian 32-bit words;
    element 8s + 2t + h is nibble s + 4h of word t; then d/32 binary16 scales."""
    rng = np.random.default_rng(11)
    m, d = 3, 256
    w = torch.from_numpy(rng.standard_normal((m, d)).astype(np.float32))
    got = wl.quantize_int4(w).numpy()
    wf = w.numpy().reshape(m, d // 32, 32)
    scale = (np.abs(wf).max(-1) / 7.0).astype(np.float16)
    scale[scale == 0] = 1
    code = np.clip(np.round(wf / scale.astype(np.float32)[..., None]), -8, 7).astype(np.int64) + 8
    want = np.zeros((m, d // 2 + d // 16), dtype=np.uint8)
    for j in range(m):
        for G in range(d // 32):
            words = [0, 0, 0, 0]
            for e in range(32):
                s, t, h = e // 8, (e % 8) // 2, e % 2
                words[t] |= int(code[j, G, e]) << (4 * (s + 4 * h))
            for t in range(4):
                for b in range(4):
                    want[j, 16 * G + 4 * t + b] = (words[t] >> (8 * b)) & 0xFF
        want[j, d // 2:] = np.frombuffer(scale[j].tobytes(), dtype=np.uint8)
    np.testing.assert_array_equal(got, want)
