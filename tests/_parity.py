"""Comparison rules shared by the GPU parity tests (CUDA path vs the fp64 oracle).

Tolerances (written here, used by every parity test):
* active sets: bit-exact, except neurons whose oracle pre-activation is within
  NEAR_ZERO of 0 (|g| for the gate set, min(|g|, |u|) for the both set); such
  excused flips are counted and returned;
* fp32 data: relative L2 error <= 1e-5;
* bf16 data: relative L2 error <= 2e-3 and max abs error <= 1e-2 * max|y_ref|.
On top of these, TIGHT_REL bounds the relative L2 error of any path that
accumulates in fp32 over identical inputs (fp32 rounding of d-term dot
products gives ~1e-6; 1e-4 leaves room and still flags one dropped row).
"""
from __future__ import annotations

import numpy as np

NEAR_ZERO = 1e-4
REL_F32 = 1e-5
REL_BF16 = 2e-3
MAXABS_BF16 = 1e-2
TIGHT_REL = 1e-4


def rel_l2(got, ref) -> float:
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    n = np.linalg.norm(ref)
    return float(np.linalg.norm(got - ref) / n) if n > 0 else float(np.linalg.norm(got))


def check_y(got, ref, dtype: str, what: str = "y") -> float:
    """Assert the output tolerance for ``dtype`` ('f32' or 'bf16'); return the relative L2 error."""
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    assert got.shape == ref.shape, f"{what}: shape {got.shape} vs {ref.shape}"
    assert np.isfinite(got).all(), f"{what}: non-finite values"
    err = rel_l2(got, ref)
    if not np.any(ref):
        assert not np.any(got), f"{what}: expected all zeros"
        return 0.0
    if dtype == "f32":
        assert err <= REL_F32, f"{what}: rel L2 {err:.3e} > {REL_F32}"
    else:
        assert err <= REL_BF16, f"{what}: rel L2 {err:.3e} > {REL_BF16}"
        mx = float(np.max(np.abs(got - ref)))
        assert mx <= MAXABS_BF16 * float(np.max(np.abs(ref))), f"{what}: max abs {mx:.3e}"
    assert err <= TIGHT_REL, f"{what}: rel L2 {err:.3e} > {TIGHT_REL} (fp32-accumulation bound)"
    return err


def check_sets(gpu_gate, gpu_both, ref: dict, token: int, rows=None) -> int:
    """Compare one token's active sets (neuron ids) with the oracle's masks; return excused flips."""
    g = ref["g"][token]
    u = ref["u"][token]
    og = np.nonzero(ref["gate_mask"][token])[0]
    ob = np.nonzero(ref["both_mask"][token])[0]
    excused = 0
    for name, got, want, near in (
        ("gate", gpu_gate, og, np.abs(g) < NEAR_ZERO),
        ("both", gpu_both, ob, (np.abs(g) < NEAR_ZERO) | (np.abs(u) < NEAR_ZERO)),
    ):
        got = np.asarray(got, np.int64)
        assert np.all(np.diff(got) > 0), f"{name} list not strictly ascending"
        diff = np.setxor1d(got, want)
        bad = diff[~near[diff]] if diff.size else diff
        assert bad.size == 0, f"token {token}: {name} set differs at {bad[:10]} (not near zero)"
        if rows is not None:
            assert np.isin(got, rows).all(), f"{name} set holds unlisted neurons"
        excused += int(diff.size)
    return excused


def union_mask(ref: dict, key: str) -> np.ndarray:
    return np.nonzero(ref[key].any(axis=0))[0]
