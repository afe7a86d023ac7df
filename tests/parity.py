"""Comparison rules between the CUDA path and the oracle.

Floating point (scores): relative error <= 2e-3 where the oracle score is at
least 2^-100; below that, where fp32 exp underflows and the oracle still
resolves 1e-40-sized values, absolute error <= 2e-3 * 2^-100.

Indices: the kept set must equal the oracle's except at tokens whose oracle
score lies within 2e-3 (relative) of the oracle's cut-off score; the GPU set
must also be exactly the top-k of the GPU's own fp32 scores (lower index first
among equals), which checks the select kernel bit-exactly.

Integer / byte outputs (scales, int8 codes, compacted rows) are bit-exact.
"""
from __future__ import annotations

import numpy as np

from oracle import taskpress_oracle as O

RTOL = 2e-3
TINY = 2.0 ** -100

#: per-test margins, reported at the end of the run (tests/conftest.py):
#: test id -> {"max_rel": worst relative score error, "units": checked rows,
#: "near_tie_diffs": kept-set differences at near-ties of the cut-off}
STATS: dict = {}

#: method-level figures (recall of planted spans and the like), reported at
#: the end of the run, not asserted
REPORTS: list = []


def _stat(key: str, value, how=max):
    import os
    test = os.environ.get("PYTEST_CURRENT_TEST", "?").split(" ")[0]
    st = STATS.setdefault(test, {"max_rel": 0.0, "units": 0, "near_tie_diffs": 0})
    st[key] = how(st[key], value) if key == "max_rel" else st[key] + value


def to_device_bf16(bits: np.ndarray):
    import torch
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).cuda()


def bf16_bits(t) -> np.ndarray:
    import torch
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def assert_scores_close(gpu: np.ndarray, ref: np.ndarray, what: str = "scores"):
    gpu = np.asarray(gpu, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert gpu.shape == ref.shape, (gpu.shape, ref.shape)
    assert np.all(np.isfinite(gpu)), f"{what}: non-finite GPU values"
    big = ref >= TINY
    _stat("units", 1)
    if big.any():
        rel = np.abs(gpu[big] - ref[big]) / ref[big]
        _stat("max_rel", float(rel.max()))
        worst = int(np.argmax(rel))
        assert rel.max() <= RTOL, (f"{what}: rel err {rel.max():.3e} at {np.flatnonzero(big)[worst]} "
                                   f"gpu={gpu[big][worst]!r} ref={ref[big][worst]!r}")
    if (~big).any():
        ab = np.abs(gpu[~big] - ref[~big]).max()
        assert ab <= RTOL * TINY, f"{what}: abs err {ab:.3e} in the underflow region"


def assert_kept(gpu_idx: np.ndarray, k: int, ref_scores: np.ndarray, gpu_scores: np.ndarray,
                what: str = "kept"):
    """gpu_idx: the row of kept indices (with -1 padding)."""
    row = np.asarray(gpu_idx)
    kept = row[row >= 0]
    assert kept.size == k, f"{what}: kept {kept.size}, want {k}"
    assert np.all(row[k:] == -1), f"{what}: padding not -1"
    assert np.all(np.diff(kept) > 0), f"{what}: kept indices not strictly ascending"
    # exact: the select kernel on the GPU's own fp32 scores
    own = O.select_topk(np.asarray(gpu_scores, dtype=np.float32).astype(np.float64), k)
    assert np.array_equal(kept, own), f"{what}: not the top-{k} of the GPU's own scores"
    # against the oracle's fp64 scores: differences only at near-ties of the cut-off
    ref = O.select_topk(ref_scores, k)
    if k == 0 or k == ref_scores.size:
        assert np.array_equal(kept, ref)
        return
    diff = np.setxor1d(kept, ref)
    _stat("near_tie_diffs", int(diff.size))
    if diff.size:
        cut = ref_scores[ref].min()
        gap = np.abs(ref_scores[diff] - cut) / max(cut, TINY)
        assert gap.max() < RTOL, f"{what}: {diff.size} differing tokens, max gap {gap.max():.3e}"
