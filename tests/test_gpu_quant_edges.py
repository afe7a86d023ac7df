"""Eq. 2 codes (b = 8 and b = 4) next to rounding boundaries, through the C ABI.

The kernels form t = v * fl(1/gamma) and round it with an adder; they take
the exact division only when t lies within 4e-5 of a half-integer (or a
clamp applies).  These rows are built so that most of their values sit that
close to a boundary k + 1/2 under an ordinary (not power-of-two) scale, plus
exact ties, so both the fast path and the exact path decide codes that a
sloppy rounding would get wrong.  Codes and scales must equal the oracle's
bit for bit, for the standalone quantiser and for the compacted cache.
"""
import numpy as np
import pytest

from oracle import taskpress_oracle as O
from tests import parity

pytestmark = pytest.mark.gpu


def _bf16_values():
    """Every finite non-negative bf16 value, as float32."""
    bits = np.arange(0, 0x7F80, dtype=np.uint32)
    return (bits << 16).view(np.float32)


def _edge_rows(d, nrows, seed=3, qmax=127):
    """Rows whose absmax a fixes an ordinary scale gamma = fl32(a / qmax) (not a
    power of two).  The other values are the bf16 values v < a with
    |v / gamma - (k + 1/2)| < 4e-5 (each scale has one or two; they are
    repeated), and values 4e-5 .. 2e-3 from a boundary (just outside the
    guard); signs alternate."""
    rng = np.random.Generator(np.random.PCG64(seed))
    vals = _bf16_values()
    rows = []
    while len(rows) < nrows:
        a = np.float32(rng.uniform(0.5, 300.0))
        a = np.float32((np.array([a]).view(np.uint32) & 0xFFFF0000).view(np.float32)[0])  # a bf16 value
        gamma = np.float32(a / np.float32(qmax))
        if np.frexp(gamma)[0] == 0.5:
            continue
        cand = vals[(vals > 0) & (vals < a)]
        t = cand.astype(np.float64) / np.float64(gamma)
        dist = np.abs(np.abs(t - np.floor(t)) - 0.5)
        near, close = cand[dist < 4e-5], cand[(dist >= 4e-5) & (dist < 2e-3)]
        if near.size == 0 or close.size == 0:
            continue
        nn = (d - 1) // 4
        pick = np.concatenate([rng.choice(near, size=nn), rng.choice(close, size=d - 1 - nn)])
        sign = np.where(np.arange(d - 1) % 2 == 0, 1.0, -1.0).astype(np.float32)
        row = np.concatenate([[a], pick * sign]).astype(np.float32)
        rng.shuffle(row)
        rows.append(row)
    r = np.stack(rows)
    return (r.view(np.uint32) >> 16).astype(np.uint16)


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("d", [64, 128])
def test_codes_at_rounding_boundaries(cuda_lib, d, bits):
    import torch
    from paper_2608_03276_gb300 import binding
    n, hkv = 384, 2
    qmax = (1 << (bits - 1)) - 1
    v = np.stack([_edge_rows(d, n, seed=10 + h, qmax=qmax) for h in range(hkv)])  # [H_kv, n, d]
    p = binding.Problem(2 * hkv, hkv, d, 4, [0, n], quant_bits=bits)
    vq = torch.empty((hkv, n, d * bits // 8), dtype=binding.code_dtype(p), device="cuda")
    g = torch.empty((hkv, n), dtype=torch.float32, device="cuda")
    binding.tp_quantize_v(p, parity.to_device_bf16(v), vq, g)
    rg, rq = O.quantize_v(v, bits)
    rq = O.pack_codes(rq, bits)
    assert np.array_equal(g.cpu().numpy().view(np.uint32), rg.view(np.uint32))
    got = vq.cpu().numpy()
    assert np.array_equal(got, rq), f"{int((got != rq).sum())} code bytes differ"

    # the same rows through the compaction kernel (every token kept, in order)
    k = np.zeros_like(v)
    idx = np.tile(np.arange(n, dtype=np.int32), (1, hkv, 1))
    kc = torch.empty((1, hkv, n, d), dtype=torch.bfloat16, device="cuda")
    vc = torch.empty_like(kc)
    vqc = torch.empty((1, hkv, n, d * bits // 8), dtype=binding.code_dtype(p), device="cuda")
    gc = torch.empty((1, hkv, n), dtype=torch.float32, device="cuda")
    binding.tp_compact(p, parity.to_device_bf16(k), parity.to_device_bf16(v),
                       torch.tensor(rg, device="cuda"), torch.tensor(idx, device="cuda"), 0.0, n,
                       kc, vc, vqc, gc)
    assert np.array_equal(vqc.cpu().numpy()[0], rq)
    assert np.array_equal(gc.cpu().numpy()[0].view(np.uint32), rg.view(np.uint32))
