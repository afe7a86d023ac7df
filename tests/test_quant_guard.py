"""The int8 code argument used by the kernels, checked on the CPU.

The kernels form t = fl32(v * fl32(1/gamma)) and take rint(t) (round half to
even, via the 1.5*2^23 adder) unless t lies within 4e-5 of a half-integer, in
which case they divide exactly.  This emulates that rule in numpy and shows,
on rows built to sit at rounding boundaries and on random data, that it never
differs from the oracle's rule (rint of the correctly rounded fp32 quotient)
outside the guard, while an unguarded version does differ.
"""
import numpy as np

from oracle import taskpress_oracle as O
from tests.test_gpu_quant_edges import _edge_rows


def _emulate(v_bits):
    f = (v_bits.astype(np.uint32) << 16).view(np.float32)
    gamma, codes = O.quantize_v(v_bits[None])
    gamma, codes = gamma[0], codes[0].astype(np.int32)
    with np.errstate(divide="ignore"):
        inv = np.where(gamma > 0, np.float32(1.0) / gamma, np.float32(0.0)).astype(np.float32)
    t = (f * inv[:, None]).astype(np.float32)
    fast = np.clip(np.rint(t), -127, 127).astype(np.int32)
    guarded = np.abs(np.abs(t - np.rint(t)) - np.float32(0.5)) < np.float32(4e-5)
    return fast, codes, guarded, gamma


def test_guard_covers_every_disagreement_at_boundaries():
    for d in (64, 128):
        fast, exact, guarded, gamma = _emulate(_edge_rows(d, 256, seed=21))
        assert (gamma > 0).all()
        differ = fast != exact
        assert differ.any(), "the rows should defeat an unguarded fast path"
        assert not (differ & ~guarded).any()


def test_guard_on_random_rows():
    rng = np.random.Generator(np.random.PCG64(5))
    x = (rng.standard_normal((4096, 128)) * np.exp(rng.uniform(-6, 6, (4096, 1)))).astype(np.float32)
    bits = (x.view(np.uint32) >> 16).astype(np.uint16)
    fast, exact, guarded, _ = _emulate(bits)
    assert not ((fast != exact) & ~guarded).any()
