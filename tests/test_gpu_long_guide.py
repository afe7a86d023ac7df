"""Guides longer than one scoring block, through the C ABI against the oracle.

A guide of more than TP_MAX_ROWS = 512 stacked rows (G * L_t: the 256- and
1024-token guides of the paper's TTFT study, Sec. 4.2.3, at G = 4) is scored
in blocks of 512 rows: each block runs both passes on its own rows and the
blocks' key scores are added in block order.  The oracle scores all rows at
once (Eq. 1 in fp64), so these cases check the block split and the addition
on every path that takes a long guide: the two-pass layer (whole blocks and a
ragged last block), the caller's normalisers, the literal normaliser (the
guide-prefix fold over whole rows), the stage entry points and both stacks of
layers.  Tolerances as everywhere: tests/parity.py.
"""
import math

import numpy as np
import pytest

from oracle import taskpress_oracle as O
from paper_2608_03276_gb300 import synth
from tests import parity
from tests.test_gpu_parity import _check_layer, _oracle, _problem, _run_compress
from tests.test_gpu_variants import _context_lse, _outputs_equal, _run_lse, _stack

pytestmark = pytest.mark.gpu


def _long(hq, hkv, d, lt, lens, **kw):
    base = dict(spans=(3, 16), v_outlier=(0.01, 16.0), key_chan_scale=(0.5, 4.0), seed=91,
                keep_ratio=0.2)
    base.update(kw)
    return synth.Workload("long-guide", hq, hkv, d, lt, tuple(lens), **base)


LONG = {
    # two whole blocks of 512 rows
    "g4-lt256-m1024": _long(8, 2, 128, 256, [3001]),
    # blocks of 512, 512 and 76 rows over ragged documents (one empty)
    "g4-lt275-m1100-ragged": _long(8, 2, 128, 275, [1500, 1, 0, 900], budget=300),
    # four blocks at d = 64, G = 8
    "g8-lt256-d64-m2048": _long(16, 2, 64, 256, [2200]),
    # the paper's longest guide: 1024 tokens at G = 4, eight blocks
    "g4-lt1024-m4096": _long(4, 1, 128, 1024, [2048]),
}


@pytest.mark.parametrize("name", sorted(LONG))
def test_long_guide_layer(cuda_lib, name):
    from paper_2608_03276_gb300 import binding
    w = LONG[name]
    assert w.rows > binding.TP_MAX_ROWS
    x = synth.make_layer(w)
    out = _run_compress(binding, w, x)
    _check_layer(w, x, out, _oracle(w, x))


@pytest.mark.parametrize("name", ["g4-lt256-m1024", "g4-lt275-m1100-ragged"])
def test_long_guide_caller_normalisers(cuda_lib, name):
    """The caller's row normalisers (extra prefix mass per row, so that the
    blocks see different normalisers): block 0's kernel also forms the Eq. 2
    scales, the later blocks add their key scores."""
    from paper_2608_03276_gb300 import binding
    w = LONG[name]
    x = synth.make_layer(w)
    lse_ctx = _context_lse(w, x)
    rng = np.random.Generator(np.random.PCG64(17))
    extra = rng.uniform(-2.0, 3.0, lse_ctx.shape)
    lse = np.logaddexp(lse_ctx.astype(np.float64), lse_ctx + extra).astype(np.float32)
    out = _run_lse(binding, w, x, lse)
    _check_layer(w, x, out, _oracle(w, x, lse=lse.astype(np.float64)))


@pytest.mark.parametrize("name", ["g4-lt275-m1100-ragged", "g8-lt256-d64-m2048"])
def test_long_guide_literal_normaliser(cuda_lib, name):
    """tp_compress_layer_guide: every block's pass 1, the fold over whole rows
    (guide keys 0..j, across block boundaries), then every block's pass 2."""
    from paper_2608_03276_gb300 import binding
    w = LONG[name]
    x = synth.make_layer(w)
    kg = synth.make_guide_keys(w)
    p = _problem(binding, w, x.doc_offsets)
    out = binding.CompressOutputs(p, w.keep_ratio, w.budget, "cuda")
    binding.compress(p, parity.to_device_bf16(x.q), parity.to_device_bf16(x.k),
                     parity.to_device_bf16(x.v), w.keep_ratio, w.budget, out,
                     k_guide=parity.to_device_bf16(kg))
    assert binding.tp_check_status(out.ws) == 0
    _check_layer(w, x, out, _oracle(w, x, k_guide_bits=kg))


def test_long_guide_stage_entry_points(cuda_lib):
    """tp_guide_lse writes every block's normalisers into their columns of
    [batch, H_kv, M] (and the Eq. 2 scales with block 0); tp_guide_scores
    matches the oracle's combined scores; the two entry points without a
    workspace refuse the long guide."""
    import torch
    from paper_2608_03276_gb300 import binding
    w = LONG["g4-lt275-m1100-ragged"]
    x = synth.make_layer(w)
    p = _problem(binding, w, x.doc_offsets)
    q, k = parity.to_device_bf16(x.q), parity.to_device_bf16(x.k)
    rows = w.rows
    lse = torch.full((w.batch, w.n_heads_kv, rows), float("nan"), dtype=torch.float32, device="cuda")
    ws = torch.empty(binding.tp_workspace_bytes(p), dtype=torch.uint8, device="cuda")
    gam = torch.empty((w.n_heads_kv, p.n_total), dtype=torch.float32, device="cuda")
    binding.tp_guide_lse(p, q, k, lse, ws, v=parity.to_device_bf16(x.v), gamma=gam)
    rg, _ = O.quantize_v(x.v)
    assert np.array_equal(gam.cpu().numpy().view(np.uint32), rg.view(np.uint32)), "gamma"
    got = lse.cpu().numpy()
    qf, kf = O.decode_bf16(x.q), O.decode_bf16(x.k)
    sigma = 1.0 / math.sqrt(w.head_dim)
    for b in range(w.batch):
        lo, hi = x.doc_offsets[b], x.doc_offsets[b + 1]
        if hi == lo:
            continue
        for h in range(w.n_heads_kv):
            want = O.guide_lse(qf[b, h * w.group:(h + 1) * w.group].reshape(rows, -1), kf[h, lo:hi], sigma)
            assert np.abs(got[b, h] - want).max() <= parity.RTOL, (b, h)
    ref = _oracle(w, x)
    s = torch.empty((w.n_heads_kv, p.n_total), dtype=torch.float32, device="cuda")
    binding.tp_guide_scores(p, q, k, torch.tensor(ref["gamma"], device="cuda"), s, ws)
    sc = s.cpu().numpy()
    for (b, h), want in ref["scores"].items():
        lo, hi = x.doc_offsets[b], x.doc_offsets[b + 1]
        parity.assert_scores_close(sc[h, lo:hi], want, f"doc {b} head {h}")
    cdll = binding.load()
    assert cdll.tp_guide_key_scores(p.ref(), q.data_ptr(), k.data_ptr(), None, lse.data_ptr(),
                                    s.data_ptr(), None, None) == binding.TP_ERR_UNSUPPORTED_SHAPE
    assert cdll.tp_guide_lse_static(p.ref(), q.data_ptr(), k.data_ptr(), None, lse.data_ptr(),
                                    None, None) == binding.TP_ERR_UNSUPPORTED_SHAPE


def test_long_guide_stacks(cuda_lib):
    """tp_compress_layers and tp_compress_layers_lse over three layers with a
    long guide equal single-layer calls bit for bit, and the oracle."""
    from paper_2608_03276_gb300 import binding
    import torch
    w = LONG["g4-lt275-m1100-ragged"]
    xs = _stack(w, 3)
    p = _problem(binding, w, xs[0].doc_offsets)
    dev = [tuple(parity.to_device_bf16(t) for t in (x.q, x.k, x.v)) for x in xs]
    outs = [binding.CompressOutputs(p, w.keep_ratio, w.budget, "cuda") for _ in xs]
    binding.tp_compress_layers(p, dev, w.keep_ratio, w.budget, outs, outs[0].ws)
    assert binding.tp_check_status(outs[0].ws) == 0
    for l, x in enumerate(xs):
        single = binding.CompressOutputs(p, w.keep_ratio, w.budget, "cuda")
        binding.compress(p, *dev[l], w.keep_ratio, w.budget, single)
        _outputs_equal(outs[l], single, f"layer {l}")
        _check_layer(w, x, single, _oracle(w, x))
    lses = [torch.tensor(_context_lse(w, x), device="cuda") for x in xs]
    outs = [binding.CompressOutputs(p, w.keep_ratio, w.budget, "cuda") for _ in xs]
    binding.tp_compress_layers_lse(p, dev, lses, w.keep_ratio, w.budget, outs, outs[0].ws)
    assert binding.tp_check_status(outs[0].ws) == 0
    for l, x in enumerate(xs):
        single = binding.CompressOutputs(p, w.keep_ratio, w.budget, "cuda")
        binding.compress(p, *dev[l], w.keep_ratio, w.budget, single, lse=lses[l])
        _outputs_equal(outs[l], single, f"lse layer {l}")
        _check_layer(w, x, single, _oracle(w, x, lse=lses[l].cpu().numpy().astype(np.float64)))
