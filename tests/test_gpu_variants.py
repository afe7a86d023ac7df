"""Scoring variants through the C ABI, against the oracle.

- The aggregation ablation's blends (Sec. 4.4): normalised add and harmonic
  mean (TP_SCORE_NORM_ADD, TP_SCORE_HARMONIC), through the fused layer and
  through tp_guide_scores.
- Single-pass scoring with the caller's row normalisers
  (tp_compress_layer_lse): with the context-only normaliser it must reproduce
  the two-pass result; with a normaliser that also counts extra guide-prefix
  mass per row (the literal prefill normaliser of Sec. 3.2) it must follow
  the oracle given the same normalisers.
"""
import math

import numpy as np
import pytest

from oracle import taskpress_oracle as O
from paper_2608_03276_gb300 import synth
from tests import parity
from tests.test_gpu_parity import SMALL, _check_layer, _oracle, _problem, _run_compress

pytestmark = pytest.mark.gpu

BLENDS = {"normadd": "TP_SCORE_NORM_ADD", "harmonic": "TP_SCORE_HARMONIC"}


@pytest.mark.parametrize("mode", sorted(BLENDS))
@pytest.mark.parametrize("name", ["c1-tiny-2k", "c2-llama-4133", "c5-ragged"])
def test_blend_fused_layer(cuda_lib, name, mode):
    from paper_2608_03276_gb300 import binding
    w = SMALL[name]
    x = synth.make_layer(w)
    out = _run_compress(binding, w, x, flags=getattr(binding, BLENDS[mode]))
    ref = _oracle(w, x, combine_mode=mode)
    _check_layer(w, x, out, ref)


@pytest.mark.parametrize("mode", sorted(BLENDS))
def test_blend_guide_scores(cuda_lib, mode):
    import torch
    from paper_2608_03276_gb300 import binding
    w = SMALL["c4-gqa7-3001"]
    x = synth.make_layer(w)
    ref = _oracle(w, x, combine_mode=mode)
    p = _problem(binding, w, x.doc_offsets, flags=getattr(binding, BLENDS[mode]))
    s = torch.empty((w.n_heads_kv, p.n_total), dtype=torch.float32, device="cuda")
    ws = torch.empty(binding.tp_workspace_bytes(p), dtype=torch.uint8, device="cuda")
    binding.tp_guide_scores(p, parity.to_device_bf16(x.q), parity.to_device_bf16(x.k),
                            torch.tensor(ref["gamma"], device="cuda"), s, ws)
    sc = s.cpu().numpy()
    for b in range(len(x.doc_offsets) - 1):
        lo, hi = x.doc_offsets[b], x.doc_offsets[b + 1]
        for h in range(w.n_heads_kv):
            parity.assert_scores_close(sc[h, lo:hi], ref["scores"][(b, h)], f"{mode} {b},{h}")


def _context_lse(w, x):
    """Each guide row's context-only normaliser [batch, H_kv, G*L_t], fp32."""
    q, k = O.decode_bf16(x.q), O.decode_bf16(x.k)
    g = w.n_heads_q // w.n_heads_kv
    sigma = 1.0 / math.sqrt(w.head_dim)
    offs = x.doc_offsets
    out = np.zeros((len(offs) - 1, w.n_heads_kv, g * w.guide_len), np.float32)
    for b in range(len(offs) - 1):
        lo, hi = int(offs[b]), int(offs[b + 1])
        if hi == lo:
            continue
        for h in range(w.n_heads_kv):
            rows = q[b, h * g:(h + 1) * g].reshape(g * w.guide_len, w.head_dim)
            out[b, h] = O.guide_lse(rows, k[h, lo:hi], sigma)
    return out


def _run_lse(binding, w, x, lse):
    import torch
    p = _problem(binding, w, x.doc_offsets)
    out = binding.CompressOutputs(p, w.keep_ratio, w.budget, "cuda")
    binding.compress(p, parity.to_device_bf16(x.q), parity.to_device_bf16(x.k),
                     parity.to_device_bf16(x.v), w.keep_ratio, w.budget, out,
                     lse=torch.tensor(lse, device="cuda"))
    assert binding.tp_check_status(out.ws) == 0
    return out


@pytest.mark.parametrize("name", ["c2-llama-4133", "c3-guide128-2053", "c5-ragged"])
def test_caller_lse_context_normaliser(cuda_lib, name):
    """The context-only normaliser supplied by the caller reproduces the
    two-pass layer (the oracle's default)."""
    from paper_2608_03276_gb300 import binding
    w = SMALL[name]
    x = synth.make_layer(w)
    lse = _context_lse(w, x)
    out = _run_lse(binding, w, x, lse)
    ref = _oracle(w, x, lse=lse.astype(np.float64))
    _check_layer(w, x, out, ref)
    ref2 = _oracle(w, x)
    for key in ref2["scores"]:
        parity.assert_scores_close(ref["scores"][key], ref2["scores"][key], f"oracle {key}")


@pytest.mark.parametrize("name", ["c2-llama-4133", "c4-gqa7-3001"])
def test_caller_lse_literal_normaliser(cuda_lib, name):
    """A normaliser that also counts guide-prefix mass (different per row, up
    to e^3 times the context mass) changes the scores and the kept sets; the
    GPU follows the oracle given the same normalisers."""
    from paper_2608_03276_gb300 import binding
    w = SMALL[name]
    x = synth.make_layer(w)
    lse_ctx = _context_lse(w, x)
    rng = np.random.Generator(np.random.PCG64(9))
    extra = rng.uniform(-2.0, 3.0, lse_ctx.shape)  # log of the prefix mass relative to the context
    lse = np.logaddexp(lse_ctx.astype(np.float64), lse_ctx + extra).astype(np.float32)
    out = _run_lse(binding, w, x, lse)
    ref = _oracle(w, x, lse=lse.astype(np.float64))
    _check_layer(w, x, out, ref)


# ---------------------------------------------------------------------------
# The literal normaliser: guide prefix folded in (tp_guide_prefix_lse,
# tp_compress_layer_guide)
# ---------------------------------------------------------------------------
def _literal_lse(w, x, kg_bits):
    q, k, kg = O.decode_bf16(x.q), O.decode_bf16(x.k), O.decode_bf16(kg_bits)
    g = w.n_heads_q // w.n_heads_kv
    sigma = 1.0 / math.sqrt(w.head_dim)
    offs = x.doc_offsets
    out = np.zeros((len(offs) - 1, w.n_heads_kv, g * w.guide_len))
    for b in range(len(offs) - 1):
        lo, hi = int(offs[b]), int(offs[b + 1])
        for h in range(w.n_heads_kv):
            out[b, h] = O.guide_lse_literal(q[b, h * g:(h + 1) * g], k[h, lo:hi], kg[b, h], sigma)
    return out


PREFIX_CASES = {
    "c1-tiny-2k": SMALL["c1-tiny-2k"],
    "c4-gqa7-3001": SMALL["c4-gqa7-3001"],
    "ragged-empty": synth.small_variant(synth.WORKLOADS[5], [300, 0, 7, 129, 1]).with_(budget=50),
    "guide-129": synth.small_variant(synth.WORKLOADS[2], [515]).with_(guide_len=129, n_heads_q=18,
                                                                      n_heads_kv=6),
}


@pytest.mark.parametrize("name", sorted(PREFIX_CASES))
def test_guide_prefix_fold(cuda_lib, name):
    """The fold alone, fed the oracle's context normalisers (fp32): each row
    must equal the oracle's literal normaliser to fp32 accuracy.  Short
    documents make one dropped or extra guide term visible (> 1e-2)."""
    import torch
    from paper_2608_03276_gb300 import binding
    w = PREFIX_CASES[name]
    x = synth.make_layer(w)
    kg = synth.make_guide_keys(w)
    p = _problem(binding, w, x.doc_offsets)
    lse = torch.tensor(_context_lse(w, x), device="cuda")
    binding.tp_guide_prefix_lse(p, parity.to_device_bf16(x.q), parity.to_device_bf16(kg), lse)
    got = lse.cpu().numpy().astype(np.float64)
    want = _literal_lse(w, x, kg)
    err = np.abs(got - want) / np.maximum(1.0, np.abs(want))
    assert err.max() <= 2e-5, f"max err {err.max():.3g} at {np.unravel_index(err.argmax(), err.shape)}"


@pytest.mark.parametrize("name", ["c2-llama-4133", "c4-gqa7-3001", "c5-ragged"])
def test_literal_normaliser_layer(cuda_lib, name):
    """tp_compress_layer_guide (pass 1, the prefix fold, pass 2, selection,
    compaction) against the oracle with the guide keys."""
    from paper_2608_03276_gb300 import binding
    w = SMALL[name]
    x = synth.make_layer(w)
    kg = synth.make_guide_keys(w)
    p = _problem(binding, w, x.doc_offsets)
    out = binding.CompressOutputs(p, w.keep_ratio, w.budget, "cuda")
    binding.compress(p, parity.to_device_bf16(x.q), parity.to_device_bf16(x.k),
                     parity.to_device_bf16(x.v), w.keep_ratio, w.budget, out,
                     k_guide=parity.to_device_bf16(kg))
    assert binding.tp_check_status(out.ws) == 0
    ref = _oracle(w, x, k_guide_bits=kg)
    _check_layer(w, x, out, ref)


# ---------------------------------------------------------------------------
# b = 4: scales absmax / 7, codes two per byte (Sec. 4 "Quantization")
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("name", ["c1-tiny-2k", "c2-llama-4133", "c5-ragged"])
def test_int4_fused_layer(cuda_lib, name):
    """The fused layer at b = 4: pass 1 forms gamma = absmax / 7, the scores use
    it (Eq. 3), and the compacted codes are packed two per byte."""
    from paper_2608_03276_gb300 import binding
    w = SMALL[name]
    x = synth.make_layer(w)
    out = _run_compress(binding, w, x, quant_bits=4)
    ref = _oracle(w, x, quant_bits=4)
    _check_layer(w, x, out, ref, bits=4)
    assert out.vqc.dtype.itemsize == 1 and out.vqc.shape[-1] == w.head_dim // 2


@pytest.mark.parametrize("name", ["c4-gqa7-3001", "c3-guide128-2053"])
def test_int4_caller_lse_layer(cuda_lib, name):
    """b = 4 through tp_compress_layer_lse, whose scales come from the key-score
    kernel's V warps: one CTA per key range at 224 guide rows, CTA pairs at 512."""
    from paper_2608_03276_gb300 import binding
    w = SMALL[name]
    x = synth.make_layer(w)
    lse = _context_lse(w, x)
    import torch
    p = _problem(binding, w, x.doc_offsets, quant_bits=4)
    out = binding.CompressOutputs(p, w.keep_ratio, w.budget, "cuda")
    binding.compress(p, parity.to_device_bf16(x.q), parity.to_device_bf16(x.k),
                     parity.to_device_bf16(x.v), w.keep_ratio, w.budget, out,
                     lse=torch.tensor(lse, device="cuda"))
    assert binding.tp_check_status(out.ws) == 0
    ref = _oracle(w, x, quant_bits=4, lse=lse.astype(np.float64))
    _check_layer(w, x, out, ref, bits=4)


@pytest.mark.parametrize("name", ["c1-tiny-2k", "c3-guide128-2053"])
def test_int4_quantize_v(cuda_lib, name):
    import torch
    from paper_2608_03276_gb300 import binding
    w = SMALL[name]
    x = synth.make_layer(w)
    p = _problem(binding, w, x.doc_offsets, quant_bits=4)
    vq = torch.empty((w.n_heads_kv, p.n_total, w.head_dim // 2), dtype=torch.uint8, device="cuda")
    g = torch.empty((w.n_heads_kv, p.n_total), dtype=torch.float32, device="cuda")
    binding.tp_quantize_v(p, parity.to_device_bf16(x.v), vq, g)
    rg, rq = O.quantize_v(x.v, 4)
    assert np.array_equal(g.cpu().numpy().view(np.uint32), rg.view(np.uint32))
    assert np.array_equal(vq.cpu().numpy(), O.pack_codes(rq, 4))


# ---------------------------------------------------------------------------
# A stack of layers in one call (tp_compress_layers) and CUDA-graph capture
# ---------------------------------------------------------------------------
def _stack(w, nl):
    return [synth.make_layer(w, l) for l in range(nl)]


def _outputs_equal(a, b, tag):
    import torch
    for name in ("idx", "kc", "vc", "vqc", "gammac"):
        assert torch.equal(getattr(a, name), getattr(b, name)), f"{tag}: {name}"


@pytest.mark.parametrize("name,bits", [("c2-llama-4133", 8), ("c5-ragged", 8), ("c1-tiny-2k", 4)])
def test_layer_stack_matches_single_layers(cuda_lib, name, bits):
    """tp_compress_layers over three layers (one workspace reset, each layer's
    pass 1 a dependent of the previous layer's last kernel) equals three
    tp_compress_layer calls bit for bit, and the oracle on every layer."""
    from paper_2608_03276_gb300 import binding
    w = SMALL[name]
    xs = _stack(w, 3)
    p = _problem(binding, w, xs[0].doc_offsets, quant_bits=bits)
    dev = [tuple(parity.to_device_bf16(t) for t in (x.q, x.k, x.v)) for x in xs]
    outs = [binding.CompressOutputs(p, w.keep_ratio, w.budget, "cuda") for _ in xs]
    binding.tp_compress_layers(p, dev, w.keep_ratio, w.budget, outs, outs[0].ws)
    assert binding.tp_check_status(outs[0].ws) == 0
    for l, x in enumerate(xs):
        single = binding.CompressOutputs(p, w.keep_ratio, w.budget, "cuda")
        binding.compress(p, *dev[l], w.keep_ratio, w.budget, single)
        _outputs_equal(outs[l], single, f"layer {l}")
        _check_layer(w, x, single, _oracle(w, x, quant_bits=bits), bits=bits)


@pytest.mark.parametrize("name,bits,nl", [("c2-llama-4133", 8, 4), ("c5-ragged", 8, 3),
                                          ("c1-tiny-2k", 4, 3), ("c3-guide128-2053", 8, 3)])
def test_lse_stack_matches_single_layers(cuda_lib, name, bits, nl):
    """tp_compress_layers_lse (each layer's scoring kernel loading and scoring
    while the previous layer's compaction finishes, then waiting for it before
    its first store; one scale and one key-score buffer; CTA pairs at 512 guide
    rows) equals one tp_compress_layer_lse call per layer bit for bit, and the
    oracle given the same normalisers on every layer.  The normalisers carry
    extra per-row mass, as a prefill's would."""
    import torch
    from paper_2608_03276_gb300 import binding
    w = SMALL[name]
    xs = _stack(w, nl)
    p = _problem(binding, w, xs[0].doc_offsets, quant_bits=bits)
    dev = [tuple(parity.to_device_bf16(t) for t in (x.q, x.k, x.v)) for x in xs]
    rng = np.random.Generator(np.random.PCG64(31))
    lses = []
    for x in xs:
        ctx = _context_lse(w, x)
        lses.append(np.logaddexp(ctx.astype(np.float64),
                                 ctx + rng.uniform(-2.0, 2.0, ctx.shape)).astype(np.float32))
    dl = [torch.tensor(t, device="cuda") for t in lses]
    outs = [binding.CompressOutputs(p, w.keep_ratio, w.budget, "cuda") for _ in xs]
    binding.tp_compress_layers_lse(p, dev, dl, w.keep_ratio, w.budget, outs, outs[0].ws)
    assert binding.tp_check_status(outs[0].ws) == 0
    for l, x in enumerate(xs):
        single = binding.CompressOutputs(p, w.keep_ratio, w.budget, "cuda")
        binding.compress(p, *dev[l], w.keep_ratio, w.budget, single, lse=dl[l])
        _outputs_equal(outs[l], single, f"layer {l}")
        _check_layer(w, x, single, _oracle(w, x, quant_bits=bits, lse=lses[l].astype(np.float64)),
                     bits=bits)


GROUPED = [("c2-llama-4133", None, 6, 4), ("c1-tiny-2k", "harmonic", 9, 8),
           ("c2-llama-4133", "key_only", 3, 3), ("c2-llama-4133", "normadd", 3, 1),
           ("c5-ragged", None, 3, 1)]


@pytest.mark.parametrize("name,mode,nl,group", GROUPED)
def test_stack_grouped_selection(cuda_lib, name, mode, nl, group):
    """With a tp_workspace_bytes_stack workspace the stacks select several
    layers per launch (four-CTA clusters, all resident): 8 units per layer on
    a 152-SM GB300 give groups of 4, 2 units groups of 8 (the last group of
    one layer), the ragged batch's 40 units no grouping, the normalised-add
    score none.  Both stacks equal one call per layer bit for bit, and the
    oracle on every layer."""
    import torch
    from paper_2608_03276_gb300 import binding
    w = SMALL[name]
    flags = {None: 0, "harmonic": binding.TP_SCORE_HARMONIC, "normadd": binding.TP_SCORE_NORM_ADD,
             "key_only": binding.TP_SCORE_KEY_ONLY}[mode]
    xs = _stack(w, nl)
    p = _problem(binding, w, xs[0].doc_offsets, flags=flags)
    ws = torch.empty(binding.tp_workspace_bytes_stack(p, w.keep_ratio, w.budget, nl), dtype=torch.uint8,
                     device="cuda")
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    got = binding.tp_stack_layers_per_selection(p, w.keep_ratio, w.budget, nl, ws.numel())
    if sms == 152:
        assert got == group, (got, group)
    dev = [tuple(parity.to_device_bf16(t) for t in (x.q, x.k, x.v)) for x in xs]
    lses = [torch.tensor(_context_lse(w, x), device="cuda") for x in xs]
    for caller_lse in (False, True):
        outs = [binding.CompressOutputs(p, w.keep_ratio, w.budget, "cuda") for _ in xs]
        if caller_lse:
            binding.tp_compress_layers_lse(p, dev, lses, w.keep_ratio, w.budget, outs, ws)
        else:
            binding.tp_compress_layers(p, dev, w.keep_ratio, w.budget, outs, ws)
        assert binding.tp_check_status(ws) == 0
        for l, x in enumerate(xs):
            single = binding.CompressOutputs(p, w.keep_ratio, w.budget, "cuda")
            binding.compress(p, *dev[l], w.keep_ratio, w.budget, single,
                             lse=lses[l] if caller_lse else None)
            _outputs_equal(outs[l], single, f"layer {l} (caller lse {caller_lse})")
            if not caller_lse:
                ref = _oracle(w, x, combine_mode=mode) if mode in BLENDS else \
                    _oracle(w, x, key_only=mode == "key_only")
                _check_layer(w, x, single, ref, key_only=mode == "key_only")


def test_full_size_lse_stack(cuda_lib):
    """Three 128K layers through tp_compress_layers_lse, the benchmark's
    caller-normaliser leg: each equals a single tp_compress_layer_lse call bit
    for bit, and every KV head of the last layer matches the oracle."""
    import torch
    from paper_2608_03276_gb300 import binding
    from tests import oracle_pool
    w = synth.WORKLOADS[3]
    xs = [synth.make_layer(w, l) for l in (0, 1, 2)]
    p = _problem(binding, w, xs[0].doc_offsets)
    dev = [tuple(parity.to_device_bf16(t) for t in (y.q, y.k, y.v)) for y in xs]
    ws = torch.empty(binding.tp_workspace_bytes(p), dtype=torch.uint8, device="cuda")
    dl = []
    for q, k, _ in dev:
        t = torch.empty((w.batch, w.n_heads_kv, w.rows), dtype=torch.float32, device="cuda")
        binding.tp_guide_lse(p, q, k, t, ws)
        dl.append(t)
    outs = [binding.CompressOutputs(p, w.keep_ratio, w.budget, "cuda") for _ in xs]
    binding.tp_compress_layers_lse(p, dev, dl, w.keep_ratio, w.budget, outs, outs[0].ws)
    assert binding.tp_check_status(outs[0].ws) == 0
    for l in range(3):
        single = binding.CompressOutputs(p, w.keep_ratio, w.budget, "cuda")
        binding.compress(p, *dev[l], w.keep_ratio, w.budget, single, lse=dl[l])
        _outputs_equal(outs[l], single, f"lse stack layer {l}")
    x = xs[2]
    ref = oracle_pool.compress_layer(x, w.n_heads_q, w.n_heads_kv, keep_ratio=w.keep_ratio,
                                     lse=dl[2].cpu().numpy().astype(np.float64))
    _check_layer(w, x, single, ref)


def test_layer_stack_graph_replay(cuda_lib):
    """The stack captured into a CUDA graph (its memset and dependent launches
    become graph nodes) and replayed on new contents of the same input
    buffers gives the eager results."""
    import torch
    from paper_2608_03276_gb300 import binding
    w = SMALL["c3-guide128-2053"]
    xs = _stack(w, 4)
    p = _problem(binding, w, xs[0].doc_offsets)
    bufs = [tuple(parity.to_device_bf16(t) for t in (x.q, x.k, x.v)) for x in xs]
    outs = [binding.CompressOutputs(p, w.keep_ratio, w.budget, "cuda", with_scores=False) for _ in xs]
    for o in outs[1:]:
        o.ws = outs[0].ws
    binding.tp_compress_layers(p, bufs, w.keep_ratio, w.budget, outs, outs[0].ws)  # eager warm-up
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        binding.tp_compress_layers(p, bufs, w.keep_ratio, w.budget, outs, outs[0].ws)
    # new contents: the layers in reverse order
    src = [tuple(parity.to_device_bf16(t) for t in (x.q, x.k, x.v)) for x in reversed(xs)]
    for dst, s_ in zip(bufs, src):
        for a, b in zip(dst, s_):
            a.copy_(b)
    g.replay()
    torch.cuda.synchronize()
    assert binding.tp_check_status(outs[0].ws) == 0
    for l in range(len(xs)):
        eager = binding.CompressOutputs(p, w.keep_ratio, w.budget, "cuda")
        binding.compress(p, *src[l], w.keep_ratio, w.budget, eager)
        _outputs_equal(outs[l], eager, f"replayed layer {l}")


# ---------------------------------------------------------------------------
# Edge shapes for the variants: empty and one-token documents, a 7-token one
# ---------------------------------------------------------------------------
EDGE = PREFIX_CASES["ragged-empty"]


@pytest.mark.parametrize("variant", ["normadd", "harmonic", "literal", "int4", "stack"])
def test_variants_on_ragged_edges(cuda_lib, variant):
    from paper_2608_03276_gb300 import binding
    w, x = EDGE, synth.make_layer(EDGE)
    if variant in BLENDS:
        out = _run_compress(binding, w, x, flags=getattr(binding, BLENDS[variant]))
        _check_layer(w, x, out, _oracle(w, x, combine_mode=variant))
    elif variant == "literal":
        kg = synth.make_guide_keys(w)
        p = _problem(binding, w, x.doc_offsets)
        out = binding.CompressOutputs(p, w.keep_ratio, w.budget, "cuda")
        binding.compress(p, parity.to_device_bf16(x.q), parity.to_device_bf16(x.k),
                         parity.to_device_bf16(x.v), w.keep_ratio, w.budget, out,
                         k_guide=parity.to_device_bf16(kg))
        assert binding.tp_check_status(out.ws) == 0
        _check_layer(w, x, out, _oracle(w, x, k_guide_bits=kg))
    elif variant == "int4":
        out = _run_compress(binding, w, x, quant_bits=4)
        _check_layer(w, x, out, _oracle(w, x, quant_bits=4), bits=4)
    else:
        xs = _stack(w, 2)
        p = _problem(binding, w, x.doc_offsets)
        dev = [tuple(parity.to_device_bf16(t) for t in (y.q, y.k, y.v)) for y in xs]
        outs = [binding.CompressOutputs(p, w.keep_ratio, w.budget, "cuda") for _ in xs]
        binding.tp_compress_layers(p, dev, w.keep_ratio, w.budget, outs, outs[0].ws)
        assert binding.tp_check_status(outs[0].ws) == 0
        for l in range(2):
            single = binding.CompressOutputs(p, w.keep_ratio, w.budget, "cuda")
            binding.compress(p, *dev[l], w.keep_ratio, w.budget, single)
            _outputs_equal(outs[l], single, f"layer {l}")


def test_full_size_stack(cuda_lib):
    """Layers 0, 15 and 31 of the 128K Llama-8B-shaped stack through
    tp_compress_layers, the benchmark's call: every layer equals a
    single-layer call bit for bit, and every KV head of every layer matches the
    oracle."""
    from paper_2608_03276_gb300 import binding
    from tests import oracle_pool
    w = synth.WORKLOADS[3]
    xs = [synth.make_layer(w, l) for l in (0, 15, 31)]
    p = _problem(binding, w, xs[0].doc_offsets)
    dev = [tuple(parity.to_device_bf16(t) for t in (y.q, y.k, y.v)) for y in xs]
    outs = [binding.CompressOutputs(p, w.keep_ratio, w.budget, "cuda") for _ in xs]
    binding.tp_compress_layers(p, dev, w.keep_ratio, w.budget, outs, outs[0].ws)
    assert binding.tp_check_status(outs[0].ws) == 0
    for l, x in enumerate(xs):
        single = binding.CompressOutputs(p, w.keep_ratio, w.budget, "cuda")
        binding.compress(p, *dev[l], w.keep_ratio, w.budget, single)
        _outputs_equal(outs[l], single, f"stack layer {l}")
        _check_layer(w, x, single, oracle_pool.compress_layer(x, w.n_heads_q, w.n_heads_kv,
                                                               keep_ratio=w.keep_ratio))


@pytest.mark.parametrize("bits", [4, 8])
def test_fully_quantised_cache(cuda_lib, bits):
    """The compacted K quantised by tp_quantize_rows (K and V both in b bits,
    as the paper's experiments store the cache): scales and codes equal the
    oracle's Eq. 2 on the kept K rows, and unused slots (zero rows) get zero
    scales and codes."""
    import torch
    from paper_2608_03276_gb300 import binding
    w = SMALL["c5-ragged"]
    x = synth.make_layer(w)
    out = _run_compress(binding, w, x, quant_bits=bits)
    shp = tuple(out.kc.shape[:-1])
    kq = torch.empty(shp + (w.head_dim * bits // 8,), dtype=binding.code_dtype(
        _problem(binding, w, x.doc_offsets, quant_bits=bits)), device="cuda")
    ks = torch.empty(shp, dtype=torch.float32, device="cuda")
    binding.tp_quantize_rows(out.kc, bits, kq, ks)
    torch.cuda.synchronize()
    rg, rq = O.quantize_v(parity.bf16_bits(out.kc), bits)
    assert np.array_equal(ks.cpu().numpy().view(np.uint32), rg.view(np.uint32))
    assert np.array_equal(kq.cpu().numpy(), O.pack_codes(rq, bits))
    idx = out.idx.cpu().numpy()
    assert not ks.cpu().numpy()[idx < 0].any()


@pytest.mark.parametrize("variant", ["caller_lse", "literal", "int4"])
def test_full_size_variants(cuda_lib, variant):
    """One 128K layer of the Llama-8B-shaped workload (8 KV heads, guide 128 x
    GQA 4) through each variant path in the benchmark's configuration; every
    KV head against the oracle."""
    import torch
    from paper_2608_03276_gb300 import binding
    from tests import oracle_pool
    w = synth.WORKLOADS[3]
    x = synth.make_layer(w)
    dev = tuple(parity.to_device_bf16(t) for t in (x.q, x.k, x.v))
    if variant == "int4":
        out = _run_compress(binding, w, x, quant_bits=4)
        ref = oracle_pool.compress_layer(x, w.n_heads_q, w.n_heads_kv, keep_ratio=w.keep_ratio,
                                         quant_bits=4)
        _check_layer(w, x, out, ref, bits=4)
        return
    p = _problem(binding, w, x.doc_offsets)
    out = binding.CompressOutputs(p, w.keep_ratio, w.budget, "cuda")
    if variant == "caller_lse":
        lse = torch.empty((w.batch, w.n_heads_kv, w.rows), dtype=torch.float32, device="cuda")
        ws = torch.empty(binding.tp_workspace_bytes(p), dtype=torch.uint8, device="cuda")
        binding.tp_guide_lse(p, dev[0], dev[1], lse, ws)
        binding.compress(p, *dev, w.keep_ratio, w.budget, out, lse=lse)
        ref = oracle_pool.compress_layer(x, w.n_heads_q, w.n_heads_kv, keep_ratio=w.keep_ratio,
                                         lse=lse.cpu().numpy().astype(np.float64))
    else:
        kg = synth.make_guide_keys(w)
        binding.compress(p, *dev, w.keep_ratio, w.budget, out, k_guide=parity.to_device_bf16(kg))
        ref = oracle_pool.compress_layer(x, w.n_heads_q, w.n_heads_kv, keep_ratio=w.keep_ratio,
                                         k_guide_bits=kg)
    assert binding.tp_check_status(out.ws) == 0
    _check_layer(w, x, out, ref)


# With the caller's normalisers, more than 256 guide rows take the key scores
# and the V scales from one kernel on CTA pairs (256-key pair tiles, so a
# document's last pair tile may be half or wholly past its end), and fall back
# to the quantiser and pass 2 when the pairs would not all be resident at once
# (here 10 documents x 8 KV heads > 76 pairs).
PAIR_WORKLOADS = {
    "pair-ragged-m512": synth.small_variant(synth.WORKLOADS[3], [1000, 300, 5000]),
    "fallback-m512-80-units": synth.small_variant(synth.WORKLOADS[3], [200] * 10),
}


@pytest.mark.parametrize("name", sorted(PAIR_WORKLOADS))
def test_caller_lse_pairs_and_fallback(cuda_lib, name):
    from paper_2608_03276_gb300 import binding
    w = PAIR_WORKLOADS[name]
    x = synth.make_layer(w)
    p = _problem(binding, w, x.doc_offsets)
    kernels = binding.tp_compress_kernel_count(p, w.keep_ratio, w.budget, binding.MODE_CALLER_LSE)
    assert kernels == (4 if name.startswith("fallback") else 3), kernels
    lse = _context_lse(w, x)
    out = _run_lse(binding, w, x, lse)
    ref = _oracle(w, x, lse=lse.astype(np.float64))
    _check_layer(w, x, out, ref)


@pytest.mark.parametrize("n", [70000, 131072])
@pytest.mark.parametrize("mode", sorted(BLENDS))
def test_blend_long_document(cuda_lib, mode, n):
    """The blends on a long document (two KV heads): the selection runs on
    twelve-CTA clusters for documents of 64K tokens or more, and at 131072
    tokens (10924 per CTA) compacts in one round of 22 tokens per thread."""
    from paper_2608_03276_gb300 import binding
    w = synth.small_variant(synth.WORKLOADS[1], [n])
    x = synth.make_layer(w)
    out = _run_compress(binding, w, x, flags=getattr(binding, BLENDS[mode]))
    ref = _oracle(w, x, combine_mode=mode)
    _check_layer(w, x, out, ref)


def test_lse_stack_graph_replay(cuda_lib):
    """The caller-normaliser stack on CTA pairs (512 guide rows: cluster launches,
    dependent launches) captured into a CUDA graph and replayed on new contents
    of the same buffers gives the eager results."""
    import torch
    from paper_2608_03276_gb300 import binding
    w = SMALL["c3-guide128-2053"]
    xs = _stack(w, 3)
    p = _problem(binding, w, xs[0].doc_offsets)
    bufs = [tuple(parity.to_device_bf16(t) for t in (x.q, x.k, x.v)) for x in xs]
    lses = [torch.tensor(_context_lse(w, x), device="cuda") for x in xs]
    outs = [binding.CompressOutputs(p, w.keep_ratio, w.budget, "cuda", with_scores=False) for _ in xs]
    for o in outs[1:]:
        o.ws = outs[0].ws
    binding.tp_compress_layers_lse(p, bufs, lses, w.keep_ratio, w.budget, outs, outs[0].ws)  # eager
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        binding.tp_compress_layers_lse(p, bufs, lses, w.keep_ratio, w.budget, outs, outs[0].ws)
    # new contents: the layers (and their normalisers) in reverse order
    for dst, s_ in zip(bufs, [tuple(parity.to_device_bf16(t) for t in (x.q, x.k, x.v)) for x in reversed(xs)]):
        for a, b in zip(dst, s_):
            a.copy_(b)
    rl = [l.clone() for l in reversed(lses)]
    for dst, s_ in zip(lses, rl):
        dst.copy_(s_)
    g.replay()
    torch.cuda.synchronize()
    assert binding.tp_check_status(outs[0].ws) == 0
    for l, x in enumerate(reversed(xs)):
        single = binding.CompressOutputs(p, w.keep_ratio, w.budget, "cuda")
        binding.compress(p, *bufs[l], w.keep_ratio, w.budget, single, lse=lses[l])
        _outputs_equal(outs[l], single, f"layer {l}")


# Guide blocks of one or two 256-row parts per key tile, whole or not, at both
# head dims.  Each (part count, whole) pair is its own compiled instance of the
# pass-2 kernels: one CTA per key range without the scales (two-pass layer) and
# with them (caller's normalisers), and the CTA-pair kernel (caller's
# normalisers above 256 rows at d 128).  Both paths are checked against the
# oracle for every shape.
PART_SHAPES = {
    # name: (query heads, KV heads, head dim, guide tokens, document lengths)
    "d128-m224": (28, 4, 128, 32, [1100]),      # one part, not whole
    "d128-m320": (10, 2, 128, 64, [700, 300]),  # two parts, the second not whole; CTA pairs
    "d128-m384": (12, 4, 128, 128, [900]),      # two parts, the second not whole; CTA pairs
    "d64-m288": (18, 2, 64, 32, [600, 257]),    # two parts at d 64: one CTA forms the scales
    "d64-m512": (8, 2, 64, 128, [513]),         # two whole parts at d 64
}


@pytest.mark.parametrize("name", sorted(PART_SHAPES))
def test_guide_part_shapes(cuda_lib, name):
    from paper_2608_03276_gb300 import binding
    hq, hkv, d, lt, lens = PART_SHAPES[name]
    w = synth.small_variant(synth.WORKLOADS[2], lens).with_(
        n_heads_q=hq, n_heads_kv=hkv, head_dim=d, guide_len=lt)
    assert w.group * lt == {"d128-m224": 224, "d128-m320": 320, "d128-m384": 384,
                            "d64-m288": 288, "d64-m512": 512}[name]
    x = synth.make_layer(w)
    p = _problem(binding, w, x.doc_offsets)
    # the scales are formed inside the scoring kernel (no separate quantiser)
    assert binding.tp_compress_kernel_count(p, w.keep_ratio, w.budget, binding.MODE_CALLER_LSE) == 3
    out = _run_compress(binding, w, x)
    _check_layer(w, x, out, _oracle(w, x))
    lse = _context_lse(w, x)
    out = _run_lse(binding, w, x, lse)
    _check_layer(w, x, out, _oracle(w, x, lse=lse.astype(np.float64)))
