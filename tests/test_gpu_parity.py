"""CUDA path vs the oracle, element by element, through the C ABI.

Small cases span several key tiles and a ragged tail; full-size cases run the
exact launch configuration the benchmark times and compare sampled heads /
documents that the oracle computes directly.  Tolerances: see tests/parity.py.
"""
import numpy as np
import pytest

from oracle import taskpress_oracle as O
from paper_2608_03276_gb300 import synth
from tests import parity

pytestmark = pytest.mark.gpu

W = synth.WORKLOADS
SMALL = {
    "c1-tiny-2k": W[1],
    "c2-llama-4133": synth.small_variant(W[2], [4133]),
    "c3-guide128-2053": synth.small_variant(W[3], [2053]),
    "c4-gqa7-3001": synth.small_variant(W[4], [3001]),
    "c5-ragged": synth.small_variant(W[5], [1500, 1, 700, 2304, 129]).with_(budget=300),
}


def _problem(binding, w, doc_offsets, **kw):
    return binding.Problem(w.n_heads_q, w.n_heads_kv, w.head_dim, w.guide_len, doc_offsets, **kw)


def _run_compress(binding, w, x, keep_ratio=None, budget=None, **kw):
    keep_ratio = w.keep_ratio if keep_ratio is None else keep_ratio
    budget = w.budget if budget is None else budget
    p = _problem(binding, w, x.doc_offsets, **kw)
    out = binding.CompressOutputs(p, keep_ratio, budget, "cuda")
    binding.compress(p, parity.to_device_bf16(x.q), parity.to_device_bf16(x.k),
                     parity.to_device_bf16(x.v), keep_ratio, budget, out)
    assert binding.tp_check_status(out.ws) == 0
    return out


def _check_layer(w, x, out, ref, heads=None, docs=None, key_only=False, bits=8):
    scores = out.scores.cpu().numpy()
    gamma = out.gamma.cpu().numpy()
    idx = out.idx.cpu().numpy()
    kc, vc = parity.bf16_bits(out.kc), parity.bf16_bits(out.vc)
    vqc, gc = out.vqc.cpu().numpy(), out.gammac.cpu().numpy()
    assert np.array_equal(gamma.view(np.uint32), ref["gamma"].view(np.uint32)), "gamma not bit-exact"
    offs = x.doc_offsets
    for b in (range(len(offs) - 1) if docs is None else docs):
        lo, hi = int(offs[b]), int(offs[b + 1])
        for h in (range(w.n_heads_kv) if heads is None else heads):
            tag = f"doc {b} head {h}"
            parity.assert_scores_close(scores[h, lo:hi], ref["scores"][(b, h)], tag)
            parity.assert_kept(idx[b, h], ref["k"][b], ref["scores"][(b, h)], scores[h, lo:hi], tag)
            k_b = ref["k"][b]
            rk, rv, rq, rg = O.gather_rows(x.k, x.v, ref["gamma"], ref["vq"], lo, h, idx[b, h, :k_b])
            rq = O.pack_codes(rq, bits)
            assert np.array_equal(kc[b, h, :k_b], rk), f"{tag}: Kc"
            assert np.array_equal(vc[b, h, :k_b], rv), f"{tag}: Vc"
            assert np.array_equal(vqc[b, h, :k_b], rq), f"{tag}: Vqc"
            assert np.array_equal(gc[b, h, :k_b], rg), f"{tag}: gammac"
            assert not kc[b, h, k_b:].any() and not vqc[b, h, k_b:].any() and not gc[b, h, k_b:].any()


def _oracle(w, x, keep_ratio=None, budget=None, heads=None, docs=None, **kw):
    return O.compress_layer(x.q, x.k, x.v, x.doc_offsets, n_heads_q=w.n_heads_q,
                            n_heads_kv=w.n_heads_kv,
                            keep_ratio=w.keep_ratio if keep_ratio is None else keep_ratio,
                            fixed_budget=w.budget if budget is None else budget,
                            heads=heads, docs=docs, **kw)


# ---------------------------------------------------------------------------
# Eq. 2 quantiser: bit-exact
# ---------------------------------------------------------------------------
def _special_v_rows(d):
    rows = np.zeros((8, d), np.float32)
    rows[1] = -0.0
    rows[2, :] = 1.0
    rows[2, 3] = np.float32(np.finfo(np.float32).max)  # bf16 rounds to inf? keep < bf16 max
    rows[2, 3] = np.float32(3.3895313892515355e38)    # bf16 max 0x7F7F
    rows[3, :] = np.float32(1e-40)                    # subnormal
    rows[4, :4] = [15.875, 0.3125, 0.4375, -0.3125]
    rows[5] = np.linspace(-3, 3, d)
    rows[6, 0] = -1.0
    rows[7] = 2.0 ** -120
    return (rows.view(np.uint32) >> 16).astype(np.uint16)


@pytest.mark.parametrize("name", ["c1-tiny-2k", "c2-llama-4133"])
def test_quantize_v_bit_exact(cuda_lib, name):
    import torch
    from paper_2608_03276_gb300 import binding
    w = SMALL[name]
    x = synth.make_layer(w)
    v = x.v.copy()
    v[0, :8] = _special_v_rows(w.head_dim)
    p = _problem(binding, w, x.doc_offsets)
    n = x.v.shape[1]
    vq = torch.empty((w.n_heads_kv, n, w.head_dim), dtype=torch.int8, device="cuda")
    g = torch.empty((w.n_heads_kv, n), dtype=torch.float32, device="cuda")
    binding.tp_quantize_v(p, parity.to_device_bf16(v), vq, g)
    rg, rq = O.quantize_v(v)
    assert np.array_equal(g.cpu().numpy().view(np.uint32), rg.view(np.uint32))
    assert np.array_equal(vq.cpu().numpy(), rq)


# ---------------------------------------------------------------------------
# Scores (Eq. 1-3) and the fused layer
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("name", sorted(SMALL))
def test_compress_layer_small(cuda_lib, name):
    from paper_2608_03276_gb300 import binding
    w = SMALL[name]
    x = synth.make_layer(w)
    out = _run_compress(binding, w, x)
    _check_layer(w, x, out, _oracle(w, x))


@pytest.mark.parametrize("name", ["c1-tiny-2k", "c5-ragged"])
def test_guide_scores_entry_point(cuda_lib, name):
    import torch
    from paper_2608_03276_gb300 import binding
    w = SMALL[name]
    x = synth.make_layer(w)
    ref = _oracle(w, x)
    for key_only in (False, True):
        p = _problem(binding, w, x.doc_offsets, flags=binding.TP_SCORE_KEY_ONLY if key_only else 0)
        n = p.n_total
        g = torch.tensor(ref["gamma"], device="cuda")
        s = torch.empty((w.n_heads_kv, n), dtype=torch.float32, device="cuda")
        ws = torch.empty(binding.tp_workspace_bytes(p), dtype=torch.uint8, device="cuda")
        binding.tp_guide_scores(p, parity.to_device_bf16(x.q), parity.to_device_bf16(x.k),
                                None if key_only else g, s, ws)
        sc = s.cpu().numpy()
        for b in range(len(x.doc_offsets) - 1):
            lo, hi = x.doc_offsets[b], x.doc_offsets[b + 1]
            for h in range(w.n_heads_kv):
                want = ref["scores"][(b, h)]
                if key_only:
                    want = O.pool(ref["key"][(b, h)], 5)
                parity.assert_scores_close(sc[h, lo:hi], want, f"key_only={key_only} {b},{h}")


@pytest.mark.parametrize("name", ["c3-guide128-2053", "c5-ragged", "c4-gqa7-3001", "c1-tiny-2k"])
def test_stage_entry_points(cuda_lib, name):
    """tp_guide_lse against the oracle's row normalisers; tp_guide_key_scores fed the
    oracle's normalisers against the oracle's unpooled key scores."""
    import math
    import torch
    from paper_2608_03276_gb300 import binding
    w = SMALL[name]
    x = synth.make_layer(w)
    p = _problem(binding, w, x.doc_offsets)
    q, k = parity.to_device_bf16(x.q), parity.to_device_bf16(x.k)
    rows = w.group * w.guide_len
    lse = torch.empty((w.batch, w.n_heads_kv, rows), dtype=torch.float32, device="cuda")
    ws = torch.empty(binding.tp_workspace_bytes(p), dtype=torch.uint8, device="cuda")
    gam = torch.empty((w.n_heads_kv, p.n_total), dtype=torch.float32, device="cuda")
    binding.tp_guide_lse(p, q, k, lse, ws, v=parity.to_device_bf16(x.v), gamma=gam)
    rg, _ = O.quantize_v(x.v)
    assert np.array_equal(gam.cpu().numpy().view(np.uint32), rg.view(np.uint32)), "fused gamma"
    lse2 = torch.empty_like(lse)
    binding.tp_guide_lse(p, q, k, lse2, ws)
    assert torch.equal(lse, lse2), "lse differs with and without the fused V scales"
    got = lse.cpu().numpy()
    qf, kf = O.decode_bf16(x.q), O.decode_bf16(x.k)
    sigma = 1.0 / math.sqrt(w.head_dim)
    ref_lse = np.zeros((w.batch, w.n_heads_kv, rows), np.float32)
    ref_key = np.zeros((w.n_heads_kv, p.n_total))
    for b in range(w.batch):
        lo, hi = x.doc_offsets[b], x.doc_offsets[b + 1]
        if hi == lo:
            continue
        for h in range(w.n_heads_kv):
            qr = qf[b, h * w.group:(h + 1) * w.group].reshape(rows, -1)
            want = O.guide_lse(qr, kf[h, lo:hi], sigma)
            assert np.abs(got[b, h] - want).max() <= parity.RTOL, (b, h)
            ref_lse[b, h] = want
            ref_key[h, lo:hi] = O.key_scores(qf[b, h * w.group:(h + 1) * w.group], kf[h, lo:hi], sigma)
    skey = torch.empty((w.n_heads_kv, p.n_total), dtype=torch.float32, device="cuda")
    binding.tp_guide_key_scores(p, q, k, torch.tensor(ref_lse, device="cuda"), skey)
    parity.assert_scores_close(skey.cpu().numpy(), ref_key, "key scores from given lse")
    # the same pass forming the Eq. 2 scales too (one CTA per key range up to 256
    # guide rows, CTA pairs above): every scale written, bit-exact, and the key
    # scores unchanged bit for bit
    skey2 = torch.empty_like(skey)
    gam2 = torch.full_like(gam, float("nan"))
    binding.tp_guide_key_scores(p, q, k, torch.tensor(ref_lse, device="cuda"), skey2,
                                v=parity.to_device_bf16(x.v), gamma=gam2)
    assert np.array_equal(gam2.cpu().numpy().view(np.uint32), rg.view(np.uint32)), "gamma of pass 2"
    assert torch.equal(skey, skey2), "key scores differ with and without the fused V scales"


def test_key_only_layer(cuda_lib):
    from paper_2608_03276_gb300 import binding
    w = SMALL["c2-llama-4133"]
    x = synth.make_layer(w)
    out = _run_compress(binding, w, x, flags=binding.TP_SCORE_KEY_ONLY)
    _check_layer(w, x, out, _oracle(w, x, key_only=True))


@pytest.mark.parametrize("pool_kernel", [1, 3, 7])
def test_pool_kernels(cuda_lib, pool_kernel):
    from paper_2608_03276_gb300 import binding
    w = SMALL["c1-tiny-2k"]
    x = synth.make_layer(w)
    out = _run_compress(binding, w, x, pool_kernel=pool_kernel)
    _check_layer(w, x, out, _oracle(w, x, pool_kernel=pool_kernel))


# ---------------------------------------------------------------------------
# Selection and compaction as separate entry points (bit-exact)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("budget", [0, 1, 2, 299, 300, 301, 5000, 9000, 13000])
def test_select_bit_exact(cuda_lib, budget):
    """Documents of 1 to 12,000 tokens (several 4096-token chunks), with tie groups
    that span chunks, zeros and negative zeros."""
    import torch
    from paper_2608_03276_gb300 import binding
    rng = np.random.Generator(np.random.PCG64(budget))
    offs = np.array([0, 300, 301, 1500, 1500, 4000, 16000, 25000])
    hkv = 3
    n = int(offs[-1])
    sc = rng.random((hkv, n)).astype(np.float32)
    sc[0, :300] = 0.5                        # all ties
    sc[1, 1500:1600] = 0.0                   # zeros
    sc[1, 1600:1610] = -0.0
    sc[2, 2000:] = np.round(sc[2, 2000:] * 8) / 8   # heavy ties across chunks
    sc[0, 4000:16000] = np.round(sc[0, 4000:16000] * 3) / 3
    sc[1, 16000:25000] = 0.25
    p = binding.Problem(hkv * 2, hkv, 64, 8, offs)
    cap = binding.tp_kept_capacity(p, 0.0, budget)
    idx = torch.empty((len(offs) - 1, hkv, cap), dtype=torch.int32, device="cuda")
    ws = torch.empty(binding.tp_workspace_bytes(p, 0.0, budget), dtype=torch.uint8, device="cuda")
    binding.tp_select(p, torch.tensor(sc, device="cuda"), 0.0, budget, idx, ws)
    got = idx.cpu().numpy()
    for b in range(len(offs) - 1):
        lo, hi = offs[b], offs[b + 1]
        for h in range(hkv):
            k = min(budget, hi - lo)
            want = O.select_topk(sc[h, lo:hi].astype(np.float64), k)
            assert np.array_equal(got[b, h, :k], want), (b, h)
            assert np.all(got[b, h, k:] == -1)


@pytest.mark.parametrize("budget", [1, 14000, 139999])
def test_select_long_document(cuda_lib, budget):
    """A document longer than the shared-memory key slices of its cluster
    (12 x 16384 tokens: the slices' keys live in the global scratch)."""
    import torch
    from paper_2608_03276_gb300 import binding
    n = 210000
    rng = np.random.Generator(np.random.PCG64(budget + 7))
    sc = np.round(rng.random((1, n)) * 64).astype(np.float32) / 64  # many ties
    p = binding.Problem(2, 1, 128, 4, [0, n])
    idx = torch.empty((1, 1, budget), dtype=torch.int32, device="cuda")
    ws = torch.empty(binding.tp_workspace_bytes(p, 0.0, budget), dtype=torch.uint8, device="cuda")
    binding.tp_select(p, torch.tensor(sc, device="cuda"), 0.0, budget, idx, ws)
    want = O.select_topk(sc[0].astype(np.float64), budget)
    assert np.array_equal(idx.cpu().numpy()[0, 0], want)


@pytest.mark.parametrize("ratio", [0.0, 0.07, 0.5, 1.0])
def test_select_ratio(cuda_lib, ratio):
    import torch
    from paper_2608_03276_gb300 import binding
    offs = np.array([0, 100, 1100, 1101])
    rng = np.random.Generator(np.random.PCG64(3))
    sc = rng.random((2, 1101)).astype(np.float32)
    p = binding.Problem(2, 2, 128, 4, offs)
    cap = binding.tp_kept_capacity(p, ratio, -1)
    idx = torch.empty((3, 2, max(cap, 0)), dtype=torch.int32, device="cuda")
    ws = torch.empty(binding.tp_workspace_bytes(p, ratio, -1), dtype=torch.uint8, device="cuda")
    binding.tp_select(p, torch.tensor(sc, device="cuda"), ratio, -1, idx if cap else None, ws)
    got = idx.cpu().numpy()
    for b in range(3):
        lo, hi = offs[b], offs[b + 1]
        k = O.budget(int(hi - lo), ratio)
        for h in range(2):
            assert np.array_equal(got[b, h, :k], O.select_topk(sc[h, lo:hi].astype(np.float64), k))


def test_compact_bit_exact(cuda_lib):
    import torch
    from paper_2608_03276_gb300 import binding
    w = SMALL["c5-ragged"]
    x = synth.make_layer(w)
    rg, rq = O.quantize_v(x.v)
    p = _problem(binding, w, x.doc_offsets)
    cap = binding.tp_kept_capacity(p, 0.0, 300)
    rng = np.random.Generator(np.random.PCG64(1))
    idx = np.full((w.batch, w.n_heads_kv, cap), -1, np.int32)
    for b in range(w.batch):
        n = int(x.doc_offsets[b + 1] - x.doc_offsets[b])
        for h in range(w.n_heads_kv):
            k = min(300, n)
            idx[b, h, :k] = np.sort(rng.choice(n, k, replace=False))
    d = w.head_dim
    kc = torch.empty((w.batch, w.n_heads_kv, cap, d), dtype=torch.bfloat16, device="cuda")
    vc, vqc = torch.empty_like(kc), torch.empty(kc.shape, dtype=torch.int8, device="cuda")
    gc = torch.empty((w.batch, w.n_heads_kv, cap), dtype=torch.float32, device="cuda")
    binding.tp_compact(p, parity.to_device_bf16(x.k), parity.to_device_bf16(x.v),
                       torch.tensor(rg, device="cuda"), torch.tensor(idx, device="cuda"), 0.0, 300,
                       kc, vc, vqc, gc)
    kcb, vcb = parity.bf16_bits(kc), parity.bf16_bits(vc)
    for b in range(w.batch):
        lo = int(x.doc_offsets[b])
        for h in range(w.n_heads_kv):
            sel = idx[b, h][idx[b, h] >= 0]
            k = sel.size
            rk, rv, rqq, rgg = O.gather_rows(x.k, x.v, rg, rq, lo, h, sel)
            assert np.array_equal(kcb[b, h, :k], rk) and np.array_equal(vcb[b, h, :k], rv)
            assert np.array_equal(vqc[b, h, :k].cpu().numpy(), rqq)
            assert np.array_equal(gc[b, h, :k].cpu().numpy(), rgg)


# ---------------------------------------------------------------------------
# Edge cases: shapes, budgets, degenerate data
# ---------------------------------------------------------------------------
def _edge_workload(hq, hkv, d, lt, lens, **kw):
    base = dict(spans=(2, 4), v_outlier=(0.02, 8.0), seed=77)
    base.update(kw)
    return synth.Workload("edge", hq, hkv, d, lt, tuple(lens), **base)


EDGE = {
    "n1": _edge_workload(4, 1, 64, 4, [1], spans=(0, 0)),
    "n127": _edge_workload(4, 2, 128, 8, [127]),
    "n129": _edge_workload(4, 2, 128, 8, [129]),
    "g1-lt1": _edge_workload(2, 2, 128, 1, [700]),
    "g1-lt129": _edge_workload(1, 1, 128, 129, [600]),
    "g8-lt64": _edge_workload(8, 1, 64, 64, [1000]),
    "g7-lt73-m511": _edge_workload(7, 1, 128, 73, [900]),
    "lt128-g4": _edge_workload(8, 2, 64, 128, [513]),
    "many-docs": _edge_workload(4, 2, 64, 4, [1, 2, 3, 128, 129, 255, 256, 257, 1000, 0, 5]),
}


@pytest.mark.parametrize("name", sorted(EDGE))
@pytest.mark.parametrize("budget", [-1, 0, 1])
def test_edge_shapes(cuda_lib, name, budget):
    from paper_2608_03276_gb300 import binding
    w = EDGE[name]
    x = synth.make_layer(w)
    out = _run_compress(binding, w, x, keep_ratio=0.3, budget=budget)
    _check_layer(w, x, out, _oracle(w, x, keep_ratio=0.3, budget=budget))


@pytest.mark.parametrize("ratio", [0.0, 1.0])
def test_ratio_extremes(cuda_lib, ratio):
    from paper_2608_03276_gb300 import binding
    w = SMALL["c5-ragged"]
    x = synth.make_layer(w)
    out = _run_compress(binding, w, x, keep_ratio=ratio, budget=-1)
    _check_layer(w, x, out, _oracle(w, x, keep_ratio=ratio, budget=-1))


def test_identical_tokens_and_zero_values(cuda_lib):
    from paper_2608_03276_gb300 import binding
    w = _edge_workload(4, 2, 128, 8, [600])
    x = synth.make_layer(w)
    x.k[0] = x.k[0, :1]          # head 0: every key identical -> every score ties
    x.v[0] = x.v[0, :1]
    x.v[1, 100:400] = 0          # head 1: zero values -> gamma 0 -> score 0
    x.v[1, 200:300] = 0x8000     # negative zeros
    out = _run_compress(binding, w, x, keep_ratio=0.25, budget=-1, pool_kernel=1)
    ref = _oracle(w, x, keep_ratio=0.25, budget=-1, pool_kernel=1)
    _check_layer(w, x, out, ref)
    assert list(out.idx[0, 0].cpu().numpy()) == list(range(150))


def test_huge_logits(cuda_lib):
    """Guide rows with large norms: logit ranges far beyond 100 (fp32 underflow region)."""
    from paper_2608_03276_gb300 import binding
    w = _edge_workload(4, 2, 128, 8, [1100])
    x = synth.make_layer(w)
    q = synth.bf16_bits_to_f32(x.q) * 40.0
    x.q = synth.f32_to_bf16_bits(q)
    out = _run_compress(binding, w, x, keep_ratio=0.2, budget=-1)
    _check_layer(w, x, out, _oracle(w, x, keep_ratio=0.2, budget=-1))


def test_repeatable(cuda_lib):
    from paper_2608_03276_gb300 import binding
    w = SMALL["c2-llama-4133"]
    x = synth.make_layer(w)
    a = _run_compress(binding, w, x)
    b = _run_compress(binding, w, x)
    assert np.array_equal(a.scores.cpu().numpy(), b.scores.cpu().numpy())
    assert np.array_equal(a.idx.cpu().numpy(), b.idx.cpu().numpy())


# ---------------------------------------------------------------------------
# Full-size workloads in the benchmark's launch configuration: every KV head
# of every document against the oracle (computed unit by unit in a pool of
# spawned processes, tests/oracle_pool.py)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("cfg,ratios", [
    (2, None),
    (3, None),
    (4, (0.05, 0.10, 0.25, 0.50)),
    (5, None),
])
def test_full_size_all_heads(cuda_lib, cfg, ratios):
    from paper_2608_03276_gb300 import binding
    from tests import oracle_pool
    w = W[cfg]
    x = synth.make_layer(w)
    for r in (ratios or (w.keep_ratio,)):
        out = _run_compress(binding, w, x, keep_ratio=r)
        ref = oracle_pool.compress_layer(x, w.n_heads_q, w.n_heads_kv, keep_ratio=r,
                                         fixed_budget=w.budget)
        _check_layer(w, x, out, ref)
