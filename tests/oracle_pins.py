"""Pins for the CPU oracle: facts fixed by the paper and by mathematics.

Each ``pin_*`` takes an oracle module and raises AssertionError when the
module disagrees with a closed form, an invariant, a special case that reduces
to a textbook routine, a hand-derived fixture, or brute force on tiny inputs.
None of them re-calls the oracle's own formula to produce its expectation.

tests/test_oracle_pins.py runs them against the oracle; tests/
test_oracle_mutations.py plants plausible mistakes in copies of the oracle and
checks that every mistake trips at least one pin.
"""
from __future__ import annotations

import itertools
import math
import os
from fractions import Fraction

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def exact_bf16(x) -> np.ndarray:
    """bf16 bits of values that bf16 represents exactly (asserts exactness)."""
    f = np.ascontiguousarray(np.asarray(x, dtype=np.float32))
    u = f.view(np.uint32)
    assert np.all((u & 0xFFFF) == 0), "value not exactly representable in bf16"
    return (u >> 16).astype(np.uint16)


def _rand(seed, shape):
    return np.random.Generator(np.random.PCG64(seed)).standard_normal(shape)


# -- Sec. 3.2: softmax over the context --------------------------------------

def pin_softmax_rows_sum_to_one(O):
    """Every guide row of A is a probability distribution over the context."""
    for seed, (m, n, d) in enumerate([(3, 17, 8), (8, 200, 16), (1, 1, 4)]):
        q, k = _rand(seed, (m, d)) * 3, _rand(seed + 100, (n, d)) * 3
        a = O.guide_attention(q, k, 1.0 / math.sqrt(d))
        assert a.shape == (m, n)
        assert np.all(a >= 0)
        assert np.allclose(a.sum(axis=1), 1.0, rtol=0, atol=1e-12)


def pin_two_key_logistic(O):
    """Two keys +-e1 and q = a*e1: A[0] is the logistic function of 2*a*sigma.

    Pins the scale 1/sqrt(d), the sign of the logits and overflow safety.
    """
    for d in (4, 16, 64):
        sigma = 1.0 / math.sqrt(d)
        k = np.zeros((2, d))
        k[0, 0], k[1, 0] = 1.0, -1.0
        for a in (0.0, 0.5, -1.25, 3.0, 40.0, 4000.0):
            q = np.zeros((1, d))
            q[0, 0] = a
            got = O.guide_attention(q, k, sigma)[0]
            t = 2.0 * a * sigma
            p0 = 1.0 / (1.0 + math.exp(-t)) if t >= 0 else math.exp(t) / (1.0 + math.exp(t))
            assert np.all(np.isfinite(got))
            assert abs(got[0] - p0) <= 1e-14 and abs(got[1] - (1.0 - p0)) <= 1e-14, (d, a, got, p0)


def pin_three_key_closed_form(O):
    """Logits 0, ln 2, ln 3 (built from exact inputs): A = (1, 2, 3) / 6."""
    d = 4
    k = np.zeros((3, d))
    k[:, 0] = [0.0, math.log(2.0), math.log(3.0)]
    q = np.zeros((1, d))
    q[0, 0] = math.sqrt(d)            # sigma * q . k_i = k_i[0]
    got = O.guide_attention(q, k, 1.0 / math.sqrt(d))[0]
    assert np.allclose(got, [1 / 6, 2 / 6, 3 / 6], rtol=0, atol=1e-14), got


def pin_default_scale_in_layer(O):
    """compress_layer scales logits by 1/sqrt(d) unless a scale is given.

    One guide token, two keys +-e1, q = a*e1: the unpooled key score of token 0
    is the logistic function of 2*a*sigma.
    """
    for d, a, scale in [(16, 4.0, 0.0), (64, 2.0, 0.0), (16, 4.0, 0.125)]:
        sigma = scale if scale > 0 else 1.0 / math.sqrt(d)
        kf = np.zeros((1, 2, d), np.float32)
        kf[0, 0, 0], kf[0, 1, 0] = 1.0, -1.0
        qf = np.zeros((1, 1, 1, d), np.float32)
        qf[0, 0, 0, 0] = a
        out = O.compress_layer(exact_bf16(qf), exact_bf16(kf), exact_bf16(np.ones((1, 2, d))), [0, 2],
                               n_heads_q=1, n_heads_kv=1, fixed_budget=1, pool_kernel=1,
                               softmax_scale=scale)
        p0 = 1.0 / (1.0 + math.exp(-2.0 * a * sigma))
        assert abs(out["key"][(0, 0)][0] - p0) <= 1e-14, (d, a, scale, out["key"][(0, 0)], p0)


def pin_row_normaliser(O):
    """lse = log n for Q = 0; two keys +-e1 and q = a*e1: lse = |t| + log1p(exp(-2|t|)), t = a*sigma."""
    for n, d in [(1, 4), (7, 8), (1000, 16)]:
        got = O.guide_lse(np.zeros((3, d)), _rand(n, (n, d)), 0.25)
        assert np.allclose(got, math.log(n), rtol=0, atol=1e-13), (got, math.log(n))
    d = 16
    k = np.zeros((2, d))
    k[0, 0], k[1, 0] = 1.0, -1.0
    for a in (0.0, 0.75, -3.0, 50.0, 9000.0):
        q = np.zeros((1, d))
        q[0, 0] = a
        t = abs(a) * 0.25
        want = t + math.log1p(math.exp(-2 * t))
        got = O.guide_lse(q, k, 0.25)[0]
        assert abs(got - want) <= 1e-12 * max(1.0, t), (a, got, want)


# -- Eq. 1: sum over guide tokens, mean over the GQA group --------------------

def pin_key_scores_total_mass(O):
    """sum_i s_key_i = L_t: each of the G*L_t rows sums to 1, averaged over G."""
    for seed, (g, lt, n, d) in enumerate([(1, 1, 9, 4), (4, 3, 50, 8), (7, 2, 33, 16)]):
        s = O.key_scores(_rand(seed, (g, lt, d)) * 2, _rand(seed + 7, (n, d)), 0.3)
        assert s.shape == (n,)
        assert abs(s.sum() - lt) <= 1e-11 * max(1, lt), (s.sum(), lt)


def pin_rows_independent_and_additive(O):
    """Each guide row's normaliser involves that row alone, and the key score
    is additive over rows: the normalisers of any block of rows equal the
    whole set's for those rows, and the per-head score of a group is the
    mean of its heads' scores, each head's a sum over its own rows.  (A
    guide longer than one scoring block is scored block by block on these two
    facts.)"""
    for seed, (g, lt, n, d) in enumerate([(4, 7, 40, 8), (3, 5, 23, 16)]):
        q = _rand(seed, (g, lt, d)) * 2
        k = _rand(seed + 11, (n, d))
        rows = q.reshape(g * lt, d)
        whole = O.guide_lse(rows, k, 0.35)
        for a, b in [(0, 1), (3, g * lt), (5, 11)]:
            part = O.guide_lse(rows[a:b], k, 0.35)
            assert np.allclose(part, whole[a:b], rtol=0, atol=1e-12), (a, b)
        heads = [O.key_scores(q[i:i + 1], k, 0.35) for i in range(g)]
        for i in range(g):  # one head: its scores sum to its L_t rows' total mass
            assert abs(heads[i].sum() - lt) <= 1e-11 * lt
        assert np.allclose(O.key_scores(q, k, 0.35), sum(heads) / g, rtol=1e-12, atol=0)


def pin_uniform_attention(O):
    """Q = 0 (or identical keys) gives A = 1/n exactly, so s_key_i = L_t / n."""
    for g, lt, n, d in [(1, 1, 5, 4), (4, 16, 64, 8), (3, 5, 7, 2)]:
        s = O.key_scores(np.zeros((g, lt, d)), _rand(n, (n, d)), 0.5)
        assert np.allclose(s, lt / n, rtol=1e-13, atol=0), (s, lt / n)
        same = np.tile(_rand(1, (1, d)), (n, 1))
        s2 = O.key_scores(_rand(2, (g, lt, d)), same, 0.5)
        assert np.allclose(s2, lt / n, rtol=1e-13, atol=0)


def pin_gqa_grouping(O):
    """Query head h feeds KV head h // G (contiguous groups, Llama/Qwen layout).

    Heads 0,1 point hard at key 3 and heads 2,3 at key 7; KV head 0 must then
    keep token 3 and KV head 1 token 7.
    """
    hq, hkv, lt, d, n = 4, 2, 2, 8, 12
    kf = np.zeros((hkv, n, d), dtype=np.float32)
    for i in range(n):
        kf[:, i, i % d] = 1.0
    qf = np.zeros((1, hq, lt, d), dtype=np.float32)
    qf[0, 0:2, :, 3] = 64.0
    qf[0, 2:4, :, 7] = 64.0
    vf = np.ones((hkv, n, d), dtype=np.float32)
    out = O.compress_layer(exact_bf16(qf), exact_bf16(kf), exact_bf16(vf), [0, n],
                           n_heads_q=hq, n_heads_kv=hkv, fixed_budget=1, pool_kernel=1)
    assert list(out["idx"][(0, 0)]) == [3], out["idx"][(0, 0)]
    assert list(out["idx"][(0, 1)]) == [7], out["idx"][(0, 1)]


# -- Eq. 1: pooling ------------------------------------------------------------

def pin_pool_delta_and_edges(O):
    """A unit impulse spreads to 1/K over the window; uniform input is damped at the edges."""
    for kern in (1, 3, 5, 7):
        half = kern // 2
        n = 11
        for j in (0, 1, 5, n - 1):
            s = np.zeros(n)
            s[j] = 1.0
            want = np.zeros(n)
            want[max(0, j - half):min(n, j + half + 1)] = 1.0 / kern
            assert np.allclose(O.pool(s, kern), want, rtol=0, atol=1e-15), (kern, j)
        c = 0.37
        got = O.pool(np.full(n, c), kern)
        for i in range(n):
            terms = min(n - 1, i + half) - max(0, i - half) + 1
            assert abs(got[i] - c * terms / kern) <= 1e-15, (kern, i)


def pin_pool_rejects_even(O):
    for kern in (0, 2, 4, -1):
        try:
            O.pool(np.ones(5), kern)
        except ValueError:
            continue
        raise AssertionError(f"pool accepted kernel {kern}")


# -- Eq. 2: quantisation scale and codes --------------------------------------

def _load_quant_cases():
    """tests/golden/quant_cases.txt: hand-derived rows (values are multiples of 2^-3)."""
    rows = []
    with open(os.path.join(GOLDEN, "quant_cases.txt")) as f:
        lines = [ln.split("#")[0].strip() for ln in f]
    lines = [ln for ln in lines if ln]
    for ln in lines:
        vals, gam, codes = ln.split("|")
        gam = gam.strip()
        g = float.fromhex(gam) if gam.startswith("0x") else float(gam)
        rows.append(([float(x) for x in vals.split()], g, [int(c) for c in codes.split()]))
    return rows


def pin_quant_golden(O):
    """Hand-derived rows: exact scales, exact codes, half-even ties, zero rows."""
    for vals, gam, codes in _load_quant_cases():
        g, q = O.quantize_v(exact_bf16([vals]), 8)
        assert g.dtype == np.float32 and q.dtype == np.int8
        assert float(g[0]) == gam, (vals, g[0], gam)
        assert list(q[0]) == codes, (vals, list(q[0]), codes)


def pin_quant_bounds(O):
    """Random rows: |q| <= 127, absmax -> +-127, |v - q*gamma| <= gamma * (1/2 + 2^-18).

    The slack is half an fp32 ulp of a quotient below 128: the code rounds the
    fp32 quotient, which may itself sit up to 2^-18 from v / gamma.
    """
    rng = np.random.Generator(np.random.PCG64(11))
    v = (rng.standard_normal((64, 96)) * np.exp(rng.uniform(-20, 20, (64, 1)))).astype(np.float32)
    bits = (v.view(np.uint32) >> 16).astype(np.uint16)
    vv = (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    g, q = O.quantize_v(bits, 8)
    a = np.abs(vv).max(axis=1)
    assert np.all(np.abs(q.astype(np.int64)) <= 127)
    assert np.allclose(g, a / 127.0, rtol=2 ** -23, atol=0)
    err = np.abs(vv - q.astype(np.float64) * g.astype(np.float64)[:, None])
    assert np.all(err <= g.astype(np.float64)[:, None] * (0.5 + 2 ** -18)), err.max()
    arg = np.argmax(np.abs(vv), axis=1)
    top = q[np.arange(64), arg].astype(np.int64)
    assert np.all(np.abs(top) == 127)
    assert np.all(np.sign(top) == np.sign(vv[np.arange(64), arg]))


def pin_quant4_golden(O):
    """b = 4 (tests/golden/quant4_cases.txt): hand-derived scales, codes and the
    two-per-byte storage (even channel in the low nibble)."""
    with open(os.path.join(GOLDEN, "quant4_cases.txt")) as f:
        lines = [ln.split("#")[0].strip() for ln in f]
    n = 0
    for ln in (x for x in lines if x):
        vals, gam, codes, packed = ln.split("|")
        gam = gam.strip()
        gw = float.fromhex(gam) if gam.startswith("0x") else float(gam)
        g, q = O.quantize_v(exact_bf16([[float(x) for x in vals.split()]]), 4)
        assert float(g[0]) == gw, (vals, g[0], gw)
        assert list(q[0]) == [int(c) for c in codes.split()], (vals, list(q[0]))
        pk = O.pack_codes(q, 4)
        assert pk.dtype == np.uint8 and pk.shape == (1, len(q[0]) // 2)
        assert [int(x) for x in pk[0]] == [int(x, 16) for x in packed.split()], (vals, list(pk[0]))
        n += 1
    assert n == 4


def pin_quant4_bounds(O):
    """Random rows at b = 4: |q| <= 7, absmax -> +-7, |v - q*gamma| <= gamma * (1/2 + 2^-18)."""
    rng = np.random.Generator(np.random.PCG64(12))
    v = (rng.standard_normal((48, 64)) * np.exp(rng.uniform(-20, 20, (48, 1)))).astype(np.float32)
    bits = (v.view(np.uint32) >> 16).astype(np.uint16)
    vv = (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    g, q = O.quantize_v(bits, 4)
    assert np.all(np.abs(q.astype(np.int64)) <= 7)
    assert np.allclose(g, np.abs(vv).max(axis=1) / 7.0, rtol=2 ** -23, atol=0)
    err = np.abs(vv - q.astype(np.float64) * g.astype(np.float64)[:, None])
    assert np.all(err <= g.astype(np.float64)[:, None] * (0.5 + 2 ** -18)), err.max()
    arg = np.argmax(np.abs(vv), axis=1)
    assert np.all(np.abs(q[np.arange(48), arg].astype(np.int64)) == 7)


# -- Eq. 3 and Sec. 3.4 selection ---------------------------------------------

def pin_combine_product(O):
    """s = s_key * gamma; the key-only ablation (Sec. 4.3.1) drops gamma."""
    a = np.array([0.5, 2.0, 0.0, 3.0])
    g = np.array([4.0, 0.25, 9.0, 1.0], dtype=np.float32)
    assert list(O.combine(a, g)) == [2.0, 0.5, 0.0, 3.0]
    assert list(O.combine(a, g, key_only=True)) == [0.5, 2.0, 0.0, 3.0]


def pin_key_scores_given_lse(O):
    """With Q = 0 every logit is 0, so exp(x - lse_r) = 1/(n + c_r) when the
    caller's normaliser lse_r = log(n + c_r) also counts guide-prefix mass c_r
    (the literal prefill normaliser, Sec. 3.2): s_i = (1/G) sum_r 1/(n + c_r).
    A shift of every normaliser by D scales every score by exp(-D); with the
    context-only normaliser the scores equal key_scores (uniform: L_t / n)."""
    g, lt, d, n = 2, 3, 8, 10
    q = np.zeros((g, lt, d))
    k = _rand(1, (n, d))
    c = np.array([0.0, 1.0, 2.0, 5.0, 0.5, 3.0])
    s = O.key_scores_given_lse(q, k, 0.3, np.log(n + c))
    want = sum(1.0 / (n + cr) for cr in c) / g
    assert np.allclose(s, want, rtol=1e-13, atol=0)
    s0 = O.key_scores_given_lse(q, k, 0.3, np.full(g * lt, math.log(n)))
    assert np.allclose(s0, lt / n, rtol=1e-13, atol=0)
    qr = _rand(2, (g, lt, d))
    lse = np.linspace(2.0, 4.0, g * lt)
    a = O.key_scores_given_lse(qr, k, 0.25, lse)
    b = O.key_scores_given_lse(qr, k, 0.25, lse + 0.75)
    assert np.allclose(b, a * math.exp(-0.75), rtol=1e-12, atol=0)


def pin_layer_given_lse_indexing(O):
    """compress_layer with caller normalisers: Q = 0 makes every logit 0, so
    the unpooled key score of document b, head h is (1/G) sum_r exp(-lse[b, h, r]).
    Two documents x two heads with distinct normalisers: a layer that reads
    another document's or head's row of lse gives another constant."""
    hq, hkv, lt, d = 4, 2, 3, 8
    g = hq // hkv
    lens = [5, 9]
    offs = [0, 5, 14]
    rng = np.random.Generator(np.random.PCG64(21))
    def b16(x):
        return (x.astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
    q = np.zeros((2, hq, lt, d), np.uint16)
    k = b16(rng.standard_normal((hkv, 14, d)))
    v = b16(rng.standard_normal((hkv, 14, d)))
    lse = np.empty((2, hkv, g * lt))
    for b in range(2):
        for h in range(hkv):
            lse[b, h] = np.log(3.0 + 10.0 * b + 4.0 * h + np.arange(g * lt))
    out = O.compress_layer(q, k, v, offs, n_heads_q=hq, n_heads_kv=hkv, keep_ratio=0.5,
                           pool_kernel=1, lse=lse)
    for b in range(2):
        for h in range(hkv):
            want = sum(1.0 / (3.0 + 10.0 * b + 4.0 * h + r) for r in range(g * lt)) / g
            got = out["key"][(b, h)]
            assert got.shape == (lens[b],)
            assert np.allclose(got, want, rtol=1e-13, atol=0), (b, h, got[0], want)


def pin_kept_count_fixed_budget(O):
    """A fixed per-(document, head) budget keeps min(budget, n) tokens (Sec. 4
    "Eviction"); budget -1 falls back to the ratio rule.  A document shorter
    than the budget keeps all of its tokens."""
    assert O.kept_count(10, 0.5, 3) == 3
    assert O.kept_count(10, 0.5, 10) == 10
    assert O.kept_count(10, 0.5, 25) == 10
    assert O.kept_count(0, 0.5, 4) == 0
    assert O.kept_count(10, 0.5, 0) == 0
    assert O.kept_count(10, 0.3, -1) == 3
    rng = np.random.Generator(np.random.PCG64(22))
    def b16(x):
        return (x.astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
    q = b16(rng.standard_normal((2, 2, 2, 8)))
    k = b16(rng.standard_normal((1, 11, 8)))
    v = b16(rng.standard_normal((1, 11, 8)))
    out = O.compress_layer(q, k, v, [0, 4, 11], n_heads_q=2, n_heads_kv=1, fixed_budget=6)
    assert out["k"] == {0: 4, 1: 6}
    assert list(out["idx"][(0, 0)]) == [0, 1, 2, 3]
    assert len(out["idx"][(1, 0)]) == 6


def pin_literal_lse_closed_form(O):
    """Q = 0: every logit is 0, so row r = (g, j) of the causal prefill map has
    n context terms and j + 1 guide terms: lse_r = log(n + j + 1), rows ordered
    query head-major (Sec. 3.2).  With no context keys only the prefix is left."""
    g, lt, d, n = 3, 4, 8, 11
    q = np.zeros((g, lt, d))
    got = O.guide_lse_literal(q, _rand(1, (n, d)), _rand(2, (lt, d)), 0.4)
    want = np.array([math.log(n + j + 1) for _ in range(g) for j in range(lt)])
    assert np.allclose(got, want, rtol=1e-14, atol=0)
    got0 = O.guide_lse_literal(q, np.zeros((0, d)), _rand(2, (lt, d)), 0.4)
    assert np.allclose(got0, [math.log(j + 1) for _ in range(g) for j in range(lt)], rtol=1e-14, atol=1e-15)


def pin_literal_lse_causal(O):
    """One scalar channel: q_r = a_g e1, context keys +-e1, guide keys c_j e1.
    Row (g, j) sums exp(+-sigma a_g) and exp(sigma a_g c_j') for j' <= j, written
    out term by term; a huge later guide key leaves earlier rows unchanged."""
    g, lt, d, sigma = 2, 3, 4, 0.5
    a = [0.7, -1.3]
    c = [2.0, -0.5, 30.0]
    q = np.zeros((g, lt, d))
    for gi in range(g):
        q[gi, :, 0] = a[gi]
    k = np.zeros((2, d))
    k[0, 0], k[1, 0] = 1.0, -1.0
    kg = np.zeros((lt, d))
    kg[:, 0] = c
    got = O.guide_lse_literal(q, k, kg, sigma)
    for gi in range(g):
        for j in range(lt):
            z = math.exp(sigma * a[gi]) + math.exp(-sigma * a[gi])
            for jj in range(j + 1):
                z += math.exp(sigma * a[gi] * c[jj])
            assert math.isclose(got[gi * lt + j], math.log(z), rel_tol=1e-13), (gi, j)


def pin_literal_key_scores_brute_force(O):
    """compress_layer with guide keys against a brute-force literal prefill row:
    for every (document, head, g, j), the causal row over [context, guide 0..j]
    is built with explicit loops, exponentiated and normalised; its context
    part, summed over rows and averaged over the group, is the key score.
    Two documents and two KV heads with distinct guide keys pin the [b, h]
    indexing of the guide keys."""
    batch, hkv, g, lt, d = 2, 2, 2, 3, 8
    offs = [0, 5, 12]
    rng = np.random.Generator(np.random.PCG64(31))
    q = rng.integers(-4, 5, (batch, hkv * g, lt, d)).astype(np.float32) / 4
    k = rng.integers(-4, 5, (hkv, offs[-1], d)).astype(np.float32) / 4
    v = rng.integers(-4, 5, (hkv, offs[-1], d)).astype(np.float32) / 4
    kg = rng.integers(-8, 9, (batch, hkv, lt, d)).astype(np.float32) / 4
    sigma = 0.5
    out = O.compress_layer(exact_bf16(q), exact_bf16(k), exact_bf16(v), offs, n_heads_q=hkv * g,
                           n_heads_kv=hkv, keep_ratio=0.5, softmax_scale=sigma,
                           k_guide_bits=exact_bf16(kg))
    for b in range(batch):
        lo, hi = offs[b], offs[b + 1]
        for h in range(hkv):
            s = [0.0] * (hi - lo)
            for gi in range(g):
                for j in range(lt):
                    qr = [float(x) for x in q[b, h * g + gi, j]]
                    ctx = [math.exp(sigma * sum(qr[c] * float(k[h, i, c]) for c in range(d)))
                           for i in range(lo, hi)]
                    pre = [math.exp(sigma * sum(qr[c] * float(kg[b, h, jj, c]) for c in range(d)))
                           for jj in range(j + 1)]
                    z = sum(ctx) + sum(pre)
                    for i in range(hi - lo):
                        s[i] += ctx[i] / z
            want = np.array(s) / g
            assert np.allclose(out["key"][(b, h)], want, rtol=1e-12, atol=0), (b, h)


def pin_combine_normadd(O):
    """Normalised add (Sec. 4.4 aggregation ablation): L2 norms over the vector.
    (3, 4) and (5, 12) have norms 5 and 13; each term is scale-free; a zero
    vector contributes nothing."""
    a, g = np.array([3.0, 4.0]), np.array([5.0, 12.0])
    s = O.combine(a, g, mode="normadd")
    assert np.allclose(s, [0.6 + 5 / 13, 0.8 + 12 / 13], rtol=1e-15, atol=0)
    assert np.allclose(O.combine(7.0 * a, 0.01 * g, mode="normadd"), s, rtol=1e-14, atol=0)
    assert np.allclose(O.combine(a, np.zeros(2), mode="normadd"), [0.6, 0.8], rtol=1e-15, atol=0)


def pin_combine_harmonic(O):
    """Harmonic mean 2ab/(a+b): (1,1) -> 1, (1,3) -> 3/2, (2,6) -> 3, (0,x) -> 0,
    and 0 where both are 0."""
    a = np.array([1.0, 1.0, 2.0, 0.0, 0.0])
    g = np.array([1.0, 3.0, 6.0, 5.0, 0.0])
    assert list(O.combine(a, g, mode="harmonic")) == [1.0, 1.5, 3.0, 0.0, 0.0]


def _brute_topk(scores, k):
    """Max-sum subset of size k; among equal sums the lexicographically smallest."""
    best, best_set = None, None
    for c in itertools.combinations(range(len(scores)), k):
        s = sum(scores[i] for i in c)
        if best is None or s > best:
            best, best_set = s, c
    return list(best_set) if best_set is not None else []


def pin_select_bruteforce(O):
    """Top-k equals brute force over all subsets (integer scores: exact sums, many ties)."""
    rng = np.random.Generator(np.random.PCG64(5))
    for n in range(0, 9):
        for trial in range(3):
            sc = rng.integers(0, 4, size=n).astype(np.float64)
            for k in range(0, n + 1):
                got = list(O.select_topk(sc, k))
                assert got == _brute_topk(list(sc), k), (sc, k, got)


def pin_select_invariants(O):
    rng = np.random.Generator(np.random.PCG64(6))
    for n, k in [(100, 7), (257, 64), (1000, 999), (50, 0), (50, 50)]:
        sc = rng.random(n)
        idx = np.asarray(O.select_topk(sc, k))
        assert idx.size == k
        assert np.all(np.diff(idx) > 0)
        mask = np.zeros(n, bool)
        mask[idx] = True
        if 0 < k < n:
            assert sc[mask].min() >= sc[~mask].max()
    same = np.full(20, 0.5)
    assert list(O.select_topk(same, 6)) == [0, 1, 2, 3, 4, 5]


# -- Sec. 4 "Eviction": uniform per-head budget --------------------------------

def pin_budget(O):
    """kept = ceil(ratio * n) exactly, for ratios written as short decimals."""
    ratios = ["0", "0.05", "0.07", "0.1", "0.2", "0.25", "0.3", "0.33", "0.5", "0.7", "0.99", "1"]
    for r in ratios:
        for n in [0, 1, 2, 3, 7, 10, 100, 129, 1000, 2048, 32768, 65536, 131072, 294911]:
            want = math.ceil(Fraction(r) * n)
            assert O.budget(n, float(r)) == want, (r, n, O.budget(n, float(r)), want)
    assert O.budget(32768, 0.2) == 6554 and O.budget(131072, 0.1) == 13108
    assert O.budget(2048, 0.25) == 512 and O.budget(65536, 0.05) == 3277
    for bad in (-0.1, 1.5, float("nan")):
        assert O.budget(10, bad) == -1


# -- special cases that reduce to a plain sort ---------------------------------

def pin_special_cases(O):
    """Q = 0 with K = 1: the selection is a sort of gamma (lower index first).
    Identical tokens: everything ties, so the first k tokens are kept."""
    rng = np.random.Generator(np.random.PCG64(9))
    hq, hkv, lt, d, n = 2, 1, 3, 8, 40
    q = np.zeros((1, hq, lt, d), np.float32)
    k = rng.standard_normal((hkv, n, d)).astype(np.float32)
    v = rng.standard_normal((hkv, n, d)).astype(np.float32)
    kb = (k.view(np.uint32) >> 16).astype(np.uint16)
    vb = (v.view(np.uint32) >> 16).astype(np.uint16)
    out = O.compress_layer(exact_bf16(q), kb, vb, [0, n], n_heads_q=hq, n_heads_kv=hkv,
                           fixed_budget=9, pool_kernel=1)
    vv = (vb.astype(np.uint32) << 16).view(np.float32)
    amax = np.abs(vv[0]).max(axis=1)
    want = sorted(sorted(range(n), key=lambda i: (-amax[i], i))[:9])
    assert list(out["idx"][(0, 0)]) == want
    kk = np.tile(k[:, :1], (1, n, 1))
    vv2 = np.tile(v[:, :1], (1, n, 1))
    kb2 = (kk.view(np.uint32) >> 16).astype(np.uint16)
    vb2 = (vv2.view(np.uint32) >> 16).astype(np.uint16)
    q2 = rng.standard_normal((1, hq, lt, d)).astype(np.float32)
    qb2 = (q2.view(np.uint32) >> 16).astype(np.uint16)
    out2 = O.compress_layer(qb2, kb2, vb2, [0, n], n_heads_q=hq, n_heads_kv=hkv,
                            fixed_budget=5, pool_kernel=1)
    assert list(out2["idx"][(0, 0)]) == [0, 1, 2, 3, 4]


def pin_ragged_docs_independent(O):
    """Documents packed along the token axis are compressed independently."""
    rng = np.random.Generator(np.random.PCG64(12))
    hq, hkv, lt, d = 4, 2, 2, 8
    lens = [13, 30, 7]
    offs = np.concatenate([[0], np.cumsum(lens)])
    n = int(offs[-1])
    def b16(x):
        return (x.astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
    q = b16(rng.standard_normal((3, hq, lt, d)))
    k = b16(rng.standard_normal((hkv, n, d)))
    v = b16(rng.standard_normal((hkv, n, d)))
    whole = O.compress_layer(q, k, v, offs, n_heads_q=hq, n_heads_kv=hkv, keep_ratio=0.5)
    for b in range(3):
        lo, hi = offs[b], offs[b + 1]
        single = O.compress_layer(q[b:b + 1], k[:, lo:hi], v[:, lo:hi], [0, hi - lo],
                                  n_heads_q=hq, n_heads_kv=hkv, keep_ratio=0.5)
        assert whole["k"][b] == math.ceil(Fraction(1, 2) * int(hi - lo))
        for h in range(hkv):
            assert list(whole["idx"][(b, h)]) == list(single["idx"][(0, h)])
            assert np.array_equal(whole["scores"][(b, h)], single["scores"][(0, h)])


def pin_gather_rows(O):
    """Compaction reads row (head, doc_lo + idx) of every tensor: rows here encode
    their own (head, token), so the gathered values name where they came from."""
    hkv, n, d = 3, 40, 4
    tok = np.arange(n)[None, :, None]
    head = np.arange(hkv)[:, None, None]
    k = (head * 1000 + tok + np.zeros((1, 1, d))).astype(np.uint16)
    v = (head * 1000 + tok + 500 + np.zeros((1, 1, d))).astype(np.uint16)
    gamma = (np.arange(hkv)[:, None] * 1000 + np.arange(n)[None, :]).astype(np.float32)
    vq = ((np.arange(n)[None, :, None] % 100) + np.zeros((hkv, 1, d))).astype(np.int8)
    idx = np.array([0, 3, 4, 9])
    kc, vc, vqc, gc = O.gather_rows(k, v, gamma, vq, 10, 2, idx)
    want_tok = 10 + idx
    assert np.array_equal(kc[:, 0], 2000 + want_tok) and np.array_equal(vc[:, 0], 2500 + want_tok)
    assert np.array_equal(gc, 2000 + want_tok) and np.array_equal(vqc[:, 0], want_tok % 100)


ALL_PINS = [v for k, v in sorted(globals().items()) if k.startswith("pin_")]
