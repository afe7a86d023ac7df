"""CPU oracle for TaskPress's prefill-time KV compression (Sec. 3, Eq. 1-3).

TEST INFRASTRUCTURE ONLY.  This module is the plain, slow, obviously correct
definition of what the CUDA path computes.  Only the tests, the smoke check
and the benchmark's CPU-baseline leg may import it; the product path never
does, and this module imports nothing from the product package (bf16 decoding
is re-implemented here on purpose).

Arithmetic is fp64 throughout, except the value quantiser, whose scale and
codes the paper defines per token in a storage precision it does not name;
that step follows the fp32 rule stated at ``quantize_v`` so that both sides
reach the same integers.

Readings of the paper used here (where it is silent or ambiguous):

* softmax normaliser - by default each guide row is normalised over the
  context keys only (the attention block the method slices out of the prefill
  map, Sec. 3.2, renormalised); given the guide's keys, the literal row of
  that causal map, context plus guide prefix (guide_lse_literal); or a
  normaliser the caller supplies;
* reduction - Eq. 1 sums over the L_t guide tokens; the G query heads sharing
  a KV head are averaged (the paper budgets per KV head, Sec. 4 "Eviction");
* pooling - the Eq. 1 window has 2*floor(K/2)+1 terms, so K must be odd; terms
  outside [0, n) are zero and the divisor stays K;
* quantiser - symmetric per-token absmax, b = 8 or 4 bits (Eq. 2); fp32
  scale; codes are round-half-even of the IEEE fp32 quotient v / gamma,
  clamped to +-(2^(b-1) - 1); gamma = 0 gives all-zero codes; 4-bit codes are
  stored two per byte, the even channel in the low nibble;
* scale - softmax scale 1/sqrt(d) unless given;
* budget - kept = ceil(ratio * n - 1e-9 * n) clamped to [0, n];
* ties - equal scores keep the lower token index; kept indices ascend;
* blends - the aggregation ablation's normalised add uses L2 norms over one
  (document, head); its harmonic mean reads the printed ',' as '+'.

Parity pins for every function live in tests/test_oracle_pins.py.
"""
from __future__ import annotations

import math
from typing import Optional, Sequence

import numpy as np


def decode_bf16(bits) -> np.ndarray:
    """Widen bf16 bit patterns (uint16) exactly to float64."""
    u = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16
    return u.view(np.float32).astype(np.float64)


def decode_bf16_f32(bits) -> np.ndarray:
    """Widen bf16 bit patterns (uint16) exactly to float32."""
    u = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16
    return u.view(np.float32)


# --------------------------------------------------------------------------
# Budget (Sec. 4 "Eviction": a uniform budget per KV head)
# --------------------------------------------------------------------------

def budget(n: int, keep_ratio: float) -> int:
    """Tokens kept per head for a keep ratio (1 - the paper's eviction ratio).

    kept = ceil(ratio*n - 1e-9*n), clamped to [0, n]; the small offset keeps
    exact decimal products such as 0.07*100 from rounding up to 8.  Returns -1
    for a ratio outside [0, 1] or NaN.
    """
    if not (0.0 <= keep_ratio <= 1.0):
        return -1
    k = math.ceil(keep_ratio * float(n) - 1e-9 * float(n))
    return int(min(max(k, 0), n))


def kept_count(n: int, keep_ratio: float, fixed_budget: int) -> int:
    """Per-(document, head) kept count: a fixed budget when >= 0, else the ratio rule."""
    if fixed_budget >= 0:
        return int(min(fixed_budget, n))
    return budget(n, keep_ratio)


# --------------------------------------------------------------------------
# Eq. 2: per-token value quantisation scale, and the int8 codes
# --------------------------------------------------------------------------

def quantize_v(v_bits, quant_bits: int = 8):
    """Per-token symmetric absmax quantisation of V (Sec. 3.3, Eq. 2).

    gamma_i = max_c |v_ic| / (2^(b-1) - 1), in fp32 with IEEE round-to-nearest
    division; q_ic = clamp(rint(v_ic / gamma_i), -(2^(b-1)-1), 2^(b-1)-1) with
    the quotient an IEEE fp32 division and rint round-half-even; gamma_i = 0
    gives q_i = 0.  Returns (gamma float32 [..., n], q int8 [..., n, d]).
    """
    qmax = (1 << (quant_bits - 1)) - 1
    v = decode_bf16_f32(v_bits)
    a = np.max(np.abs(v), axis=-1)
    gamma = (a.astype(np.float32) / np.float32(qmax)).astype(np.float32)
    safe = np.where(gamma > 0, gamma, np.float32(1.0)).astype(np.float32)
    quot = (v / safe[..., None]).astype(np.float32)
    q = np.clip(np.rint(quot), -qmax, qmax)
    q = np.where(gamma[..., None] > 0, q, 0.0)
    return gamma, q.astype(np.int8)


def pack_codes(q, quant_bits: int = 8) -> np.ndarray:
    """Storage form of the Eq. 2 codes.  b = 8: one int8 per value.  b = 4 (the
    4-bit KV of the paper's experiments, Sec. 4 "Quantization"): two codes per
    byte, channel 2i in the low nibble and channel 2i+1 in the high nibble,
    each in 4-bit two's complement.  Returns int8 [..., d] or uint8 [..., d/2]."""
    q = np.asarray(q)
    if quant_bits == 8:
        return q.astype(np.int8)
    if quant_bits == 4:
        u = q.astype(np.int64) & 0xF
        return (u[..., 0::2] | (u[..., 1::2] << 4)).astype(np.uint8)
    raise ValueError("quant_bits must be 4 or 8")


# --------------------------------------------------------------------------
# Sec. 3.2: guide-to-context attention and Eq. 1
# --------------------------------------------------------------------------

def guide_attention(q_rows: np.ndarray, k_ctx: np.ndarray, sigma: float) -> np.ndarray:
    """A[r, i] = softmax_i(sigma * q_r . k_i) over the context keys of one head.

    q_rows: [M, d] float64 guide query rows; k_ctx: [n, d] float64 keys.
    An explicit full softmax per row (max, exp, sum, divide) in fp64.
    """
    x = (q_rows @ k_ctx.T) * sigma
    m = np.max(x, axis=1, keepdims=True)
    e = np.exp(x - m)
    z = np.sum(e, axis=1, keepdims=True)
    return e / z


def guide_lse(q_rows: np.ndarray, k_ctx: np.ndarray, sigma: float) -> np.ndarray:
    """lse[r] = log sum_i exp(sigma * q_r . k_i): each guide row's softmax normaliser."""
    x = (q_rows @ k_ctx.T) * sigma
    m = np.max(x, axis=1)
    return m + np.log(np.sum(np.exp(x - m[:, None]), axis=1))


def key_scores(q_group: np.ndarray, k_ctx: np.ndarray, sigma: float) -> np.ndarray:
    """Unpooled key importance of every context token for one KV head.

    q_group: [G, L_t, d] float64 (the G query heads sharing the KV head);
    returns s[i] = (1/G) * sum_g sum_j A_g[j, i]  (Eq. 1's inner sum over j,
    averaged over the GQA group).
    """
    g, lt, d = q_group.shape
    a = guide_attention(q_group.reshape(g * lt, d), k_ctx, sigma)
    return a.sum(axis=0) / g


def key_scores_given_lse(q_group: np.ndarray, k_ctx: np.ndarray, sigma: float,
                         lse_rows: np.ndarray) -> np.ndarray:
    """key_scores with each row's softmax normaliser supplied by the caller.

    s[i] = (1/G) * sum_r exp(sigma * q_r . k_i - lse_r) over the G*L_t rows
    r = (g, j).  The method slices A out of the full prefill attention map
    (Sec. 3.2), whose row normaliser also covers the guide's own causal prefix;
    a caller that keeps the prefill's per-row log-sum-exp passes it here, which
    gives that literal normaliser and needs no normalisation pass.  With lse_r =
    guide_lse(...) this equals key_scores.
    """
    g, lt, d = q_group.shape
    x = (q_group.reshape(g * lt, d) @ k_ctx.T) * sigma
    return np.exp(x - np.asarray(lse_rows, dtype=np.float64)[:, None]).sum(axis=0) / g


def guide_lse_literal(q_group: np.ndarray, k_ctx: np.ndarray, k_guide: np.ndarray,
                      sigma: float) -> np.ndarray:
    """Each guide row's normaliser over its whole causal row of the prefill map.

    The prefill attends over the context followed by the guide, causally, so
    guide token j sees every context key and the guide keys 0..j (itself
    included).  A is sliced out of that map (Sec. 3.2), so row r = (g, j) of
    the stacked group (query head-major, then guide token) is normalised by
      lse[r] = log( sum_i exp(sigma q_r . k_i) + sum_{j' <= j} exp(sigma q_r . kg_j') ).
    q_group [G, L_t, d], k_ctx [n, d], k_guide [L_t, d] float64 (post-RoPE).
    Each row is written out as its own logit vector: context part, then the
    guide prefix; then max, exp, sum, log.
    """
    g, lt, d = q_group.shape
    out = np.empty(g * lt)
    for gi in range(g):
        for j in range(lt):
            qr = q_group[gi, j]
            x = np.concatenate([k_ctx @ qr, k_guide[: j + 1] @ qr]) * sigma
            m = np.max(x)
            out[gi * lt + j] = m + math.log(float(np.sum(np.exp(x - m))))
    return out


def pool(s: np.ndarray, kernel: int) -> np.ndarray:
    """Eq. 1's 1-D average pooling with window K (odd), zero outside [0, n)."""
    if kernel < 1 or kernel % 2 == 0:
        raise ValueError("pool kernel must be odd and >= 1")
    n = s.shape[0]
    half = kernel // 2
    out = np.zeros(n, dtype=np.float64)
    for off in range(-half, half + 1):
        lo = max(0, -off)
        hi = min(n, n - off)
        out[lo:hi] += s[lo + off:hi + off]
    return out / kernel


COMBINE_MODES = ("mul", "normadd", "harmonic")


def combine(pooled: np.ndarray, gamma: np.ndarray, key_only: bool = False,
            mode: str = "mul") -> np.ndarray:
    """Eq. 3: s_i = s_key_i * s_value_i with s_value_i = gamma_i (Sec. 3.3-3.4).

    The two other blends of the aggregation ablation (Sec. 4.4, "Score
    aggregation strategy"), over one (document, head):
      normadd   s_key_i / ||s_key||_2 + s_value_i / ||s_value||_2, a term whose
                norm is 0 contributing 0;
      harmonic  2 s_key_i s_value_i / (s_key_i + s_value_i), 0 where the sum
                is 0 (the printed formula has ',' for '+').
    key_only drops s_value (Sec. 4.3.1, the key-only row of Tab. 8).
    """
    if key_only:
        return pooled.copy()
    a = np.asarray(pooled, dtype=np.float64)
    b = np.asarray(gamma, dtype=np.float64)
    if mode == "mul":
        return a * b
    if mode == "normadd":
        na, nb = math.sqrt(float(np.sum(a * a))), math.sqrt(float(np.sum(b * b)))
        return (a / na if na > 0 else 0.0 * a) + (b / nb if nb > 0 else 0.0 * b)
    if mode == "harmonic":
        den = a + b
        out = np.zeros_like(a)
        nz = den != 0
        out[nz] = 2.0 * a[nz] * b[nz] / den[nz]
        return out
    raise ValueError(f"unknown combine mode {mode!r}")


# --------------------------------------------------------------------------
# Sec. 3.4 / Sec. 4: top-budget selection per head, then compaction
# --------------------------------------------------------------------------

def select_topk(scores: np.ndarray, k: int) -> np.ndarray:
    """Indices of the k largest scores, lower index first among equals, ascending."""
    n = scores.shape[0]
    k = int(min(max(k, 0), n))
    order = np.lexsort((np.arange(n), -scores))  # primary: score desc; then index asc
    return np.sort(order[:k]).astype(np.int64)


def compress_layer(q_bits, k_bits, v_bits, doc_offsets: Sequence[int], *,
                   n_heads_q: int, n_heads_kv: int, keep_ratio: float = 0.25,
                   fixed_budget: int = -1, pool_kernel: int = 5, quant_bits: int = 8,
                   softmax_scale: float = 0.0, key_only: bool = False, combine_mode: str = "mul",
                   lse=None, k_guide_bits=None, heads: Optional[Sequence[int]] = None,
                   docs: Optional[Sequence[int]] = None):
    """The whole compression of one layer (Sec. 3.1-3.4 with Sec. 4 budgets).

    q_bits [batch, H_q, L_t, d], k_bits / v_bits [H_kv, N_total, d] (bf16 bits),
    doc_offsets [batch+1].  ``lse`` [batch, H_kv, G*L_t] (natural log), when
    given, replaces each guide row's normaliser (key_scores_given_lse);
    ``k_guide_bits`` [batch, H_kv, L_t, d] (bf16 bits), when given, gives each
    row the literal normaliser of guide_lse_literal instead (not with ``lse``);
    ``combine_mode`` selects the blend of ``combine``.  Returns a dict:
      gamma  [H_kv, N_total] float32, vq [H_kv, N_total, d] int8,
      scores {(b, h): float64 [n_b]}  combined scores s_i,
      key    {(b, h): float64 [n_b]}  unpooled key scores,
      idx    {(b, h): int64 [k_b]}    kept doc-local indices, ascending,
      k      {b: k_b}.
    ``heads`` / ``docs`` restrict the (expensive) scoring to a subset.
    """
    if lse is not None and k_guide_bits is not None:
        raise ValueError("give either lse or k_guide_bits")
    q = decode_bf16(q_bits)
    k_all = decode_bf16(k_bits)
    kg = None if k_guide_bits is None else decode_bf16(k_guide_bits)
    batch, hq, lt, d = q.shape
    g = n_heads_q // n_heads_kv
    sigma = softmax_scale if softmax_scale > 0 else 1.0 / math.sqrt(d)
    gamma, vq = quantize_v(v_bits, quant_bits)
    out = {"gamma": gamma, "vq": vq, "scores": {}, "key": {}, "idx": {}, "k": {}}
    heads = range(n_heads_kv) if heads is None else heads
    docs = range(batch) if docs is None else docs
    for b in docs:
        lo, hi = int(doc_offsets[b]), int(doc_offsets[b + 1])
        n = hi - lo
        kb = kept_count(n, keep_ratio, fixed_budget)
        out["k"][b] = kb
        for h in heads:
            qg = q[b, h * g:(h + 1) * g]
            # an empty document has no context tokens: nothing to score or keep
            if n == 0:
                s_key = np.zeros(0)
            elif kg is not None:
                lse_rows = guide_lse_literal(qg, k_all[h, lo:hi], kg[b, h], sigma)
                s_key = key_scores_given_lse(qg, k_all[h, lo:hi], sigma, lse_rows)
            elif lse is None:
                s_key = key_scores(qg, k_all[h, lo:hi], sigma)
            else:
                s_key = key_scores_given_lse(qg, k_all[h, lo:hi], sigma, np.asarray(lse)[b, h])
            s = combine(pool(s_key, pool_kernel), gamma[h, lo:hi], key_only, combine_mode)
            out["key"][(b, h)] = s_key
            out["scores"][(b, h)] = s
            out["idx"][(b, h)] = select_topk(s, kb)
    return out


def gather_rows(k_bits, v_bits, gamma, vq, doc_lo: int, head: int, idx: np.ndarray):
    """Compaction of one (document, head): kept K, V, int8 V and scales in token order."""
    tok = doc_lo + np.asarray(idx, dtype=np.int64)
    return (np.asarray(k_bits)[head, tok], np.asarray(v_bits)[head, tok],
            np.asarray(vq)[head, tok], np.asarray(gamma)[head, tok])
