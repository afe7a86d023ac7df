"""Seeded synthetic inputs for the TaskPress compression path.

This module only *makes inputs*: it holds none of the method's arithmetic
(no attention, no scores, no quantisation).  Both the oracle tests and the
CUDA path consume what it produces, so the two sides see the same bytes.

The paper evaluates on LongBench / RULER prompts run through LLaMA-3.1-8B and
Qwen3 (Sec. 4); none of that is available offline, so these seeded tensors
stand in for the post-RoPE guide queries and the context K/V of one layer.
The recipe, per configuration, is:

* guide queries  Q ~ N(0, 1), shape [batch, H_q, L_t, d]
* keys           K ~ N(0, 1) (or Student-t nu=3 scaled to unit variance),
                 optionally times a per-(KV head, channel) scale drawn
                 log-uniform in [lo, hi]; shape [H_kv, N_total, d]
* planted spans  S spans of L_s tokens at random non-overlapping aligned
                 slots (shared by all heads of a document); each span key is
                 replaced by |k| * (0.6 u + 0.8 w), u the normalised mean of
                 the KV head's group guide queries and w a random unit vector
                 orthogonal to u (so cos(k, u) = 0.6)
* values         V ~ N(0, 1); a fraction f of tokens per KV head get one random
                 channel multiplied by a factor ("outlier token")

Everything is drawn on the host with numpy's PCG64 in float32 and rounded to
bf16 with round-to-nearest-even; tensors are returned as uint16 bf16 bit
patterns.  ``make_layer_torch`` draws the same recipe with torch's generator
on a device (distributionally identical, not bitwise) for large benchmark
stacks that would take minutes to draw on the host.
"""
from __future__ import annotations

import hashlib
import math
from dataclasses import dataclass, field, replace
from typing import Optional, Sequence

import numpy as np


@dataclass(frozen=True)
class Workload:
    """Shape and value recipe of one synthetic compression workload."""

    name: str
    n_heads_q: int
    n_heads_kv: int
    head_dim: int
    guide_len: int
    doc_lens: tuple            # context length of each document (batch = len)
    layers: int = 1
    keep_ratio: float = 0.25   # used when budget < 0
    budget: int = -1           # fixed per-(document, head) budget when >= 0
    seed: int = 0
    key_dist: str = "normal"   # "normal" or "student_t3"
    key_chan_scale: Optional[tuple] = None   # (lo, hi) log-uniform per (head, channel)
    spans: tuple = (0, 0)      # (count, length) per document
    v_outlier: tuple = (0.0, 1.0)  # (fraction of tokens per head, factor)
    per_doc_seed: bool = False     # doc b uses seed + b (else one stream)
    keep_ratios: tuple = field(default_factory=tuple)  # extra ratios swept

    @property
    def batch(self) -> int:
        return len(self.doc_lens)

    @property
    def group(self) -> int:
        return self.n_heads_q // self.n_heads_kv

    @property
    def rows(self) -> int:
        """Stacked guide rows per KV head (GQA group size x guide length)."""
        return self.group * self.guide_len

    @property
    def n_total(self) -> int:
        return int(sum(self.doc_lens))

    def doc_offsets(self) -> np.ndarray:
        return np.concatenate([[0], np.cumsum(self.doc_lens)]).astype(np.int64)

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)


def _ragged_lengths(seed: int, batch: int, lo: int, hi: int) -> tuple:
    rng = np.random.Generator(np.random.PCG64(seed))
    return tuple(int(x) for x in rng.integers(lo, hi + 1, size=batch))


#: The five workloads the path is measured and checked on.
WORKLOADS = {
    1: Workload("tiny-gqa4-d64-2k", 8, 2, 64, 16, (2048,), keep_ratio=0.25, seed=0,
                spans=(4, 32), v_outlier=(0.01, 20.0)),
    2: Workload("llama8b-layer-32k", 32, 8, 128, 64, (32768,), keep_ratio=0.20,
                seed=2000, key_chan_scale=(0.5, 4.0), spans=(64, 64),
                v_outlier=(0.005, 16.0)),
    3: Workload("llama8b-stack32-128k", 32, 8, 128, 128, (131072,), layers=32,
                keep_ratio=0.10, seed=3000, key_chan_scale=(0.5, 4.0),
                spans=(64, 64), v_outlier=(0.005, 16.0)),
    4: Workload("qwen-gqa7-64k", 28, 4, 128, 32, (65536,), keep_ratio=0.05,
                seed=4000, key_dist="student_t3", v_outlier=(0.02, 32.0),
                keep_ratios=(0.05, 0.10, 0.25, 0.50)),
    5: Workload("ragged8-8k-64k", 32, 8, 128, 64,
                _ragged_lengths(5000, 8, 8192, 65536), budget=2048, seed=5000,
                key_chan_scale=(0.5, 4.0), spans=(64, 64), v_outlier=(0.005, 16.0),
                per_doc_seed=True),
}


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bf16 (round-to-nearest-even), returned as uint16 bits."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    rounded = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return rounded.astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float32 (input plumbing only)."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


@dataclass
class LayerInputs:
    """One layer of synthetic inputs as bf16 bit patterns (uint16)."""

    q: np.ndarray          # [batch, H_q, L_t, d]
    k: np.ndarray          # [H_kv, N_total, d]
    v: np.ndarray          # [H_kv, N_total, d]
    doc_offsets: np.ndarray  # [batch + 1] int64
    spans: list            # per document: array of planted span start tokens (doc-local)

    def digest(self) -> str:
        h = hashlib.sha256()
        for a in (self.q, self.k, self.v, self.doc_offsets):
            h.update(np.ascontiguousarray(a).tobytes())
        return h.hexdigest()[:16]


def _draw_doc(rng, w: Workload, n: int):
    """Draw (q, k, v, span_starts) float32 for one document."""
    hq, hkv, d, lt, g = w.n_heads_q, w.n_heads_kv, w.head_dim, w.guide_len, w.group
    q = rng.standard_normal((hq, lt, d), dtype=np.float32)
    if w.key_dist == "normal":
        k = rng.standard_normal((hkv, n, d), dtype=np.float32)
    elif w.key_dist == "student_t3":
        k = (rng.standard_t(3.0, size=(hkv, n, d)) / math.sqrt(3.0)).astype(np.float32)
    else:
        raise ValueError(w.key_dist)
    if w.key_chan_scale is not None:
        lo, hi = w.key_chan_scale
        s = np.exp(rng.uniform(math.log(lo), math.log(hi), size=(hkv, 1, d))).astype(np.float32)
        k *= s
    n_spans, span_len = w.spans
    starts = np.zeros(0, dtype=np.int64)
    if n_spans > 0 and span_len > 0 and n // span_len > 0:
        slots = n // span_len
        m = min(n_spans, slots)
        starts = np.sort(rng.choice(slots, size=m, replace=False)).astype(np.int64) * span_len
        tok = (starts[:, None] + np.arange(span_len)[None, :]).reshape(-1)
        for h in range(hkv):
            u = q[h * g:(h + 1) * g].reshape(-1, d).astype(np.float64).mean(axis=0)
            u /= max(np.linalg.norm(u), 1e-30)
            wv = rng.standard_normal((tok.size, d))
            wv -= np.outer(wv @ u, u)
            wv /= np.maximum(np.linalg.norm(wv, axis=1, keepdims=True), 1e-30)
            norms = np.linalg.norm(k[h, tok].astype(np.float64), axis=1, keepdims=True)
            k[h, tok] = (norms * (0.6 * u[None, :] + 0.8 * wv)).astype(np.float32)
    v = rng.standard_normal((hkv, n, d), dtype=np.float32)
    frac, factor = w.v_outlier
    n_out = int(round(frac * n))
    if n_out > 0:
        for h in range(hkv):
            toks = rng.choice(n, size=n_out, replace=False)
            chans = rng.integers(0, d, size=n_out)
            v[h, toks, chans] *= np.float32(factor)
    return q, k, v, starts


def make_layer(w: Workload, layer: int = 0) -> LayerInputs:
    """Seeded host inputs for one layer of workload ``w``."""
    docs_q, docs_k, docs_v, spans = [], [], [], []
    base = w.seed + layer * 1000003
    rng = np.random.Generator(np.random.PCG64(base))
    for b, n in enumerate(w.doc_lens):
        if w.per_doc_seed:
            rng = np.random.Generator(np.random.PCG64(base + b))
        q, k, v, st = _draw_doc(rng, w, int(n))
        docs_q.append(q)
        docs_k.append(k)
        docs_v.append(v)
        spans.append(st)
    q = np.stack(docs_q, axis=0)
    k = np.concatenate(docs_k, axis=1)
    v = np.concatenate(docs_v, axis=1)
    return LayerInputs(f32_to_bf16_bits(q), f32_to_bf16_bits(k), f32_to_bf16_bits(v),
                       w.doc_offsets(), spans)


def make_layer_torch(w: Workload, layer: int, device, generator=None):
    """Same recipe drawn with torch on ``device``; returns bf16 (q, k, v) tensors.

    Used where drawing on the host would dominate a run (the 32-layer, 128K
    stack is 16 GiB of K/V).  Distributionally identical to ``make_layer``,
    not bitwise.
    """
    import torch

    gen = generator or torch.Generator(device=device)
    gen.manual_seed(w.seed + layer * 1000003)
    hq, hkv, d, lt, g = w.n_heads_q, w.n_heads_kv, w.head_dim, w.guide_len, w.group
    qs, ks, vs = [], [], []
    for n in w.doc_lens:
        n = int(n)
        q = torch.randn((hq, lt, d), generator=gen, device=device, dtype=torch.float32)
        if w.key_dist == "normal":
            k = torch.randn((hkv, n, d), generator=gen, device=device, dtype=torch.float32)
        else:
            # Student-t(3) = N / sqrt(chi2_3 / 3), chi2_3 = sum of 3 squared normals
            z = torch.randn((hkv, n, d), generator=gen, device=device)
            c = torch.randn((3, hkv, n, d), generator=gen, device=device).square().sum(0)
            k = z / torch.sqrt(c / 3.0) / math.sqrt(3.0)
        if w.key_chan_scale is not None:
            lo, hi = w.key_chan_scale
            u = torch.rand((hkv, 1, d), generator=gen, device=device)
            k *= torch.exp(math.log(lo) + u * (math.log(hi) - math.log(lo)))
        n_spans, span_len = w.spans
        if n_spans > 0 and span_len > 0 and n // span_len > 0:
            slots = n // span_len
            m = min(n_spans, slots)
            starts = torch.randperm(slots, generator=gen, device=device)[:m] * span_len
            tok = (starts[:, None] + torch.arange(span_len, device=device)[None, :]).reshape(-1)
            for h in range(hkv):
                u = q[h * g:(h + 1) * g].reshape(-1, d).mean(0)
                u = u / u.norm().clamp_min(1e-30)
                wv = torch.randn((tok.numel(), d), generator=gen, device=device)
                wv = wv - (wv @ u)[:, None] * u[None, :]
                wv = wv / wv.norm(dim=1, keepdim=True).clamp_min(1e-30)
                norms = k[h, tok].norm(dim=1, keepdim=True)
                k[h, tok] = norms * (0.6 * u[None, :] + 0.8 * wv)
        v = torch.randn((hkv, n, d), generator=gen, device=device, dtype=torch.float32)
        frac, factor = w.v_outlier
        n_out = int(round(frac * n))
        if n_out > 0:
            for h in range(hkv):
                toks = torch.randperm(n, generator=gen, device=device)[:n_out]
                chans = torch.randint(0, d, (n_out,), generator=gen, device=device)
                v[h, toks, chans] *= factor
        qs.append(q)
        ks.append(k)
        vs.append(v)
    q = torch.stack(qs, 0).to(torch.bfloat16).contiguous()
    k = torch.cat(ks, 1).to(torch.bfloat16).contiguous()
    v = torch.cat(vs, 1).to(torch.bfloat16).contiguous()
    return q, k, v


#: standard deviation of the synthetic guide keys.  With unit-variance guide
#: queries and the 1/sqrt(d) scale, a guide-prefix logit is N(0, 4), so each
#: prefix term has mean mass e^2, against e^(1/2) for a unit-variance context key
GUIDE_KEY_STD = 2.0


def make_guide_keys(w: Workload, layer: int = 0) -> np.ndarray:
    """Seeded host guide keys [batch, H_kv, L_t, d] (bf16 bits): the post-RoPE
    keys of the guide tokens themselves, N(0, GUIDE_KEY_STD^2)."""
    rng = np.random.Generator(np.random.PCG64(w.seed + layer * 1000003 + 424243))
    x = rng.standard_normal((w.batch, w.n_heads_kv, w.guide_len, w.head_dim), dtype=np.float32)
    return f32_to_bf16_bits(x * np.float32(GUIDE_KEY_STD))


def make_guide_keys_torch(w: Workload, layer: int, device):
    """The guide-key recipe drawn with torch on ``device`` (bf16)."""
    import torch

    gen = torch.Generator(device=device)
    gen.manual_seed(w.seed + layer * 1000003 + 424243)
    x = torch.randn((w.batch, w.n_heads_kv, w.guide_len, w.head_dim), generator=gen, device=device)
    return (x * GUIDE_KEY_STD).to(torch.bfloat16).contiguous()


def small_variant(w: Workload, doc_lens: Sequence[int], layers: int = 1) -> Workload:
    """The same recipe at oracle-friendly sizes (spans shrink to fit)."""
    n_spans, span_len = w.spans
    m = min(doc_lens)
    if span_len and n_spans:
        span_len = min(span_len, max(1, m // 16))
        n_spans = min(n_spans, max(1, m // (4 * span_len)))
    return w.with_(doc_lens=tuple(int(x) for x in doc_lens), layers=layers,
                   spans=(n_spans, span_len))
