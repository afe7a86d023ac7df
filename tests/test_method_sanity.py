"""Method-level sanity of the oracle on the planted workloads (not parity).

The synthetic inputs plant spans of keys aligned with the guide queries
(cos 0.6) and give a few tokens a V outlier channel.  The method should then
keep the planted spans (guide attention, Eq. 1) and, under a guide that
attends to nothing in particular, keep the outlier tokens first (the scale
signal, Eq. 2-3).  As the number of planted spans grows at a fixed budget,
recall of them falls: the attention dilution the paper discusses for dense
needle tasks (App. B).  The GPU path matches the oracle's kept sets (the
parity tests), so these figures hold for it too.
"""
import numpy as np

from oracle import taskpress_oracle as O
from paper_2608_03276_gb300 import synth
from tests import parity


def _recall(out, x, w, h):
    span = np.concatenate([np.arange(s, s + w.spans[1]) for s in x.spans[0]])
    kept = set(out["idx"][(0, h)].tolist())
    return float(np.mean([t in kept for t in span]))


def _layer(w, **kw):
    x = synth.make_layer(w)
    return x, O.compress_layer(x.q, x.k, x.v, x.doc_offsets, n_heads_q=w.n_heads_q,
                               n_heads_kv=w.n_heads_kv, keep_ratio=w.keep_ratio,
                               fixed_budget=w.budget, **kw)


def test_planted_spans_are_kept():
    """Tiny workload (4 spans of 32 aligned keys in 2048 tokens, keep 25%): the
    guide-attention score alone keeps every planted token; weighted by the
    scales (Eq. 3) it still keeps most of them."""
    w = synth.WORKLOADS[1]
    x, key_only = _layer(w, key_only=True)
    _, product = _layer(w)
    for h in range(w.n_heads_kv):
        assert _recall(key_only, x, w, h) >= 0.95
        assert _recall(product, x, w, h) >= 0.8
        parity.REPORTS.append(f"tiny workload head {h}: planted-span recall {_recall(product, x, w, h):.3f} "
                              f"(key-only {_recall(key_only, x, w, h):.3f})")


def test_outliers_kept_first_under_a_flat_guide():
    """With a zero guide every token gets the same attention, so the ranking is
    the scale's: every token with a V outlier channel (absmax far above the
    rest) is kept while the budget lasts."""
    w = synth.WORKLOADS[1]
    x = synth.make_layer(w)
    q = np.zeros_like(x.q)
    out = O.compress_layer(q, x.k, x.v, x.doc_offsets, n_heads_q=w.n_heads_q,
                           n_heads_kv=w.n_heads_kv, keep_ratio=w.keep_ratio)
    vmax = np.abs(O.decode_bf16(x.v)).max(axis=-1)
    for h in range(w.n_heads_kv):
        outliers = np.flatnonzero(vmax[h] > 8.0)
        assert 0 < outliers.size <= out["k"][0]
        assert set(outliers.tolist()) <= set(out["idx"][(0, h)].tolist())


def test_dilution_with_more_spans():
    """Fixed budget of 128 tokens, 1 / 4 / 16 / 64 planted spans of 32 tokens:
    recall of the planted tokens falls as they outnumber the budget."""
    recalls = []
    for ns in (1, 4, 16, 64):
        w = synth.WORKLOADS[1].with_(spans=(ns, 32), seed=11, budget=128)
        x, out = _layer(w)
        recalls.append(float(np.mean([_recall(out, x, w, h) for h in range(w.n_heads_kv)])))
    parity.REPORTS.append("dilution (budget 128, spans 1/4/16/64 of 32 tokens): recall "
                          + " / ".join(f"{r:.3f}" for r in recalls))
    assert all(a >= b for a, b in zip(recalls, recalls[1:]))
    assert recalls[0] > 0.8 and recalls[-1] < 0.2
