"""The pooled oracle (one process per (document, KV head) unit, used by the
full-size GPU parity tests) gives exactly what oracle.compress_layer gives on
the whole layer: units are independent."""
import numpy as np

from oracle import taskpress_oracle as O
from paper_2608_03276_gb300 import synth
from tests import oracle_pool


def test_pooled_oracle_equals_whole_layer():
    w = synth.small_variant(synth.WORKLOADS[5], [300, 0, 177]).with_(budget=50)
    x = synth.make_layer(w)
    lse = np.random.Generator(np.random.PCG64(3)).uniform(2.0, 6.0, (w.batch, w.n_heads_kv, w.rows))
    for kw in ({}, {"lse": lse}, {"quant_bits": 4}):
        whole = O.compress_layer(x.q, x.k, x.v, x.doc_offsets, n_heads_q=w.n_heads_q,
                                 n_heads_kv=w.n_heads_kv, fixed_budget=w.budget, **kw)
        pooled = oracle_pool.compress_layer(x, w.n_heads_q, w.n_heads_kv, fixed_budget=w.budget, **kw)
        assert np.array_equal(whole["gamma"].view(np.uint32), pooled["gamma"].view(np.uint32))
        assert np.array_equal(whole["vq"], pooled["vq"])
        assert whole["k"] == pooled["k"]
        for key in whole["scores"]:
            assert np.array_equal(whole["scores"][key], pooled["scores"][key])
            assert np.array_equal(whole["key"][key], pooled["key"][key])
            assert np.array_equal(whole["idx"][key], pooled["idx"][key])
