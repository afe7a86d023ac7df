"""The seeded generator is deterministic and follows its stated recipe."""
import numpy as np

from paper_2608_03276_gb300 import synth


def test_deterministic_and_shapes():
    w = synth.small_variant(synth.WORKLOADS[2], [1000, 333])
    a, b = synth.make_layer(w), synth.make_layer(w)
    assert a.digest() == b.digest()
    assert a.q.shape == (2, 32, 64, 128) and a.k.shape == (8, 1333, 128) and a.v.shape == a.k.shape
    assert list(a.doc_offsets) == [0, 1000, 1333]
    c = synth.make_layer(w, layer=1)
    assert c.digest() != a.digest()


def test_planted_span_alignment():
    w = synth.small_variant(synth.WORKLOADS[1], [2048])
    x = synth.make_layer(w)
    q = synth.bf16_bits_to_f32(x.q).astype(np.float64)
    k = synth.bf16_bits_to_f32(x.k).astype(np.float64)
    g = w.group
    starts = x.spans[0]
    assert len(starts) == w.spans[0]
    for h in range(w.n_heads_kv):
        u = q[0, h * g:(h + 1) * g].reshape(-1, w.head_dim).mean(0)
        u /= np.linalg.norm(u)
        for s in starts:
            kk = k[h, s:s + w.spans[1]]
            cos = kk @ u / np.linalg.norm(kk, axis=1)
            assert np.all(np.abs(cos - 0.6) < 0.02), cos


def test_value_outliers():
    w = synth.small_variant(synth.WORKLOADS[1], [2048])
    x = synth.make_layer(w)
    v = np.abs(synth.bf16_bits_to_f32(x.v))
    per_tok = v.max(-1)
    for h in range(w.n_heads_kv):
        n_out = int(round(0.01 * 2048))
        assert n_out * 0.5 <= (per_tok[h] > 6.0).sum() <= n_out + 2


def test_ragged_workload():
    w = synth.WORKLOADS[5]
    assert w.batch == 8 and all(8192 <= n <= 65536 for n in w.doc_lens)
    assert w.budget == 2048


def test_bf16_round_to_nearest_even():
    x = np.array([1.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -2.5, 0.0], np.float32)
    got = synth.bf16_bits_to_f32(synth.f32_to_bf16_bits(x))
    assert list(got) == [1.0, 1.0, 1.0 + 4 * 2 ** -8, -2.5, 0.0]
