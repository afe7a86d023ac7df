"""The benchmark's accounting, on the CPU: the algorithmic bytes and flops it
divides by, the HBM fraction it reports, and the ncu traffic record it quotes.

The expected figures are the workloads' own arithmetic, written out here
independently of bench.py: K + V read once (4 d bytes per token and head),
the guide read once, 648 bytes per kept token and head written (K, V, 8-bit V
codes, scale, index at d = 128), and one QK^T of 2 M n d flops per head.
"""
import os

import pytest

import bench
from paper_2608_03276_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.parametrize("cfg,kept_per_head,read,write,flops", [
    # Llama-3-8B-shaped 128K layer, guide 128, keep 10%: 13108 kept per head
    (3, 13108, 8 * 131072 * 512 + 2 * 128 * 32 * 128, 648 * 13108 * 8, 2 * 512 * 128 * 131072 * 8),
    # 32K layer, guide 64, keep 20%: 6554 kept per head
    (2, 6554, 8 * 32768 * 512 + 2 * 128 * 32 * 64, 648 * 6554 * 8, 2 * 256 * 128 * 32768 * 8),
    # 64K wide-GQA layer (28 q / 4 KV heads), guide 32, keep 5%: 3277 kept per head
    (4, 3277, 4 * 65536 * 512 + 2 * 128 * 28 * 32, 648 * 3277 * 4, 2 * 224 * 128 * 65536 * 4),
])
def test_layer_algorithmic(cfg, kept_per_head, read, write, flops):
    w = synth.WORKLOADS[cfg]
    got = bench.layer_algorithmic(w, kept_per_head * w.n_heads_kv)
    assert got == (read, write, flops)


def test_headline_bytes_match_the_stated_figures():
    """605,871,360 bytes per 128K layer (537 MB of K and V, 1 MB of guide, 68 MB
    of cache) and 168,717,952 per 32K layer."""
    w3, w2 = synth.WORKLOADS[3], synth.WORKLOADS[2]
    assert sum(bench.layer_algorithmic(w3, 13108 * 8)[:2]) == 605_871_360
    assert sum(bench.layer_algorithmic(w2, 6554 * 8)[:2]) == 168_717_952


def test_hbm_fraction():
    w = synth.WORKLOADS[3]
    r = bench.hbm_fused_of(w, 13108 * 8, 100e-6, 6000.0, "measured")
    assert r["algorithmic_bytes"] == 605_871_360
    assert r["achieved_gbs"] == pytest.approx(605_871_360 / 100e-6 / 1e9)
    assert r["frac"] == pytest.approx(r["achieved_gbs"] / 6000.0)
    assert r["frac_of_nominal_8tbs"] == pytest.approx(r["achieved_gbs"] / 8000.0)


def test_traffic_record_follows_the_kernel_source():
    """The committed ncu traffic is quoted only while score_tc.cu is the source
    it was captured from (its hash is in the summary's third column)."""
    import hashlib
    src = os.path.join(ROOT, "paper_2608_03276_gb300", "csrc", "score_tc.cu")
    sha = hashlib.sha256(open(src, "rb").read()).hexdigest()[:12]
    rows = {}
    with open(os.path.join(ROOT, "profiles", "ncu_traffic.txt")) as f:
        for line in f:
            parts = line.split()
            if len(parts) >= 4 and not line.startswith("#"):
                rows[(parts[0], parts[1], parts[2])] = float(parts[3])
    want = rows.get(("tp_lse_kernel", "llama8b-stack32-128k", sha))
    assert bench.traffic_record("tp_lse_kernel", "llama8b-stack32-128k") == want
    assert bench.traffic_record("no_such_kernel", "llama8b-stack32-128k") is None
