"""One layer compressed by a plain C program through the C ABI
(tests/c/compress_layer.c: cudaMalloc, tp_compress_layer, tp_check_status, no
Python in the call path).  Its kept indices, int8 codes and scales must equal
the Python binding's on the same inputs bit for bit, and its kept sets must
be the oracle's."""
import os
import shutil
import struct
import subprocess

import numpy as np
import pytest

from paper_2608_03276_gb300 import synth
from tests import parity
from tests.test_gpu_parity import SMALL, _oracle, _run_compress

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _cuda_home():
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    return os.path.dirname(os.path.dirname(os.path.realpath(nvcc)))


@pytest.mark.parametrize("name", ["c2-llama-4133", "c5-ragged"])
def test_c_caller_layer(cuda_lib, tmp_path, name):
    from paper_2608_03276_gb300 import binding, build
    if shutil.which("gcc") is None:
        pytest.skip("gcc not available")
    lib = build.build()
    cuda = _cuda_home()
    exe = tmp_path / "compress_layer"
    cmd = ["gcc", "-std=c99", "-Wall", "-Werror", "-I", os.path.join(ROOT, "include"),
           "-I", os.path.join(cuda, "include"), os.path.join(ROOT, "tests", "c", "compress_layer.c"),
           "-o", str(exe), "-L", os.path.dirname(lib), "-ltaskpress", "-L", os.path.join(cuda, "lib64"),
           "-lcudart", "-Wl,-rpath," + os.path.dirname(lib), "-Wl,-rpath," + os.path.join(cuda, "lib64")]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr

    w = SMALL[name]
    x = synth.make_layer(w)
    offs = np.asarray(x.doc_offsets, dtype=np.int64)
    inp, out = tmp_path / "in.bin", tmp_path / "out.bin"
    with open(inp, "wb") as f:
        f.write(struct.pack("<5i", w.n_heads_q, w.n_heads_kv, w.head_dim, w.guide_len, len(offs) - 1))
        f.write(struct.pack("<d", w.keep_ratio))
        f.write(offs.tobytes())
        for t in (x.q, x.k, x.v):
            f.write(np.ascontiguousarray(t, dtype=np.uint16).tobytes())
    r = subprocess.run([str(exe), str(inp), str(out)], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stdout + r.stderr

    raw = open(out, "rb").read()
    cap = struct.unpack_from("<q", raw, 0)[0]
    batch, hkv, d = len(offs) - 1, w.n_heads_kv, w.head_dim
    m = batch * hkv * cap
    o = 8
    idx = np.frombuffer(raw, np.int32, m, o).reshape(batch, hkv, cap)
    o += 4 * m
    vqc = np.frombuffer(raw, np.int8, m * d, o).reshape(batch, hkv, cap, d)
    o += m * d
    gc = np.frombuffer(raw, np.float32, m, o).reshape(batch, hkv, cap)

    ref = _run_compress(binding, w, x, budget=-1)  # the same call through the Python binding
    assert np.array_equal(idx, ref.idx.cpu().numpy())
    assert np.array_equal(vqc, ref.vqc.cpu().numpy())
    assert np.array_equal(gc.view(np.uint32), ref.gammac.cpu().numpy().view(np.uint32))
    orc = _oracle(w, x, budget=-1)
    scores = ref.scores.cpu().numpy()
    for b in range(batch):
        lo, hi = int(offs[b]), int(offs[b + 1])
        for h in range(hkv):
            parity.assert_kept(idx[b, h], orc["k"][b], orc["scores"][(b, h)], scores[h, lo:hi],
                               f"doc {b} head {h}")
