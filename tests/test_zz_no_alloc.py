"""tp_guide_lse_static: pass 1 without a caller-provided workspace.

Some callers cannot allocate device memory (for example code running inside a
CUDA stream capture or a framework hook that hands over only a stream and the
tensors).  This entry point uses the library's fixed device scratch instead of
a workspace; its results must match tp_guide_lse, which uses one.  Two calls in
a row check that leftover scratch contents from the first call do not leak
into the second.  Collected last so that a failure here cannot hide the
other tests of a run that stops at the first failure.
"""
import numpy as np
import pytest

from paper_2608_03276_gb300 import synth
from tests import parity

pytestmark = pytest.mark.gpu


def test_static_scratch_matches_workspace_entry(cuda_lib):
    import torch
    from paper_2608_03276_gb300 import binding
    for w in (synth.small_variant(synth.WORKLOADS[2], [4133]),
              synth.small_variant(synth.WORKLOADS[5], [1500, 1, 700, 2304])):
        x = synth.make_layer(w)
        p = binding.Problem(w.n_heads_q, w.n_heads_kv, w.head_dim, w.guide_len, x.doc_offsets)
        q, k, v = (parity.to_device_bf16(a) for a in (x.q, x.k, x.v))
        shape = (w.batch, w.n_heads_kv, w.rows)
        ws = torch.empty(binding.tp_workspace_bytes(p), dtype=torch.uint8, device="cuda")
        ref = torch.empty(shape, dtype=torch.float32, device="cuda")
        ref_g = torch.empty((w.n_heads_kv, p.n_total), dtype=torch.float32, device="cuda")
        binding.tp_guide_lse(p, q, k, ref, ws, v=v, gamma=ref_g)
        for _ in range(2):
            got = torch.full(shape, float("nan"), dtype=torch.float32, device="cuda")
            got_g = torch.full_like(ref_g, float("nan"))
            binding.tp_guide_lse_static(p, q, k, got, v=v, gamma=got_g)
            torch.cuda.synchronize()
            # the same kernel on the same inputs, its partials merged in a fixed
            # CTA order: the normalisers must agree bit for bit
            a, b = got.cpu().numpy(), ref.cpu().numpy()
            assert np.all(np.isfinite(a))
            assert np.array_equal(a.view(np.uint32), b.view(np.uint32))
            assert np.array_equal(got_g.cpu().numpy().view(np.uint32),
                                  ref_g.cpu().numpy().view(np.uint32))


def test_static_scratch_rejects_oversized_problem(cuda_lib):
    import torch
    from paper_2608_03276_gb300 import binding
    # 256 documents x 64 KV heads: the per-CTA partials exceed the 2 MiB scratch
    offs = np.arange(0, 257 * 4096, 4096, dtype=np.int64)
    p = binding.Problem(512, 64, 128, 1, offs)
    cdll = binding.load()
    dummy = torch.zeros(16, dtype=torch.float32, device="cuda")
    st = cdll.tp_guide_lse_static(p.ref(), dummy.data_ptr(), dummy.data_ptr(), None,
                                  dummy.data_ptr(), None, None)
    assert st == binding.TP_ERR_WORKSPACE
