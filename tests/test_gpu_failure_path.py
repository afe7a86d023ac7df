"""The failure path every kernel shares, provoked without a fault: a bounded
mbarrier wait on a barrier that nothing arrives at gives up after its limit,
the kernel records TP_ERR_TIMEOUT in the workspace status word and returns,
and the context keeps working."""
import time

import pytest

from paper_2608_03276_gb300 import synth
from tests.test_gpu_parity import SMALL, _check_layer, _oracle, _run_compress

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("limit_ms", [5, 50])
def test_bounded_wait_reports_timeout(cuda_lib, limit_ms):
    import torch
    from paper_2608_03276_gb300 import binding
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    binding.tp_selftest_wait_timeout(ws, limit_ms * 1_000_000)
    st = binding.tp_check_status(ws)
    waited = time.perf_counter() - t0
    assert st == binding.TP_ERR_TIMEOUT, binding.tp_status_string(st)
    assert waited >= limit_ms * 1e-3 * 0.9, waited  # it really waited out its limit
    assert waited < limit_ms * 1e-3 + 5.0

    # the context is intact: a layer right after compresses correctly
    w = SMALL["c1-tiny-2k"]
    x = synth.make_layer(w)
    out = _run_compress(binding, w, x)
    _check_layer(w, x, out, _oracle(w, x))
