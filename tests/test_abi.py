"""C ABI checks that need no GPU: the library loads, exports every declared
symbol, and its host-side logic (budget rule, capacity, workspace sizing,
argument validation) behaves as include/taskpress.h states."""
import math
import os
import re
from fractions import Fraction

import pytest

from oracle import taskpress_oracle as O

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2608_03276_gb300 import build as b
    from paper_2608_03276_gb300 import binding
    b.build()
    return binding


def declared_symbols():
    with open(os.path.join(ROOT, "include", "taskpress.h")) as f:
        src = f.read()
    return sorted(set(re.findall(r"^\s*(?:[\w\*]+\s+)+\**(tp_\w+)\s*\(", src, re.M)))


def test_exports_every_declared_symbol(lib):
    names = declared_symbols()
    assert len(names) == 23, names
    assert sorted(lib.EXPORTS) == names
    cdll = lib.load()
    for n in names:
        assert hasattr(cdll, n), n


def test_missing_library_fails_loudly(tmp_path):
    """The binding has no fallback: without the built library every call
    raises (a fresh copy of the module, pointed at a path with no library)."""
    import importlib.util
    spec = importlib.util.spec_from_file_location(
        "binding_copy", os.path.join(ROOT, "paper_2608_03276_gb300", "binding.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    with pytest.raises(RuntimeError, match="not built"):
        mod.load(str(tmp_path / "libtaskpress.so"))


def test_budget_matches_oracle_and_exact_decimals(lib):
    for r in ["0", "0.05", "0.07", "0.1", "0.2", "0.25", "0.33", "0.5", "0.9", "1"]:
        for n in [0, 1, 2, 7, 100, 129, 2048, 32768, 65536, 131072, 294912]:
            got = lib.tp_budget(n, float(r))
            assert got == O.budget(n, float(r)) == math.ceil(Fraction(r) * n), (r, n, got)
    assert lib.tp_budget(10, -0.5) == -1 and lib.tp_budget(10, 1.01) == -1
    assert lib.tp_budget(10, float("nan")) == -1 and lib.tp_budget(-1, 0.5) == -1


def _prob(lib, offs, **kw):
    args = dict(n_heads_q=8, n_heads_kv=2, head_dim=64, guide_len=16, doc_offsets=offs)
    args.update(kw)
    return lib.Problem(**args)


def test_capacity_and_workspace(lib):
    p = _prob(lib, [0, 1000, 1001, 3000])
    assert lib.tp_kept_capacity(p, 0.25, -1) == 500
    assert lib.tp_kept_capacity(p, 0.0, 300) == 300
    assert lib.tp_kept_capacity(p, 0.0, 5000) == 1999
    assert lib.tp_kept_capacity(p, 1.5, -1) == -1
    assert lib.tp_workspace_bytes(p, 0.25, -1) > 3000 * 2 * 12
    assert lib.tp_workspace_bytes(p, 0.25, -1) % 256 == 0


@pytest.mark.parametrize("kw", [
    dict(head_dim=96), dict(head_dim=256), dict(pool_kernel=4), dict(pool_kernel=0), dict(pool_kernel=35),
    dict(quant_bits=2), dict(quant_bits=16), dict(n_heads_q=7), dict(guide_len=0), dict(guide_len=1025, n_heads_q=16),
])
def test_rejects_unsupported(lib, kw):
    p = _prob(lib, [0, 100], **kw)
    assert lib.tp_kept_capacity(p, 0.5, -1) == -1
    assert lib.tp_workspace_bytes(p, 0.5, -1) == 0


def test_long_guide_plan(lib):
    """More than TP_MAX_ROWS stacked guide rows run in blocks of 512: the
    workspace adds one fp32 normaliser per row, document and head and one
    fp32 key score per token and head; the two entry points without a
    workspace refuse such guides before any launch; above TP_MAX_GUIDE_ROWS
    nothing takes them.  The addresses below are never dereferenced."""
    offs = [0, 1000, 3000]
    shape = dict(n_heads_q=8, n_heads_kv=2, head_dim=128)
    w512 = lib.tp_workspace_bytes(_prob(lib, offs, guide_len=128, **shape), 0.25, -1)  # M 512
    p1024 = _prob(lib, offs, guide_len=256, **shape)                                   # M 1024
    up = lambda b: (b + 255) // 256 * 256
    assert lib.tp_workspace_bytes(p1024, 0.25, -1) == w512 + up(4 * 2 * 2 * 1024) + up(4 * 2 * 3000)
    assert lib.TP_MAX_GUIDE_ROWS == 8192
    assert lib.tp_workspace_bytes(_prob(lib, offs, guide_len=2048, **shape), 0.25, -1) > 0   # M 8192
    assert lib.tp_workspace_bytes(_prob(lib, offs, guide_len=2049, **shape), 0.25, -1) == 0  # M 8196
    cdll = lib.load()
    ok = 0x10000
    assert cdll.tp_guide_key_scores(p1024.ref(), ok, ok, None, ok, ok, None, None) == \
        lib.TP_ERR_UNSUPPORTED_SHAPE
    assert cdll.tp_guide_lse_static(p1024.ref(), ok, ok, None, ok, None, None) == \
        lib.TP_ERR_UNSUPPORTED_SHAPE
    # per further block: pass 1, pass 2 and the addition of its key scores
    # (two-pass); pass 2 and the addition (caller's normalisers)
    p = lib.Problem(32, 8, 128, 275, [0, 65536])  # M 1100: blocks of 512, 512, 76
    assert lib.tp_compress_kernel_count(p, 0.1, -1, lib.MODE_TWO_PASS) == 4 + 2 * 3
    assert lib.tp_compress_kernel_count(p, 0.1, -1, lib.MODE_LITERAL) == 5 + 2 * 3
    import torch
    if not torch.cuda.is_available():
        assert lib.tp_compress_kernel_count(p, 0.1, -1, lib.MODE_CALLER_LSE) == 4 + 2 * 2


def test_stack_workspace(lib):
    """tp_workspace_bytes_stack adds, for documents of at most 65536 tokens and
    up to 7 further layers, one more layer's key scores, scales and selection
    scratch (3 x 4 bytes per token and head, each array 256-byte aligned);
    above 65536 tokens, or for one layer, it is tp_workspace_bytes.  The
    grouping query answers 1 where the workspace has no room, for the
    normalised-add score, and without a device to ask."""
    offs = [0, 1000, 3000]
    p = _prob(lib, offs)
    base = lib.tp_workspace_bytes(p, 0.25, -1)
    slot = 3 * ((4 * 2 * 3000 + 255) // 256 * 256)
    assert lib.tp_workspace_bytes_stack(p, 0.25, -1, 1) == base
    assert lib.tp_workspace_bytes_stack(p, 0.25, -1, 4) == base + 3 * slot
    assert lib.tp_workspace_bytes_stack(p, 0.25, -1, 40) == base + 7 * slot
    long_doc = _prob(lib, [0, 65537])
    assert lib.tp_workspace_bytes_stack(long_doc, 0.25, -1, 4) == lib.tp_workspace_bytes(long_doc, 0.25, -1)
    assert lib.load().tp_workspace_bytes_stack(p.ref(), 0.25, -1, -1) == 0
    assert lib.tp_stack_layers_per_selection(p, 0.25, -1, 4, base) == 1
    nadd = _prob(lib, offs, flags=lib.TP_SCORE_NORM_ADD)
    assert lib.tp_stack_layers_per_selection(nadd, 0.25, -1, 4, base + 3 * slot) == 1
    import torch
    if not torch.cuda.is_available():
        assert lib.tp_stack_layers_per_selection(p, 0.25, -1, 4, base + 3 * slot) == 1
    with pytest.raises(lib.TaskPressError):
        lib.tp_stack_layers_per_selection(p, 0.25, -1, 0, base)


def test_rejects_bad_offsets(lib):
    assert lib.tp_kept_capacity(_prob(lib, [1, 100]), 0.5, -1) == -1
    assert lib.tp_kept_capacity(_prob(lib, [0, 100, 50]), 0.5, -1) == -1
    assert lib.tp_kept_capacity(_prob(lib, list(range(0, 258))), 0.5, -1) == -1


def test_score_flags(lib):
    for f in (0, lib.TP_SCORE_KEY_ONLY, lib.TP_SCORE_NORM_ADD, lib.TP_SCORE_HARMONIC):
        assert lib.tp_kept_capacity(_prob(lib, [0, 100], flags=f), 0.5, -1) == 50
    for f in (lib.TP_SCORE_NORM_ADD | lib.TP_SCORE_HARMONIC, lib.TP_SCORE_KEY_ONLY | lib.TP_SCORE_NORM_ADD,
              0x8, 0x100):
        assert lib.tp_kept_capacity(_prob(lib, [0, 100], flags=f), 0.5, -1) == -1


def test_null_pointers_rejected_before_any_launch(lib):
    cdll = lib.load()
    p = _prob(lib, [0, 100])
    assert cdll.tp_quantize_v(p.ref(), None, None, None, None) == lib.TP_ERR_INVALID_ARG
    assert cdll.tp_compress_layer(p.ref(), None, None, None, 0.5, -1, None, None, None, None, None,
                                  None, None, None, 0, None) == lib.TP_ERR_INVALID_ARG
    assert cdll.tp_compress_layer_lse(p.ref(), None, None, None, None, 0.5, -1, None, None, None, None,
                                      None, None, None, None, 0, None) == lib.TP_ERR_INVALID_ARG
    assert cdll.tp_compress_layer_guide(p.ref(), None, None, None, None, 0.5, -1, None, None, None,
                                        None, None, None, None, None, 0, None) == lib.TP_ERR_INVALID_ARG
    assert cdll.tp_guide_prefix_lse(p.ref(), None, None, None, None) == lib.TP_ERR_INVALID_ARG
    assert cdll.tp_select(p.ref(), None, 0.5, -1, None, None, 0, None) == lib.TP_ERR_INVALID_ARG
    assert cdll.tp_status_string(-5) == b"device-side wait timed out"


def test_layer_stack_arguments_rejected_before_any_launch(lib):
    """tp_compress_layers checks every layer's pointers (present, 16-byte
    aligned) and the workspace before it enqueues anything.  The addresses
    below are never dereferenced."""
    from ctypes import c_void_p
    cdll = lib.load()
    p = _prob(lib, [0, 100])

    def arr(*xs):
        a = (c_void_p * len(xs))()
        for i, x in enumerate(xs):
            a[i] = x
        return a

    good = 0x10000
    q, k, v, idx = arr(good, good), arr(good, good), arr(good, good), arr(good, good)
    call = lambda n, q_, k_, v_, idx_, ws, ws_bytes: cdll.tp_compress_layers(
        p.ref(), n, q_, k_, v_, 0.5, -1, idx_, None, None, None, None, ws, ws_bytes, None)
    assert call(-1, q, k, v, idx, good, 1 << 30) == lib.TP_ERR_INVALID_ARG
    assert call(2, None, k, v, idx, good, 1 << 30) == lib.TP_ERR_INVALID_ARG
    assert call(2, arr(good, None), k, v, idx, good, 1 << 30) == lib.TP_ERR_INVALID_ARG
    assert call(2, q, arr(good, good + 8), v, idx, good, 1 << 30) == lib.TP_ERR_INVALID_ARG
    assert call(2, q, k, v, arr(good, None), good, 1 << 30) == lib.TP_ERR_INVALID_ARG
    assert call(2, q, k, v, idx, None, 1 << 30) == lib.TP_ERR_WORKSPACE
    assert call(2, q, k, v, idx, good, 16) == lib.TP_ERR_WORKSPACE
    assert call(0, None, None, None, None, good, 1 << 30) == 0  # an empty stack is a no-op


def test_code_buffer_alignment(lib):
    """b = 4 code buffers need 4-byte alignment, b = 8 ones 8-byte."""
    cdll = lib.load()
    for bits, bad in ((8, 0x10004), (4, 0x10002)):
        p = _prob(lib, [0, 100], quant_bits=bits)
        assert cdll.tp_quantize_v(p.ref(), 0x10000, bad, 0x10000, None) == lib.TP_ERR_INVALID_ARG


def test_quantize_rows_arguments(lib):
    cdll = lib.load()
    ok = 0x10000
    assert cdll.tp_quantize_rows(ok, -1, 128, 8, ok, ok, None) == lib.TP_ERR_INVALID_ARG
    assert cdll.tp_quantize_rows(ok, 10, 96, 8, ok, ok, None) == lib.TP_ERR_UNSUPPORTED_SHAPE
    assert cdll.tp_quantize_rows(ok, 10, 128, 6, ok, ok, None) == lib.TP_ERR_UNSUPPORTED_SHAPE
    assert cdll.tp_quantize_rows(ok + 8, 10, 128, 8, ok, ok, None) == lib.TP_ERR_INVALID_ARG
    assert cdll.tp_quantize_rows(ok, 10, 128, 8, ok + 4, ok, None) == lib.TP_ERR_INVALID_ARG
    assert cdll.tp_quantize_rows(ok, 10, 128, 4, ok, None, None) == lib.TP_ERR_INVALID_ARG
    assert cdll.tp_quantize_rows(None, 0, 128, 4, None, None, None) == 0  # nothing to do


def test_selftest_arguments(lib):
    cdll = lib.load()
    assert cdll.tp_selftest_wait_timeout(None, 256, 1000, None) == lib.TP_ERR_WORKSPACE
    assert cdll.tp_selftest_wait_timeout(0x10000, 2, 1000, None) == lib.TP_ERR_WORKSPACE
    assert cdll.tp_selftest_wait_timeout(0x10000, 256, 0, None) == lib.TP_ERR_INVALID_ARG
    assert cdll.tp_selftest_wait_timeout(0x10000, 256, 2_000_000_000, None) == lib.TP_ERR_INVALID_ARG


def test_kernel_count_query(lib):
    """The fused calls launch pass 1, [the prefix fold,] pass 2, the selection
    and, when anything is kept, the compaction.  With the caller's normalisers
    pass 2 also forms the V scales where that kernel fits (up to 256 guide
    rows on one CTA per key range: a plan decision, known without a GPU; more
    rows need co-resident CTA pairs, which a host without a GPU cannot
    confirm, so it counts the separate V-scale pass)."""
    p = lib.Problem(32, 8, 128, 128, [0, 131072])
    assert lib.tp_compress_kernel_count(p, 0.1, -1, lib.MODE_TWO_PASS) == 4
    import torch
    if not torch.cuda.is_available():
        assert lib.tp_compress_kernel_count(p, 0.1, -1, lib.MODE_CALLER_LSE) == 4
    p256 = lib.Problem(32, 8, 128, 64, [0, 32768])
    assert lib.tp_compress_kernel_count(p256, 0.1, -1, lib.MODE_CALLER_LSE) == 3
    assert lib.tp_compress_kernel_count(p256, 0.1, -1, lib.MODE_TWO_PASS) == 4
    assert lib.tp_compress_kernel_count(p, 0.1, -1, lib.MODE_LITERAL) == 5
    assert lib.tp_compress_kernel_count(p, 0.0, -1, lib.MODE_TWO_PASS) == 3
    empty = lib.Problem(4, 1, 128, 16, [0, 0])
    assert lib.tp_compress_kernel_count(empty, 0.1, -1, lib.MODE_TWO_PASS) == 1
    with pytest.raises(lib.TaskPressError):
        lib.tp_compress_kernel_count(p, 1.5, -1)
