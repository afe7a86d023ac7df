"""Canary guard bands around every output and the workspace (a stand-in for a
memory sanitizer): each buffer the library writes sits between two 4 KiB bands
of a known byte, and after the call every band must be untouched.  Covers the
fused layer (both blend kernels, 8- and 4-bit codes, ragged documents with an
empty one), the caller-normaliser and literal-normaliser layers, the stack of
layers (also with the stack workspace, whose short layers are selected four
per launch, and with a guide longer than one 512-row block), and the
stand-alone selection and compaction."""
import numpy as np
import pytest

from paper_2608_03276_gb300 import synth
from tests import parity

pytestmark = pytest.mark.gpu

G = 4096          # guard bytes on each side (keeps every view 256-byte aligned)
CANARY = 0xA5


class Guarded:
    def __init__(self):
        self.bufs = []

    def make(self, shape, dtype):
        import torch
        n = int(np.prod(shape)) * torch.empty((), dtype=dtype).element_size()
        buf = torch.full((G + n + G,), CANARY, dtype=torch.uint8, device="cuda")
        self.bufs.append((buf, n))
        return buf[G:G + n].view(dtype).view(shape)

    def check(self, what):
        import torch
        torch.cuda.synchronize()
        for i, (buf, n) in enumerate(self.bufs):
            head, tail = buf[:G].cpu().numpy(), buf[G + n:].cpu().numpy()
            assert (head == CANARY).all() and (tail == CANARY).all(), f"{what}: buffer {i} guard band written"


def _outputs(binding, gd, p, w, keep_ratio, budget, scores=True):
    import torch
    cap = binding.tp_kept_capacity(p, keep_ratio, budget)
    shp = (w.batch, w.n_heads_kv, cap)
    d, bits = w.head_dim, p.c.quant_bits
    o = type("Out", (), {})()
    o.idx = gd.make(shp, torch.int32)
    o.kc = gd.make(shp + (d,), torch.bfloat16)
    o.vc = gd.make(shp + (d,), torch.bfloat16)
    o.vqc = gd.make(shp + (d * bits // 8,), binding.code_dtype(p))
    o.gammac = gd.make(shp, torch.float32)
    o.scores = gd.make((w.n_heads_kv, w.n_total), torch.float32) if scores else None
    o.gamma = gd.make((w.n_heads_kv, w.n_total), torch.float32) if scores else None
    o.ws = gd.make((binding.tp_workspace_bytes(p, keep_ratio, budget),), torch.uint8)
    return o


RAGGED = synth.small_variant(synth.WORKLOADS[5], [1500, 0, 700, 129, 1]).with_(budget=300)


@pytest.mark.parametrize("flags,bits", [(0, 8), ("TP_SCORE_NORM_ADD", 8), ("TP_SCORE_HARMONIC", 4)])
def test_fused_layer_stays_in_bounds(cuda_lib, flags, bits):
    from paper_2608_03276_gb300 import binding
    w, x = RAGGED, synth.make_layer(RAGGED)
    fl = getattr(binding, flags) if flags else 0
    p = binding.Problem(w.n_heads_q, w.n_heads_kv, w.head_dim, w.guide_len, x.doc_offsets,
                        quant_bits=bits, flags=fl)
    gd = Guarded()
    q, k, v = (parity.to_device_bf16(a) for a in (x.q, x.k, x.v))
    o = _outputs(binding, gd, p, w, w.keep_ratio, w.budget)
    binding.compress(p, q, k, v, w.keep_ratio, w.budget, o)
    assert binding.tp_check_status(o.ws) == 0
    gd.check(f"tp_compress_layer flags={flags} bits={bits}")


@pytest.mark.parametrize("variant", ["lse", "literal"])
def test_normaliser_layers_stay_in_bounds(cuda_lib, variant):
    import torch
    from paper_2608_03276_gb300 import binding
    w, x = RAGGED, synth.make_layer(RAGGED)
    p = binding.Problem(w.n_heads_q, w.n_heads_kv, w.head_dim, w.guide_len, x.doc_offsets)
    gd = Guarded()
    q, k, v = (parity.to_device_bf16(a) for a in (x.q, x.k, x.v))
    o = _outputs(binding, gd, p, w, w.keep_ratio, w.budget)
    if variant == "lse":
        lse = gd.make((w.batch, w.n_heads_kv, w.rows), torch.float32)
        binding.tp_guide_lse(p, q, k, lse, o.ws)
        binding.compress(p, q, k, v, w.keep_ratio, w.budget, o, lse=lse)
    else:
        kg = parity.to_device_bf16(synth.make_guide_keys(w))
        binding.compress(p, q, k, v, w.keep_ratio, w.budget, o, k_guide=kg)
    assert binding.tp_check_status(o.ws) == 0
    gd.check(f"compress ({variant})")


def test_stack_and_stages_stay_in_bounds(cuda_lib):
    import torch
    from paper_2608_03276_gb300 import binding
    w = synth.small_variant(synth.WORKLOADS[2], [3001])
    xs = [synth.make_layer(w, l) for l in range(3)]
    p = binding.Problem(w.n_heads_q, w.n_heads_kv, w.head_dim, w.guide_len, xs[0].doc_offsets)
    gd = Guarded()
    dev = [tuple(parity.to_device_bf16(t) for t in (y.q, y.k, y.v)) for y in xs]
    outs = [_outputs(binding, gd, p, w, w.keep_ratio, w.budget, scores=False) for _ in xs]
    binding.tp_compress_layers(p, dev, w.keep_ratio, w.budget, outs, outs[0].ws)
    assert binding.tp_check_status(outs[0].ws) == 0
    gd.check("tp_compress_layers")
    # the stages on their own
    q, k, v = dev[0]
    o = outs[0]
    gamma = gd.make((w.n_heads_kv, w.n_total), torch.float32)
    scores = gd.make((w.n_heads_kv, w.n_total), torch.float32)
    vq = gd.make((w.n_heads_kv, w.n_total, w.head_dim), torch.int8)
    binding.tp_quantize_v(p, v, vq, gamma)
    binding.tp_guide_scores(p, q, k, gamma, scores, o.ws)
    binding.tp_select(p, scores, w.keep_ratio, w.budget, o.idx, o.ws)
    binding.tp_compact(p, k, v, gamma, o.idx, w.keep_ratio, w.budget, o.kc, o.vc, o.vqc, o.gammac)
    gd.check("stand-alone stages")


@pytest.mark.parametrize("lt", [64, 160])
def test_grouped_and_long_guide_stacks_stay_in_bounds(cuda_lib, lt):
    """Both stacks with the stack workspace (the later layers' key scores,
    scales and selection scratch in slots after the single-layer workspace):
    guide 64 (256 rows) selects layers several per launch, guide 160 (640
    rows) also scores in blocks of 512 rows."""
    import torch
    from paper_2608_03276_gb300 import binding
    w = synth.small_variant(synth.WORKLOADS[2], [3001]).with_(guide_len=lt)
    nl = 5
    xs = [synth.make_layer(w, l) for l in range(nl)]
    p = binding.Problem(w.n_heads_q, w.n_heads_kv, w.head_dim, w.guide_len, xs[0].doc_offsets)
    gd = Guarded()
    dev = [tuple(parity.to_device_bf16(t) for t in (y.q, y.k, y.v)) for y in xs]
    ws = gd.make((binding.tp_workspace_bytes_stack(p, w.keep_ratio, w.budget, nl),), torch.uint8)
    outs = [_outputs(binding, gd, p, w, w.keep_ratio, w.budget, scores=False) for _ in xs]
    binding.tp_compress_layers(p, dev, w.keep_ratio, w.budget, outs, ws)
    assert binding.tp_check_status(ws) == 0
    gd.check(f"tp_compress_layers, stack workspace, guide {lt}")
    lses = [gd.make((w.batch, w.n_heads_kv, w.rows), torch.float32) for _ in xs]
    for (q, k, _), lse in zip(dev, lses):
        binding.tp_guide_lse(p, q, k, lse, outs[0].ws)
    binding.tp_compress_layers_lse(p, dev, lses, w.keep_ratio, w.budget, outs, ws)
    assert binding.tp_check_status(ws) == 0
    gd.check(f"tp_compress_layers_lse, stack workspace, guide {lt}")
