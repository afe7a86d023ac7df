"""Plant plausible mistakes in copies of the oracle; each must trip some pin.

Every mutation is a literal source edit of oracle/taskpress_oracle.py, loaded
as a separate module on the CPU.  A mutation that no pin catches would mean
the pins leave that part of the oracle unchecked.
"""
import inspect
import types

import pytest

from oracle import taskpress_oracle as O
from tests import oracle_pins

SRC = inspect.getsource(O)

MUTATIONS = {
    "softmax over the wrong axis": ("z = np.sum(e, axis=1, keepdims=True)", "z = np.sum(e, axis=0, keepdims=True)"),
    "scale 1/d instead of 1/sqrt(d)": ("1.0 / math.sqrt(d)\n    gamma", "1.0 / d\n    gamma"),
    "no max subtraction": ("e = np.exp(x - m)", "e = np.exp(x)"),
    "row normaliser drops the max": ("return m + np.log(np.sum(np.exp(x - m[:, None]), axis=1))", "return np.log(np.sum(np.exp(x), axis=1))"),
    "row normaliser summed over every row": ("return m + np.log(np.sum(np.exp(x - m[:, None]), axis=1))", "return m + np.log(np.sum(np.exp(x - m[:, None])))"),
    "row normaliser log2": ("return m + np.log(np.sum(np.exp(x - m[:, None]), axis=1))", "return m + np.log2(np.sum(np.exp(x - m[:, None]), axis=1))"),
    "sum over the GQA group": ("return a.sum(axis=0) / g", "return a.sum(axis=0)"),
    "mean over guide tokens": ("return a.sum(axis=0) / g", "return a.mean(axis=0)"),
    "interleaved GQA heads": ("qg = q[b, h * g:(h + 1) * g]", "qg = q[b, h::n_heads_kv]"),
    "pool renormalised at edges": ("return out / kernel", "return out / np.convolve(np.ones(n), np.ones(kernel), 'same')"),
    "pool window one short": ("for off in range(-half, half + 1):", "for off in range(-half, half):"),
    "pool accepts even kernels": ("if kernel < 1 or kernel % 2 == 0:", "if kernel < 1:"),
    "quant divisor 2^(b-1)": ("qmax = (1 << (quant_bits - 1)) - 1", "qmax = (1 << (quant_bits - 1))"),
    "quant rounds half away from zero": ("q = np.clip(np.rint(quot), -qmax, qmax)", "q = np.clip(np.trunc(quot + np.copysign(0.5, quot)), -qmax, qmax)"),
    "quant truncates": ("q = np.clip(np.rint(quot), -qmax, qmax)", "q = np.clip(np.trunc(quot), -qmax, qmax)"),
    "quant uses mean |v|": ("a = np.max(np.abs(v), axis=-1)", "a = np.mean(np.abs(v), axis=-1)"),
    "additive combine": ("        return a * b\n", "        return a + b\n"),
    "ties keep the higher index": ("order = np.lexsort((np.arange(n), -scores))", "order = np.lexsort((-np.arange(n), -scores))"),
    "selects the smallest scores": ("order = np.lexsort((np.arange(n), -scores))", "order = np.lexsort((np.arange(n), scores))"),
    "kept indices not ascending": ("return np.sort(order[:k]).astype(np.int64)", "return order[:k].astype(np.int64)"),
    "naive ceil budget": ("k = math.ceil(keep_ratio * float(n) - 1e-9 * float(n))", "k = math.ceil(keep_ratio * float(n))"),
    "budget rounds down": ("k = math.ceil(keep_ratio * float(n) - 1e-9 * float(n))", "k = math.floor(keep_ratio * float(n))"),
    "gather ignores the document offset": ("tok = doc_lo + np.asarray(idx, dtype=np.int64)", "tok = np.asarray(idx, dtype=np.int64)"),
    "documents not offset": ("s_key = key_scores(qg, k_all[h, lo:hi], sigma)\n", "s_key = key_scores(qg, k_all[h, 0:n], sigma)\n"),
    "given normaliser added": ("np.exp(x - np.asarray(lse_rows", "np.exp(x + np.asarray(lse_rows"),
    "given normalisers of document 0": ("key_scores_given_lse(qg, k_all[h, lo:hi], sigma, np.asarray(lse)[b, h])", "key_scores_given_lse(qg, k_all[h, lo:hi], sigma, np.asarray(lse)[0, h])"),
    "given normalisers of head 0": ("key_scores_given_lse(qg, k_all[h, lo:hi], sigma, np.asarray(lse)[b, h])", "key_scores_given_lse(qg, k_all[h, lo:hi], sigma, np.asarray(lse)[b, 0])"),
    "fixed budget not clamped to n": ("return int(min(fixed_budget, n))", "return int(fixed_budget)"),
    "given-normaliser scores not averaged over G": ("[:, None]).sum(axis=0) / g", "[:, None]).sum(axis=0)"),
    "guide prefix excludes the token itself": ("x = np.concatenate([k_ctx @ qr, k_guide[: j + 1] @ qr]) * sigma", "x = np.concatenate([k_ctx @ qr, k_guide[:j] @ qr]) * sigma"),
    "whole guide, no causal mask": ("x = np.concatenate([k_ctx @ qr, k_guide[: j + 1] @ qr]) * sigma", "x = np.concatenate([k_ctx @ qr, k_guide @ qr]) * sigma"),
    "literal normaliser drops the context": ("x = np.concatenate([k_ctx @ qr, k_guide[: j + 1] @ qr]) * sigma", "x = k_guide[: j + 1] @ qr * sigma"),
    "literal rows token-major": ("out[gi * lt + j] = m", "out[j * g + gi] = m"),
    "guide keys of document 0": ("lse_rows = guide_lse_literal(qg, k_all[h, lo:hi], kg[b, h], sigma)", "lse_rows = guide_lse_literal(qg, k_all[h, lo:hi], kg[0, h], sigma)"),
    "guide keys of head 0": ("lse_rows = guide_lse_literal(qg, k_all[h, lo:hi], kg[b, h], sigma)", "lse_rows = guide_lse_literal(qg, k_all[h, lo:hi], kg[b, 0], sigma)"),
    "4-bit nibbles swapped": ("return (u[..., 0::2] | (u[..., 1::2] << 4)).astype(np.uint8)", "return (u[..., 1::2] | (u[..., 0::2] << 4)).astype(np.uint8)"),
    "4-bit codes sign-magnitude": ("u = q.astype(np.int64) & 0xF", "u = np.abs(q).astype(np.int64) | np.where(q < 0, 8, 0)"),
    "normalised add with L1 norms": ("na, nb = math.sqrt(float(np.sum(a * a))), math.sqrt(float(np.sum(b * b)))", "na, nb = float(np.sum(np.abs(a))), float(np.sum(np.abs(b)))"),
    "harmonic mean without the factor 2": ("out[nz] = 2.0 * a[nz] * b[nz] / den[nz]", "out[nz] = a[nz] * b[nz] / den[nz]"),
    "harmonic mean divides by a zero sum": ("nz = den != 0", "nz = den == den"),
}


def _mutant(old, new):
    assert SRC.count(old) == 1, f"mutation anchor not unique/found: {old!r}"
    mod = types.ModuleType("oracle_mutant")
    exec(compile(SRC.replace(old, new), "oracle_mutant", "exec"), mod.__dict__)
    return mod


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_mutation_is_caught(name):
    mod = _mutant(*MUTATIONS[name])
    caught = []
    for pin in oracle_pins.ALL_PINS:
        try:
            pin(mod)
        except Exception as e:  # AssertionError or a crash both count as caught
            caught.append(pin.__name__)
    assert caught, f"no pin catches mutation: {name}"
