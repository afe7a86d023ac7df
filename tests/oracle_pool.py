"""The oracle over many (document, KV head) units at once, for the full-size
parity tests: one spawned worker process per unit, BLAS single-threaded.

Each unit runs oracle.compress_layer on its own slice (one document, one KV
head and its G query heads), which is exactly how the oracle treats units:
documents and heads are independent (Sec. 4 "Eviction").  The results are put
back into the dictionary layout of oracle.compress_layer.  Inputs reach the
workers through memory-mapped .npy files, not pickles.
"""
from __future__ import annotations

import atexit
import multiprocessing as mp
import os
import shutil
import tempfile

import numpy as np

_pool = None


def _init():
    os.environ["OPENBLAS_NUM_THREADS"] = "1"
    os.environ["OMP_NUM_THREADS"] = "1"


def _unit(args):
    qf, kf, vf, lf, gf, g, kw = args
    from oracle import taskpress_oracle as O
    q, k, v = np.load(qf), np.load(kf, mmap_mode="r"), np.load(vf, mmap_mode="r")
    extra = dict(kw)
    if lf:
        extra["lse"] = np.load(lf)
    if gf:
        extra["k_guide_bits"] = np.load(gf)
    out = O.compress_layer(q, k, v, [0, k.shape[1]], n_heads_q=g, n_heads_kv=1, **extra)
    return (out["gamma"][0], out["vq"][0], out["scores"][(0, 0)], out["key"][(0, 0)],
            out["idx"][(0, 0)], out["k"][0])


def pool():
    """The session's worker pool (spawned: safe after CUDA is initialised)."""
    global _pool
    if _pool is None:
        _pool = mp.get_context("spawn").Pool(processes=os.cpu_count() or 1, initializer=_init)
        atexit.register(_pool.terminate)
    return _pool


def compress_layer(x, n_heads_q: int, n_heads_kv: int, *, heads=None, docs=None, lse=None,
                   k_guide_bits=None, quant_bits: int = 8, **kw):
    """oracle.compress_layer(x.q, x.k, x.v, x.doc_offsets, ...) restricted to
    `heads` x `docs` (all when None), computed unit by unit in the pool.  The
    returned gamma / vq cover the units' tokens (other entries are zero)."""
    g = n_heads_q // n_heads_kv
    offs = np.asarray(x.doc_offsets, dtype=np.int64)
    heads = list(range(n_heads_kv)) if heads is None else list(heads)
    docs = list(range(len(offs) - 1)) if docs is None else list(docs)
    tmp = tempfile.mkdtemp(prefix="tp_parity_")
    try:
        jobs = []
        for b in docs:
            lo, hi = int(offs[b]), int(offs[b + 1])
            for h in heads:
                stem = os.path.join(tmp, f"{b}_{h}_")
                np.save(stem + "q.npy", np.ascontiguousarray(x.q[b:b + 1, h * g:(h + 1) * g]))
                np.save(stem + "k.npy", np.ascontiguousarray(x.k[h:h + 1, lo:hi]))
                np.save(stem + "v.npy", np.ascontiguousarray(x.v[h:h + 1, lo:hi]))
                lf = gf = ""
                if lse is not None:
                    lf = stem + "lse.npy"
                    np.save(lf, np.ascontiguousarray(np.asarray(lse)[b:b + 1, h:h + 1]))
                if k_guide_bits is not None:
                    gf = stem + "kg.npy"
                    np.save(gf, np.ascontiguousarray(np.asarray(k_guide_bits)[b:b + 1, h:h + 1]))
                jobs.append(((b, h, lo, hi),
                             (stem + "q.npy", stem + "k.npy", stem + "v.npy", lf, gf, g,
                              dict(kw, quant_bits=quant_bits))))
        results = pool().map(_unit, [j for _, j in jobs], chunksize=1)
    finally:
        shutil.rmtree(tmp, ignore_errors=True)
    n_total, d = x.k.shape[1], x.k.shape[2]
    out = {"gamma": np.zeros((n_heads_kv, n_total), np.float32),
           "vq": np.zeros((n_heads_kv, n_total, d), np.int8),
           "scores": {}, "key": {}, "idx": {}, "k": {}}
    for ((b, h, lo, hi), _), (gam, vq, sc, key, idx, kb) in zip(jobs, results):
        out["gamma"][h, lo:hi] = gam
        out["vq"][h, lo:hi] = vq
        out["scores"][(b, h)] = sc
        out["key"][(b, h)] = key
        out["idx"][(b, h)] = idx
        out["k"][b] = kb
    return out
