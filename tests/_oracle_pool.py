"""Whole-tensor oracle checks spread over worker processes (test infrastructure).

The workers are started with the 'spawn' method, so none of them inherits the
CUDA context of the test process, and each runs single-threaded BLAS. A task is
one (b, hq) head: the worker evaluates the oracle's full two-view attention of
that head (every row, seed rows through their explicit leave-one-out views)
and compares it with the kernel's output of the head, element by element.
"""
import concurrent.futures as cf
import multiprocessing as mp
import os

import numpy as np

_THREAD_VARS = ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS")


def _head_check(task):
    import oracle
    from paper_2602_06161_gb300 import workloads as W
    q, kc, vc, km, vm, seeds, out_bits, lse_dev = task
    f = lambda a: W.bf16_bits_to_f64(a)[None, None]  # noqa: E731
    ref, ref_lse = oracle.override_attention(f(q), f(kc), f(vc), f(km), f(vm), seeds[None])
    d = np.abs(W.bf16_bits_to_f64(out_bits) - ref[0, 0])
    dl = np.abs(lse_dev.astype(np.float64) - ref_lse[0, 0])
    return float(d.max()), float(d.sum()), int(d.size), float(dl.max())


def check_heads(tasks, n_tasks: int):
    """Runs _head_check over the tasks; returns (max |d|, mean |d|, max lse |d|, heads)."""
    n = max(1, min(os.cpu_count() or 1, 16, n_tasks))
    saved = {k: os.environ.get(k) for k in _THREAD_VARS}
    os.environ.update({k: "1" for k in _THREAD_VARS})
    try:
        # a worker that dies raises BrokenProcessPool here instead of being restarted forever
        with cf.ProcessPoolExecutor(max_workers=n, mp_context=mp.get_context("spawn")) as ex:
            res = list(ex.map(_head_check, tasks))
    finally:
        for k, v in saved.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v
    dmax = max(r[0] for r in res)
    dmean = sum(r[1] for r in res) / sum(r[2] for r in res)
    lmax = max(r[3] for r in res)
    return dmax, dmean, lmax, len(res)
