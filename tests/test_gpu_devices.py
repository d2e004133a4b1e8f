"""Entry points on more than one device in the same process.

A kernel's shared-memory limit and a __device__ symbol's address hold only in
the context they were set or looked up in; the library keeps them per context.
With two visible devices every family of entry points runs on both, in both
orders, and must give the same results; with one device the test is skipped.
"""
import numpy as np
import pytest
import torch

from paper_2602_06161_gb300 import api
from paper_2602_06161_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def _run_on(dev, inp, sinp):
    with torch.cuda.device(dev):
        t = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(dev).view(torch.bfloat16)  # noqa: E731
        seeds = torch.from_numpy(inp.seed_idx).to(dev)
        out, lse = api.cover_attn_fwd(t(inp.q), t(inp.k_cached), t(inp.v_cached), t(inp.k_seedmask),
                                      t(inp.v_seedmask), seeds)
        logits = t(sinp.logits)
        s1 = api.cover_score_fwd(logits, sinp.n_seq, sinp.topk)
        s2 = api.cover_score_fwd_noalloc(logits, sinp.n_seq, sinp.topk)
        torch.cuda.synchronize(dev)
        assert api.cover_device_status() == 0
        return [out.cpu(), lse.cpu(), s1["topk_idx"].cpu(), s2["topk_idx"].cpu(), s1["entropy"].cpu()]


def test_two_devices_same_results():
    if torch.cuda.device_count() < 2:
        pytest.skip("needs two visible GPUs")
    inp = W.make_attn_inputs(1, 4, 2, 384, 128, 8, seed=3, dtype="bf16")
    sinp = W.make_score_inputs(512, 5000, 2, 8, seed=4)
    a = _run_on(0, inp, sinp)
    b = _run_on(1, inp, sinp)
    c = _run_on(0, inp, sinp)
    for x, y, z in zip(a, b, c):
        assert torch.equal(x, y) and torch.equal(x, z)
