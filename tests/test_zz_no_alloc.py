"""The allocation-free scoring entry point, cover_score_fwd_noalloc.

Some callers cannot allocate device memory for a workspace (a serving loop
that reserves all of its GPU memory at start-up, a plugin interface that is
handed inputs and outputs but no allocator). cover_score_fwd_noalloc keeps the
per-sequence counters in a fixed device array of the library instead. These
tests call it through the C ABI and check it against cover_score_fwd on two
calls in a row. The file is named so that pytest collects it last.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2602_06161_gb300 import _lib, api, build
from paper_2602_06161_gb300 import workloads as W

MAX_SEQ = 4096


def _dev(a, kind):
    if kind == "bf16":
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda().view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _empty_out(N, n_seq, k):
    return dict(maxprob=torch.empty(N, device="cuda"), entropy=torch.empty(N, device="cuda"),
                argmax=torch.empty(N, dtype=torch.int32, device="cuda"), score=torch.empty(N, device="cuda"),
                topk_idx=torch.empty((n_seq, k), dtype=torch.int32, device="cuda"),
                topk_score=torch.empty((n_seq, k), device="cuda"))


def _call_noalloc(lib, logits, n_seq, k, side, out):
    p = lambda t: None if t is None else t.data_ptr()  # noqa: E731
    N, V = logits.shape
    return lib.cover_score_fwd_noalloc(
        p(logits), N, V, n_seq, p(side.get("cur_tok")), p(side.get("d_in")), p(side.get("d_out")),
        p(side.get("eligible")), k, p(out["maxprob"]), p(out["entropy"]), p(out["argmax"]), p(out["score"]),
        p(out["topk_idx"]), p(out["topk_score"]), torch.cuda.current_stream().cuda_stream)


def _same(a, b):
    assert torch.equal(a["argmax"], b["argmax"])
    assert torch.equal(a["topk_idx"], b["topk_idx"])
    for key in ("maxprob", "entropy", "score", "topk_score"):
        x, y = a[key].double(), b[key].double()
        finite = torch.isfinite(y)
        assert torch.equal(torch.isfinite(x), finite), key
        assert (x[finite] - y[finite]).abs().max().item() <= 1e-5 if finite.any() else True, key


@pytest.mark.gpu
@pytest.mark.parametrize("N,V,n_seq,k", [(1024, 9000, 4, 24), (MAX_SEQ, 64, MAX_SEQ, 1)])
def test_noalloc_matches_workspace_entry_point_twice(N, V, n_seq, k):
    inp = W.make_score_inputs(N, V, n_seq, k, seed=31, spike_frac=0.05, with_cur_tok=True, with_dio=True,
                              eligible_frac=0.7)
    logits = _dev(inp.logits, "bf16")
    side = dict(cur_tok=_dev(inp.cur_tok, "i32"), d_in=_dev(inp.d_in, "f32"), d_out=_dev(inp.d_out, "f32"),
                eligible=_dev(inp.eligible, "u8"))
    ref = api.cover_score_fwd(logits, n_seq, k, **side)
    torch.cuda.synchronize()
    lib = _lib.load()
    for _ in range(2):          # the second call finds the array as the first one left it
        out = _empty_out(N, n_seq, k)
        assert _call_noalloc(lib, logits, n_seq, k, side, out) == 0
        torch.cuda.synchronize()
        assert api.cover_device_status() == 0
        _same(out, ref)


@pytest.mark.gpu
def test_noalloc_after_a_call_of_another_segment_shape():
    # the shared array's counters serve whichever segments a call has: a call with many one-row
    # segments is followed by one with a few long segments, whose top-k must still be right
    lib = _lib.load()
    for (N, V, n_seq, k) in [(MAX_SEQ, 64, MAX_SEQ, 1), (1024, 9000, 4, 24), (1024, 2000, 256, 3)]:
        inp = W.make_score_inputs(N, V, n_seq, k, seed=37 + n_seq, spike_frac=0.05, with_cur_tok=True,
                                  with_dio=True, eligible_frac=0.7)
        logits = _dev(inp.logits, "bf16")
        side = dict(cur_tok=_dev(inp.cur_tok, "i32"), d_in=_dev(inp.d_in, "f32"), d_out=_dev(inp.d_out, "f32"),
                    eligible=_dev(inp.eligible, "u8"))
        ref = api.cover_score_fwd(logits, n_seq, k, **side)
        out = _empty_out(N, n_seq, k)
        assert _call_noalloc(lib, logits, n_seq, k, side, out) == 0
        torch.cuda.synchronize()
        assert api.cover_device_status() == 0
        _same(out, ref)


def test_noalloc_rejects_more_sequences_than_the_array_holds():
    build.build()
    lib = ctypes.CDLL(build.LIB)
    fn = lib.cover_score_fwd_noalloc
    fn.restype = ctypes.c_int
    fn.argtypes = _lib._SIGNATURES["cover_score_fwd_noalloc"][1]
    P = 0x10000   # fake aligned pointers; the size check returns before any use
    n = MAX_SEQ + 1
    assert fn(P, n, 8, n, None, None, None, None, 1, P, P, P, P, P, P, None) == -1
    assert fn(P, MAX_SEQ, 8, MAX_SEQ, None, None, None, None, 2, P, P, P, P, P, P, None) == -1   # k > rows
