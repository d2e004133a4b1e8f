"""GPU parity of the fused scoring + top-k kernel against the fp64 oracle."""
import numpy as np
import pytest
import torch

import oracle
from paper_2602_06161_gb300 import api
from paper_2602_06161_gb300 import workloads as W
from tests import _gpu as H

pytestmark = pytest.mark.gpu

TOL = 1e-5   # fp32 outputs, max |d|


def run_score(inp: W.ScoreInputs, workspace=None):
    logits = H.to_dev(inp.logits, "bf16")
    kw = {}
    if inp.cur_tok is not None:
        kw["cur_tok"] = H.to_dev(inp.cur_tok, "i32")
    if inp.d_in is not None:
        kw["d_in"] = H.to_dev(inp.d_in, "f32")
        kw["d_out"] = H.to_dev(inp.d_out, "f32")
    if inp.eligible is not None:
        kw["eligible"] = torch.from_numpy(inp.eligible).cuda()
    r = api.cover_score_fwd(logits, inp.n_seq, inp.topk, workspace=workspace, **kw)
    torch.cuda.synchronize()
    assert api.cover_device_status() == 0
    return {k: v.cpu().numpy() for k, v in r.items()}


def check(inp: W.ScoreInputs, r, what=""):
    ref = oracle.score_rows(inp.logits_f64(), cur_tok=inp.cur_tok, d_in=inp.d_in, d_out=inp.d_out)
    assert np.array_equal(r["argmax"], ref["argmax"]), what
    for k in ("maxprob", "entropy", "score"):
        d = np.abs(r[k].astype(np.float64) - ref[k]).max()
        assert d <= TOL, f"{what} {k} max |d| {d:.3e}"
    # the top-k decision taken on the kernel's own fp32 scores must be bit-exact
    idx, val = oracle.topk_select(r["score"], inp.n_seq, inp.topk, inp.eligible)
    assert np.array_equal(r["topk_idx"], idx), what
    assert np.array_equal(r["topk_score"], val.astype(np.float32)), what
    # against the fp64 selection: identical wherever the oracle's margin is clear
    ref_idx, _ = oracle.topk_select(ref["score"], inp.n_seq, inp.topk, inp.eligible)
    gaps = oracle.topk_margin(ref["score"], inp.n_seq, inp.topk, inp.eligible)
    for g in range(inp.n_seq):
        if gaps[g] > 4 * TOL:
            assert set(r["topk_idx"][g].tolist()) == set(ref_idx[g].tolist()), f"{what} segment {g}"
    return ref


@pytest.mark.parametrize("N,V,n_seq,k", [
    (1, 1, 1, 1), (3, 7, 1, 2), (16, 1000, 4, 3), (64, 4099, 2, 32), (8, 8, 8, 1), (37, 20001, 1, 37),
])
def test_score_shapes(N, V, n_seq, k):
    inp = W.make_score_inputs(N, V, n_seq, k, seed=N + V, spike_frac=0.1)
    check(inp, run_score(inp), f"N{N} V{V}")


def test_score_side_inputs_and_eligibility():
    inp = W.make_score_inputs(96, 5003, 3, 10, seed=7, with_cur_tok=True, with_dio=True, eligible_frac=0.4)
    check(inp, run_score(inp))


@pytest.mark.parametrize("per,k,frac", [(1000, 32, 0.012), (300, 20, 0.012), (1000, 6, 0.003)])
def test_score_topk_fewer_eligible_than_k(per, k, frac):
    """General path with fewer eligible rows than k: the list ends in -1 / -inf."""
    inp = W.make_score_inputs(2 * per, 300, 2, k, seed=per, eligible_frac=frac)
    r = run_score(inp)
    check(inp, r)
    n_elig = inp.eligible.reshape(2, per).sum(axis=1)
    assert (n_elig < k).all()
    for g in range(2):
        assert (r["topk_idx"][g, n_elig[g]:] == -1).all() and (r["topk_idx"][g, :n_elig[g]] >= 0).all()


def test_score_no_eligible_rows():
    inp = W.make_score_inputs(32, 512, 2, 4, seed=8, eligible_frac=0.0)
    r = run_score(inp)
    assert (r["topk_idx"] == -1).all() and np.isneginf(r["topk_score"]).all()


def test_score_ties_and_uniform_rows():
    inp = W.make_score_inputs(16, 3000, 1, 16, seed=9)
    x = inp.logits.copy()
    x[0, :] = W.f32_to_bf16_bits(np.full(3000, 0.5, np.float32))      # all equal: argmax 0
    x[1, :] = W.f32_to_bf16_bits(np.full(3000, -1.0, np.float32))
    x[1, [17, 2000, 2999]] = W.f32_to_bf16_bits(np.float32([3.0, 3.0, 3.0]))  # tie: lowest index 17
    x[2] = x[1]                                                           # equal scores: lower row first
    inp.logits = x
    r = run_score(inp)
    assert r["argmax"][0] == 0 and r["argmax"][1] == 17
    check(inp, r)


@pytest.mark.parametrize("V", [40000, 40001])   # bulk-copy kernel (V % 8 == 0), register-load kernel
def test_score_argmax_ties_across_batches(V):
    """The first index of the row maximum when it occurs several times: in different chunks, in one
    thread's batch (different vectors), in one thread's batches of different chunks, at the row's
    first and last element, and as -0.0 before +0.0."""
    placed = [
        [39999, 12345, 8192 + 3, 20000],       # several chunks: 8195
        [2 * 2048 + 5 * 8 + 3, 5 * 8 + 6],     # one thread, one batch, vectors 2 and 0: 46
        [3 * 8192 + 7 * 8 + 1, 8192 + 7 * 8 + 2],
        [0, V - 1],
        [V - 1],
        [8 * 4096 + 11, 4096 + 3, 2 * 4096 + 3],
    ]
    inp = W.make_score_inputs(len(placed) + 1, V, 1, 3, seed=V)
    x = inp.logits.copy()
    for r, pos in enumerate(placed):
        x[r, pos] = W.f32_to_bf16_bits(np.full(len(pos), 9.5, np.float32))
    zr = len(placed)
    x[zr, :] = W.f32_to_bf16_bits(np.full(V, -2.0, np.float32))
    x[zr, 30000] = np.uint16(0x8000)   # -0.0
    x[zr, 31000] = np.uint16(0x0000)   # +0.0
    x[zr, 500] = np.uint16(0x8000)
    inp.logits = x
    r = run_score(inp)
    expect = [min(p) for p in placed] + [500]
    assert r["argmax"].tolist() == expect
    check(inp, r)


def test_score_max_segment_and_workspace_reuse():
    inp = W.make_score_inputs(4096, 64, 1, 256, seed=10)
    ws = api.score_workspace(1)
    r1 = run_score(inp, workspace=ws)
    r2 = run_score(inp, workspace=ws)
    assert int(ws.abs().sum().item()) == 0
    for k in r1:
        assert np.array_equal(r1[k], r2[k])
    check(inp, r1)


@pytest.mark.parametrize("name", ["dream_gqa_l1024", "llada_b8_l2048"])
def test_score_named_workloads_full(name):
    inp = W.WORKLOADS[name].score_inputs()
    r = run_score(inp)
    ref = check(inp, r, name)
    gaps = oracle.topk_margin(ref["score"], inp.n_seq, inp.topk)
    print(f"{name}: top-k margins min {gaps.min():.3e}")


@pytest.mark.parametrize("per,V,k", [
    (288, 1000, 40),    # one row per thread of the bulk-copy kernel: selection by rank
    (289, 1000, 20),    # the general path, a short list: warp sorts and merges
    (289, 1000, 40),    # the general path, a long list: the bitonic sort
    (512, 1001, 33),    # the register-load kernel (512 threads): selection by rank
    (513, 1001, 32),    # and one row past it: warp sorts and merges
    (4096, 136, 32),    # the largest segment, k = 32
    (600, 300, 9),      # the fewest keys taken by warp sorts
    (600, 300, 8),      # the most taken by rounds of a CTA-wide maximum
    (777, 200, 1),      # k = 1
    (600, 1001, 5),     # the register-load kernel's general path (16 warps), rounds
])
def test_score_topk_on_both_sides_of_the_fast_path(per, V, k):
    inp = W.make_score_inputs(2 * per, V, 2, k, seed=per + k, spike_frac=0.1, eligible_frac=0.8)
    check(inp, run_score(inp), f"per {per} V {V} k {k}")
