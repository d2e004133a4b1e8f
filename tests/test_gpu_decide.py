"""GPU parity of the fused scoring + decision step (Sections 5.2, 3 and 5.3).

The decisions (drafting, Keep / Replace / ReMask, the adaptive seed count and
the selection) turn floating-point comparisons into integers, so they are
compared bit-exactly with the oracle's decision function applied to the
kernel's own fp32 per-row values (c, y_hat, H, u). Those fp32 values, and the
seed scores, are compared with the fp64 oracle within the scoring tolerance.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2602_06161_gb300 import api
from paper_2602_06161_gb300 import workloads as W
from tests import _gpu as H

pytestmark = pytest.mark.gpu

TOL = 1e-5   # fp32 outputs, max |d|
F32 = np.float32


def _params(**kw):
    p = dict(tau_draft=0.8, draft_budget=15, remask_budget=5, min_one=True, pos0=0, max_seeds=16)
    p.update(kw)
    return p


def run_decide(di: W.DecideInputs, p, *, dio=True, draft_ok=True, stats=True, workspace=None):
    logits = H.to_dev(di.logits, "bf16")
    tok = torch.from_numpy(di.tok.copy()).cuda()
    flags = torch.from_numpy(di.flags.copy()).cuda()
    rc = torch.from_numpy(di.remask_cnt.copy()).cuda()
    kw = {}
    if dio:
        kw["d_in"] = H.to_dev(di.d_in, "f32")
        kw["d_out"] = H.to_dev(di.d_out, "f32")
    if draft_ok:
        kw["draft_ok"] = torch.from_numpy(di.draft_ok).cuda()
    r = api.cover_score_decide_fwd(logits, di.n_seq, tok, flags, rc, mask_id=di.mask_id, workspace=workspace,
                                   **p, **kw)
    torch.cuda.synchronize()
    assert api.cover_device_status() == 0
    out = {k: v.cpu().numpy() for k, v in r.items()}
    if not stats:
        out.pop("stats")
    out.update(tok=tok.cpu().numpy(), flags=flags.cpu().numpy(), remask_cnt=rc.cpu().numpy())
    # the kernel's fp32 u of the current token and of the greedy token (= ln Z), from the
    # plain scoring entry point, whose per-row arithmetic is the same
    cur = api.cover_score_fwd(logits, di.n_seq, 0, cur_tok=torch.from_numpy(di.tok).cuda())
    top = api.cover_score_fwd(logits, di.n_seq, 0)
    torch.cuda.synchronize()
    out["u_cur"] = cur["score"].cpu().numpy()
    out["u_top"] = top["score"].cpu().numpy()
    for k in ("maxprob", "entropy", "argmax"):
        assert np.array_equal(out[k], cur[k].cpu().numpy()), k
    return out


def check(di: W.DecideInputs, p, r, *, dio=True, draft_ok=True, fp64_rows=None, what=""):
    n = di.N
    per = n // di.n_seq
    d_in = di.d_in if dio else None
    d_out = di.d_out if dio else None
    dok = di.draft_ok if draft_ok else None
    outs = oracle.decide_step(r["maxprob"], r["argmax"], r["entropy"], r["u_cur"], r["u_top"], d_in, d_out,
                              di.tok, di.flags, di.remask_cnt, dok, di.n_seq, tau=F32(p["tau_draft"]),
                              budget=p["draft_budget"], m_remask=p["remask_budget"], mask_id=di.mask_id,
                              min_one=p["min_one"], pos0=p["pos0"], max_seeds=p["max_seeds"])
    for g, o in enumerate(outs):
        sl = slice(g * per, (g + 1) * per)
        assert np.array_equal(r["tok"][sl], o["tok"]), f"{what} seq {g} tok"
        assert np.array_equal(r["flags"][sl], o["flags"]), f"{what} seq {g} flags"
        assert np.array_equal(r["remask_cnt"][sl], o["remask_cnt"]), f"{what} seq {g} remask"
        assert np.array_equal(r["score"][sl], o["score"].astype(F32)), f"{what} seq {g} score"
        seeds = o["seeds"] + [-1] * (p["max_seeds"] - len(o["seeds"]))
        if p["max_seeds"] > 0:
            assert r["seed_idx"][g].tolist() == seeds, f"{what} seq {g} seeds"
        assert r["n_seeds"][g] == o["n_select"], f"{what} seq {g} n_seeds"
        if "stats" in r:
            want = [len(o["drafted"]), len(o["kept"]), len(o["replaced"]), len(o["remasked"]), o["n_t"],
                    o["n_above"]]
            assert r["stats"][g].tolist() == want, f"{what} seq {g} stats"
    # the kernel's fp32 per-row values and seed scores against the fp64 definition
    rows = np.arange(n) if fp64_rows is None else fp64_rows
    new_tok = r["tok"][rows].astype(np.int64)
    unmasked = new_tok != di.mask_id
    ref = oracle.score_rows(di.logits_f64(rows), cur_tok=np.where(unmasked, new_tok, 0),
                            d_in=None if d_in is None else d_in[rows], d_out=None if d_out is None else d_out[rows])
    assert np.array_equal(r["argmax"][rows], ref["argmax"]), what
    for k in ("maxprob", "entropy"):
        d = np.abs(r[k][rows].astype(np.float64) - ref[k]).max()
        assert d <= TOL, f"{what} {k} max |d| {d:.3e}"
    s = r["score"][rows].astype(np.float64)
    assert np.isneginf(s[~unmasked]).all(), what
    if unmasked.any():
        d = np.abs(s[unmasked] - ref["score"][unmasked]).max()
        assert d <= TOL, f"{what} score max |d| {d:.3e}"
    return outs


@pytest.mark.parametrize("N,V,n_seq,block", [
    (1, 300, 1, 1), (16, 1000, 2, 4), (64, 4096, 4, 8), (96, 5003, 3, 16), (256, 2048, 1, 64),
    (512, 1000, 2, 64),
])
def test_decide_shapes(N, V, n_seq, block):
    for seed in range(3):
        di = W.make_decide_inputs(N, V, n_seq, seed=17 * seed + N, block_len=block)
        p = _params(draft_budget=max(1, block // 4), max_seeds=8)
        check(di, p, run_decide(di, p), what=f"N{N} V{V} seed {seed}")


def test_decide_variants_of_the_inputs():
    di = W.make_decide_inputs(128, 4000, 2, seed=5, block_len=32)
    for kw in (dict(dio=False), dict(draft_ok=False), dict(stats=False)):
        p = _params()
        check(di, p, run_decide(di, p, **kw), dio=kw.get("dio", True), draft_ok=kw.get("draft_ok", True),
              what=str(kw))


@pytest.mark.parametrize("pkw", [
    dict(draft_budget=0), dict(draft_budget=0, min_one=False), dict(tau_draft=0.0), dict(tau_draft=1.0),
    dict(max_seeds=0), dict(max_seeds=1), dict(remask_budget=0), dict(remask_budget=255), dict(pos0=1792),
    dict(draft_budget=10000),
])
def test_decide_parameters(pkw):
    di = W.make_decide_inputs(192, 3000, 3, seed=11, block_len=32)
    p = _params(**pkw)
    check(di, p, run_decide(di, p), what=str(pkw))


def test_decide_degenerate_states():
    di = W.make_decide_inputs(96, 2000, 3, seed=21, block_len=32)
    per = 32
    # sequence 0: everything masked (no seeds, no unmasked rows); sequence 1: nothing masked
    di.tok[:per] = di.mask_id
    di.flags[:per] = 0
    di.tok[per:2 * per][di.tok[per:2 * per] == di.mask_id] = 7
    # sequence 2: uniform logits (every confidence 1/V, equal scores: nothing above the mean)
    di.logits[2 * per:] = W.f32_to_bf16_bits(np.zeros((per, 2000), np.float32))
    di.d_in[2 * per:] = 0.0
    di.d_out[2 * per:] = 0.0
    p = _params(tau_draft=0.5)
    outs = check(di, p, run_decide(di, p), what="degenerate")
    assert outs[0]["n_t"] == len(outs[0]["drafted"])
    assert outs[2]["n_above"] == 0 and outs[2]["n_select"] == 0


def test_decide_longest_segment_and_workspace_reuse():
    di = W.make_decide_inputs(4096, 512, 1, seed=23, block_len=512)
    p = _params(max_seeds=64)
    ws = api.decide_workspace(4096, 1)
    for _ in range(2):
        check(di, p, run_decide(di, p, workspace=ws), what="4096 rows")


def test_decide_register_path_odd_vocab():
    di = W.make_decide_inputs(48, 3001, 2, seed=29, block_len=8)   # V % 8 != 0: the register-load kernel
    p = _params()
    check(di, p, run_decide(di, p), what="odd V")


def test_decide_chained_steps():
    """Three decoding steps with fresh logits, the state carried on the device."""
    base = W.make_decide_inputs(128, 3000, 2, seed=31, block_len=32)
    p = _params(draft_budget=4, max_seeds=6)
    tok, flags, rc = base.tok.copy(), base.flags.copy(), base.remask_cnt.copy()
    for step in range(3):
        di = W.make_decide_inputs(128, 3000, 2, seed=100 + step, block_len=32)
        di.tok, di.flags, di.remask_cnt, di.draft_ok = tok, flags, rc, base.draft_ok
        r = run_decide(di, p)
        check(di, p, r, what=f"step {step}")
        tok, flags, rc = r["tok"], r["flags"], r["remask_cnt"]


def test_decide_named_workload_full():
    wl = W.WORKLOADS["llada_b8_l2048"]
    di = wl.decide_inputs()
    p = _params(max_seeds=64, pos0=wl.L - wl.score_N // wl.score_n_seq)
    rng = np.random.default_rng(0)
    rows = np.sort(rng.choice(di.N, size=128, replace=False))
    check(di, p, run_decide(di, p), fp64_rows=rows, what=wl.name)


@pytest.mark.parametrize("per,V", [
    (288, 1000),    # one row per thread of the bulk-copy kernel (288 threads): the fast path
    (289, 1000),    # one row more than its threads: the general path
    (1153, 1000),   # the general path, four rows per thread and one more
    (512, 1001),    # the register-load kernel (odd vocabulary, 512 threads): its fast-path limit
    (513, 1001),    # and one row past it
    (2049, 1001),   # a segment of 2049 rows: 48 KB of keys and scores in shared memory
])
def test_decide_both_sides_of_the_fast_path(per, V):
    # the per-sequence decision has a one-row-per-thread path and a general one; on both sides
    # of the switch the decisions equal the oracle's, with a drafting budget that forces the
    # ranking (more candidates than the budget) and a seed cap above 32 (rank or sort instead of
    # the short selections)
    di = W.make_decide_inputs(2 * per, V, 2, seed=per, block_len=64)
    for p in (_params(draft_budget=15, max_seeds=8), _params(draft_budget=2, tau_draft=0.05, max_seeds=40)):
        check(di, p, run_decide(di, p), what=f"per {per} V {V} B {p['draft_budget']}")


@pytest.mark.parametrize("per", [256, 512, 513, 1024, 2049])
def test_update_then_select_both_paths(per):
    # the split order (update phase, then the selection launch with the caller's d_in / d_out):
    # the selection launch has 512 threads, so 512 rows take its fast path and 513 the general
    # one; 2049 rows need 48 KB of shared memory for the keys and scores
    di = W.make_decide_inputs(2 * per, 1000, 2, seed=per + 1, block_len=32)
    p = _params(max_seeds=12)
    logits = H.to_dev(di.logits, "bf16")
    tok = torch.from_numpy(di.tok.copy()).cuda()
    flags = torch.from_numpy(di.flags.copy()).cuda()
    rc = torch.from_numpy(di.remask_cnt.copy()).cuda()
    ws = api.decide_workspace(di.N, di.n_seq)
    kw = dict(tau_draft=p["tau_draft"], draft_budget=p["draft_budget"], remask_budget=p["remask_budget"],
              mask_id=di.mask_id, min_one=p["min_one"], pos0=p["pos0"], max_seeds=p["max_seeds"])
    upd = api.cover_score_decide_fwd(logits, di.n_seq, tok, flags, rc, phase=api.COVER_DECIDE_UPDATE,
                                     workspace=ws, draft_ok=torch.from_numpy(di.draft_ok).cuda(), **kw)
    d_in, d_out = H.to_dev(di.d_in, "f32"), H.to_dev(di.d_out, "f32")
    sel = api.cover_seed_select_fwd(di.n_seq, tok, flags, rc, ws, remask_budget=p["remask_budget"],
                                    mask_id=di.mask_id, pos0=p["pos0"], max_seeds=p["max_seeds"], d_in=d_in,
                                    d_out=d_out)
    torch.cuda.synchronize()
    assert api.cover_device_status() == 0
    u_cur = api.cover_score_fwd(logits, di.n_seq, 0, cur_tok=torch.from_numpy(di.tok).cuda())["score"].cpu().numpy()
    u_top = api.cover_score_fwd(logits, di.n_seq, 0)["score"].cpu().numpy()
    h = {k: v.cpu().numpy() for k, v in upd.items()}
    outs = oracle.decide_step(h["maxprob"], h["argmax"], h["entropy"], u_cur, u_top, di.d_in, di.d_out, di.tok,
                              di.flags, di.remask_cnt, di.draft_ok, di.n_seq, tau=F32(p["tau_draft"]),
                              budget=p["draft_budget"], m_remask=p["remask_budget"], mask_id=di.mask_id,
                              min_one=p["min_one"], pos0=p["pos0"], max_seeds=p["max_seeds"])
    t, fl, r_, sc = tok.cpu().numpy(), flags.cpu().numpy(), rc.cpu().numpy(), sel["score"].cpu().numpy()
    for g, o in enumerate(outs):
        sl = slice(g * per, (g + 1) * per)
        assert np.array_equal(t[sl], o["tok"]) and np.array_equal(r_[sl], o["remask_cnt"]), (per, g)
        assert np.array_equal(fl[sl], o["flags"]), (per, g)
        assert np.array_equal(sc[sl], o["score"].astype(F32)), (per, g)
        seeds = o["seeds"] + [-1] * (p["max_seeds"] - len(o["seeds"]))
        assert sel["seed_idx"][g].cpu().tolist() == seeds, (per, g)
        assert int(sel["n_seeds"][g]) == o["n_select"], (per, g)
