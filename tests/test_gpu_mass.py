"""GPU parity of d_in / d_out (Section 5.3) and of the three-phase decision step.

d_in / d_out come from the head-averaged attention weights of the current pass,
recomputed on the tensor cores from the attention kernel's q, K', masked keys
and lse; they are compared with the fp64 oracle (which runs the full softmax of
every view), and the decisions of the update -> mass -> select pipeline are
compared bit-exactly with the oracle's decisions on the kernel's own values.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2602_06161_gb300 import api
from paper_2602_06161_gb300 import workloads as W
from tests import _gpu as H

pytestmark = pytest.mark.gpu

F32 = np.float32


def _mass_tol(d):
    return 2e-3 * np.maximum(1.0, np.abs(d))


def _attention(inp):
    args = [H.to_dev(inp.q, "bf16"), H.to_dev(inp.k_cached, "bf16"), H.to_dev(inp.v_cached, "bf16")]
    if inp.S:
        args += [H.to_dev(inp.k_seedmask, "bf16"), H.to_dev(inp.v_seedmask, "bf16"), H.to_dev(inp.seed_idx, "i32")]
    out, lse = api.cover_attn_fwd(*args)
    return args, lse


def _state(B, per, rng, mask_id=7):
    tok = rng.integers(0, 6, size=B * per).astype(np.int32)
    masked = rng.random(B * per) < 0.4
    tok[masked] = mask_id
    flags = np.zeros(B * per, np.uint8)
    drafted = (~masked) & (rng.random(B * per) < 0.3)
    flags[drafted] |= 2
    return tok, flags, masked.reshape(B, per), drafted.reshape(B, per)


def run_mass(inp, tok, flags, pos0, per, mask_id=7):
    args, lse = _attention(inp)
    kw = dict(k_seedmask=args[3], seed_idx=args[5]) if inp.S else {}
    d_in, d_out = api.cover_attn_mass_fwd(args[0], args[1], lse, torch.from_numpy(tok).cuda(),
                                          torch.from_numpy(flags).cuda(), mask_id=mask_id, pos0=pos0, per=per, **kw)
    torch.cuda.synchronize()
    assert api.cover_device_status() == 0
    return d_in.cpu().numpy(), d_out.cpu().numpy()


def oracle_mass(inp, masked, drafted, pos0, batches=None):
    f = W.bf16_bits_to_f64
    bs = range(inp.q.shape[0]) if batches is None else batches
    ins, outs = [], []
    for b in bs:
        sl = slice(b, b + 1)
        seeds = inp.seed_idx[sl] if inp.S else None
        km = f(inp.k_seedmask[sl]) if inp.S else None
        di, do = oracle.attention_mass(f(inp.q[sl]), f(inp.k_cached[sl]), km, seeds, masked[sl], drafted[sl], pos0)
        ins.append(di[0])
        outs.append(do[0])
    return np.stack(ins), np.stack(outs)


@pytest.mark.parametrize("B,Hq,Hkv,L,S,pos0,per", [
    (2, 4, 2, 384, 8, 128, 256),      # response block of two row tiles, seeds inside and outside
    (1, 4, 4, 300, 6, 44, 256),       # ragged last key tile
    (1, 4, 4, 200, 4, 0, 200),        # the whole memory is the response
    (1, 7, 1, 160, 5, 31, 129),       # GQA 7:1, one row past a tile
    (2, 2, 2, 64, 3, 63, 1),          # a single response position
    (1, 2, 2, 256, 0, 64, 192),       # no seeds
    (1, 4, 2, 1100, 10, 460, 640),    # five tiles each way: the two-stage rings wrap twice
])
def test_mass_against_oracle(B, Hq, Hkv, L, S, pos0, per):
    inp = W.make_attn_inputs(B, Hq, Hkv, L, 128, S, dtype="bf16", seed=L + per, seed_lo=0, seed_hi=L)
    rng = np.random.default_rng(L * 3 + per)
    tok, flags, masked, drafted = _state(B, per, rng)
    d_in, d_out = run_mass(inp, tok, flags, pos0, per)
    ref_in, ref_out = oracle_mass(inp, masked, drafted, pos0)
    assert np.all(np.abs(d_in - ref_in.ravel()) <= _mass_tol(ref_in.ravel())), np.abs(d_in - ref_in.ravel()).max()
    assert np.all(np.abs(d_out - ref_out.ravel()) <= _mass_tol(ref_out.ravel())), np.abs(d_out - ref_out.ravel()).max()


def test_mass_whole_memory_sums_to_the_masked_count():
    # with every position a response position each masked row spreads mass 1 over the keys
    B, Hq, Hkv, L, S = 2, 4, 2, 640, 16
    inp = W.make_attn_inputs(B, Hq, Hkv, L, 128, S, dtype="bf16", seed=3, seed_lo=0, seed_hi=L)
    rng = np.random.default_rng(4)
    tok, flags, masked, drafted = _state(B, L, rng)
    d_in, d_out = run_mass(inp, tok, flags, 0, L)
    sums = d_in.reshape(B, L).sum(axis=1)
    assert np.allclose(sums, masked.sum(axis=1), rtol=2e-3)
    assert np.all(d_out >= 0) and np.all(d_out <= 1 + 1e-3)


def test_mass_named_workload_sampled():
    wl = W.WORKLOADS["llada_b8_l2048"]
    inp = wl.attn_inputs()
    per = wl.score_N // wl.score_n_seq
    pos0 = wl.L - per
    rng = np.random.default_rng(5)
    tok, flags, masked, drafted = _state(wl.B, per, rng)
    d_in, d_out = run_mass(inp, tok, flags, pos0, per)
    ref_in, ref_out = oracle_mass(inp, masked, drafted, pos0, batches=[0, wl.B - 1])
    for k, b in enumerate([0, wl.B - 1]):
        sl = slice(b * per, (b + 1) * per)
        assert np.all(np.abs(d_in[sl] - ref_in[k]) <= _mass_tol(ref_in[k]))
        assert np.all(np.abs(d_out[sl] - ref_out[k]) <= _mass_tol(ref_out[k]))


def test_decide_update_mass_select_pipeline():
    """Section 5.3's order: update the state, take d_in / d_out of the updated state, then select."""
    B, Hq, Hkv, L, S = 2, 4, 2, 512, 12
    per, n_seq = 128, 2
    pos0 = L - per
    inp = W.make_attn_inputs(B, Hq, Hkv, L, 128, S, dtype="bf16", seed=9, seed_lo=0, seed_hi=L)
    di = W.make_decide_inputs(B * per, 3000, n_seq, seed=10, block_len=32)
    p = dict(tau_draft=0.8, draft_budget=6, remask_budget=5, mask_id=di.mask_id, min_one=True, pos0=pos0,
             max_seeds=8)
    logits = H.to_dev(di.logits, "bf16")
    tok = torch.from_numpy(di.tok.copy()).cuda()
    flags = torch.from_numpy(di.flags.copy()).cuda()
    rc = torch.from_numpy(di.remask_cnt.copy()).cuda()
    ws = api.decide_workspace(B * per, n_seq)
    draft_ok = torch.from_numpy(di.draft_ok).cuda()
    upd = api.cover_score_decide_fwd(logits, n_seq, tok, flags, rc, phase=api.COVER_DECIDE_UPDATE, workspace=ws,
                                     draft_ok=draft_ok, **p)
    torch.cuda.synchronize()
    tok_u, flags_u, rc_u = tok.cpu().numpy(), flags.cpu().numpy(), rc.cpu().numpy()
    args, lse = _attention(inp)
    d_in, d_out = api.cover_attn_mass_fwd(args[0], args[1], lse, tok, flags, mask_id=di.mask_id, pos0=pos0, per=per,
                                          k_seedmask=args[3], seed_idx=args[5])
    sel = api.cover_seed_select_fwd(n_seq, tok, flags, rc, ws, remask_budget=5, mask_id=di.mask_id, pos0=pos0,
                                    max_seeds=8, d_in=d_in, d_out=d_out)
    torch.cuda.synchronize()
    assert api.cover_device_status() == 0
    # the kernel's fp32 per-row values, read back through the plain scoring entry point
    u_cur = api.cover_score_fwd(logits, n_seq, 0, cur_tok=torch.from_numpy(di.tok).cuda())["score"].cpu().numpy()
    u_top = api.cover_score_fwd(logits, n_seq, 0)["score"].cpu().numpy()
    h = {k: v.cpu().numpy() for k, v in upd.items()}
    din, dout = d_in.cpu().numpy(), d_out.cpu().numpy()
    outs = oracle.decide_step(h["maxprob"], h["argmax"], h["entropy"], u_cur, u_top, din, dout, di.tok, di.flags,
                              di.remask_cnt, di.draft_ok, n_seq, tau=F32(0.8), budget=6, m_remask=5,
                              mask_id=di.mask_id, min_one=True, pos0=pos0, max_seeds=8)
    # the update phase: drafted rows carry flag bit 1, the previous seeds still bit 0
    drafted = np.zeros(B * per, bool)
    for g, o in enumerate(outs):
        sl = slice(g * per, (g + 1) * per)
        assert np.array_equal(tok_u[sl], o["tok"]) and np.array_equal(rc_u[sl], o["remask_cnt"])
        drafted[g * per + np.array(o["drafted"], dtype=int)] = True
    assert np.array_equal((flags_u & 2) != 0, drafted)
    assert np.array_equal(flags_u & 1, di.flags & 1 & ~drafted)
    # the select phase: final state, seeds and scores
    fl, sc = flags.cpu().numpy(), sel["score"].cpu().numpy()
    for g, o in enumerate(outs):
        sl = slice(g * per, (g + 1) * per)
        assert np.array_equal(fl[sl], o["flags"])
        assert np.array_equal(sc[sl], o["score"].astype(F32))
        assert sel["seed_idx"][g].tolist() == o["seeds"] + [-1] * (8 - len(o["seeds"]))
        assert sel["n_seeds"][g].item() == o["n_select"]
        assert sel["stats"][g, 4:].tolist() == [o["n_t"], o["n_above"]]
    # d_in / d_out of the updated state against the fp64 oracle
    masked = (tok_u == di.mask_id).reshape(B, per)
    ref_in, ref_out = oracle_mass(inp, masked, drafted.reshape(B, per), pos0)
    assert np.all(np.abs(din - ref_in.ravel()) <= _mass_tol(ref_in.ravel()))
    assert np.all(np.abs(dout - ref_out.ravel()) <= _mass_tol(ref_out.ravel()))
