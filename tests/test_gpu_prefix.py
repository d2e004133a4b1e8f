"""GPU parity of the prefix-cache window attention (Section 6.6) against the fp64 oracle."""
import numpy as np
import pytest
import torch

import oracle
from paper_2602_06161_gb300 import api
from paper_2602_06161_gb300 import workloads as W
from tests import _gpu as H

pytestmark = pytest.mark.gpu


def _case(B, Hq, Hkv, Lk, D, S, q0, Lq, dtype, seed, inside):
    """Memory of Lk positions; `inside` of the S seeds fall in the window [q0, q0 + Lq)."""
    inp = W.make_attn_inputs(B, Hq, Hkv, Lk, D, 0, dtype=dtype, seed=seed, seed_lo=0, seed_hi=Lk)
    rng = np.random.default_rng(seed + 100)
    seeds = np.zeros((B, S), np.int32)
    for b in range(B):
        win = rng.choice(np.arange(q0, q0 + Lq), size=min(inside, Lq), replace=False)
        rest = np.setdiff1d(np.arange(Lk), win)
        out = rng.choice(rest, size=S - len(win), replace=False)
        seeds[b] = rng.permutation(np.concatenate([win, out]))
    side = W.make_attn_inputs(B, Hq, Hkv, S, D, 0, dtype=dtype, seed=seed + 1, seed_lo=0, seed_hi=S)
    return inp.q, inp.k_cached, inp.v_cached, side.k_cached, side.v_cached, seeds


def run_window(q_full, kc, vc, km, vm, seeds, q0, Lq, dtype):
    dt = dtype
    q = q_full[:, :, q0:q0 + Lq]
    fn = api.cover_attn_fwd_prefix if dt == "bf16" else api.cover_attn_fwd_prefix_f32
    out, lse = fn(H.to_dev(np.ascontiguousarray(q), dt), H.to_dev(kc, dt), H.to_dev(vc, dt), H.to_dev(km, dt),
                  H.to_dev(vm, dt), H.to_dev(seeds, "i32"), q0=q0)
    torch.cuda.synchronize()
    assert api.cover_device_status() == 0
    return out.float().cpu().numpy(), lse.cpu().numpy()


@pytest.mark.parametrize("B,Hq,Hkv,Lk,Lq,q0,S,inside", [
    (1, 4, 2, 300, 64, 236, 6, 3),          # window at the end, not 128-aligned
    (2, 4, 4, 1000, 100, 450, 12, 5),       # window in the middle, diagonal crossing a KV tile
    (1, 2, 1, 2048, 64, 1984, 16, 8),       # LLaDA-like active block of 64 at the end of the memory
    (2, 28, 4, 1024, 32, 512, 32, 4),       # Dream-like GQA 28/4, block of 32
    (1, 2, 2, 513, 513, 0, 8, 8),           # the whole memory: the square case
    (1, 2, 2, 400, 1, 257, 3, 1),           # a single query row that is a seed
    (1, 2, 2, 700, 300, 200, 0, 0),         # no seeds
    # 320 one-tile units: CTAs run two or three back to back
    (8, 40, 40, 128, 64, 64, 8, 4),         # one KV tile per unit
    (8, 40, 8, 100, 30, 70, 6, 3),          # one ragged KV tile, GQA 5:1
    (8, 40, 40, 256, 64, 192, 8, 4),        # two KV tiles per unit
    (8, 40, 40, 768, 100, 600, 8, 4),       # six KV tiles: three per warpgroup in every split unit
    (2, 4, 2, 768, 128, 640, 10, 6),        # a full 128-row window tile, GQA 2:1
])
def test_window_bf16(B, Hq, Hkv, Lk, Lq, q0, S, inside):
    q, kc, vc, km, vm, seeds = _case(B, Hq, Hkv, Lk, 128, S, q0, Lq, "bf16", Lk + Lq, inside)
    out, lse = run_window(q, kc, vc, km, vm, seeds, q0, Lq, "bf16")
    f = W.bf16_bits_to_f64
    ref, ref_lse = oracle.override_attention_window(f(q[:, :, q0:q0 + Lq]), f(kc), f(vc), f(km), f(vm),
                                                    seeds if S else None, q0)
    d = np.abs(out - ref)
    assert d.max() <= H.TOL_BF16_MAX and d.mean() <= H.TOL_BF16_MEAN, (d.max(), d.mean())
    assert np.abs(lse - ref_lse).max() <= H.TOL_LSE


@pytest.mark.parametrize("D,Lk,Lq,q0", [(64, 100, 30, 70), (128, 77, 20, 3)])
def test_window_f32(D, Lk, Lq, q0):
    q, kc, vc, km, vm, seeds = _case(2, 4, 2, Lk, D, 6, q0, Lq, "f32", D + Lk, 3)
    out, lse = run_window(q, kc, vc, km, vm, seeds, q0, Lq, "f32")
    ref, ref_lse = oracle.override_attention_window(q[:, :, q0:q0 + Lq].astype(np.float64), kc.astype(np.float64),
                                                    vc.astype(np.float64), km.astype(np.float64),
                                                    vm.astype(np.float64), seeds, q0)
    assert np.abs(out - ref).max() <= H.TOL_F32 and np.abs(lse - ref_lse).max() <= H.TOL_F32


def test_window_rows_equal_square_rows_bit_exactly():
    # a query row's arithmetic does not depend on where its tile starts: the window rows
    # are bit-identical to the same rows of the square launch (an odd number of KV tiles,
    # so the square launch does not split any unit's keys over two CTAs). The windows run on the
    # square kernel through the fault entry with no planted load: the prefix call itself may take
    # the packed grouped-query kernel, whose rows agree up to rounding (test_gpu_window_gqa.py)
    B, Hq, Hkv, Lk, S = 2, 4, 2, 1100, 20
    q, kc, vc, km, vm, seeds = _case(B, Hq, Hkv, Lk, 128, S, 300, 200, "bf16", 7, 10)
    dq, dk, dv, dkm, dvm = (H.to_dev(x, "bf16") for x in (q, kc, vc, km, vm))
    ds = H.to_dev(seeds, "i32")
    full, full_lse = api.cover_attn_fwd(dq, dk, dv, dkm, dvm, ds)
    for q0, Lq in ((300, 200), (0, 1100), (1099, 1), (130, 257)):
        win, win_lse = api.cover_debug_attn_fault(dq[:, :, q0:q0 + Lq].contiguous(), dk, dv, dkm, dvm, ds, q0=q0,
                                                  fault_cta=-1, fault_entry=-1, limit_us=1000000)
        torch.cuda.synchronize()
        assert torch.equal(win, full[:, :, q0:q0 + Lq]), (q0, Lq)
        assert torch.equal(win_lse, full_lse[:, :, q0:q0 + Lq]), (q0, Lq)
    assert api.cover_device_status() == 0


def test_window_rows_match_split_square_rows():
    # with an even number of KV tiles and few units the square launch splits every unit's keys
    # over two CTAs (merged in the epilogue); the window rows then agree up to rounding
    B, Hq, Hkv, Lk, S = 2, 4, 2, 1000, 20
    q, kc, vc, km, vm, seeds = _case(B, Hq, Hkv, Lk, 128, S, 300, 200, "bf16", 7, 10)
    dq, dk, dv, dkm, dvm = (H.to_dev(x, "bf16") for x in (q, kc, vc, km, vm))
    ds = H.to_dev(seeds, "i32")
    full, full_lse = api.cover_attn_fwd(dq, dk, dv, dkm, dvm, ds)
    for q0, Lq in ((300, 200), (999, 1)):
        win, win_lse = api.cover_attn_fwd_prefix(dq[:, :, q0:q0 + Lq].contiguous(), dk, dv, dkm, dvm, ds, q0=q0)
        torch.cuda.synchronize()
        d = (win.float() - full[:, :, q0:q0 + Lq].float()).abs()
        assert d.max().item() <= H.TOL_BF16_MAX and d.mean().item() <= H.TOL_BF16_MEAN, (q0, Lq)
        assert (win_lse - full_lse[:, :, q0:q0 + Lq]).abs().max().item() <= H.TOL_LSE, (q0, Lq)
    assert api.cover_device_status() == 0
