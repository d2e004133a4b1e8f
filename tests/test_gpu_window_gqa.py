"""GPU parity of the packed grouped-query window kernel (the prefix-cache window of Section 6.6
for G = Hq / Hkv >= 2) against the fp64 oracle, and the choice between it and the square kernel.

cover_attn_fwd_prefix runs a window of grouped-query heads on the packed kernel where a launch-time
model predicts it to be faster; cover_debug_attn_prefix_packed runs the packed kernel on every
shape it supports, which the parity cases below use.

The kernel packs a KV head's G query heads into common 128-row Q tiles and splits the keys over
the CTAs of a cluster (T = ceil(nkv / 8) KV tiles per CTA, nsplit = ceil(nkv / T) CTAs), which
combine their partial (m, l, O) through distributed shared memory and merge a seed row's masked
self term there. The cases below reach one and several KV steps per CTA, clusters of 1 to 8
CTAs, one and two Q tiles, packed-row counts that end inside a 32-row warp, a ragged last KV
tile, a seed whose diagonal is the only key of its split, and routing of repeated and
out-of-range seed entries."""
import numpy as np
import pytest
import torch

import oracle
from paper_2602_06161_gb300 import CoverError, api
from paper_2602_06161_gb300 import workloads as W
from tests import _gpu as H
from tests.test_gpu_prefix import _case

pytestmark = pytest.mark.gpu


def _packed(q, kc, vc, km, vm, seeds, q0, Lq):
    out, lse = api.cover_debug_attn_prefix_packed(
        H.to_dev(np.ascontiguousarray(q[:, :, q0:q0 + Lq]), "bf16"), H.to_dev(kc, "bf16"), H.to_dev(vc, "bf16"),
        H.to_dev(km, "bf16"), H.to_dev(vm, "bf16"), H.to_dev(seeds, "i32"), q0=q0)
    torch.cuda.synchronize()
    assert api.cover_device_status() == 0
    return out.float().cpu().numpy(), lse.cpu().numpy()


def _check(q, kc, vc, km, vm, seeds, q0, Lq):
    out, lse = _packed(q, kc, vc, km, vm, seeds, q0, Lq)
    f = W.bf16_bits_to_f64
    ref, ref_lse = oracle.override_attention_window(f(q[:, :, q0:q0 + Lq]), f(kc), f(vc), f(km), f(vm),
                                                    seeds if seeds.shape[1] else None, q0)
    d = np.abs(out - ref)
    assert np.isfinite(out).all() and np.isfinite(lse).all()
    assert d.max() <= H.TOL_BF16_MAX and d.mean() <= H.TOL_BF16_MEAN, (d.max(), d.mean())
    assert np.abs(lse - ref_lse).max() <= H.TOL_LSE


@pytest.mark.parametrize("B,Hq,Hkv,Lk,Lq,q0,S,inside", [
    (1, 28, 4, 1024, 32, 992, 32, 6),      # Dream active block at the end: 8 one-step CTAs, 2 Q tiles
    (1, 28, 4, 1024, 32, 992, 0, 0),       # the same without seeds
    (1, 8, 2, 1100, 20, 1080, 12, 5),      # 9 KV tiles: 5 CTAs of 2, 1 steps; ragged tail holds diagonals
    (1, 8, 2, 8192, 32, 8160, 16, 8),      # 64 KV tiles: 8 CTAs of 8 steps each
    (1, 4, 2, 700, 128, 300, 10, 6),       # 256 packed rows (the limit), window in the middle
    (2, 9, 3, 333, 37, 100, 7, 3),         # 111 packed rows: the last warp's rows end mid-warp
    (1, 16, 2, 640, 16, 624, 5, 2),        # G = 8: one full Q tile
    (3, 10, 5, 90, 3, 40, 4, 2),           # one ragged KV tile: a cluster of one CTA
    (1, 28, 4, 1024, 128, 896, 32, 20),    # 896 packed rows: 7 Q tiles per KV head
    (2, 28, 4, 2048, 64, 1984, 24, 10),    # 16 KV tiles: 8 CTAs of 2 steps, 4 Q tiles
])
def test_packed_window_matches_oracle(B, Hq, Hkv, Lk, Lq, q0, S, inside):
    q, kc, vc, km, vm, seeds = _case(B, Hq, Hkv, Lk, 128, S, q0, Lq, "bf16", 3 * Lk + Lq, inside)
    _check(q, kc, vc, km, vm, seeds, q0, Lq)


def test_packed_window_seed_alone_in_its_split():
    # Lk = 129: the second KV tile holds one key, position 128, which is the window's row and a
    # seed; its cached diagonal is excluded, so that split has no key left for the row and the
    # combine must take the row from the other split and the masked self term alone
    B, Hq, Hkv, Lk, Lq, q0 = 2, 6, 2, 129, 1, 128
    q, kc, vc, km, vm, seeds = _case(B, Hq, Hkv, Lk, 128, 3, q0, Lq, "bf16", 41, 1)
    assert all(128 in seeds[b] for b in range(B))
    _check(q, kc, vc, km, vm, seeds, q0, Lq)


def test_packed_window_repeated_and_out_of_range_seeds():
    # a position named by two slots takes the lower slot's masked row; entries outside [0, Lk)
    # are ignored
    B, Hq, Hkv, Lk, Lq, q0, S = 2, 12, 4, 520, 40, 480, 10
    q, kc, vc, km, vm, seeds = _case(B, Hq, Hkv, Lk, 128, S, q0, Lq, "bf16", 57, 5)
    for b in range(B):
        inside = [s for s in seeds[b, :S - 3] if q0 <= s < q0 + Lq]
        assert inside
        seeds[b, -1] = inside[0]          # a later slot repeats a window seed
        seeds[b, -2] = -1
        seeds[b, -3] = Lk + 5
    _check(q, kc, vc, km, vm, seeds, q0, Lq)


def test_packed_window_rows_match_square_rows():
    # the packed kernel's rows agree with the same rows of the square launch up to rounding, and
    # back-to-back calls give identical bits
    B, Hq, Hkv, Lk, S = 2, 8, 2, 1100, 20
    q, kc, vc, km, vm, seeds = _case(B, Hq, Hkv, Lk, 128, S, 300, 200, "bf16", 7, 10)
    dq, dk, dv, dkm, dvm = (H.to_dev(x, "bf16") for x in (q, kc, vc, km, vm))
    ds = H.to_dev(seeds, "i32")
    full, full_lse = api.cover_attn_fwd(dq, dk, dv, dkm, dvm, ds)
    for q0, Lq in ((1099, 1), (300, 32), (1068, 32), (0, 64)):
        qw = dq[:, :, q0:q0 + Lq].contiguous()
        win, win_lse = api.cover_debug_attn_prefix_packed(qw, dk, dv, dkm, dvm, ds, q0=q0)
        again, again_lse = api.cover_debug_attn_prefix_packed(qw, dk, dv, dkm, dvm, ds, q0=q0)
        torch.cuda.synchronize()
        d = (win.float() - full[:, :, q0:q0 + Lq].float()).abs()
        assert d.max().item() <= H.TOL_BF16_MAX and d.mean().item() <= H.TOL_BF16_MEAN, (q0, Lq)
        assert (win_lse - full_lse[:, :, q0:q0 + Lq]).abs().max().item() <= H.TOL_LSE, (q0, Lq)
        assert torch.equal(win, again) and torch.equal(win_lse, again_lse), (q0, Lq)
    assert api.cover_device_status() == 0


@pytest.mark.parametrize("B,Hq,Hkv,Lk,Lq,packed", [
    (1, 28, 4, 1024, 32, True),     # Dream active block: 8 clusters of 8 one-step CTAs
    (1, 32, 8, 8192, 32, True),     # long memory: 8 steps per packed CTA against 32 per warpgroup
    (3, 10, 5, 90, 3, False),       # one KV tile: the square kernel's short chain wins
    (8, 32, 8, 2048, 64, False),    # 128 clusters: many waves of packed CTAs
])
def test_prefix_call_picks_the_predicted_kernel(B, Hq, Hkv, Lk, Lq, packed):
    # the call's result equals, bit for bit, the kernel the launch-time model picks for the shape
    q0 = Lk - Lq
    q, kc, vc, km, vm, seeds = _case(B, Hq, Hkv, Lk, 128, 6, q0, Lq, "bf16", 5 + Lk, 2)
    dev = [H.to_dev(np.ascontiguousarray(q[:, :, q0:]), "bf16"), H.to_dev(kc, "bf16"), H.to_dev(vc, "bf16"),
           H.to_dev(km, "bf16"), H.to_dev(vm, "bf16"), H.to_dev(seeds, "i32")]
    prod, prod_lse = api.cover_attn_fwd_prefix(*dev, q0=q0)
    pk, pk_lse = api.cover_debug_attn_prefix_packed(*dev, q0=q0)
    sq, sq_lse = api.cover_debug_attn_fault(*dev, q0=q0, fault_cta=-1, fault_entry=-1, limit_us=1000000)
    torch.cuda.synchronize()
    assert api.cover_device_status() == 0
    ref = (pk, pk_lse) if packed else (sq, sq_lse)
    assert torch.equal(prod, ref[0]) and torch.equal(prod_lse, ref[1])
    assert (pk.float() - sq.float()).abs().max().item() <= H.TOL_BF16_MAX


def test_packed_entry_refuses_what_the_packed_kernel_does_not_run():
    q, kc, vc, km, vm, seeds = _case(1, 4, 4, 256, 128, 4, 192, 64, "bf16", 9, 2)
    dev = [H.to_dev(kc, "bf16"), H.to_dev(vc, "bf16"), H.to_dev(km, "bf16"), H.to_dev(vm, "bf16"),
           H.to_dev(seeds, "i32")]
    with pytest.raises(CoverError) as e:   # G = 1: no query heads to pack
        api.cover_debug_attn_prefix_packed(H.to_dev(np.ascontiguousarray(q[:, :, 192:]), "bf16"), *dev, q0=192)
    assert e.value.code == -2
    q, kc, vc, km, vm, seeds = _case(1, 4, 2, 256, 128, 4, 0, 256, "bf16", 9, 2)
    with pytest.raises(CoverError) as e:   # the square call
        api.cover_debug_attn_prefix_packed(H.to_dev(q, "bf16"), H.to_dev(kc, "bf16"), H.to_dev(vc, "bf16"),
                                           H.to_dev(km, "bf16"), H.to_dev(vm, "bf16"), H.to_dev(seeds, "i32"),
                                           q0=0)
    assert e.value.code == -2


def test_packed_planted_missing_load_aborts_cleanly():
    # The packed kernel's self-test instance: CTA 0 (key split 0 of Q tile 0 of KV head 0) leaves
    # out its first K load and every wait gives up after 20 ms. Its waits for that tile time out,
    # or the waits of its cluster's CTAs for its partial block, every role leaves its loop, the cluster's copies and barriers still
    # complete, and the launch returns well within a second. The rows CTA 0's cluster combines
    # (packed rows 0..127 of KV head 0: query heads 0..3 of the Dream shape) are unspecified;
    # every other row is bit-identical to a clean launch, and so is the next clean launch.
    import time
    B, Hq, Hkv, Lk, Lq, q0, S = 1, 28, 4, 1024, 32, 992, 32
    q, kc, vc, km, vm, seeds = _case(B, Hq, Hkv, Lk, 128, S, q0, Lq, "bf16", 71, 6)
    dev = [H.to_dev(np.ascontiguousarray(q[:, :, q0:]), "bf16"), H.to_dev(kc, "bf16"), H.to_dev(vc, "bf16"),
           H.to_dev(km, "bf16"), H.to_dev(vm, "bf16"), H.to_dev(seeds, "i32")]
    clean, clean_lse = api.cover_debug_attn_prefix_packed(*dev, q0=q0)
    torch.cuda.synchronize()
    assert api.cover_debug_status_detail() == (0, 0, 0)
    out = torch.full_like(clean, float("nan"))
    lse = torch.full_like(clean_lse, float("nan"))
    t0 = time.perf_counter()
    api.cover_debug_attn_prefix_packed(*dev, q0=q0, fault_cta=0, limit_us=20000, out=out, lse=lse)
    code, site, block = api.cover_debug_status_detail()
    elapsed = time.perf_counter() - t0
    # the first wait to give up: CTA 0's MMA thread waiting for the tile (60) or its softmax warps
    # waiting for the product (61), or a CTA of its cluster waiting for CTA 0's block of its rows
    # (62); all have the same limit
    assert code == -4 and (site in (60, 61) and block == 0 or site == 62 and 0 < block < 8), (code, site, block)
    assert elapsed < 0.5
    assert api.cover_debug_status_detail() == (0, 0, 0)
    G = Hq // Hkv
    mine = torch.zeros((B, Hq, Lq), dtype=torch.bool, device="cuda")
    mine.view(B, Hkv, G * Lq)[0, 0, :128] = True
    assert torch.equal(out[~mine], clean[~mine]) and torch.equal(lse[~mine], clean_lse[~mine])
    again, again_lse = api.cover_debug_attn_prefix_packed(*dev, q0=q0)
    torch.cuda.synchronize()
    assert api.cover_device_status() == 0
    assert torch.equal(again, clean) and torch.equal(again_lse, clean_lse)
