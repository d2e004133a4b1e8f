"""GPU parity of the override-attention kernels against the fp64 oracle.

Everything goes through the C ABI (via the ctypes binding). Inputs come from
the seeded generators; expected values come only from oracle/.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2602_06161_gb300 import api
from paper_2602_06161_gb300 import workloads as W
from tests import _gpu as H
from tests import _oracle_pool as OP

pytestmark = pytest.mark.gpu


# ----------------------------------------------------------------------------
# building blocks
# ----------------------------------------------------------------------------

def test_umma_tile_operand_layouts():
    g = torch.Generator().manual_seed(0)
    a, b, p, v = [torch.randn(128, 128, generator=g).to(torch.bfloat16) for _ in range(4)]
    c1, c2 = api.cover_debug_umma_tile(a.cuda(), b.cuda(), p.cuda(), v.cuda())
    torch.cuda.synchronize()
    assert api.cover_device_status() == 0
    r1 = a.double() @ b.double().T
    r2 = p.double() @ v.double()
    e1 = (c1.cpu().double() - r1).abs().max().item()
    e2 = (c2.cpu().double() - r2).abs().max().item()
    assert e1 < 1e-3 and e2 < 1e-3, (e1, e2, c1[:2, :4].tolist(), r1[:2, :4].tolist(), c2[:2, :4].tolist(),
                                     r2[:2, :4].tolist())


@pytest.mark.parametrize("route", [api.cover_seed_route, api.cover_seed_route_debug])
def test_seed_routing_bit_exact(route):
    L = 300
    seeds = np.array([[5, 130, 5, -1, 300, 127, 128, 299],
                      [0, 0, 0, 1, 2, 3, 255, 1000]], dtype=np.int32)
    slot, bitmap, n_inv = route(H.to_dev(seeds, "i32"), 2, L)
    ref_slot, ref_bitmap, ref_inv = oracle.route_seeds(seeds, L)
    assert np.array_equal(slot.cpu().numpy(), ref_slot)
    assert np.array_equal(bitmap.cpu().numpy().view(np.uint32), ref_bitmap)
    assert int(n_inv.item()) == ref_inv


def test_seed_routing_random():
    rng = np.random.default_rng(5)
    B, L, S = 3, 1000, 400
    seeds = rng.integers(-20, L + 20, size=(B, S)).astype(np.int32)
    slot, bitmap, n_inv = api.cover_seed_route(H.to_dev(seeds, "i32"), B, L)
    ref_slot, ref_bitmap, ref_inv = oracle.route_seeds(seeds, L)
    assert np.array_equal(slot.cpu().numpy(), ref_slot)
    assert np.array_equal(bitmap.cpu().numpy().view(np.uint32), ref_bitmap)
    assert int(n_inv.item()) == ref_inv


def test_bounded_wait_reports_timeout_and_context_survives():
    api.cover_debug_wait_timeout(20000)  # 20 ms
    assert api.cover_device_status() == -4
    assert api.cover_device_status() == 0   # cleared
    inp = W.make_attn_inputs(1, 2, 2, 64, 64, 4, dtype="f32", seed=0, seed_lo=32, seed_hi=64)
    out, lse = H.run_attn(inp)
    ref, ref_lse = H.oracle_full(inp)
    H.assert_f32_close(out, ref, lse, ref_lse)


# ----------------------------------------------------------------------------
# fp32 path
# ----------------------------------------------------------------------------

def test_tiny_f32_workload():
    inp = W.WORKLOADS["tiny_f32_l64"].attn_inputs()
    out, lse = H.run_attn(inp)
    ref, ref_lse = H.oracle_full(inp)
    H.assert_f32_close(out, ref, lse, ref_lse, "tiny_f32_l64")


@pytest.mark.parametrize("B,Hq,Hkv,L,D,S", [
    (1, 1, 1, 1, 64, 1), (1, 2, 1, 3, 64, 3), (2, 4, 2, 37, 128, 5), (1, 7, 1, 130, 64, 0), (1, 2, 2, 65, 128, 65),
])
def test_f32_shapes(B, Hq, Hkv, L, D, S):
    inp = W.make_attn_inputs(B, Hq, Hkv, L, D, S, dtype="f32", seed=L + S)
    out, lse = H.run_attn(inp)
    ref, ref_lse = H.oracle_full(inp)
    H.assert_f32_close(out, ref, lse, ref_lse)


# ----------------------------------------------------------------------------
# bf16 tcgen05 path: small shapes, ragged tails, seeds in every position class
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("B,Hq,Hkv,L,S", [
    (1, 1, 1, 128, 0),        # one tile, no seeds
    (1, 1, 1, 256, 7),        # two Q tiles in one CTA
    (1, 2, 1, 512, 16),       # several KV tiles, GQA G=2
    (2, 7, 1, 384, 40),       # G=7, second Q tile of the last CTA out of range
    (1, 2, 2, 1, 1),          # L = 1: a seed row sees only its masked pair
    (1, 1, 1, 5, 2),          # tiny ragged
    (1, 2, 1, 129, 3),        # one key in the tail tile
    (1, 4, 2, 300, 300),      # every row a seed
    (2, 4, 4, 1000, 33),      # ragged, several CTAs
    (1, 8, 2, 768, 20),       # GQA 4:1, every unit split over two CTAs (few units, even KV count)
])
def test_bf16_shapes(B, Hq, Hkv, L, S):
    inp = W.make_attn_inputs(B, Hq, Hkv, L, 128, S, dtype="bf16", seed=B * 1000 + L + S)
    out, lse = H.run_attn(inp)
    ref, ref_lse = H.oracle_full(inp)
    H.assert_bf16_close(out, ref, lse, ref_lse, f"B{B} Hq{Hq} Hkv{Hkv} L{L} S{S}")


def test_bf16_seed_in_tail_tile_diagonal():
    # seeds at the last position and at the only key of a one-key tail tile
    inp = W.make_attn_inputs(1, 2, 1, 257, 128, 3, dtype="bf16", seed=3)
    inp.seed_idx[0] = [256, 255, 0]
    out, lse = H.run_attn(inp)
    ref, ref_lse = H.oracle_full(inp)
    H.assert_bf16_close(out, ref, lse, ref_lse)


def test_bf16_dominant_diagonal():
    # a seed row whose cached diagonal would hold almost all the weight (alpha > 0.999)
    inp = W.make_attn_inputs(1, 1, 1, 256, 128, 4, dtype="bf16", seed=4)
    q = W.bf16_bits_to_f32(inp.q)
    kc = W.bf16_bits_to_f32(inp.k_cached)
    for i in inp.seed_idx[0]:
        kc[0, 0, i] = q[0, 0, i] / np.linalg.norm(q[0, 0, i]) * 60.0
    inp.k_cached = W.f32_to_bf16_bits(kc)
    out, lse = H.run_attn(inp)
    ref, ref_lse = H.oracle_full(inp)
    H.assert_bf16_close(out, ref, lse, ref_lse)


def test_bf16_gqa_several_rounds_and_split_sampled():
    """GQA 5:1 with more units than SMs: every CTA runs several whole units back to back (its
    pipelines carried across unit boundaries), then the last round's units are split over two
    CTAs each. Seed rows and a sample of other rows of heads in the first, a middle and the
    split last round against the oracle."""
    B, Hq, Hkv, L, S = 2, 40, 8, 1536, 48
    inp = W.make_attn_inputs(B, Hq, Hkv, L, 128, S, dtype="bf16", seed=21)
    out, lse = H.run_attn(inp)
    rng = np.random.default_rng(22)
    for b, hq in [(0, 0), (0, 17), (1, 39)]:
        seeds = [int(x) for x in inp.seed_idx[b] if 0 <= x < L]
        others = rng.choice(np.setdiff1d(np.arange(L), seeds), size=48, replace=False).tolist()
        rows = sorted(set(seeds)) + others
        ref, ref_lse = H.oracle_head_rows(inp, b, hq, rows)
        H.assert_bf16_close(out[b, hq, rows], ref, lse[b, hq, rows], ref_lse, f"b{b} h{hq}")


def test_bf16_split_last_round():
    """More units than SMs with a small remainder: the units of the last round are split
    over two CTAs each (the two KV halves merged in the epilogue). Every row of the last head
    (split units) and of the first head (whole units) against the oracle."""
    B, Hq, Hkv, L, S = 1, 39, 39, 1024, 24
    inp = W.make_attn_inputs(B, Hq, Hkv, L, 128, S, dtype="bf16", seed=11)
    out, lse = H.run_attn(inp)
    rows = list(range(L))
    for hq in (0, Hq - 1):
        ref, ref_lse = H.oracle_head_rows(inp, 0, hq, rows)
        H.assert_bf16_close(out[0, hq], ref, lse[0, hq], ref_lse, f"head {hq}")


@pytest.mark.parametrize("B,Hq,L,heads", [
    # one KV tile per unit, 320 units: CTAs run two or three units back to back, every ring
    # entry reusing a stage that still holds the output of the unit two entries back
    (8, 40, 128, [(0, 0), (3, 30), (7, 39)]),
    # two KV tiles per unit, 160 units: one whole unit per CTA, then the last 8 units split over
    # two CTAs each with a single KV step per warpgroup
    (4, 40, 256, [(0, 0), (3, 31), (3, 32), (3, 39)]),
])
def test_bf16_short_units_several_per_cta(B, Hq, L, heads):
    inp = W.make_attn_inputs(B, Hq, Hq, L, 128, 12, dtype="bf16", seed=B * 100 + L)
    out, lse = H.run_attn(inp)
    rows = list(range(L))
    for b, hq in heads:
        ref, ref_lse = H.oracle_head_rows(inp, b, hq, rows)
        H.assert_bf16_close(out[b, hq], ref, lse[b, hq], ref_lse, f"L{L} b{b} h{hq}")


@pytest.mark.parametrize("name", ["llada_mha_l512", "dream_gqa_l1024"])
def test_bf16_named_workloads_full(name):
    inp = W.WORKLOADS[name].attn_inputs()
    out, lse = H.run_attn(inp)
    ref, ref_lse = H.oracle_full(inp)
    H.assert_bf16_close(out, ref, lse, ref_lse, name)


@pytest.mark.parametrize("name", ["llada_b8_l2048", "gqa_l8192_stress"])
def test_bf16_named_workloads_sampled(name):
    """Full-size launch; the oracle checks every seed row and a random sample of
    other rows of a few heads, one explicit view per row."""
    inp = W.WORKLOADS[name].attn_inputs()
    out, lse = H.run_attn(inp)
    rng = np.random.default_rng(99)
    heads = [(0, 0), (inp.B - 1, inp.Hq - 1), (inp.B // 2, inp.Hq // 2 + 1)]
    for b, hq in heads:
        seeds = [int(s) for s in inp.seed_idx[b]]
        others = rng.choice(np.setdiff1d(np.arange(inp.L), seeds), size=64, replace=False).tolist()
        rows = seeds + others
        ref, ref_lse = H.oracle_head_rows(inp, b, hq, rows)
        H.assert_bf16_close(out[b, hq, rows], ref, lse[b, hq, rows], ref_lse, f"{name} b{b} h{hq}")


@pytest.mark.parametrize("name", ["llada_b8_l2048", "gqa_l8192_stress"])
def test_bf16_named_workloads_whole_tensor(name):
    """Full-size launch compared with the oracle on every element of out and lse (every head,
    every row; the oracle's heads run in spawned worker processes)."""
    inp = W.WORKLOADS[name].attn_inputs()
    args = _dev_inputs(inp)
    out, lse = api.cover_attn_fwd(*args)
    torch.cuda.synchronize()
    assert api.cover_device_status() == 0
    out_bits = out.view(torch.int16).cpu().numpy().view(np.uint16)
    lse_h = lse.cpu().numpy()
    del out, lse, args
    G = inp.Hq // inp.Hkv
    heads = [(b, hq) for b in range(inp.B) for hq in range(inp.Hq)]
    tasks = ((inp.q[b, hq], inp.k_cached[b, hq // G], inp.v_cached[b, hq // G], inp.k_seedmask[b, hq // G],
              inp.v_seedmask[b, hq // G], inp.seed_idx[b], out_bits[b, hq], lse_h[b, hq]) for b, hq in heads)
    dmax, dmean, lmax, n = OP.check_heads(tasks, len(heads))
    print(f"{name}: {n} heads, max |d| {dmax:.3e}, mean |d| {dmean:.3e}, lse max |d| {lmax:.3e}")
    assert n == len(heads)
    assert dmax <= H.TOL_BF16_MAX and dmean <= H.TOL_BF16_MEAN and lmax <= H.TOL_LSE, (dmax, dmean, lmax)


# ----------------------------------------------------------------------------
# invariances (bit-exact on the GPU) and determinism
# ----------------------------------------------------------------------------

def _dev_inputs(inp):
    return [H.to_dev(inp.q, "bf16"), H.to_dev(inp.k_cached, "bf16"), H.to_dev(inp.v_cached, "bf16"),
            H.to_dev(inp.k_seedmask, "bf16"), H.to_dev(inp.v_seedmask, "bf16"), H.to_dev(inp.seed_idx, "i32")]


def test_bf16_dominant_self_term():
    """Seed rows whose masked self score lies far above the row's other scores: the self term's
    weight relative to the running maximum is ~2^45 for some rows and 2^140 to 2^175 for others
    (beyond the bf16 range of the probabilities P; the merge rescales O instead)."""
    inp = W.make_attn_inputs(1, 2, 1, 384, 128, 12, dtype="bf16", seed=5)
    q = W.bf16_bits_to_f32(inp.q)
    km = W.bf16_bits_to_f32(inp.k_seedmask)
    for s, i in enumerate(inp.seed_idx[0]):
        lam = 35.0 if s % 2 == 0 else 115.0
        # head 0's query of row i sets the direction; the masked key is shared by both query heads
        km[0, 0, s] = q[0, 0, i] / np.linalg.norm(q[0, 0, i]) * lam
    inp.k_seedmask = W.f32_to_bf16_bits(km)
    out, lse = H.run_attn(inp)
    ref, ref_lse = H.oracle_full(inp)
    H.assert_bf16_close(out, ref, lse, ref_lse)


def test_bf16_invariances_bit_exact():
    inp = W.make_attn_inputs(2, 4, 2, 640, 128, 24, dtype="bf16", seed=21)
    args = _dev_inputs(inp)
    out0, lse0 = api.cover_attn_fwd(*args)
    # a seed row must not change at all when its own cached pair changes (other rows do see it)
    for b, s in [(0, 0), (0, 5), (1, 11), (1, 23)]:
        i = int(inp.seed_idx[b, s])
        kc, vc = args[1].clone(), args[2].clone()
        kc[b, :, i] = kc[b, :, i] * 3 + 1
        vc[b, :, i] = -vc[b, :, i] + 2
        out1, lse1 = api.cover_attn_fwd(args[0], kc, vc, *args[3:])
        torch.cuda.synchronize()
        assert torch.equal(out0[b, :, i], out1[b, :, i])
        assert torch.equal(lse0[b, :, i], lse1[b, :, i])
        j = (i + 1) % 640
        assert not torch.equal(out0[b, :, j], out1[b, :, j])
    # non-seed rows must not change at all when the masked buffer changes
    out2, lse2 = api.cover_attn_fwd(*args[:3], args[3] * 5 - 1, args[4] + 3, args[5])
    torch.cuda.synchronize()
    seed_mask = np.zeros((2, 640), bool)
    for b in range(2):
        seed_mask[b, inp.seed_idx[b]] = True
    sm = torch.from_numpy(seed_mask).cuda()
    for b in range(2):
        assert torch.equal(out0[b][:, ~sm[b]], out2[b][:, ~sm[b]])
        assert torch.equal(lse0[b][:, ~sm[b]], lse2[b][:, ~sm[b]])
        assert not torch.equal(out0[b][:, sm[b]], out2[b][:, sm[b]])


def test_bf16_deterministic_and_guard_bands():
    inp = W.make_attn_inputs(1, 4, 2, 700, 128, 9, dtype="bf16", seed=22)
    args = _dev_inputs(inp)
    n = 1 * 4 * 700 * 128
    guard = 4096
    buf = torch.full((n + 2 * guard,), float("nan"), dtype=torch.bfloat16, device="cuda")
    lbuf = torch.full((4 * 700 + 2 * guard,), float("nan"), dtype=torch.float32, device="cuda")
    out = buf[guard:guard + n].view(1, 4, 700, 128)
    lse = lbuf[guard:guard + 4 * 700].view(1, 4, 700)
    api.cover_attn_fwd(*args, out=out, lse=lse)
    out_b, lse_b = api.cover_attn_fwd(*args)
    torch.cuda.synchronize()
    assert torch.equal(out, out_b) and torch.equal(lse, lse_b)
    assert torch.isnan(buf[:guard].float()).all() and torch.isnan(buf[guard + n:].float()).all()
    assert torch.isnan(lbuf[:guard]).all() and torch.isnan(lbuf[guard + 4 * 700:]).all()
    assert not torch.isnan(out.float()).any()


def test_no_seed_path_equals_sdpa_shape():
    # zero seeds: plain attention over K', V' (the overhead baseline of the benchmark)
    inp = W.make_attn_inputs(1, 8, 2, 1024, 128, 0, dtype="bf16", seed=23)
    out, lse = H.run_attn(inp)
    ref, ref_lse = H.oracle_full(inp)
    H.assert_bf16_close(out, ref, lse, ref_lse)
