"""GPU parity of the seed K/V cache kernels (Section 5.1): bit-exact against the oracle."""
import numpy as np
import pytest
import torch

import oracle
from paper_2602_06161_gb300 import api
from paper_2602_06161_gb300 import workloads as W
from tests import _gpu as H

pytestmark = pytest.mark.gpu


def _bits(shape, rng, dtype):
    if dtype == "bf16":
        return rng.integers(0, 1 << 16, size=shape, dtype=np.uint16)
    return rng.standard_normal(shape).astype(np.float32)


def _dev(a, dtype):
    return H.to_dev(a, dtype)


def _host(t, dtype):
    if dtype == "bf16":
        return t.view(torch.int16).cpu().numpy().view(np.uint16)
    return t.cpu().numpy()


def _seeds(B, S, L, rng, invalid=True):
    seeds = np.stack([rng.choice(L, size=min(S, L), replace=False) for _ in range(B)]).astype(np.int32)
    if seeds.shape[1] < S:
        seeds = np.concatenate([seeds, np.full((B, S - seeds.shape[1]), -1, np.int32)], axis=1)
    if invalid and S >= 4:
        seeds[0, -1] = -1                # padding, as the decision step writes it
        seeds[-1, -2] = L + 3            # out of range
        seeds[-1, -3] = seeds[-1, 0]     # repeats a lower slot's position
    return seeds


@pytest.mark.parametrize("B,Hkv,L,D,S,dtype", [
    (1, 1, 1, 64, 1, "bf16"), (2, 4, 300, 128, 7, "bf16"), (3, 2, 129, 8, 40, "bf16"), (2, 3, 50, 4, 9, "f32"),
    (1, 2, 64, 64, 64, "f32"), (8, 32, 2048, 128, 64, "bf16"), (4, 8, 8192, 128, 256, "bf16"),
])
def test_gather_and_override(B, Hkv, L, D, S, dtype):
    rng = np.random.default_rng(B * 1000 + S)
    k, v = _bits((B, Hkv, L, D), rng, dtype), _bits((B, Hkv, L, D), rng, dtype)
    kbar, vbar = _bits((B, Hkv, S, D), rng, dtype), _bits((B, Hkv, S, D), rng, dtype)
    seeds = _seeds(B, S, L, rng)
    dk, dv, ds = _dev(k, dtype), _dev(v, dtype), _dev(seeds, "i32")
    # gather
    gk, gv = api.cover_seed_kv_gather(dk, dv, ds)
    torch.cuda.synchronize()
    rk, rv = oracle.seed_kv_gather(k, v, seeds)
    assert np.array_equal(_host(gk, dtype), rk) and np.array_equal(_host(gv, dtype), rv)
    # override (in place)
    ck, cv = _dev(kbar, dtype), _dev(vbar, dtype)
    api.cover_seed_kv_override(dk, dv, ds, ck, cv)
    torch.cuda.synchronize()
    assert api.cover_device_status() == 0
    k2, v2, km, vm = oracle.seed_kv_override(k, v, seeds, kbar, vbar)
    assert np.array_equal(_host(dk, dtype), k2) and np.array_equal(_host(dv, dtype), v2)
    assert np.array_equal(_host(ck, dtype), km) and np.array_equal(_host(cv, dtype), vm)
    # swapping again restores every buffer
    api.cover_seed_kv_override(dk, dv, ds, ck, cv)
    torch.cuda.synchronize()
    assert np.array_equal(_host(dk, dtype), k) and np.array_equal(_host(ck, dtype), kbar)


def test_no_seeds_leaves_memory_alone():
    rng = np.random.default_rng(3)
    k = _bits((1, 2, 32, 128), rng, "bf16")
    dk, dv = _dev(k, "bf16"), _dev(k, "bf16")
    api.cover_seed_kv_override(dk, dv, None, None, None)
    torch.cuda.synchronize()
    assert np.array_equal(_host(dk, "bf16"), k)


def test_cache_then_override_then_attention():
    """Step t-1 caches the new seeds' states; step t overrides the masked-input memory with them and runs
    the two-view attention on the result: equal to the oracle's leave-one-out views of Section 5.1."""
    B, Hq, Hkv, L, D, S = 2, 4, 2, 384, 128, 12
    rng = np.random.default_rng(5)
    prev = W.make_attn_inputs(B, Hq, Hkv, L, D, S, dtype="bf16", seed=6, seed_lo=0, seed_hi=L)
    new = W.make_attn_inputs(B, Hq, Hkv, L, D, S, dtype="bf16", seed=7, seed_lo=0, seed_hi=L)
    seeds = prev.seed_idx
    # step t-1: cache the seeds' states from that step's memory
    kc, vc = api.cover_seed_kv_gather(_dev(prev.k_cached, "bf16"), _dev(prev.v_cached, "bf16"), _dev(seeds, "i32"))
    # step t: the layer's states from the input with the seeds masked, then the override swap
    dk, dv = _dev(new.k_cached, "bf16"), _dev(new.v_cached, "bf16")
    api.cover_seed_kv_override(dk, dv, _dev(seeds, "i32"), kc, vc)
    q = _dev(new.q, "bf16")
    out, lse = api.cover_attn_fwd(q, dk, dv, kc, vc, _dev(seeds, "i32"))
    torch.cuda.synchronize()
    assert api.cover_device_status() == 0
    # oracle: the same pipeline in fp64 on the stored values
    f = W.bf16_bits_to_f64
    rk, rv = oracle.seed_kv_gather(prev.k_cached, prev.v_cached, seeds)
    k2, v2, km, vm = oracle.seed_kv_override(new.k_cached, new.v_cached, seeds, rk, rv)
    ref, ref_lse = oracle.override_attention(f(new.q), f(k2), f(v2), f(km), f(vm), seeds)
    d = np.abs(out.float().cpu().numpy() - ref)
    assert d.max() <= H.TOL_BF16_MAX and d.mean() <= H.TOL_BF16_MEAN
    assert np.abs(lse.cpu().numpy() - ref_lse).max() <= H.TOL_LSE
    # the seed rows saw the previous step's states on every other column, their own masked-input pair
    # on the diagonal
    for b in range(B):
        for s, j in enumerate(seeds[b]):
            assert np.array_equal(_host(dk, "bf16")[b, :, j], prev.k_cached[b, :, j])
            assert np.array_equal(_host(kc, "bf16")[b, :, s], new.k_cached[b, :, j])
