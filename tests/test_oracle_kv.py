"""Pins of the seed K/V cache oracle (Section 5.1, KV cache override) that need no GPU."""
import numpy as np
import pytest

import oracle.cover_oracle as orc


def _states(B, H, L, D, seed, dtype=np.float64):
    rng = np.random.default_rng(seed)
    return rng.standard_normal((B, H, L, D)).astype(dtype), rng.standard_normal((B, H, L, D)).astype(dtype)


def test_override_matches_the_case_definition():
    # K'_j = cached state if j is a seed position, else the fresh state (Section 5.1)
    B, H, L, D, S = 2, 3, 11, 4, 4
    k, v = _states(B, H, L, D, 0)
    kbar, vbar = _states(B, H, S, D, 1)
    seeds = np.array([[3, 9, 0, 5], [10, 2, 7, 1]])
    k2, v2, km, vm = orc.seed_kv_override(k, v, seeds, kbar, vbar)
    for b in range(B):
        slot_of = {int(seeds[b, s]): s for s in range(S)}
        for j in range(L):
            if j in slot_of:
                assert np.array_equal(k2[b, :, j], kbar[b, :, slot_of[j]])
                assert np.array_equal(v2[b, :, j], vbar[b, :, slot_of[j]])
                assert np.array_equal(km[b, :, slot_of[j]], k[b, :, j])
                assert np.array_equal(vm[b, :, slot_of[j]], v[b, :, j])
            else:
                assert np.array_equal(k2[b, :, j], k[b, :, j]) and np.array_equal(v2[b, :, j], v[b, :, j])


def test_override_is_an_involution():
    k, v = _states(1, 2, 16, 8, 2)
    kbar, vbar = _states(1, 2, 5, 8, 3)
    seeds = np.array([[4, 15, 0, 8, 9]])
    once = orc.seed_kv_override(k, v, seeds, kbar, vbar)
    twice = orc.seed_kv_override(*once[:2], seeds, *once[2:])
    for a, b in zip(twice, (k, v, kbar, vbar)):
        assert np.array_equal(a, b)


def test_gather_then_override_restores_the_cached_states():
    # states of step t-1 cached at selection reappear in the seed columns at step t
    k_prev, v_prev = _states(2, 2, 12, 4, 4)
    k_new, v_new = _states(2, 2, 12, 4, 5)
    seeds = np.array([[1, 6, 11], [0, 5, 7]])
    kc, vc = orc.seed_kv_gather(k_prev, v_prev, seeds)
    for b in range(2):
        for s in range(3):
            assert np.array_equal(kc[b, :, s], k_prev[b, :, seeds[b, s]])
    k2, v2, km, vm = orc.seed_kv_override(k_new, v_new, seeds, kc, vc)
    for b in range(2):
        for s, j in enumerate(seeds[b]):
            assert np.array_equal(k2[b, :, j], k_prev[b, :, j]) and np.array_equal(v2[b, :, j], v_prev[b, :, j])
            assert np.array_equal(km[b, :, s], k_new[b, :, j]) and np.array_equal(vm[b, :, s], v_new[b, :, j])


def test_override_feeds_the_leave_one_out_views():
    # attention over the overridden memory with the swapped-out rows as diagonal pairs equals the
    # explicit view of Section 5.1: K'/V' everywhere, (k_i, v_i) of the masked input on the diagonal
    B, Hq, H, L, D = 1, 2, 1, 9, 4
    rng = np.random.default_rng(6)
    q = rng.standard_normal((B, Hq, L, D))
    k_new, v_new = _states(B, H, L, D, 7)
    kbar, vbar = _states(B, H, 3, D, 8)
    seeds = np.array([[2, 8, 5]])
    k2, v2, km, vm = orc.seed_kv_override(k_new, v_new, seeds, kbar, vbar)
    out, _ = orc.override_attention(q, k2, v2, km, vm, seeds)
    for hq in range(Hq):
        for i in range(L):
            K = k2[0, 0].copy()
            V = v2[0, 0].copy()
            if i in seeds[0]:
                K[i], V[i] = k_new[0, 0, i], v_new[0, 0, i]
            z = q[0, hq, i] @ K.T / np.sqrt(D)
            w = np.exp(z - z.max())
            w /= w.sum()
            assert np.allclose(out[0, hq, i], w @ V, atol=1e-13)


def test_invalid_and_repeated_slots():
    k, v = _states(1, 1, 6, 2, 9)
    kbar, vbar = _states(1, 1, 4, 2, 10)
    seeds = np.array([[2, -1, 2, 6]])                      # slot 2 repeats slot 0; -1 and 6 are out of range
    k2, v2, km, vm = orc.seed_kv_override(k, v, seeds, kbar, vbar)
    assert np.array_equal(k2[0, 0, 2], kbar[0, 0, 0])      # the lowest slot wins
    assert np.array_equal(km[0, 0, 0], k[0, 0, 2])
    for s in (1, 2, 3):                                    # the others keep their cache rows
        assert np.array_equal(km[0, 0, s], kbar[0, 0, s]) and np.array_equal(vm[0, 0, s], vbar[0, 0, s])
    changed = [j for j in range(6) if not np.array_equal(k2[0, 0, j], k[0, 0, j])]
    assert changed == [2]
    kc, vc = orc.seed_kv_gather(k, v, seeds)
    assert np.array_equal(kc[0, 0, 0], k[0, 0, 2]) and np.array_equal(kc[0, 0, 2], k[0, 0, 2])
    assert not kc[0, 0, 1].any() and not kc[0, 0, 3].any()


@pytest.mark.parametrize("dtype", [np.uint16, np.float32])
def test_no_seeds_and_exact_copies(dtype):
    rng = np.random.default_rng(11)
    k = rng.integers(0, 65535, (1, 2, 5, 8)).astype(dtype)
    v = rng.integers(0, 65535, (1, 2, 5, 8)).astype(dtype)
    empty = np.zeros((1, 0), dtype=np.int64)
    k2, v2, km, vm = orc.seed_kv_override(k, v, empty, k[:, :, :0], v[:, :, :0])
    assert np.array_equal(k2, k) and np.array_equal(v2, v) and km.shape[2] == 0
    kc, _ = orc.seed_kv_gather(k, v, np.array([[4, 0]]))
    assert kc.dtype == k.dtype and np.array_equal(kc[0, :, 0], k[0, :, 4])
