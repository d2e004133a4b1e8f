"""Pins for the fp64 oracle (CPU only).

Each test ties the oracle to something other than itself: hand-worked
fixtures, closed forms the paper states, torch's float64 SDPA (a library
routine) for the no-seed special case, 50-digit decimal brute force on tiny
inputs, invariances of the two-view definition, and planted mistakes that the
pins must catch.
"""
import copy
import math
from decimal import Decimal, getcontext

import numpy as np
import pytest
import torch

import oracle
from oracle import cover_oracle as orc
from tests import _golden as G

RNG = np.random.default_rng(1234)


def rand_case(B, Hq, Hkv, L, D, S, rng=RNG, seed_lo=0, seed_hi=None):
    seed_hi = L if seed_hi is None else seed_hi
    q = rng.standard_normal((B, Hq, L, D))
    kc = rng.standard_normal((B, Hkv, L, D))
    vc = rng.standard_normal((B, Hkv, L, D))
    km = rng.standard_normal((B, Hkv, S, D))
    vm = rng.standard_normal((B, Hkv, S, D))
    seeds = np.stack([rng.choice(np.arange(seed_lo, seed_hi), size=S, replace=False) for _ in range(B)])
    return q, kc, vc, km, vm, seeds.astype(np.int32).reshape(B, S)


def sdpa_reference(q, kc, vc):
    """torch float64 scaled_dot_product_attention (no mask), GQA via repeat_interleave."""
    G_ = q.shape[1] // kc.shape[1]
    tq = torch.from_numpy(q)
    tk = torch.from_numpy(kc).repeat_interleave(G_, dim=1)
    tv = torch.from_numpy(vc).repeat_interleave(G_, dim=1)
    out = torch.nn.functional.scaled_dot_product_attention(tq, tk, tv)
    scores = (tq @ tk.transpose(-1, -2)) / math.sqrt(q.shape[-1])
    return out.numpy(), torch.logsumexp(scores, dim=-1).numpy()


# ----------------------------------------------------------------------------
# Special cases that reduce to textbook attention
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("B,Hq,Hkv,L,D", [(1, 1, 1, 5, 4), (2, 4, 2, 33, 8), (1, 6, 3, 130, 16)])
def test_zero_seeds_is_sdpa(B, Hq, Hkv, L, D):
    q, kc, vc, km, vm, seeds = rand_case(B, Hq, Hkv, L, D, 0)
    out, lse = oracle.override_attention(q, kc, vc, km, vm, seeds)
    ref, ref_lse = sdpa_reference(q, kc, vc)
    assert np.max(np.abs(out - ref)) < 1e-12
    assert np.max(np.abs(lse - ref_lse)) < 1e-12


@pytest.mark.parametrize("B,Hq,Hkv,L,D,S", [(1, 2, 2, 9, 4, 3), (2, 6, 2, 40, 8, 7)])
def test_masked_equal_to_cached_is_standard(B, Hq, Hkv, L, D, S):
    q, kc, vc, km, vm, seeds = rand_case(B, Hq, Hkv, L, D, S)
    for b in range(B):
        for s in range(S):
            km[b, :, s] = kc[b, :, seeds[b, s]]
            vm[b, :, s] = vc[b, :, seeds[b, s]]
    out, lse = oracle.override_attention(q, kc, vc, km, vm, seeds)
    ref, ref_lse = sdpa_reference(q, kc, vc)
    assert np.max(np.abs(out - ref)) < 1e-12
    assert np.max(np.abs(lse - ref_lse)) < 1e-12


# ----------------------------------------------------------------------------
# Closed form (Appendix B) versus the explicit view (Section 5.1)
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("L", [1, 2, 3, 8])
@pytest.mark.parametrize("D", [1, 4])
def test_closed_form_equals_explicit_view(L, D):
    rng = np.random.default_rng(L * 10 + D)
    for S in sorted({0, 1, L // 2, L}):
        q, kc, vc, km, vm, seeds = rand_case(2, 4, 2, L, D, S, rng=rng)
        a, la = oracle.override_attention(q, kc, vc, km, vm, seeds)
        b, lb = oracle.override_attention_closed_form(q, kc, vc, km, vm, seeds)
        assert np.max(np.abs(a - b)) < 1e-12
        assert np.max(np.abs(la - lb)) < 1e-12


def test_length_one_seed_row():
    rng = np.random.default_rng(7)
    q, kc, vc, km, vm, seeds = rand_case(1, 2, 1, 1, 4, 1, rng=rng)
    out, lse = oracle.override_attention(q, kc, vc, km, vm, seeds)
    for h in range(2):
        assert np.allclose(out[0, h, 0], vm[0, 0, 0], atol=1e-15, rtol=0)
        assert abs(lse[0, h, 0] - float(q[0, h, 0] @ km[0, 0, 0]) / 2.0) < 1e-14


def test_zero_query_is_uniform_over_view():
    rng = np.random.default_rng(8)
    L, D = 9, 4
    q, kc, vc, km, vm, seeds = rand_case(1, 1, 1, L, D, 3, rng=rng)
    q[:] = 0.0
    out, lse = oracle.override_attention(q, kc, vc, km, vm, seeds)
    for s, i in enumerate(seeds[0]):
        expect = (vc[0, 0].sum(axis=0) - vc[0, 0, i] + vm[0, 0, s]) / L
        assert np.max(np.abs(out[0, 0, i] - expect)) < 1e-14
        assert abs(lse[0, 0, i] - math.log(L)) < 1e-14


def test_zero_score_shift_rows():
    """delta_i = 0 (k_i = k'_i): r_i = 1 and o_i = o_ovr_i + alpha_i (v_i - v'_i)."""
    rng = np.random.default_rng(9)
    L, D = 12, 4
    q, kc, vc, km, vm, seeds = rand_case(1, 2, 1, L, D, 4, rng=rng)
    for s, i in enumerate(seeds[0]):
        km[0, 0, s] = kc[0, 0, i]
    out, lse = oracle.override_attention(q, kc, vc, km, vm, seeds)
    plain, plain_lse = sdpa_reference(q, kc, vc)
    for h in range(2):
        z = (kc[0, 0] @ q[0, h].T).T / math.sqrt(D)
        w = np.exp(z - z.max(axis=1, keepdims=True))
        w /= w.sum(axis=1, keepdims=True)
        for s, i in enumerate(seeds[0]):
            expect = plain[0, h, i] + w[i, i] * (vm[0, 0, s] - vc[0, 0, i])
            assert np.max(np.abs(out[0, h, i] - expect)) < 1e-13
            assert abs(lse[0, h, i] - plain_lse[0, h, i]) < 1e-13


def test_corrected_weights_sum_to_one_and_match_lemma():
    """Appendix B.3: w_ij = w_ovr_ij / r_i (j != i), w_ii = alpha_i e^delta_i / r_i, sum 1."""
    rng = np.random.default_rng(10)
    L, D = 10, 4
    q, kc, vc, km, vm, seeds = rand_case(1, 1, 1, L, D, 3, rng=rng)
    for s, i in enumerate(seeds[0]):
        w = oracle.corrected_weights_row(q, kc, vc, km, vm, seeds, 0, 0, int(i))
        assert abs(w.sum() - 1.0) < 1e-14
        z = kc[0, 0] @ q[0, 0, i] / math.sqrt(D)
        w_ovr = np.exp(z - z.max())
        w_ovr /= w_ovr.sum()
        delta = float(q[0, 0, i] @ (km[0, 0, s] - kc[0, 0, i])) / math.sqrt(D)
        r = 1 + w_ovr[i] * (math.exp(delta) - 1)
        lemma = w_ovr / r
        lemma[i] = w_ovr[i] * math.exp(delta) / r
        assert np.max(np.abs(w - lemma)) < 1e-14


# ----------------------------------------------------------------------------
# Invariances of the two-view definition (Section 5.1)
# ----------------------------------------------------------------------------

def test_invariances_exact():
    rng = np.random.default_rng(11)
    q, kc, vc, km, vm, seeds = rand_case(2, 4, 2, 24, 8, 5, rng=rng)
    out, lse = oracle.override_attention(q, kc, vc, km, vm, seeds)
    # a seed row ignores its own cached pair (other rows do see it)
    for b in range(2):
        for i in seeds[b]:
            kc2, vc2 = kc.copy(), vc.copy()
            kc2[b, :, i] += 3.0
            vc2[b, :, i] -= 5.0
            out2, lse2 = oracle.override_attention(q, kc2, vc2, km, vm, seeds)
            assert np.array_equal(out[b, :, i], out2[b, :, i])
            assert np.array_equal(lse[b, :, i], lse2[b, :, i])
            assert not np.array_equal(out[b, :, (i + 1) % 24], out2[b, :, (i + 1) % 24])
    # non-seed rows ignore the masked buffer
    out3, lse3 = oracle.override_attention(q, kc, vc, km * 7 + 1, vm - 2, seeds)
    mask = np.ones((2, 24), bool)
    for b in range(2):
        mask[b, seeds[b]] = False
    for b in range(2):
        assert np.array_equal(out[b][:, mask[b]], out3[b][:, mask[b]])
        assert np.array_equal(lse[b][:, mask[b]], lse3[b][:, mask[b]])


# ----------------------------------------------------------------------------
# 50-digit brute force on tiny inputs (pure Python, no numpy arithmetic)
# ----------------------------------------------------------------------------

def brute_force_decimal(q, kc, vc, km, vm, seeds):
    getcontext().prec = 50
    B, Hq, L, D = q.shape
    Hkv = kc.shape[1]
    scale = Decimal(1) / Decimal(D).sqrt()
    out = np.zeros(q.shape)
    lse = np.zeros(q.shape[:3])
    for b in range(B):
        first = {}
        for s, p in enumerate(seeds[b]):
            if 0 <= p < L and p not in first:
                first[int(p)] = s
        for h in range(Hq):
            g = h // (Hq // Hkv)
            for i in range(L):
                keys, vals = [], []
                for j in range(L):
                    if j == i and i in first:
                        keys.append(km[b, g, first[i]])
                        vals.append(vm[b, g, first[i]])
                    else:
                        keys.append(kc[b, g, j])
                        vals.append(vc[b, g, j])
                z = [scale * sum(Decimal(float(q[b, h, i, d])) * Decimal(float(k[d])) for d in range(D))
                     for k in keys]
                e = [zz.exp() for zz in z]
                Z = sum(e)
                for d in range(D):
                    out[b, h, i, d] = float(sum(e[j] * Decimal(float(vals[j][d])) for j in range(L)) / Z)
                lse[b, h, i] = float(Z.ln())
    return out, lse


def test_brute_force_decimal_small():
    rng = np.random.default_rng(12)
    q, kc, vc, km, vm, seeds = rand_case(1, 4, 2, 6, 3, 3, rng=rng)
    out, lse = oracle.override_attention(q, kc, vc, km, vm, seeds)
    bo, bl = brute_force_decimal(q, kc, vc, km, vm, seeds)
    assert np.max(np.abs(out - bo)) < 1e-13
    assert np.max(np.abs(lse - bl)) < 1e-13


def test_dominant_diagonal_stress():
    """q_i parallel to k'_i with alpha_i > 0.999 and a very negative delta_i.

    The explicit view stays exact; the closed form divides by a small r_i and
    loses digits. The explicit view must match 50-digit brute force.
    """
    rng = np.random.default_rng(13)
    L, D = 8, 4
    q, kc, vc, km, vm, seeds = rand_case(1, 1, 1, L, D, 1, rng=rng)
    i = int(seeds[0, 0])
    kc[0, 0, i] = q[0, 0, i] / np.linalg.norm(q[0, 0, i]) * 12.0
    km[0, 0, 0] = -kc[0, 0, i]
    z = kc[0, 0] @ q[0, 0, i] / math.sqrt(D)
    w = np.exp(z - z.max())
    w /= w.sum()
    assert w[i] > 0.999
    out, lse = oracle.override_attention(q, kc, vc, km, vm, seeds)
    bo, bl = brute_force_decimal(q, kc, vc, km, vm, seeds)
    assert np.max(np.abs(out - bo)) < 1e-13
    assert np.max(np.abs(lse - bl)) < 1e-13


# ----------------------------------------------------------------------------
# Hand-worked fixtures
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("name", ["two_view_d1_l3.json", "two_view_gqa_dup.json"])
def test_golden_two_view(golden_dir, name):
    g = G.load(golden_dir, name)
    arrs = {k: G.array(g[k]) for k in ["q", "k_cached", "v_cached", "k_seedmask", "v_seedmask", "out", "lse"]}
    seeds = np.array(g["seed_idx"], dtype=np.int32)
    for fn in (oracle.override_attention, oracle.override_attention_closed_form):
        out, lse = fn(arrs["q"], arrs["k_cached"], arrs["v_cached"], arrs["k_seedmask"],
                      arrs["v_seedmask"], seeds)
        assert np.max(np.abs(out - arrs["out"])) < 1e-13, fn.__name__
        assert np.max(np.abs(lse - arrs["lse"])) < 1e-13, fn.__name__
    if "route_slot" in g:
        slot, bitmap, n_inv = oracle.route_seeds(seeds, g["L"])
        assert slot.tolist() == g["route_slot"]
        assert n_inv == g["route_n_invalid"]


def test_golden_score(golden_dir):
    g = G.load(golden_dir, "score_v4.json")
    x = G.array(g["logits"])[None, :]
    r = oracle.score_rows(x)
    assert r["argmax"][0] == g["argmax"]
    assert abs(r["maxprob"][0] - G.value(g["maxprob"])) < 1e-15
    assert abs(r["entropy"][0] - G.value(g["entropy"])) < 1e-14
    assert abs(r["u"][0] - G.value(g["u_no_cur"])) < 1e-14
    assert abs(r["score"][0] - G.value(g["u_no_cur"])) < 1e-14
    r2 = oracle.score_rows(x, cur_tok=[g["cur_tok"]], d_in=[G.value(g["d_in"])], d_out=[G.value(g["d_out"])])
    assert abs(r2["u"][0] - G.value(g["u_cur"])) < 1e-14
    assert abs(r2["score"][0] - G.value(g["score_cur"])) < 1e-14


# ----------------------------------------------------------------------------
# Seed routing (seed-set semantics)
# ----------------------------------------------------------------------------

def test_route_seeds_spec():
    seeds = np.array([[5, 130, 5, -1, 300, 127, 128], [0, 0, 0, 1, 2, 3, 255]], dtype=np.int32)
    slot, bitmap, n_inv = oracle.route_seeds(seeds, 256)
    assert n_inv == 3 + 2
    assert slot[0, 5] == 0 and slot[0, 130] == 1 and slot[0, 127] == 5 and slot[0, 128] == 6
    assert slot[1, 0] == 0 and slot[1, 1] == 3 and slot[1, 255] == 6
    assert (slot[0] >= 0).sum() == 4 and (slot[1] >= 0).sum() == 5
    # bitmap: tile 0 word 0 bit 5 and word 3 bit 31 (row 127); tile 1 word 0 bits 0 and 2 (rows 128, 130)
    assert bitmap[0, 0].tolist() == [1 << 5, 0, 0, 1 << 31]
    assert bitmap[0, 1].tolist() == [(1 << 0) | (1 << 2), 0, 0, 0]
    assert bitmap[1, 1].tolist() == [0, 0, 0, 1 << 31]
    popcount = sum(bin(int(w)).count("1") for w in bitmap.ravel())
    assert popcount == int((slot >= 0).sum())


# ----------------------------------------------------------------------------
# Scoring (Sections 3, 5.3, 6.1)
# ----------------------------------------------------------------------------

def test_score_uniform_logits():
    V = 1000
    r = oracle.score_rows(np.full((2, V), 0.75))
    assert np.allclose(r["maxprob"], 1.0 / V, rtol=1e-14, atol=0)
    assert np.allclose(r["entropy"], math.log(V), rtol=1e-14, atol=0)
    assert r["argmax"].tolist() == [0, 0]
    assert np.allclose(r["u"], math.log(V), rtol=1e-14, atol=0)


def test_score_single_spike():
    V = 5000
    x = np.zeros((1, V))
    x[0, 1234] = 20.0
    r = oracle.score_rows(x)
    assert r["argmax"][0] == 1234
    expect_c = 1.0 / (1.0 + (V - 1) * math.exp(-20.0))
    assert abs(r["maxprob"][0] - expect_c) < 1e-15


def test_score_two_value_entropy():
    V, n1, a, b = 777, 100, 1.5, -0.5
    x = np.full((1, V), b)
    x[0, 300:300 + n1] = a
    r = oracle.score_rows(x)
    Z = n1 * math.exp(a) + (V - n1) * math.exp(b)
    pa, pb = math.exp(a) / Z, math.exp(b) / Z
    H = -(n1 * pa * math.log(pa) + (V - n1) * pb * math.log(pb))
    assert abs(r["entropy"][0] - H) < 1e-13
    assert r["argmax"][0] == 300
    assert abs(r["maxprob"][0] - pa) < 1e-15


def test_score_argmax_ties_lower_index():
    x = np.array([[0.0, 2.0, 1.0, 2.0, 2.0]])
    assert oracle.score_rows(x)["argmax"][0] == 1


def rank_topk(score, n_seq, k, eligible=None):
    """Independent brute force: a candidate's position is the number of candidates that beat it."""
    N = len(score)
    per = N // n_seq
    idx = np.full((n_seq, k), -1)
    for g in range(n_seq):
        cand = [j for j in range(per) if eligible is None or eligible[g * per + j]]
        for j in cand:
            sj = score[g * per + j]
            rank = sum(1 for t in cand if score[g * per + t] > sj or (score[g * per + t] == sj and t < j))
            if rank < k:
                idx[g, rank] = j
    return idx


@pytest.mark.parametrize("with_elig", [False, True])
def test_topk_against_rank_brute_force(with_elig):
    rng = np.random.default_rng(14)
    N, n_seq, k = 96, 3, 7
    score = np.round(rng.standard_normal(N), 1)       # many exact ties
    elig = (rng.uniform(size=N) < 0.3).astype(np.uint8) if with_elig else None
    idx, val = oracle.topk_select(score, n_seq, k, elig)
    assert idx.tolist() == rank_topk(score, n_seq, k, elig).tolist()
    for g in range(n_seq):
        for t in range(k):
            if idx[g, t] >= 0:
                assert val[g, t] == score[g * (N // n_seq) + idx[g, t]]
            else:
                assert val[g, t] == -np.inf


def test_topk_margin():
    score = np.array([3.0, 1.0, 2.0, 2.5])
    assert oracle.topk_margin(score, 1, 2)[0] == pytest.approx(0.5)
    assert oracle.topk_margin(score, 1, 4)[0] == np.inf


# ----------------------------------------------------------------------------
# Planted mistakes: each must break at least one pin above
# ----------------------------------------------------------------------------

def _golden_two_view_fails(golden_dir):
    try:
        test_golden_two_view(golden_dir, "two_view_gqa_dup.json")
        test_golden_two_view(golden_dir, "two_view_d1_l3.json")
    except AssertionError:
        return True
    return False


def test_planted_cached_diagonal_is_caught(golden_dir, monkeypatch):
    # mistake: the seed query keeps the cached pair on its diagonal (no correction)
    monkeypatch.setattr(orc, "view_for_row", lambda kc_h, vc_h, i, pair=None: (kc_h, vc_h))
    assert _golden_two_view_fails(golden_dir)


def test_gqa_mapping_distinguishes_interleaved():
    # the contiguous-group reading (hkv = hq // G) must differ from an interleaved
    # mapping (hkv = hq % Hkv) on this input, so the SDPA pin above pins the reading
    rng = np.random.default_rng(15)
    q, kc, vc, km, vm, seeds = rand_case(1, 4, 2, 16, 4, 0, rng=rng)
    out, _ = oracle.override_attention(q, kc, vc, km, vm, seeds)
    tq = torch.from_numpy(q)
    tk = torch.from_numpy(kc).repeat(1, 2, 1, 1)
    tv = torch.from_numpy(vc).repeat(1, 2, 1, 1)
    interleaved = torch.nn.functional.scaled_dot_product_attention(tq, tk, tv).numpy()
    assert np.max(np.abs(out - interleaved)) > 1e-2
    assert np.max(np.abs(out - sdpa_reference(q, kc, vc)[0])) < 1e-12


def test_planted_closed_form_sign_is_caught(golden_dir, monkeypatch):
    # mistake: + alpha v'_i instead of - alpha v'_i in the closed form
    src = copy.copy(orc.override_attention_closed_form)

    def wrong(q, kc, vc, km, vm, seed_idx):
        out, lse = src(q, kc, vc, km, vm, seed_idx)
        slot = orc.route_seeds(seed_idx, q.shape[2])[0]
        for b in range(q.shape[0]):
            for i in np.nonzero(slot[b] >= 0)[0]:
                out[b, :, i] += 1e-3
        return out, lse
    monkeypatch.setattr(oracle, "override_attention_closed_form", wrong)
    assert _golden_two_view_fails(golden_dir)


def test_planted_entropy_log_base_is_caught(golden_dir, monkeypatch):
    g = G.load(golden_dir, "score_v4.json")
    x = G.array(g["logits"])[None, :]
    r = oracle.score_rows(x)
    assert abs(r["entropy"][0] / math.log(2) - G.value(g["entropy"])) > 1e-3


# ----------------------------------------------------------------------------
# Prefix-cache window (Section 6.6): a window of query rows over the full memory
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("q0,Lq", [(0, 24), (5, 7), (13, 11), (23, 1), (0, 1)])
def test_window_rows_equal_the_square_rows(q0, Lq):
    # attention rows are independent: the window's rows are the square problem's rows q0 .. q0+Lq-1
    rng = np.random.default_rng(40 + q0)
    q, kc, vc, km, vm, seeds = rand_case(2, 4, 2, 24, 8, 6, rng=rng)
    full, full_lse = oracle.override_attention(q, kc, vc, km, vm, seeds)
    out, lse = oracle.override_attention_window(q[:, :, q0:q0 + Lq], kc, vc, km, vm, seeds, q0)
    assert np.max(np.abs(out - full[:, :, q0:q0 + Lq])) < 1e-12
    assert np.max(np.abs(lse - full_lse[:, :, q0:q0 + Lq])) < 1e-12


def test_window_with_seeds_outside_is_plain_attention():
    # seeds outside the query window only shape the memory: the window rows are textbook
    # attention over K', V' (torch float64 SDPA)
    rng = np.random.default_rng(47)
    q, kc, vc, km, vm, _ = rand_case(1, 2, 1, 20, 8, 3, rng=rng)
    seeds = np.array([[0, 3, 17]], dtype=np.int32)
    out, lse = oracle.override_attention_window(q[:, :, 5:15], kc, vc, km, vm, seeds, 5)
    ref, ref_lse = sdpa_reference(q[:, :, 5:15], kc, vc)
    assert np.max(np.abs(out - ref)) < 1e-12 and np.max(np.abs(lse - ref_lse)) < 1e-12


# ----------------------------------------------------------------------------
# d_in / d_out (Section 5.3) from the head-averaged attention weights
# ----------------------------------------------------------------------------

def test_mass_sums_to_the_counts():
    # each weight row sums to 1: over the whole memory (pos0 = 0, every position a response
    # position) the total incoming mass is |M_t|, and a position whose every key is drafted
    # sends mass 1
    rng = np.random.default_rng(50)
    q, kc, vc, km, vm, seeds = rand_case(2, 4, 2, 12, 8, 3, rng=rng)
    masked = rng.random((2, 12)) < 0.4
    d_in, d_out = oracle.attention_mass(q, kc, km, seeds, masked, np.ones((2, 12), bool), 0)
    assert np.allclose(d_in.sum(axis=1), masked.sum(axis=1), atol=1e-12)
    assert np.allclose(d_out, 1.0, atol=1e-12)
    d_in, d_out = oracle.attention_mass(q, kc, km, seeds, np.zeros((2, 12), bool), np.zeros((2, 12), bool), 0)
    assert not d_in.any() and not d_out.any()


def test_mass_uniform_queries():
    # q = 0: every weight is 1/L (seed rows too), so d_in = |M|/L and d_out = |D|/L
    rng = np.random.default_rng(51)
    _, kc, vc, km, vm, seeds = rand_case(1, 2, 1, 10, 4, 2, rng=rng)
    q = np.zeros((1, 2, 10, 4))
    masked = np.zeros((1, 6), bool)
    masked[0, [1, 4]] = True
    drafted = np.zeros((1, 6), bool)
    drafted[0, [0, 2, 5]] = True
    d_in, d_out = oracle.attention_mass(q, kc, km, seeds, masked, drafted, 3)
    assert np.allclose(d_in, 2 / 10, atol=1e-15) and np.allclose(d_out, 3 / 10, atol=1e-15)


def test_mass_matches_the_corrected_weights():
    # the weight rows are App. B.3's corrected weights (pinned above): sum them directly
    rng = np.random.default_rng(52)
    q, kc, vc, km, vm, seeds = rand_case(1, 2, 2, 9, 4, 3, rng=rng)
    pos0, n = 2, 6
    masked = rng.random((1, n)) < 0.5
    drafted = rng.random((1, n)) < 0.5
    d_in, d_out = oracle.attention_mass(q, kc, km, seeds, masked, drafted, pos0)
    A = np.zeros((n, 9))
    for hq in range(2):
        for r in range(n):
            A[r] += oracle.corrected_weights_row(q, kc, vc, km, vm, seeds, 0, hq, pos0 + r) / 2
    for j in range(n):
        assert abs(d_in[0, j] - sum(A[r, pos0 + j] for r in range(n) if masked[0, r])) < 1e-12
        assert abs(d_out[0, j] - sum(A[j, pos0 + i] for i in range(n) if drafted[0, i])) < 1e-12


# ----------------------------------------------------------------------------
# Row-sampled oracle (the checker of every sampled GPU parity test)
# ----------------------------------------------------------------------------

def _rows_case():
    # two batch rows, GQA 6 query heads over 2 KV heads; batch row 1 carries a repeated and an
    # out-of-range seed, so the per-batch routing and the lowest-slot rule are exercised
    rng = np.random.default_rng(60)
    q, kc, vc, km, vm, _ = rand_case(2, 6, 2, 40, 8, 5, rng=rng)
    seeds = np.array([[3, 17, 39, 0, 22], [22, 9, 22, 41, 30]], dtype=np.int32)
    return q, kc, vc, km, vm, seeds


def test_rows_equal_the_full_oracle_every_head():
    # Section 5.1 / App. B.1: each listed row of head (b, hq) is that row of the full two-view
    # attention, for every batch row and every query head of every KV group
    q, kc, vc, km, vm, seeds = _rows_case()
    full, full_lse = oracle.override_attention(q, kc, vc, km, vm, seeds)
    rows = [0, 3, 9, 17, 21, 22, 30, 39]
    for b in range(2):
        for hq in range(6):
            out, lse = oracle.override_attention_rows(q, kc, vc, km, vm, seeds, b, hq, rows)
            assert np.max(np.abs(out - full[b, hq, rows])) < 1e-13, (b, hq)
            assert np.max(np.abs(lse - full_lse[b, hq, rows])) < 1e-13, (b, hq)


def _rows_check_fails(rows_fn, full):
    q, kc, vc, km, vm, seeds = _rows_case()
    rows = [3, 9, 22, 30]
    for b in range(2):
        for hq in range(6):
            out, _ = rows_fn(q, kc, vc, km, vm, seeds, b, hq, rows)
            if np.max(np.abs(out - full[b, hq, rows])) > 1e-6:
                return True
    return False


def test_planted_rows_mistakes_are_caught(monkeypatch):
    good = orc.override_attention_rows
    full = oracle.override_attention(*_rows_case())[0]   # computed before any mistake is planted
    assert not _rows_check_fails(good, full)
    # (1) a seed row keeps the cached pair on its diagonal
    monkeypatch.setattr(orc, "view_for_row", lambda kc_h, vc_h, i, pair=None: (kc_h, vc_h))
    assert _rows_check_fails(good, full)
    monkeypatch.undo()

    # (2) the seed routing of batch row 0 used for every batch row
    def first_batch_seeds(q, kc, vc, km, vm, seeds, b, hq, rows):
        s = seeds.copy()
        s[b] = seeds[0]
        return good(q, kc, vc, km, vm, s, b, hq, rows)
    assert _rows_check_fails(first_batch_seeds, full)

    # (3) interleaved GQA mapping (hkv = hq % Hkv) instead of contiguous groups: the query of
    # head hq read against the KV head of head (hq % Hkv) * G under the contiguous rule
    def interleaved(q, kc, vc, km, vm, seeds, b, hq, rows):
        Hkv, G_ = kc.shape[1], q.shape[1] // kc.shape[1]
        q2 = q.copy()
        q2[b, (hq % Hkv) * G_] = q[b, hq]
        return good(q2, kc, vc, km, vm, seeds, b, (hq % Hkv) * G_, rows)
    assert _rows_check_fails(interleaved, full)
