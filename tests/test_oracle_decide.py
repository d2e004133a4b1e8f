"""Pins of the decision-step oracle (Sections 3, 5.2 and 5.3) that do not need a GPU.

The oracle's decision function is checked against a hand-worked fixture, the
paper's set identities, closed forms of the adaptive revision rate, the
revision rule case by case, order properties of both selections, and source
mutations that plant plausible mistakes.
"""
import inspect
import math
from fractions import Fraction

import numpy as np
import pytest

import oracle.cover_oracle as orc
from tests import _golden as G

F32 = np.float32


def _f32(lst):
    return np.array([F32(G.value(x)) for x in lst], dtype=F32)


def _golden_inputs(golden_dir):
    g = G.load(golden_dir, "decide_seq10.json")
    p = dict(g["params"])
    params = dict(tau=F32(G.value(p["tau"])), budget=p["budget"], m_remask=p["m_remask"], mask_id=p["mask_id"],
                  min_one=bool(p["min_one"]), pos0=p["pos0"], max_seeds=p["max_seeds"])
    args = (_f32(g["conf"]), np.array(g["yhat"]), _f32(g["entropy"]), _f32(g["u_cur"]), _f32(g["u_top"]),
            _f32(g["d_in"]), _f32(g["d_out"]), np.array(g["tok"]), np.array(g["flags"]),
            np.array(g["remask_cnt"]), np.array(g["draft_ok"]))
    return g, args, params


def _check_golden(fn, golden_dir):
    g, args, params = _golden_inputs(golden_dir)
    r = fn(*args, **params)
    e = g["expect"]
    for key in ("tok", "remask_cnt", "flags"):
        assert list(r[key]) == e[key], key
    for key in ("drafted", "kept", "replaced", "remasked", "seeds"):
        assert list(r[key]) == e[key], key
    for key in ("n_t", "n_above", "n_select"):
        assert r[key] == e[key], key
    want = [-np.inf if s == "-inf" else G.value(s) for s in e["score"]]
    assert [float(x) for x in r["score"]] == want


def _check_strict_threshold(fn):
    # confidence exactly tau neither drafts (Section 5.2, "exceeds") nor replaces
    tau = F32(0.8)
    above = np.nextafter(tau, F32(1))
    conf = np.array([tau, above, tau, above], F32)
    yhat = np.array([1, 2, 3, 4])
    tok = np.array([9, 9, 5, 6])                    # rows 2, 3: previous seeds re-predicting another token
    flags = np.array([0, 0, 1, 1])
    z = np.zeros(4, F32)
    r = fn(conf, yhat, z, z, z, z, z, tok, flags, np.zeros(4, np.int64), np.ones(4, np.int64), tau=tau, budget=4,
           m_remask=3, mask_id=9, min_one=False, pos0=0, max_seeds=4)
    assert r["drafted"] == [1]
    assert r["remasked"] == [2] and r["replaced"] == [3]


def _check_mean_ties(fn):
    # scores equal to their mean are not "above" it: F_t(mean) counts s_j <= mean
    n = 5
    s = np.array([1.0, 3.0, 2.0, 2.0, 2.0], F32)    # mean 2: only the 3 is above
    z = np.zeros(n, F32)
    r = fn(np.full(n, 0.5, F32), np.zeros(n, np.int64), z, s, s, z, z, np.zeros(n, np.int64),
           np.zeros(n, np.int64), np.zeros(n, np.int64), np.ones(n, np.int64), tau=F32(0.8), budget=1, m_remask=1,
           mask_id=-1, min_one=False, pos0=0, max_seeds=5)
    assert r["n_above"] == 1 and r["n_select"] == 1 and r["seeds"] == [1]


def _check_all(fn, golden_dir):
    _check_golden(fn, golden_dir)
    _check_strict_threshold(fn)
    _check_mean_ties(fn)


def test_golden_decide(golden_dir):
    _check_all(orc.decide_sequence, golden_dir)


def _mutant(old, new):
    """decide_sequence with one source edit (a planted mistake)."""
    src = inspect.getsource(orc.decide_sequence)
    assert src.count(old) >= 1, old
    ns = dict(vars(orc))
    exec(compile(src.replace(old, new), "<mutant>", "exec"), ns)
    return ns["decide_sequence"]


@pytest.mark.parametrize("old,new", [
    ("conf[i] > tau]", "conf[i] >= tau]"),                                # threshold not strict
    ("(-float(conf[i]), i)", "(-float(conf[i]), -i)"),                     # ties to the higher index
    ("over[:max(budget, 0)]", "over[:max(budget, 0) + 1]"),               # budget off by one
    ("elif conf[i] > tau:", "elif conf[i] > 0.0:"),                       # Replace without the threshold
    ("elif conf[i] > tau:", "elif conf[i] >= tau:"),                      # Replace threshold not strict
    ("new_rc[i] += 1", "new_rc[i] += 0"),                                 # ReMask not counted
    ("if i in changed else", "if False else"),                            # u of the old token after a change
    ("dtype(one + din)) / dtype(one + dout)", "dtype(one + dout)) / dtype(one + din)"),  # inverted influence
    ("if vals[i] <= mean", "if vals[i] < mean"),                          # CDF not inclusive
    ("i not in prev and", ""),                                            # previous seeds not excluded
    ("new_rc[i] < m_remask", "new_rc[i] <= m_remask"),                     # ReMask budget off by one
    ("(-float(score[i]), i)", "(float(score[i]), i)"),                     # lowest scores selected
])
def test_planted_decide_mistakes_are_caught(golden_dir, old, new):
    with pytest.raises(AssertionError):
        _check_all(_mutant(old, new), golden_dir)


def _case(n, rng, mask_id=1000, n_seed=3):
    tok = rng.integers(0, 50, n)
    masked = rng.random(n) < 0.4
    tok[masked] = mask_id
    unm = np.nonzero(~masked)[0]
    flags = np.zeros(n, dtype=np.int64)
    if len(unm):
        flags[rng.choice(unm, size=min(n_seed, len(unm)), replace=False)] = orc.FLAG_SEED
    conf = rng.choice(np.array([0.3, 0.5, 0.75, 0.8, 0.85, 0.9, 0.95], dtype=F32), n)
    yhat = np.where(rng.random(n) < 0.5, tok, rng.integers(0, 50, n))
    yhat[masked] = rng.integers(0, 50, masked.sum())
    ent = rng.choice(np.array([0.5, 1.0, 2.0], dtype=F32), n)
    u_top = rng.choice(np.array([0.125, 0.25, 1.0, 2.0, 3.0], dtype=F32), n)
    u_cur = np.where(yhat == tok, u_top, rng.choice(np.array([0.5, 1.5, 4.0], dtype=F32), n)).astype(F32)
    d_in = rng.choice(np.array([0.0, 0.5, 1.0], dtype=F32), n)
    d_out = rng.choice(np.array([0.0, 0.25, 1.0], dtype=F32), n)
    rc = rng.integers(0, 3, n)
    draft_ok = (rng.random(n) < 0.8).astype(np.int64)
    return conf, yhat, ent, u_cur, u_top, d_in, d_out, tok, flags, rc, draft_ok


@pytest.mark.parametrize("seed", range(40))
def test_decide_identities(seed):
    rng = np.random.default_rng(seed)
    n = int(rng.integers(1, 24))
    mask_id = 1000
    args = _case(n, rng, mask_id)
    conf, yhat, ent, u_cur, u_top, d_in, d_out, tok, flags, rc, draft_ok = args
    tau = F32(0.8)
    budget = int(rng.integers(0, 5))
    m_remask = int(rng.integers(1, 4))
    max_seeds = int(rng.integers(0, 6))
    r = orc.decide_sequence(*args, tau=tau, budget=budget, m_remask=m_remask, mask_id=mask_id, min_one=False,
                            pos0=7, max_seeds=max_seeds)
    M0 = {i for i in range(n) if tok[i] == mask_id}
    U0 = set(range(n)) - M0
    S0 = {i for i in U0 if flags[i] & orc.FLAG_SEED}
    D, R = set(r["drafted"]), set(r["remasked"])
    U1 = {i for i in range(n) if r["tok"][i] != mask_id}
    # Section 3: U_t = (U_{t-1} u D_t) \ R_t, D_t within M_{t-1}, R_t within S_{t-1}
    assert U1 == (U0 | D) - R
    assert D <= M0 and R <= S0
    assert set(r["kept"]) | set(r["replaced"]) | R == S0
    # drafting: only draftable positions above tau; the budget; order property
    over = [i for i in M0 if draft_ok[i] and conf[i] > tau]
    assert len(D) == min(budget, len(over)) and D <= set(over)
    for i in D:
        for j in set(over) - D:
            assert conf[i] > conf[j] or (conf[i] == conf[j] and i < j)
    # revision rule case by case
    for i in S0:
        if yhat[i] == tok[i]:
            assert i in r["kept"] and r["tok"][i] == tok[i]
        elif conf[i] > tau:
            assert i in r["replaced"] and r["tok"][i] == yhat[i]
        else:
            assert i in R and r["tok"][i] == mask_id and r["remask_cnt"][i] == rc[i] + 1
    # seed score of the updated token, computed directly in float32
    for i in range(n):
        if i not in U1:
            assert r["score"][i] == -np.inf
            continue
        u = u_top[i] if (i in D or i in r["replaced"]) else u_cur[i]
        assert r["score"][i] == F32(F32(u * F32(1 + d_in[i])) / F32(1 + d_out[i]))
    # adaptive rate: n_t pi_t = #{s_j : n s_j > sum s}; |S_t| = ceil(sqrt(.)) capped
    s = {i: Fraction(float(r["score"][i])) for i in U1}
    total = sum(s.values())
    above = sum(1 for i in U1 if len(U1) * s[i] > total)
    assert r["n_t"] == len(U1) and r["n_above"] == above
    k = 0
    while k * k < above:
        k += 1
    elig = [i for i in U1 if i not in S0 and r["remask_cnt"][i] < m_remask]
    assert r["n_select"] == min(k, max_seeds, len(elig))
    chosen = [p - 7 for p in r["seeds"]]
    assert set(chosen) <= set(elig) and len(set(chosen)) == len(chosen)
    for a, b in zip(chosen, chosen[1:]):
        assert r["score"][a] > r["score"][b] or (r["score"][a] == r["score"][b] and a < b)
    for i in chosen:
        for j in set(elig) - set(chosen):
            assert r["score"][i] > r["score"][j] or (r["score"][i] == r["score"][j] and i < j)
    assert {i for i in range(n) if r["flags"][i] & orc.FLAG_SEED} == set(chosen)


def _unmasked_only(scores, **kw):
    n = len(scores)
    s = np.asarray(scores, dtype=F32)
    z = np.zeros(n, dtype=F32)
    args = (np.full(n, 0.5, F32), np.zeros(n, np.int64), np.ones(n, F32), s, s, z, z, np.zeros(n, np.int64),
            np.zeros(n, np.int64), np.zeros(n, np.int64), np.ones(n, np.int64))
    p = dict(tau=F32(0.8), budget=4, m_remask=5, mask_id=-7, min_one=False, pos0=0, max_seeds=64)
    p.update(kw)
    return orc.decide_sequence(*args, **p)


@pytest.mark.parametrize("scores,n_above,k", [
    ([2.0] * 9, 0, 0),                      # all equal: F(mean) = 1, pi = 0, nothing selected
    ([1.0] * 8 + [3.0], 1, 1),              # one above the mean
    ([1.0, 2.0, 3.0, 4.0], 2, 2),           # mean 2.5: two above, ceil(sqrt 2) = 2
    ([0.0] * 6 + [1.0] * 10, 10, 4),        # mean 10/16: ten above, ceil(sqrt 10) = 4
    ([0.0] * 7 + [1.0] * 9, 9, 3),          # a perfect square: sqrt 9 = 3 exactly
    ([5.0], 0, 0),                          # a single unmasked position equals its mean
])
def test_adaptive_rate_closed_forms(scores, n_above, k):
    r = _unmasked_only(scores)
    assert r["n_t"] == len(scores) and r["n_above"] == n_above and r["n_select"] == k
    assert r["n_select"] == math.ceil(math.sqrt(n_above) - 1e-12)


def test_adaptive_rate_capped_by_output_size():
    r = _unmasked_only([0.0] * 6 + [1.0] * 10, max_seeds=3)
    assert r["n_above"] == 10 and r["n_select"] == 3


def test_min_one_takes_lowest_entropy():
    n = 6
    conf = np.full(n, 0.5, F32)                     # nobody above tau
    ent = np.array([3.0, 0.25, 2.0, 0.25, 0.125, 1.0], F32)
    tok = np.array([9, 9, 9, 9, 4, 9])              # row 4 is unmasked
    draft_ok = np.array([1, 1, 1, 1, 1, 0])
    z = np.zeros(n, F32)
    base = (conf, np.arange(n), ent, z, z, z, z, tok, np.zeros(n, np.int64), np.zeros(n, np.int64), draft_ok)
    p = dict(tau=F32(0.8), budget=3, m_remask=2, mask_id=9, pos0=0, max_seeds=4)
    r = orc.decide_sequence(*base, min_one=True, **p)
    assert r["drafted"] == [1]                      # entropy tie 1 / 3 goes to the lower index
    assert r["tok"][1] == 1
    r = orc.decide_sequence(*base, min_one=False, **p)
    assert r["drafted"] == [] and list(r["tok"]) == list(tok)


def test_decide_step_segments():
    rng = np.random.default_rng(3)
    a = _case(12, rng)
    b = _case(12, rng)
    both = tuple(np.concatenate([x, y]) for x, y in zip(a, b))
    p = dict(tau=F32(0.8), budget=2, m_remask=2, mask_id=1000, min_one=True, pos0=5, max_seeds=3)
    outs = orc.decide_step(*both, n_seq=2, **p)
    ra = orc.decide_sequence(*a, **p)
    rb = orc.decide_sequence(*b, **p)
    assert list(outs[0]["tok"]) == list(ra["tok"]) and list(outs[1]["tok"]) == list(rb["tok"])
    assert outs[0]["seeds"] == ra["seeds"] and outs[1]["seeds"] == rb["seeds"]
