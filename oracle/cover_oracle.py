"""Plain, slow, fp64 CPU oracle for COVER's override-attention and seed-scoring path.

TEST INFRASTRUCTURE ONLY. Nothing in the product path may import this module:
only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline /
reference leg use it. It shares no code with the CUDA kernels or their host
glue; it works on numpy float64 arrays that the caller widened exactly from the
stored (fp32 or bf16) inputs.

Everything here is written from the paper's definitions:

* §5.1 "Dual-View Feed Forward through KV Cache Override": the overridden memory
  K', V' (seed columns hold the cached states), attention of every query over
  K', V' with softmax scale 1/sqrt(d), and, for a seed query i, the
  leave-one-out key/value set whose diagonal entry is restored to the pair
  (k_i, v_i) computed from the masked input.
* Appendix B (B.1 notation, Lemma B.1, B.3 weights, B.4 outputs): the closed
  form diagonal correction alpha_i, delta_i, r_i and the corrected output.
* §3 (drafting): greedy token argmax p and confidence max p.
* §6.1: entropy-ordered greedy unmasking (Shannon entropy of p).
* §5.3: uncertainty u(j) = -log p_j(y_j), Score(j) = u (1 + d_in)/(1 + d_out),
  top-k seed selection over eligible positions.
* §5.2 and §3 (one step's decisions): threshold drafting capped at B, the
  Keep / Replace / ReMask revision of the previous seeds, the state update;
  §5.3: the seed score on the updated state, the adaptive revision rate
  |S_t| = ceil(sqrt(n_t pi_t)) and the exclusions from seed selection.
* §5.3 (d_in, d_out): attention mass from masked queries into a position and
  from a position into the drafted ones, over the head-averaged weights.
* §5.1 (seed K/V cache): the states of the new seeds cached at selection and
  written over the seed columns of the next step's memory, the masked-input
  states moving into the diagonal side buffer.

Readings of points the paper leaves open (numbered as in the design notes):
the cached inputs already hold the overridden memory K', V' (R1); the masked
pairs (k_i, v_i) come as a compact [B, Hkv, S, D] buffer whose row s belongs to
position seed_idx[b, s] (R2); grouped-query heads map hkv = hq // (Hq/Hkv)
(R3); no causal mask (R4); scale 1/sqrt(D) (R5); the lse of a seed row is that
of its corrected distribution (R6); out-of-range seeds are ignored and, among
duplicates, the lowest slot wins (R7); ties in argmax / top-k go to the lower
index (R9); entropy is natural-log Shannon entropy at temperature 1 (R10);
without current tokens y = argmax (R11); absent d_in / d_out are 0 (R12);
top-k takes the largest scores (R13). For the decision step: when no masked
position passes the drafting threshold, the lowest-entropy one is drafted if
the caller asks for guaranteed progress (R21); n_t, the mean and the empirical
CDF run over every unmasked position of the updated state with a finite score,
and the exclusions apply only to the selection (R22); |S_t| is further capped
by the caller's seed capacity and the number of eligible positions (R23);
"selected in the previous step" means S_{t-1} (R24); the seed score uses the
uncertainty of the updated token, so a drafted or replaced position takes
-log p(greedy token) (R25); drafting is limited to a caller-given set of
positions, the active block of semi-autoregressive decoding (R26). With a
prefix cache (§6.6) only the active block's queries are computed: query row r
is memory position q0 + r, and a seed outside that window only overrides the
memory (R27).

Every function is pinned by ``tests/test_oracle_pins.py`` against closed forms,
hand-worked fixtures, a library routine (torch float64 SDPA) and brute force.
"""
from __future__ import annotations

import math
from typing import Optional, Sequence

import numpy as np

TILE_ROWS = 128  # row-tile height of the seed bitmap (a build structure, not the paper's)


# ----------------------------------------------------------------------------
# Seed routing (seed set semantics, §3 "Decoding protocol" and §5.1)
# ----------------------------------------------------------------------------

def route_seeds(seed_idx: np.ndarray, L: int):
    """Map each position of each batch row to the slot of the seed that names it.

    seed_idx: int [B, S]. Returns (slot [B, L] int32 with -1 for non-seeds,
    bitmap [B, ceil(L/128), 4] uint32 with bit (r % 32) of word (r % 128) // 32
    of tile r // 128 set iff slot[r] >= 0, n_invalid = number of entries that
    are out of [0, L) or repeat an earlier slot's position).
    """
    seed_idx = np.asarray(seed_idx)
    B = seed_idx.shape[0]
    S = seed_idx.shape[1] if seed_idx.ndim == 2 else 0
    slot = np.full((B, L), -1, dtype=np.int32)
    n_invalid = 0
    for b in range(B):
        for s in range(S):
            p = int(seed_idx[b, s])
            if p < 0 or p >= L:
                n_invalid += 1
                continue
            if slot[b, p] >= 0:
                n_invalid += 1          # duplicate: the earlier (lower) slot keeps the position
                continue
            slot[b, p] = s
    n_tiles = (L + TILE_ROWS - 1) // TILE_ROWS
    bitmap = np.zeros((B, n_tiles, 4), dtype=np.uint32)
    for b in range(B):
        for r in range(L):
            if slot[b, r] >= 0:
                t, w, bit = r // TILE_ROWS, (r % TILE_ROWS) // 32, r % 32
                bitmap[b, t, w] |= np.uint32(1) << np.uint32(bit)
    return slot, bitmap, n_invalid


# ----------------------------------------------------------------------------
# Attention: the explicit two-view definition (§5.1, Appendix B.1)
# ----------------------------------------------------------------------------

def _softmax_row(z: np.ndarray):
    """Naive softmax with max subtraction; returns (weights, natural-log lse)."""
    m = np.max(z)
    e = np.exp(z - m)
    Z = np.sum(e)
    return e / Z, m + math.log(Z)


def view_for_row(kc_h: np.ndarray, vc_h: np.ndarray, i: int, masked_pair=None):
    """Key/value set seen by query i (§5.1, Appendix B.1).

    kc_h, vc_h: [L, D] overridden memory K', V' of one KV head. For a seed query
    the diagonal entry is restored to the masked-input pair (k_i, v_i); every
    other entry stays K', V'. Non-seed queries see K', V' unchanged.
    """
    if masked_pair is None:
        return kc_h, vc_h
    K = kc_h.copy()
    V = vc_h.copy()
    K[i] = masked_pair[0]
    V[i] = masked_pair[1]
    return K, V


def attention_row(q_i: np.ndarray, K: np.ndarray, V: np.ndarray):
    """o_i = softmax(K q_i / sqrt(d)) V and its lse, for one query over one key/value set."""
    d = q_i.shape[-1]
    z = (K @ q_i) / math.sqrt(d)
    w, lse = _softmax_row(z)
    return w @ V, lse, w


def override_attention_rows(q, kc, vc, km, vm, seed_idx, b: int, hq: int, rows: Sequence[int]):
    """Outputs of the listed query rows of head (b, hq), each from its own explicit view."""
    B, Hq, L, D = q.shape
    Hkv = kc.shape[1]
    hkv = hq // (Hq // Hkv)
    slot, _, _ = route_seeds(seed_idx[b:b + 1], L) if seed_idx is not None and seed_idx.size else (
        np.full((1, L), -1, np.int32), None, 0)
    out = np.zeros((len(rows), D))
    lse = np.zeros(len(rows))
    for n, i in enumerate(rows):
        s = int(slot[0, i])
        pair = (km[b, hkv, s], vm[b, hkv, s]) if s >= 0 else None
        K, V = view_for_row(kc[b, hkv], vc[b, hkv], i, pair)
        out[n], lse[n], _ = attention_row(q[b, hq, i], K, V)
    return out, lse


def override_attention(q, kc, vc, km, vm, seed_idx):
    """Full two-view attention output and lse for every (b, hq, i).

    q [B,Hq,L,D], kc/vc [B,Hkv,L,D] (= K', V'), km/vm [B,Hkv,S,D],
    seed_idx [B,S]. Non-seed rows are plain attention over K', V' (computed a
    head at a time with a matmul); seed rows go through their explicit
    leave-one-out view one by one.
    """
    B, Hq, L, D = q.shape
    Hkv = kc.shape[1]
    G = Hq // Hkv
    S = 0 if seed_idx is None else seed_idx.shape[1]
    slot = route_seeds(seed_idx, L)[0] if S else np.full((B, L), -1, np.int32)
    out = np.zeros((B, Hq, L, D))
    lse = np.zeros((B, Hq, L))
    for b in range(B):
        for hq in range(Hq):
            hkv = hq // G
            Kp, Vp = kc[b, hkv], vc[b, hkv]
            z = (q[b, hq] @ Kp.T) / math.sqrt(D)          # [L, L]
            m = z.max(axis=1, keepdims=True)
            e = np.exp(z - m)
            Z = e.sum(axis=1, keepdims=True)
            out[b, hq] = (e / Z) @ Vp
            lse[b, hq] = (m + np.log(Z))[:, 0]
            for i in np.nonzero(slot[b] >= 0)[0]:
                s = int(slot[b, i])
                K, V = view_for_row(Kp, Vp, int(i), (km[b, hkv, s], vm[b, hkv, s]))
                out[b, hq, i], lse[b, hq, i], _ = attention_row(q[b, hq, i], K, V)
    return out, lse


def override_attention_window(q, kc, vc, km, vm, seed_idx, q0: int):
    """Two-view attention for a window of query rows (§6.6 prefix cache; reading R27).

    q [B,Hq,Lq,D] holds the queries of memory positions q0 .. q0+Lq-1 (the
    active block); kc/vc [B,Hkv,Lk,D] are K', V' over every position; seeds are
    memory positions in [0, Lk). Row r is computed as memory position q0 + r:
    attention over K', V', or, when that position is a seed, over its
    leave-one-out view. Seeds outside the window change nothing here.
    """
    B, Hq, Lq, D = q.shape
    Hkv, Lk = kc.shape[1], kc.shape[2]
    G = Hq // Hkv
    S = 0 if seed_idx is None else seed_idx.shape[1]
    slot = route_seeds(seed_idx, Lk)[0] if S else np.full((B, Lk), -1, np.int32)
    out = np.zeros((B, Hq, Lq, D))
    lse = np.zeros((B, Hq, Lq))
    for b in range(B):
        for hq in range(Hq):
            hkv = hq // G
            for r in range(Lq):
                i = q0 + r
                s = int(slot[b, i])
                pair = (km[b, hkv, s], vm[b, hkv, s]) if s >= 0 else None
                K, V = view_for_row(kc[b, hkv], vc[b, hkv], i, pair)
                out[b, hq, r], lse[b, hq, r], _ = attention_row(q[b, hq, r], K, V)
    return out, lse


def attention_mass(q, kc, km, seed_idx, masked, drafted, pos0: int):
    """d_in and d_out of §5.3 from the head-averaged attention of the current pass.

    q [B,Hq,L,D] and kc [B,Hkv,L,D] (= K') cover every memory position; km
    [B,Hkv,S,D] holds the masked-input keys of the seeds (seed_idx [B,S]).
    The weight row of a query is its softmax over its own key set (§5.1: K',
    with the diagonal restored to k_i for a seed), i.e. the corrected weights
    of App. B.3. A = mean over the Hq heads of those weight matrices.
    masked / drafted [B, n] flag the response positions pos0 .. pos0+n-1 that
    are in M_t (masked after the update) and D_t (drafted this step). Returns
    d_in, d_out [B, n]: d_in[j] = sum over masked q of A[q -> j], d_out[j] =
    sum over drafted i of A[j -> i], for the response positions j.
    """
    B, Hq, L, D = q.shape
    Hkv = kc.shape[1]
    G = Hq // Hkv
    n = masked.shape[1]
    S = 0 if seed_idx is None else seed_idx.shape[1]
    slot = route_seeds(seed_idx, L)[0] if S else np.full((B, L), -1, np.int32)
    d_in = np.zeros((B, n))
    d_out = np.zeros((B, n))
    for b in range(B):
        A = np.zeros((n, L))                       # head-averaged weight rows of the response queries
        for hq in range(Hq):
            hkv = hq // G
            for r in range(n):
                i = pos0 + r
                s = int(slot[b, i])
                K = kc[b, hkv]
                if s >= 0:
                    K = K.copy()
                    K[i] = km[b, hkv, s]
                z = K @ q[b, hq, i] / math.sqrt(D)
                w = np.exp(z - z.max())
                A[r] += w / w.sum() / Hq
        cols = A[:, pos0:pos0 + n]                 # attention from response queries to response keys
        d_in[b] = cols[np.asarray(masked[b], bool)].sum(axis=0)
        d_out[b] = cols[:, np.asarray(drafted[b], bool)].sum(axis=1)
    return d_in, d_out


def override_attention_closed_form(q, kc, vc, km, vm, seed_idx):
    """The same result through Appendix B's closed form (Lemma B.1, B.3, B.4).

    One attention pass over K', V' for all rows, then for each seed row:
    alpha_i = w_ovr[i, i], delta_i = q_i (k_i - k'_i) / sqrt(d),
    r_i = 1 + alpha_i (exp(delta_i) - 1),
    o_i = (o_ovr_i - alpha_i v'_i + alpha_i exp(delta_i) v_i) / r_i,
    lse_i = lse_ovr_i + ln r_i (the normaliser changes by the factor r_i).
    """
    B, Hq, L, D = q.shape
    Hkv = kc.shape[1]
    G = Hq // Hkv
    S = 0 if seed_idx is None else seed_idx.shape[1]
    slot = route_seeds(seed_idx, L)[0] if S else np.full((B, L), -1, np.int32)
    out = np.zeros((B, Hq, L, D))
    lse = np.zeros((B, Hq, L))
    for b in range(B):
        for hq in range(Hq):
            hkv = hq // G
            Kp, Vp = kc[b, hkv], vc[b, hkv]
            s_ovr = (q[b, hq] @ Kp.T) / math.sqrt(D)
            m = s_ovr.max(axis=1, keepdims=True)
            e = np.exp(s_ovr - m)
            Z = e.sum(axis=1, keepdims=True)
            w_ovr = e / Z
            o_ovr = w_ovr @ Vp
            lse_ovr = (m + np.log(Z))[:, 0]
            out[b, hq] = o_ovr
            lse[b, hq] = lse_ovr
            for i in np.nonzero(slot[b] >= 0)[0]:
                s = int(slot[b, i])
                k_i, v_i = km[b, hkv, s], vm[b, hkv, s]
                alpha = w_ovr[i, i]
                delta = float(q[b, hq, i] @ (k_i - Kp[i])) / math.sqrt(D)
                r = 1.0 + alpha * (math.exp(delta) - 1.0)
                out[b, hq, i] = (o_ovr[i] - alpha * Vp[i] + alpha * math.exp(delta) * v_i) / r
                lse[b, hq, i] = lse_ovr[i] + math.log(r)
    return out, lse


def corrected_weights_row(q, kc, vc, km, vm, seed_idx, b: int, hq: int, i: int):
    """Attention weights of row i under its own view (Appendix B.3), for sum-to-one checks."""
    B, Hq, L, D = q.shape
    hkv = hq // (Hq // kc.shape[1])
    slot = route_seeds(seed_idx[b:b + 1], L)[0][0] if seed_idx is not None and seed_idx.size else (
        np.full(L, -1, np.int32))
    s = int(slot[i])
    pair = (km[b, hkv, s], vm[b, hkv, s]) if s >= 0 else None
    K, V = view_for_row(kc[b, hkv], vc[b, hkv], i, pair)
    return attention_row(q[b, hq, i], K, V)[2]


# ----------------------------------------------------------------------------
# Per-position scoring (§3 drafting, §6.1 entropy, §5.3 seed score)
# ----------------------------------------------------------------------------

def score_rows(logits: np.ndarray, cur_tok=None, d_in=None, d_out=None):
    """Per-row confidence, entropy, greedy token, uncertainty and seed score.

    logits: float64 [N, V] (exact widening of the bf16 values). For each row,
    p = softmax(x) at temperature 1; c = max_v p(v) (§3); y_hat = the first
    index attaining the maximum logit (§3, ties to the lower index); H =
    -sum_v p(v) ln p(v) (§6.1); u = -ln p(y) with y = cur_tok, or y_hat when no
    current tokens are given (§5.3); Score = u (1 + d_in) / (1 + d_out) with
    absent d_in / d_out taken as 0 (§5.3).
    Returns dict of float64 / int64 arrays: maxprob, entropy, argmax, u, score.
    """
    x = np.asarray(logits, dtype=np.float64)
    N, V = x.shape
    maxprob = np.zeros(N)
    entropy = np.zeros(N)
    argmax = np.zeros(N, dtype=np.int64)
    u = np.zeros(N)
    score = np.zeros(N)
    for n in range(N):
        row = x[n]
        m = row.max()
        y_hat = int(np.argmax(row))            # first occurrence of the maximum
        e = np.exp(row - m)
        Z = e.sum()
        p = e / Z
        logp = (row - m) - math.log(Z)
        maxprob[n] = p.max()
        entropy[n] = -np.sum(p * logp)
        argmax[n] = y_hat
        y = y_hat if cur_tok is None else int(cur_tok[n])
        u[n] = -logp[y]
        din = 0.0 if d_in is None else float(d_in[n])
        dout = 0.0 if d_out is None else float(d_out[n])
        score[n] = u[n] * (1.0 + din) / (1.0 + dout)
    return dict(maxprob=maxprob, entropy=entropy, argmax=argmax, u=u, score=score)


def topk_select(score: np.ndarray, n_seq: int, k: int, eligible=None):
    """Top-k seed selection per sequence segment (§5.3).

    The N rows split into n_seq equal consecutive segments. Within a segment the
    eligible rows are ordered by score, largest first, ties to the lower index;
    the first k are taken. Returned indices are offsets within the segment;
    missing entries (fewer than k eligible rows) are -1 with score -inf.
    """
    score = np.asarray(score)
    N = score.shape[0]
    per = N // n_seq
    idx = np.full((n_seq, k), -1, dtype=np.int64)
    val = np.full((n_seq, k), -np.inf)
    for g in range(n_seq):
        cand = [j for j in range(per) if eligible is None or eligible[g * per + j]]
        ranked = sorted(cand, key=lambda j: (-float(score[g * per + j]), j))
        for t, j in enumerate(ranked[:k]):
            idx[g, t] = j
            val[g, t] = score[g * per + j]
    return idx, val


def topk_margin(score: np.ndarray, n_seq: int, k: int, eligible=None):
    """Per segment, the gap between the k-th and (k+1)-th largest eligible score (inf if none)."""
    score = np.asarray(score, dtype=np.float64)
    N = score.shape[0]
    per = N // n_seq
    gaps = np.full(n_seq, np.inf)
    for g in range(n_seq):
        vals = [score[g * per + j] for j in range(per) if eligible is None or eligible[g * per + j]]
        vals.sort(reverse=True)
        if len(vals) > k:
            gaps[g] = vals[k - 1] - vals[k]
    return gaps


# ----------------------------------------------------------------------------
# One decoding step's decisions after scoring: §5.2 (threshold drafting with a
# budget, the Keep / Replace / ReMask revision rule), §3 (state update) and
# §5.3 (stability-aware seed score on the updated state, adaptive revision
# rate |S_t| = ceil(sqrt(n_t pi_t)), exclusion of the previous seeds and of
# positions that used up their ReMask budget).
# ----------------------------------------------------------------------------

FLAG_SEED = 1   # bit of the per-position flag byte: "in the seed set"


def decide_sequence(conf, yhat, ent, u_cur, u_top, d_in, d_out, tok, flags, remask_cnt, draft_ok, *,
                    tau: float, budget: int, m_remask: int, mask_id: int, min_one: bool, pos0: int,
                    max_seeds: int):
    """Decisions of one step for one sequence (rows = its response positions).

    Per row i the scoring pass of this step supplies c_i = max_v p_i(v)
    (``conf``), the greedy token (``yhat``), the entropy H_i (``ent``),
    u_cur = -log p_i(y_i^(t-1)) for the current token and u_top = -log p_i(yhat_i).
    ``tok`` holds y^(t-1) with ``mask_id`` for [MASK]; bit FLAG_SEED of
    ``flags`` marks S_{t-1}; ``remask_cnt`` counts each position's ReMasks so
    far; ``draft_ok`` marks the positions the drafting rule may unmask (the
    active block of semi-autoregressive decoding); d_in / d_out are the
    influence terms of the seed score (None = 0).

    The seed score is formed in the floating-point type of ``u_cur`` / ``u_top``
    as (u * (1 + d_in)) / (1 + d_out); every comparison that follows (the
    threshold, the orderings, the mean of the adaptive rate) is exact on those
    values (the mean is a Fraction).

    Returns a dict: tok, remask_cnt, flags (new arrays), drafted / kept /
    replaced / remasked (sorted index lists), score (per row, -inf where the
    new state is [MASK] or the score is not finite), n_t, n_above, n_select,
    seeds (positions pos0 + i in selection order).
    """
    from fractions import Fraction

    n = len(tok)
    tok = np.asarray(tok, dtype=np.int64)
    flags = np.asarray(flags, dtype=np.int64)
    remask_cnt = np.asarray(remask_cnt, dtype=np.int64)
    conf = np.asarray(conf)
    dtype = np.asarray(u_cur).dtype.type

    # masked / unmasked sets at the start of the step (§3)
    masked = [i for i in range(n) if tok[i] == mask_id]
    unmasked = [i for i in range(n) if tok[i] != mask_id]
    seeds_prev = [i for i in unmasked if flags[i] & FLAG_SEED]

    # drafting (§5.2): masked positions whose confidence exceeds tau, at most
    # `budget` of them, the largest confidences kept (ties to the lower index)
    draftable = [i for i in masked if draft_ok is None or draft_ok[i]]
    over = [i for i in draftable if conf[i] > tau]
    over.sort(key=lambda i: (-float(conf[i]), i))
    drafted = sorted(over[:max(budget, 0)])
    if not drafted and min_one and draftable:
        # guaranteed progress: the lowest-entropy masked position (§6.1)
        drafted = [min(draftable, key=lambda i: (float(ent[i]), i))]

    # revision of the previous seeds (§5.2): Keep / Replace / ReMask
    kept, replaced, remasked = [], [], []
    for i in seeds_prev:
        if yhat[i] == tok[i]:
            kept.append(i)
        elif conf[i] > tau:
            replaced.append(i)
        else:
            remasked.append(i)

    # state update (§3)
    new_tok = tok.copy()
    new_rc = remask_cnt.copy()
    for i in drafted + replaced:
        new_tok[i] = yhat[i]
    for i in remasked:
        new_tok[i] = mask_id
        new_rc[i] += 1
    changed = set(drafted) | set(replaced)

    # seed score on the updated state (§5.3): u = -log p(y^(t))
    score = np.full(n, -np.inf)
    scored = []
    one = dtype(1)
    for i in range(n):
        if new_tok[i] == mask_id:
            continue
        u = dtype(u_top[i]) if i in changed else dtype(u_cur[i])
        din = dtype(0) if d_in is None else dtype(d_in[i])
        dout = dtype(0) if d_out is None else dtype(d_out[i])
        s = dtype(dtype(u * dtype(one + din)) / dtype(one + dout))
        if np.isfinite(s):
            score[i] = s
            scored.append(i)

    # adaptive revision rate (§5.3): n_t, the empirical CDF at the mean, pi_t
    n_t = len(scored)
    n_select = 0
    n_above = 0
    if n_t > 0:
        vals = {i: Fraction(float(score[i])) for i in scored}
        mean = sum(vals.values()) / n_t
        F = Fraction(sum(1 for i in scored if vals[i] <= mean), n_t)
        pi = 1 - F
        n_above = int(n_t * pi)                  # n_t * pi_t is a whole number
        n_select = math.isqrt(n_above)
        if n_select * n_select < n_above:
            n_select += 1                        # ceil(sqrt(n_t pi_t))
    n_select = min(n_select, max_seeds)

    # selection: previous seeds and positions at the ReMask budget are excluded
    prev = set(seeds_prev)
    eligible = [i for i in scored if i not in prev and new_rc[i] < m_remask]
    eligible.sort(key=lambda i: (-float(score[i]), i))
    chosen = eligible[:n_select]

    new_flags = flags & ~FLAG_SEED
    for i in chosen:
        new_flags[i] |= FLAG_SEED
    return dict(tok=new_tok, remask_cnt=new_rc, flags=new_flags, drafted=drafted, kept=sorted(kept),
                replaced=sorted(replaced), remasked=sorted(remasked), score=score, n_t=n_t, n_above=n_above,
                n_select=len(chosen), seeds=[pos0 + i for i in chosen])


def decide_step(conf, yhat, ent, u_cur, u_top, d_in, d_out, tok, flags, remask_cnt, draft_ok, n_seq: int,
                **params):
    """decide_sequence over the n_seq equal consecutive segments of N rows."""
    N = len(tok)
    per = N // n_seq
    outs = []
    for g in range(n_seq):
        sl = slice(g * per, (g + 1) * per)
        pick = (lambda a: None if a is None else np.asarray(a)[sl])
        outs.append(decide_sequence(pick(conf), pick(yhat), pick(ent), pick(u_cur), pick(u_top), pick(d_in),
                                    pick(d_out), pick(tok), pick(flags), pick(remask_cnt), pick(draft_ok),
                                    **params))
    return outs


# ----------------------------------------------------------------------------
# Seed K/V cache (§5.1 "KV cache override yields a stable drafting view"):
# at selection the per-layer key / value states of the new seeds are cached;
# at the next step the memory is overridden at the seed positions with them,
# while the states computed from the masked input at those positions become
# the diagonal pairs (k_i, v_i) of the leave-one-out views.
# ----------------------------------------------------------------------------

def _seed_slots(seed_idx, L: int):
    """Per batch row, the (slot, position) pairs that name a position: in range and
    not repeating an earlier slot's position (the lowest slot wins, as in R7)."""
    out = []
    for b in range(seed_idx.shape[0]):
        seen, pairs = set(), []
        for s in range(seed_idx.shape[1]):
            j = int(seed_idx[b, s])
            if 0 <= j < L and j not in seen:
                seen.add(j)
                pairs.append((s, j))
        out.append(pairs)
    return out


def seed_kv_gather(k, v, seed_idx):
    """Cache at selection: cache[b, h, s] = state[b, h, seed_idx[b, s]] for k and v.

    k, v: [B, Hkv, L, D] (any dtype; values are copied, never computed).
    A slot whose position is out of [0, L) holds zeros; a repeated position is
    cached again in every slot that names it.
    """
    B, H, L, D = k.shape
    S = seed_idx.shape[1]
    kc = np.zeros((B, H, S, D), dtype=k.dtype)
    vc = np.zeros((B, H, S, D), dtype=v.dtype)
    for b in range(B):
        for s in range(S):
            j = int(seed_idx[b, s])
            if 0 <= j < L:
                kc[b, :, s] = k[b, :, j]
                vc[b, :, s] = v[b, :, j]
    return kc, vc


def seed_kv_override(k, v, seed_idx, k_cache, v_cache):
    """Override at the next step.

    k, v: the layer's states from the masked input, [B, Hkv, L, D];
    k_cache, v_cache: the states cached at selection, [B, Hkv, S, D].
    Returns (k', v', k_mask, v_mask): k'/v' equal k/v except that row j of
    every seed (b, s, j) holds the cached row s; k_mask/v_mask row s holds the
    masked-input state at j (the pair (k_j, v_j) restored on the diagonal).
    Slots that do not name a position (out of range, or a position already
    named by a lower slot) keep their cache row and change no memory row.
    """
    L = k.shape[2]
    k2, v2 = k.copy(), v.copy()
    km, vm = k_cache.copy(), v_cache.copy()
    for b, pairs in enumerate(_seed_slots(seed_idx, L)):
        for s, j in pairs:
            k2[b, :, j] = k_cache[b, :, s]
            v2[b, :, j] = v_cache[b, :, s]
            km[b, :, s] = k[b, :, j]
            vm[b, :, s] = v[b, :, j]
    return k2, v2, km, vm
