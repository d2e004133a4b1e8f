"""Seeded synthetic inputs for the override-attention and scoring path.

This module is shared by the oracle-side tests and the CUDA path. It holds
no arithmetic of the method itself: it only draws random numbers, rounds them
to the storage precision, and places seed positions.

Input recipe (the paper's workloads are LLaDA-8B / Dream-7B forward passes
over HumanEval/MBPP/GSM8K/MATH500 prompts, §6.1; none of those weights or
datasets are used, synthetic tensors of the same shapes stand in):

* ``numpy.random.default_rng(seed)`` draws, in this order, q [B,Hq,L,D],
  k_cached [B,Hkv,L,D], v_cached [B,Hkv,L,D], k_seedmask [B,Hkv,S,D],
  v_seedmask [B,Hkv,S,D] (all standard normal, float32, C order), then the
  seed positions per batch row.
* Optional scaling of q/k_cached/v_cached by ``in_scale`` (the LLaDA L=512
  workload uses 1/D**0.25); the masked side buffer is never scaled.
* bf16 workloads round every float32 draw to bf16 with round-to-nearest-even;
  the rounded values are what both the oracle and the kernels see.
* Logits come from a separate ``default_rng(seed + 1)``: N(0, 2) means
  variance 2 (standard deviation sqrt(2)). Spiked rows get +8 added to one
  uniformly chosen vocabulary entry before bf16 rounding.
* Decision-step state (make_decide_inputs, ``default_rng(seed + 2)``): per
  sequence of ``per`` response positions an active block of ``block_len``
  positions (64 for LLaDA-shaped, 32 for Dream-shaped workloads, §6.1) starts
  at a uniformly drawn multiple of ``block_len``; positions before it hold
  tokens, positions inside it are masked with probability 1/2, positions after
  it are masked. ceil(sqrt(unmasked)) unmasked positions carry the
  previous-seed flag; unmasked positions have ReMask counts uniform in
  [0, m_remask]. [MASK] is token V - 128. Logits are N(0, var) plus, on one
  token per row, a spike uniform in [0, max_spike): the current token with
  probability 1/2 for previous seeds, else a uniform token. d_in and d_out are
  uniform in [0, 2).
* Seed positions: "uniform" draws S distinct positions from [lo, hi) without
  replacement, in draw order (slot s <-> draw s). "runs" draws the starts of
  ``n_runs`` contiguous runs uniformly from [lo, hi - run_len] and rejects a
  start that overlaps an earlier run; slots follow run order then position.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import numpy as np


# ----------------------------------------------------------------------------
# bf16 storage helpers (input preparation only)
# ----------------------------------------------------------------------------

def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bf16 (round-to-nearest-even); return uint16 bits."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    rounded = u + (np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1)))
    return (rounded >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float32."""
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def bf16_bits_to_f64(b: np.ndarray) -> np.ndarray:
    return bf16_bits_to_f32(b).astype(np.float64)


# ----------------------------------------------------------------------------
# Seed placement
# ----------------------------------------------------------------------------

def draw_seeds_uniform(rng: np.random.Generator, S: int, lo: int, hi: int) -> np.ndarray:
    if S > hi - lo:
        raise ValueError(f"cannot draw {S} distinct seeds from [{lo}, {hi})")
    return rng.choice(np.arange(lo, hi, dtype=np.int64), size=S, replace=False).astype(np.int32)


def draw_seeds_runs(rng: np.random.Generator, n_runs: int, run_len: int, lo: int, hi: int) -> np.ndarray:
    starts: list[int] = []
    guard = 0
    while len(starts) < n_runs:
        a = int(rng.integers(lo, hi - run_len + 1))
        guard += 1
        if guard > 100000:
            raise RuntimeError("could not place disjoint seed runs")
        if all(abs(a - b) >= run_len for b in starts):
            starts.append(a)
    return np.concatenate([np.arange(a, a + run_len, dtype=np.int32) for a in starts])


# ----------------------------------------------------------------------------
# Attention inputs
# ----------------------------------------------------------------------------

@dataclasses.dataclass
class AttnInputs:
    B: int
    Hq: int
    Hkv: int
    L: int
    D: int
    S: int
    dtype: str                    # "f32" or "bf16"
    # storage arrays: float32 for "f32", uint16 bf16 bits for "bf16"
    q: np.ndarray
    k_cached: np.ndarray
    v_cached: np.ndarray
    k_seedmask: np.ndarray
    v_seedmask: np.ndarray
    seed_idx: np.ndarray          # int32 [B, S]

    def as_f64(self, name: str) -> np.ndarray:
        a = getattr(self, name)
        if self.dtype == "bf16":
            return bf16_bits_to_f64(a)
        return a.astype(np.float64)


def _store(x: np.ndarray, dtype: str) -> np.ndarray:
    if dtype == "bf16":
        return f32_to_bf16_bits(x)
    if dtype == "f32":
        return np.ascontiguousarray(x, dtype=np.float32)
    raise ValueError(dtype)


def make_attn_inputs(B: int, Hq: int, Hkv: int, L: int, D: int, S: int, *, dtype: str = "bf16",
                     seed: int = 0, seed_lo: int = 0, seed_hi: Optional[int] = None,
                     placement: str = "uniform", n_runs: int = 4, run_len: int = 64,
                     in_scale: float = 1.0) -> AttnInputs:
    """Draw one attention workload following the recipe in the module docstring."""
    if seed_hi is None:
        seed_hi = L
    rng = np.random.default_rng(seed)
    q = rng.standard_normal((B, Hq, L, D), dtype=np.float32)
    kc = rng.standard_normal((B, Hkv, L, D), dtype=np.float32)
    vc = rng.standard_normal((B, Hkv, L, D), dtype=np.float32)
    km = rng.standard_normal((B, Hkv, S, D), dtype=np.float32)
    vm = rng.standard_normal((B, Hkv, S, D), dtype=np.float32)
    if in_scale != 1.0:
        s = np.float32(in_scale)
        q *= s
        kc *= s
        vc *= s
    seeds = np.zeros((B, S), dtype=np.int32)
    for b in range(B):
        if S == 0:
            continue
        if placement == "uniform":
            seeds[b] = draw_seeds_uniform(rng, S, seed_lo, seed_hi)
        elif placement == "runs":
            if n_runs * run_len != S:
                raise ValueError("runs placement needs S == n_runs * run_len")
            seeds[b] = draw_seeds_runs(rng, n_runs, run_len, seed_lo, seed_hi)
        else:
            raise ValueError(placement)
    return AttnInputs(B, Hq, Hkv, L, D, S, dtype,
                      _store(q, dtype), _store(kc, dtype), _store(vc, dtype),
                      _store(km, dtype), _store(vm, dtype), seeds)


# ----------------------------------------------------------------------------
# Scoring inputs
# ----------------------------------------------------------------------------

@dataclasses.dataclass
class ScoreInputs:
    N: int
    V: int
    n_seq: int
    topk: int
    logits: np.ndarray            # uint16 bf16 bits [N, V]
    spiked_rows: np.ndarray       # int64 rows that received the +8 spike (informational)
    cur_tok: Optional[np.ndarray] = None     # int32 [N] or None
    d_in: Optional[np.ndarray] = None        # float32 [N] or None
    d_out: Optional[np.ndarray] = None       # float32 [N] or None
    eligible: Optional[np.ndarray] = None    # uint8 [N] or None

    def logits_f64(self, rows=None) -> np.ndarray:
        x = self.logits if rows is None else self.logits[rows]
        return bf16_bits_to_f64(x)


def make_score_inputs(N: int, V: int, n_seq: int, topk: int, *, seed: int = 0, var: float = 2.0,
                      spike_frac: float = 0.0, spike: float = 8.0,
                      with_cur_tok: bool = False, with_dio: bool = False,
                      eligible_frac: Optional[float] = None) -> ScoreInputs:
    """Draw bf16 logits N(0, var) with optional spiked rows (recipe in the module docstring).

    Optional side inputs (current tokens, d_in/d_out, eligibility mask) are drawn
    after the logits from the same generator, in that order.
    """
    rng = np.random.default_rng(seed + 1)
    x = rng.standard_normal((N, V), dtype=np.float32)
    x *= np.float32(math.sqrt(var))
    n_spike = int(round(spike_frac * N))
    rows = np.zeros(0, dtype=np.int64)
    if n_spike > 0:
        rows = rng.choice(N, size=n_spike, replace=False)
        cols = rng.integers(0, V, size=n_spike)
        x[rows, cols] += np.float32(spike)
    logits = f32_to_bf16_bits(x)
    del x
    inp = ScoreInputs(N, V, n_seq, topk, logits, rows)
    if with_cur_tok:
        inp.cur_tok = rng.integers(0, V, size=N).astype(np.int32)
    if with_dio:
        inp.d_in = rng.uniform(0.0, 3.0, size=N).astype(np.float32)
        inp.d_out = rng.uniform(0.0, 3.0, size=N).astype(np.float32)
    if eligible_frac is not None:
        inp.eligible = (rng.uniform(size=N) < eligible_frac).astype(np.uint8)
    return inp


@dataclasses.dataclass
class DecideInputs:
    """Logits and decoding state for one step of the decision epilogue."""
    N: int
    V: int
    n_seq: int
    mask_id: int
    logits: np.ndarray       # uint16 bf16 bits [N, V]
    tok: np.ndarray          # int32 [N]; mask_id marks [MASK]
    flags: np.ndarray        # uint8 [N]; bit 0 marks the previous seeds
    remask_cnt: np.ndarray   # uint8 [N]
    draft_ok: np.ndarray     # uint8 [N]; the active block
    d_in: np.ndarray         # float32 [N]
    d_out: np.ndarray        # float32 [N]

    def logits_f64(self, rows=None) -> np.ndarray:
        b = self.logits if rows is None else self.logits[rows]
        return bf16_bits_to_f64(b)


def make_decide_inputs(N: int, V: int, n_seq: int, *, seed: int = 0, block_len: int = 64, var: float = 2.0,
                       max_spike: float = 16.0, m_remask: int = 5) -> DecideInputs:
    """Draw one decoding step's state and its logits (recipe in the module docstring)."""
    rng = np.random.default_rng(seed + 2)
    per = N // n_seq
    mask_id = V - 128 if V > 128 else V - 1
    tok = rng.integers(0, V - 1, size=N).astype(np.int32)
    tok[tok >= mask_id] += 1                              # real tokens never equal [MASK]
    flags = np.zeros(N, dtype=np.uint8)
    remask = np.zeros(N, dtype=np.uint8)
    draft_ok = np.zeros(N, dtype=np.uint8)
    n_blocks = max(1, -(-per // block_len))
    for g in range(n_seq):
        base = g * per
        lo = int(rng.integers(0, n_blocks)) * block_len
        hi = min(per, lo + block_len)
        in_block = rng.uniform(size=hi - lo) < 0.5
        seg = tok[base:base + per]
        seg[hi:] = mask_id
        seg[lo:hi][in_block] = mask_id
        draft_ok[base + lo:base + hi] = 1
        unmasked = np.nonzero(seg != mask_id)[0]
        if len(unmasked):
            k = int(math.ceil(math.sqrt(len(unmasked))))
            pick = rng.choice(unmasked, size=k, replace=False)
            flags[base + pick] = 1
            remask[base + unmasked] = rng.integers(0, m_remask + 1, size=len(unmasked))
    x = rng.standard_normal((N, V), dtype=np.float32)
    x *= np.float32(math.sqrt(var))
    spike_tok = rng.integers(0, V, size=N)
    keep = (flags == 1) & (rng.uniform(size=N) < 0.5)
    spike_tok[keep] = tok[keep]
    spike = rng.uniform(0.0, max_spike, size=N).astype(np.float32)
    x[np.arange(N), spike_tok] += spike
    logits = f32_to_bf16_bits(x)
    del x
    d_in = rng.uniform(0.0, 2.0, size=N).astype(np.float32)
    d_out = rng.uniform(0.0, 2.0, size=N).astype(np.float32)
    return DecideInputs(N, V, n_seq, mask_id, logits, tok, flags, remask, draft_ok, d_in, d_out)


# ----------------------------------------------------------------------------
# The five named workloads
# ----------------------------------------------------------------------------

@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    B: int
    Hq: int
    Hkv: int
    L: int
    D: int
    S: int
    dtype: str
    seed_lo: int
    seed_hi: int
    placement: str = "uniform"
    in_scale: float = 1.0
    # scoring part (None when the workload has no logits)
    score_N: Optional[int] = None
    score_V: Optional[int] = None
    score_n_seq: Optional[int] = None
    score_topk: Optional[int] = None
    score_spike_frac: float = 0.0
    decide_block: int = 64
    seed: int = 0

    @property
    def attn_flops(self) -> float:
        """Algorithmic flops of one override-attention pass: 4*B*Hq*L^2*D."""
        return 4.0 * self.B * self.Hq * self.L * self.L * self.D

    def attn_inputs(self) -> AttnInputs:
        return make_attn_inputs(self.B, self.Hq, self.Hkv, self.L, self.D, self.S, dtype=self.dtype,
                                seed=self.seed, seed_lo=self.seed_lo, seed_hi=self.seed_hi,
                                placement=self.placement, in_scale=self.in_scale)

    def score_inputs(self) -> Optional[ScoreInputs]:
        if self.score_N is None:
            return None
        return make_score_inputs(self.score_N, self.score_V, self.score_n_seq, self.score_topk,
                                 seed=self.seed, spike_frac=self.score_spike_frac)


    def decide_inputs(self) -> Optional[DecideInputs]:
        if self.score_N is None:
            return None
        return make_decide_inputs(self.score_N, self.score_V, self.score_n_seq, seed=self.seed,
                                  block_len=self.decide_block)


WORKLOADS = {
    # tiny fp32 check
    "tiny_f32_l64": Workload("tiny_f32_l64", 1, 2, 2, 64, 64, 4, "f32", 32, 64),
    # LLaDA-8B-shaped layer, MHA 32x128, L = 256 prompt + 256 generated, seeds in one 32-block
    "llada_mha_l512": Workload("llada_mha_l512", 1, 32, 32, 512, 128, 8, "bf16", 256, 288,
                               in_scale=1.0 / 128 ** 0.25),
    # Dream-7B-shaped GQA layer 28/4 x 128, L = 512 + 512, plus vocab-152064 scoring
    "dream_gqa_l1024": Workload("dream_gqa_l1024", 1, 28, 4, 1024, 128, 32, "bf16", 512, 1024,
                                score_N=1024, score_V=152064, score_n_seq=1, score_topk=32,
                                score_spike_frac=0.05, decide_block=32),
    # batched LLaDA-shaped, B=8, L=2048, plus vocab-126464 scoring of 8 x 256 rows
    "llada_b8_l2048": Workload("llada_b8_l2048", 8, 32, 32, 2048, 128, 64, "bf16", 1024, 2048,
                               score_N=8 * 256, score_V=126464, score_n_seq=8, score_topk=64),
    # long-context GQA 32/8 stress, 4 runs of 64 seeds in the second half
    "gqa_l8192_stress": Workload("gqa_l8192_stress", 4, 32, 8, 8192, 128, 256, "bf16", 4096, 8192,
                                 placement="runs"),
}
