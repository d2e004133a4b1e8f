// attn_bf16_sm103.cu - two-view override attention, bf16, tcgen05 tensor cores.
//
// What it computes (Section 5.1, Appendix B): for every query row i of head
// (b, hq), attention over the overridden memory K', V' of KV head
// hq / (Hq / Hkv), scale 1/sqrt(d), no causal mask; for a seed row the
// diagonal entry uses the masked-input pair (k_i, v_i) instead of (k'_i, v'_i)
// (leave-one-out view). The diagonal correction of Appendix B is applied in
// exclusion form: the cached diagonal score of a seed row is set to -inf
// inside the online softmax (only in the one KV tile that holds the diagonal),
// and the masked self term e^{s_self - m} v_i is merged into (m, l, O) in the
// epilogue. Equal to the closed form in exact arithmetic; it never divides by
// r_i, and a seed row never reads k'_i, v'_i while a non-seed row never reads
// the masked buffer.
//
// Structure: a persistent grid of one CTA per SM; a work unit is 256 query
// rows (two Q tiles of 128) of one head, and CTA c takes units c, c + grid,
// c + 2 grid, ... The pipelines below run across unit boundaries, so one
// unit's epilogue overlaps the next unit's loads and first products. When the
// last round of units would leave at least half of the SMs idle, its units
// are split over two CTAs each (one Q tile per CTA, the two softmax
// warpgroups on the two halves of the keys, merged in the epilogue).
//   warps 0-3  softmax + epilogue of Q tile 0 (thread = row)
//   warps 4-7  softmax + epilogue of Q tile 1
//   warp  8    tensor-memory allocation; lane 0 issues tcgen05.mma
//   warp  9    lane 0 issues every TMA copy (Q per unit, K/V through a 2-stage ring,
//              the staged output rows)
//   warp  10   seed routing of the next unit (double-buffered slot table)
//   warp  11   seed self scores q_i . k_i of the next unit; copies its masked value
//              rows v_i into shared memory for the epilogue's merge
// Registers: launched at 168 per thread (12 warps); the producer warpgroup
// gives back down to 136 and the two softmax warpgroups take 184 each
// (setmaxnreg), so the 128-column softmax rows stay in registers without
// spilling.
// Tensor memory (512 columns): S0 | S1 | O0 | O1, 128 fp32 columns each; the
// bf16 probabilities P of tile t overwrite the first 64 columns of S_t and
// feed the P.V product straight from tensor memory.
// Per KV tile j the MMA issue order is PV(0, j-1), S(0, j), PV(1, j-1), S(1, j)
// so that one Q tile's softmax overlaps the other tile's products.
// The running max is updated lazily: O is rescaled only when a row's max grows
// by more than 2^8.
#include <cuda_bf16.h>
#include <math.h>

#include "context.cuh"
#include "kernels.cuh"
#include "ptx.cuh"
#include "route.cuh"
#include "tmap.cuh"

namespace cover {
namespace {

constexpr int kD = 128;
constexpr int kBM = 128;                  // rows per Q tile
constexpr int kBN = 128;                  // keys per KV tile
constexpr int kNQ = 2;                    // Q tiles per CTA
constexpr int kRowsPerCta = kNQ * kBM;
constexpr int kStages = 2;
constexpr int kTileBytes = kBM * kD * 2;  // 32 KB
constexpr int kBoxBytes = kTileBytes / 2; // one 64-column, 128-byte-swizzled box
constexpr int kThreads = 384;
constexpr int kLaunchRegs = 168;          // registers per thread at launch (65536 / 384, rounded to 8)
constexpr int kSoftmaxRegs = 184;         // 2 * 128 * 184 + 128 * 136 == 384 * 168
constexpr int kProducerRegs = 136;
static_assert(2 * 128 * kSoftmaxRegs + 128 * kProducerRegs <= kThreads * kLaunchRegs, "register split");
constexpr int kMmaWarp = 8;
constexpr int kTmaWarp = 9;
constexpr int kRouteWarp = 10;
constexpr int kSeedWarp = 11;
constexpr float kRescaleThreshold = 8.0f;  // log2 units
// A seed row's self term e^{s_self} is merged at the row's reference m as (O + p v) / (l + p),
// p = 2^(s_self - m) (equal to rescaling all three to max(m, s_self)), while s_self <= m + 64
// keeps p and O + p v far inside fp32; above that (m, l, O) is rescaled to s_self instead.
constexpr float kSelfInPlace = 64.0f;      // log2 units
constexpr int kVStageRows = 32;            // masked value rows of a unit staged in shared memory
constexpr int kNotStaged = 255;

// A work unit is 256 query rows (two Q tiles) of one head (b, hq); the grid is
// persistent and CTA c takes units c, c + gridDim.x, ... in order.
struct Unit {
  int mblk, hq, b;
  int split;   // 1: only Q tile ts of the unit, both softmax warpgroups on halves of its KV tiles
  int ts;
};

// Wait limit of every bounded wait of the launch, and a load the TMA thread leaves out on
// purpose: CTA `cta` does not issue the K tile of its ring entry `entry` (its entry-th KV tile
// over all its units). A normal launch has cta = -1 and the one-second limit; the self-test
// entry point plants the missing load with a short limit to drive the kernel's abort path.
struct Fault {
  int cta, entry;
  uint64_t wait_ns;
};

// Division by a launch-invariant divisor d >= 1 through a multiply-high (the round-up method of
// Granlund and Montgomery, "Division by invariant integers using multiplication", PLDI 1994):
// for 0 <= u < 2^31, u / d == (umulhi(u, m) + u) >> s with s = ceil(log2 d) and
// m = floor(2^32 (2^s - d) / d) + 1 (m < 2^32; the sum stays below 2^32). The per-unit index
// arithmetic then runs on the integer pipes instead of the special-function unit, which the
// softmax warps' exponentials keep busy.
struct FastDiv {
  uint32_t d, m, s;
  __device__ __forceinline__ uint32_t div(uint32_t u) const { return (__umulhi(u, m) + u) >> s; }
};

// The persistent grid's unit space: n_reg whole units, n_split split ones, and the divisors
// that decompose a unit index (n_mblk row blocks per head, Hq heads) and map a query head to
// its KV head (Hq / Hkv query heads per KV head).
struct UnitGrid {
  int n_reg, n_split;
  FastDiv mblk, hq, group;
};

// Iteration it of this CTA. Units c, c + grid, ... below n_reg are whole units. When the
// last round would leave at least half of the SMs idle, its n_split units are split instead:
// CTA c < 2 n_split takes Q tile (c & 1) of unit n_reg + c / 2 as one more iteration, and
// its two softmax warpgroups each take half of the KV tiles (merged in the epilogue).
// kSplitAll (the window instance with one Q tile): when n_split > 0 every unit is split, and
// CTA c takes units c, c + grid, ... whole, both warpgroups on the two halves of the keys.
template <bool kSplitAll>
__device__ __forceinline__ bool work_of(int it, const UnitGrid& ug, Unit& w) {
  const int n_reg = ug.n_reg, n_split = ug.n_split;
  const int c = static_cast<int>(blockIdx.x), g = static_cast<int>(gridDim.x);
  int u = c + it * g;
  w.split = 0;
  w.ts = 0;
  if (kSplitAll && n_split > 0) {
    if (u >= n_split) return false;
    w.split = 1;
  } else if (u >= n_reg) {
    if (n_split == 0 || it * g != n_reg || c >= 2 * n_split) return false;
    u = n_reg + (c >> 1);
    w.split = 1;
    w.ts = c & 1;
  }
  const uint32_t t = ug.mblk.div(static_cast<uint32_t>(u));   // (b, hq) index
  const uint32_t b = ug.hq.div(t);
  w.mblk = u - static_cast<int>(t * ug.mblk.d);
  w.hq = static_cast<int>(t - b * ug.hq.d);
  w.b = static_cast<int>(b);
  return true;
}

// first query row of Q tile t of a unit
__device__ __forceinline__ int tile_row0(const Unit& w, int t) {
  return w.mblk * kRowsPerCta + (w.split ? w.ts : t) * kBM;
}

struct AttnSmem {
  uint8_t q[kNQ][kTileBytes];
  uint8_t k[kStages][kTileBytes];
  uint8_t v[kStages][kTileBytes];
  uint64_t bar_q_full[kNQ];
  uint64_t bar_q_empty[kNQ];       // the unit's last Q.K^T product has read Q tile t (tcgen05.commit)
  uint64_t bar_q_read[kNQ];        // the seed-score warp is done reading Q tile t
  uint64_t bar_k_full[kStages];
  uint64_t bar_k_empty[kStages];
  uint64_t bar_v_full[kStages];
  uint64_t bar_v_empty[kStages];
  // a stage whose KV tile ended a unit holds that unit's output until the TMA thread
  // has stored it: K stage for Q tile 0, V stage for Q tile 1
  uint64_t bar_ostage_full[kNQ];   // the tile's four softmax warps have staged the unit's output
  uint64_t bar_s_full[kNQ];
  uint64_t bar_p_full[kNQ];
  uint64_t bar_o_full[kNQ];
  uint64_t bar_slot_full[2];       // routing of a unit written (double-buffered by unit parity)
  uint64_t bar_slot_empty[2];      // a unit's routing and self scores consumed (softmax warps, seed warp)
  uint64_t bar_sself_full[2];      // a unit's seed self scores written
  uint64_t bar_drain;
  uint32_t tmem_base;
  int abort;
  int slot[2][kRowsPerCta];
  Unit unit[2];                    // coordinates of the unit whose routing is in slot[sb]
  float sself[2][kRowsPerCta];     // s_self = q_i . k_i (log2-scaled) of the unit's seed rows
  float split_m[2][kBM];           // a split unit: running max and sum per row of each KV half
  float split_l[2][kBM];
  uint64_t bar_split;              // ... written (all eight softmax warps)
  uint8_t vidx[2][kRowsPerCta];    // a seed row's staged value row, or kNotStaged
  alignas(16) uint8_t vstage[2][kVStageRows][kD * 2];   // masked-input value rows v_i, bf16
};

__device__ __forceinline__ uint32_t col_s(int qt) { return qt * 128u; }
__device__ __forceinline__ uint32_t col_o(int qt) { return 256u + qt * 128u; }

// Sets s[32 * K + i] to -inf where bit i of sel is set (K a compile-time chunk index).
template <int K>
__device__ __forceinline__ void exclude_in_chunk(float* s, uint32_t sel) {
#pragma unroll
  for (int i = 0; i < 32; ++i)
    if ((sel >> i) & 1u) s[32 * K + i] = -INFINITY;
}

__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort, uint64_t limit_ns) {
  const bool ok = mbar_wait(bar, parity, abort, limit_ns);
  return __all_sync(0xffffffffu, ok);
}

__device__ __forceinline__ void raise_abort(AttnSmem& sm, int* status, int site) {
  report_status(status, kStatusTimeout, site);
  sm.abort = 1;
}

// NQ: Q tiles holding query rows (1 for a window of at most 128 rows, else 2).
// kWindow: query row r sits at memory position q0 + r of an Lk-long memory;
// otherwise Lq = Lk and q0 = 0 are compile-time facts.
// kFault: the self-test instance that takes its wait limit and a planted missing load from
// `flt`; the production instances wait up to one second and load every tile.
template <int NQ, bool kWindow, bool kFault>
__global__ void __launch_bounds__(kThreads, 1)
    attn_bf16_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                     const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_o,
                     const __nv_bfloat16* __restrict__ k_seedmask,
                     const __nv_bfloat16* __restrict__ v_seedmask, const int32_t* __restrict__ seed_idx, int n_seeds,
                     int Hq, int Hkv, int Lq_arg, int Lk, int q0_arg, const UnitGrid ug,
                     float scale_log2,
                     __nv_bfloat16* __restrict__ out, float* __restrict__ lse, int* status, const Fault flt) {
  extern __shared__ uint8_t smem_raw[];
  AttnSmem& sm = *reinterpret_cast<AttnSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));

  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;
  const int nkv = (Lk + kBN - 1) / kBN;
  constexpr int nqt = NQ;
  const uint64_t wait_ns = kFault ? flt.wait_ns : kWaitLimitNs;
  const int Lq = kWindow ? Lq_arg : Lk;
  const int q0 = kWindow ? q0_arg : 0;
  const int tail_valid = Lk - (nkv - 1) * kBN;   // valid keys in the last KV tile (1..128)
  // a window of at most 128 rows has one Q tile; with an even number of KV tiles its units are
  // all split, so the second softmax warpgroup takes half of every unit's keys
  constexpr bool kSplitAll = kWindow && NQ == 1;
  const bool all_split = kSplitAll && ug.n_split > 0;

  // ---------------- prologue ----------------
  if (warp == kTmaWarp && lane == 0) {
    for (int t = 0; t < kNQ; ++t) {
      mbar_init(&sm.bar_q_full[t], 1);
      mbar_init(&sm.bar_q_empty[t], 1);
      mbar_init(&sm.bar_q_read[t], 1);
      mbar_init(&sm.bar_s_full[t], 1);
      mbar_init(&sm.bar_p_full[t], kBM);
      mbar_init(&sm.bar_o_full[t], 1);
      mbar_init(&sm.bar_ostage_full[t], 4);
    }
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&sm.bar_k_full[s], 1);
      mbar_init(&sm.bar_k_empty[s], 1);
      mbar_init(&sm.bar_v_full[s], 1);
      mbar_init(&sm.bar_v_empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&sm.bar_slot_full[s], 32);
      mbar_init(&sm.bar_slot_empty[s], 4 * (all_split ? 2 : nqt) + 1);
      mbar_init(&sm.bar_sself_full[s], 1);
    }
    mbar_init(&sm.bar_drain, 1);
    mbar_init(&sm.bar_split, 8);
    sm.abort = 0;
    fence_mbar_init();
    tma_prefetch_desc(&tm_q);
    tma_prefetch_desc(&tm_k);
    tma_prefetch_desc(&tm_v);
    tma_prefetch_desc(&tm_o);
  }
  if (warp == kMmaWarp) {
    tmem_alloc(&sm.tmem_base, 512);
    tmem_relinquish();
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tbase = sm.tmem_base;
  // Launched as a programmatic dependent of the stream's previous kernel: the set-up above
  // overlaps that kernel's tail, and nothing global is read or written before its results are
  // complete and visible here.
  griddep_wait();

  if (warp >= kMmaWarp) {
   setmaxnreg_dec<kProducerRegs>();
   if (warp == kTmaWarp) {
    // ---------------- TMA producer ----------------
    // K/V tiles run through the two-stage ring across unit boundaries (G counts the
    // CTA's KV tiles); Q tile t of a unit is loaded once the previous unit's last
    // Q.K^T product and the tile's seed self scores are done with it.
    if (lane == 0) {
      int G = 0;
      int last_kg = -1, last_vg = -1;         // last KV tiles whose K / V loads were issued
      int last_qit[kNQ] = {-1, -1};           // last units whose Q tiles were issued
      int n_stored = 0;                       // units whose output the thread has stored
      int skipped_kg = -1;                    // the K load left out by a planted fault
      const int fault_entry = kFault && static_cast<int>(blockIdx.x) == flt.cta ? flt.entry : -1;
      bool ok = true;
      // Stores unit n's output of Q tile t from the stage its last KV tile used, once the
      // tile's softmax warps have staged it; returns after the copies have read the stage.
      auto store_unit = [&](int n, int t) {
        Unit wn;
        work_of<kSplitAll>(n, ug, wn);
        if (!mbar_wait(&sm.bar_ostage_full[t], n & 1, &sm.abort, wait_ns)) return false;
        // a split unit's one tile was staged by both warpgroups (one 64-column box each)
        if (wn.split && !mbar_wait(&sm.bar_ostage_full[1], n & 1, &sm.abort, wait_ns)) return false;
        const int sig = (n * nkv + nkv - 1) & 1;
        const uint8_t* stage = t == 0 ? sm.k[sig] : sm.v[sig];
        for (int wq = 0; wq < 4; ++wq) {
          const int wrow = tile_row0(wn, t) + wq * 32;
          if (wrow < Lq) {   // rows at or past Lq fall outside the tensor and are not written
            tma_store_4d(&tm_o, stage + wq * 8192, 0, wrow, wn.hq, wn.b);
            tma_store_4d(&tm_o, stage + wq * 8192 + 4096, 64, wrow, wn.hq, wn.b);
          }
        }
        bulk_commit_group();
        bulk_wait_group_read0();
        return true;
      };
      const int half = nkv >> 1;
      for (int it = 0; ok; ++it) {
        Unit w;
        if (!work_of<kSplitAll>(it, ug, w)) break;
        const int hkv = static_cast<int>(ug.group.div(static_cast<uint32_t>(w.hq)));
        // Q tile t of the unit: wait until the previous unit is done with the buffer
        auto load_q = [&](int t) {
          if (it > 0 && (!mbar_wait(&sm.bar_q_empty[t], (it - 1) & 1, &sm.abort, wait_ns) ||
                         !mbar_wait(&sm.bar_q_read[t], (it - 1) & 1, &sm.abort, wait_ns)))
            return false;
          mbar_arrive_expect_tx(&sm.bar_q_full[t], kTileBytes);
          for (int h = 0; h < 2; ++h)
            tma_load_4d(sm.q[t] + h * kBoxBytes, &tm_q, &sm.bar_q_full[t], 64 * h, tile_row0(w, t), w.hq, w.b);
          last_qit[t] = it;
          return true;
        };
        if (w.split) {
          // Split unit (the CTA's last): ring entry e = 2 s + t holds KV tile t * half + s of
          // warpgroup t's step s. Each K and V tile has one user, so K loads run a step ahead of
          // V loads in the order the products free their stages: V(e) after P.V of step s - 1,
          // K(e + 2) after Q.K^T of step s.
          const int g0 = G;
          auto load_k = [&](int e) {
            const int g = g0 + e, st = g & 1, n = g >> 1;
            if (n >= 1 && !mbar_wait(&sm.bar_k_empty[st], (n - 1) & 1, &sm.abort, wait_ns)) return false;
            // entry 1 reuses the stage of the previous unit's last KV tile, which holds its output
            if (g >= 2 && e == 1 && !store_unit(n_stored, 0)) return false;
            if (kFault && g == fault_entry) {
              skipped_kg = g;
              return true;
            }
            mbar_arrive_expect_tx(&sm.bar_k_full[st], kTileBytes);
            for (int h = 0; h < 2; ++h)
              tma_load_4d(sm.k[st] + h * kBoxBytes, &tm_k, &sm.bar_k_full[st], 64 * h,
                          ((e & 1) * half + (e >> 1)) * kBN, hkv, w.b);
            last_kg = g;
            return true;
          };
          auto load_v = [&](int e) {
            const int g = g0 + e, st = g & 1, n = g >> 1;
            if (n >= 1 && !mbar_wait(&sm.bar_v_empty[st], (n - 1) & 1, &sm.abort, wait_ns)) return false;
            if (g >= 2 && e == 1) {
              if (nqt > 1 && !store_unit(n_stored, 1)) return false;
              ++n_stored;
            }
            mbar_arrive_expect_tx(&sm.bar_v_full[st], kTileBytes);
            for (int h = 0; h < 2; ++h)
              tma_load_4d(sm.v[st] + h * kBoxBytes, &tm_v, &sm.bar_v_full[st], 64 * h,
                          ((e & 1) * half + (e >> 1)) * kBN, hkv, w.b);
            last_vg = g;
            return true;
          };
          ok = load_k(0) && load_q(0) && load_k(1);
          for (int sp = 0; sp < half && ok; ++sp) {
            ok = load_v(2 * sp) && (sp + 1 == half || load_k(2 * sp + 2)) && load_v(2 * sp + 1) &&
                 (sp + 1 == half || load_k(2 * sp + 3));
          }
          G = g0 + nkv;
          continue;
        }
        // K and V tiles of ring entry jj; `staged`: the entry's stage holds the output of the unit
        // whose last KV tile it took two entries ago, which is stored before the stage is reloaded
        // (entry 1 of a unit). With one KV tile per unit (`store_prev`) the previous unit's output
        // is stored instead between this entry's K and V loads: that unit can stage its output
        // without any further load, while the next one cannot before its V tile arrives, so the
        // staging barrier never runs two phases ahead of this thread's wait.
        auto kv_entry = [&](int jj, bool staged, bool first, bool store_prev) {
          const int st = G & 1, n = G >> 1;
          if (n >= 1 && !mbar_wait(&sm.bar_k_empty[st], (n - 1) & 1, &sm.abort, wait_ns)) return false;
          if (staged && !store_unit(n_stored, 0)) return false;
          if (kFault && G == fault_entry) {
            skipped_kg = G;
          } else {
            mbar_arrive_expect_tx(&sm.bar_k_full[st], kTileBytes);
            for (int h = 0; h < 2; ++h)
              tma_load_4d(sm.k[st] + h * kBoxBytes, &tm_k, &sm.bar_k_full[st], 64 * h, jj * kBN, hkv, w.b);
            last_kg = G;
          }
          if (first && !load_q(0)) return false;
          if (store_prev) {
            if (!store_unit(n_stored, 0) || (nqt > 1 && !store_unit(n_stored, 1))) return false;
            ++n_stored;
          }
          if (n >= 1 && !mbar_wait(&sm.bar_v_empty[st], (n - 1) & 1, &sm.abort, wait_ns)) return false;
          if (staged) {
            if (nqt > 1 && !store_unit(n_stored, 1)) return false;
            ++n_stored;
          }
          mbar_arrive_expect_tx(&sm.bar_v_full[st], kTileBytes);
          for (int h = 0; h < 2; ++h)
            tma_load_4d(sm.v[st] + h * kBoxBytes, &tm_v, &sm.bar_v_full[st], 64 * h, jj * kBN, hkv, w.b);
          last_vg = G;
          return true;
        };
        ok = kv_entry(0, false, true, nkv == 1 && G >= 1);
        for (int t = 1; t < nqt && ok; ++t) ok = load_q(t);
        if (!ok) break;
        {
          // the next unit's Q tiles go to L2 now, so their loads at the boundary are short
          Unit wn;
          if (work_of<kSplitAll>(it + 1, ug, wn))
            for (int t = 0; t < (wn.split ? 1 : nqt); ++t)
              for (int h = 0; h < 2; ++h) tma_prefetch_l2_4d(&tm_q, 64 * h, tile_row0(wn, t), wn.hq, wn.b);
        }
        ++G;
        if (nkv > 1) {
          ok = kv_entry(1, G >= 2, false, false);
          ++G;
        }
        for (int jj = 2; jj < nkv && ok; ++jj, ++G) ok = kv_entry(jj, false, false, false);
        if (!ok) break;
      }
      // the units whose stages were not needed again (a split unit stores its one merged tile)
      for (; ok; ++n_stored) {
        Unit wn;
        if (!work_of<kSplitAll>(n_stored, ug, wn)) break;
        for (int t = 0; t < (wn.split ? 1 : nqt) && ok; ++t) ok = store_unit(n_stored, t);
      }
      bulk_wait_group0();
      if (!ok) {
        raise_abort(sm, status, 10);
        // let every copy already issued land before the CTA's shared memory is released
        for (int t = 0; t < nqt; ++t)
          if (last_qit[t] >= 0) mbar_wait(&sm.bar_q_full[t], last_qit[t] & 1, nullptr, wait_ns);
        for (int g = max(0, last_kg - 1); g <= last_kg; ++g)
          if (!kFault || g != skipped_kg) mbar_wait(&sm.bar_k_full[g & 1], (g >> 1) & 1, nullptr, wait_ns);
        for (int g = max(0, last_vg - 1); g <= last_vg; ++g)
          mbar_wait(&sm.bar_v_full[g & 1], (g >> 1) & 1, nullptr, wait_ns);
      }
    }
   } else if (warp == kRouteWarp) {
    // ---------------- seed routing ----------------
    // slot[r] of a unit = lowest seed slot naming the unit's row r, written one unit
    // ahead of the softmax warps into a double buffer.
    for (int it = 0;; ++it) {
      Unit w;
      if (!work_of<kSplitAll>(it, ug, w)) break;
      const int sb = it & 1;
      if (it >= 2 && !warp_wait(&sm.bar_slot_empty[sb], ((it >> 1) - 1) & 1, &sm.abort, wait_ns)) {
        if (lane == 0 && !sm.abort) raise_abort(sm, status, 40);
        break;
      }
      if (lane == 0) sm.unit[sb] = w;
      // slot[t * 128 + r] belongs to query row tile_row0(w, t) + r, at memory position q0 + that
      const int rows = w.split ? kBM : kRowsPerCta;
      route_clear(sm.slot[sb], rows, lane, 32);
      __syncwarp();
      route_scan(sm.slot[sb], seed_idx + static_cast<size_t>(w.b) * n_seeds, n_seeds, q0 + tile_row0(w, 0), rows,
                 Lk, lane, 32);
      if (w.split) {
        // both warpgroups of a split unit work on the same rows
        __syncwarp();
        for (int r = lane; r < kBM; r += 32) sm.slot[sb][kBM + r] = sm.slot[sb][r];
      }
      mbar_arrive(&sm.bar_slot_full[sb]);
    }
   } else if (warp == kSeedWarp) {
    // ---------------- seed self scores ----------------
    // For each seed row of a unit: s_self = q_i . k_i with the masked-input key (log2-scaled),
    // one row per warp pass (lane l takes dimensions 4l .. 4l+3), and the masked-input value
    // row v_i copied into shared memory for the epilogue's merge (the unit's first 32 seed
    // rows; the epilogue reads any others from global memory). Runs one unit ahead of the
    // softmax warps, off their critical path.
    for (int it = 0;; ++it) {
      Unit wk;
      if (!work_of<kSplitAll>(it, ug, wk)) break;
      const int sb = it & 1;
      if (!warp_wait(&sm.bar_slot_full[sb], (it >> 1) & 1, &sm.abort, wait_ns)) {
        if (lane == 0 && !sm.abort) raise_abort(sm, status, 50);
        break;
      }
      const Unit w = sm.unit[sb];
      const size_t mbase = (static_cast<size_t>(w.b) * Hkv + ug.group.div(static_cast<uint32_t>(w.hq))) * n_seeds;
      int n_staged = 0;
      bool ok = true;
      for (int t = 0; t < (w.split ? 1 : nqt); ++t) {
        if (!warp_wait(&sm.bar_q_full[t], it & 1, &sm.abort, wait_ns)) {
          ok = false;
          break;
        }
        // byte offset of this lane's 8 bytes inside a row of the 128-byte-swizzled Q tile
        const int h = lane >> 4, c8 = (lane & 15) >> 1, half = (lane & 1) * 8;
        for (int rc = 0; rc < kBM; rc += 32) {
          const int rr = rc + lane;
          const int sl = sm.slot[sb][t * kBM + rr];
          const bool seed_row = sl != kNoSlot && tile_row0(w, t) + rr < Lq;
          uint32_t pending = __ballot_sync(0xffffffffu, seed_row);
          while (pending != 0u) {
            // up to four seed rows at a time, their loads in flight together
            int row[4];
            uint2 kv[4], vv[4];
#pragma unroll
            for (int g = 0; g < 4; ++g) {
              row[g] = -1;
              if (pending != 0u) {
                const int src = __ffs(pending) - 1;
                pending &= pending - 1u;
                row[g] = rc + src;
                const size_t mrow = (mbase + __shfl_sync(0xffffffffu, sl, src)) * kD;
                kv[g] = __ldg(reinterpret_cast<const uint2*>(k_seedmask + mrow) + lane);
                vv[g] = __ldg(reinterpret_cast<const uint2*>(v_seedmask + mrow) + lane);
              }
            }
#pragma unroll
            for (int g = 0; g < 4; ++g) {
              if (row[g] < 0) continue;
              const uint2 qv = *reinterpret_cast<const uint2*>(sm.q[t] + h * kBoxBytes + row[g] * 128 +
                                                               ((c8 ^ (row[g] & 7)) * 16) + half);
              const __nv_bfloat162* qp = reinterpret_cast<const __nv_bfloat162*>(&qv);
              const __nv_bfloat162* kp = reinterpret_cast<const __nv_bfloat162*>(&kv[g]);
              const float2 q01 = __bfloat1622float2(qp[0]), q23 = __bfloat1622float2(qp[1]);
              const float2 k01 = __bfloat1622float2(kp[0]), k23 = __bfloat1622float2(kp[1]);
              float dot = fmaf(q01.x, k01.x, q01.y * k01.y) + fmaf(q23.x, k23.x, q23.y * k23.y);
#pragma unroll
              for (int o = 16; o >= 1; o >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, o);
              // the first kVStageRows seed rows of the unit keep v_i in shared memory
              const int vi = n_staged < kVStageRows ? n_staged++ : kNotStaged;
              if (vi != kNotStaged) reinterpret_cast<uint2*>(sm.vstage[sb][vi])[lane] = vv[g];
              if (lane == 0) {
                sm.sself[sb][t * kBM + row[g]] = dot * scale_log2;
                sm.vidx[sb][t * kBM + row[g]] = static_cast<uint8_t>(vi);
              }
            }
          }
        }
        // this warp no longer reads Q tile t of the unit
        __syncwarp();
        if (lane == 0) mbar_arrive(&sm.bar_q_read[t]);
      }
      if (!ok) {
        if (lane == 0 && !sm.abort) raise_abort(sm, status, 51);
        break;
      }
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&sm.bar_sself_full[sb]);
        mbar_arrive(&sm.bar_slot_empty[sb]);   // done reading the unit's routing
      }
    }
   } else if (warp == kMmaWarp) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      constexpr uint32_t id_qk = idesc_bf16_f32(kBM, kBN, false, false);
      constexpr uint32_t id_pv = idesc_bf16_f32(kBM, kD, false, true);
      // descriptors of stage / tile 0; the others are one tile (kTileBytes >> 4 units) further
      constexpr uint64_t kTileDesc = kTileBytes >> 4;
      const uint64_t dq0 = sdesc_sw128(smem_u32(sm.q[0]), 16, 1024);
      const uint64_t dk0 = sdesc_sw128(smem_u32(sm.k[0]), 16, 1024);
      const uint64_t dv0 = sdesc_sw128(smem_u32(sm.v[0]), kBoxBytes, 1024);
      // O_t (+)= P_t . V(stage); P from tensor memory, V MN-major from shared memory
      auto issue_pv = [&](int t, int vst, bool acc) {
#pragma unroll
        for (int ks = 0; ks < kBN / 16; ++ks)
          umma_ts(tbase + col_o(t), tbase + col_s(t) + 8 * ks,
                  dv0 + vst * kTileDesc + static_cast<uint64_t>((ks * 2048) >> 4), id_pv,
                  (acc || ks > 0) ? 1u : 0u);
      };
      // One stream of steps over the CTA's units. Inside a unit, KV tile j issues
      // PV(0, j-1), S(0, j), PV(1, j-1), S(1, j); at a unit boundary the previous
      // unit's last products PV(0), PV(1) go first, then the new unit's S(0, 0),
      // S(1, 0), so one unit's epilogue overlaps the next unit's first products.
      // Each wait sits right after a group of products has been queued.
      // S_t = Q(qbuf) . K(stage)^T, both K-major with 128-byte swizzle
      auto issue_s = [&](int t, int qbuf, int kst) {
#pragma unroll
        for (int ks = 0; ks < kD / 16; ++ks) {
          const uint64_t off = static_cast<uint64_t>(((ks >> 2) * kBoxBytes + (ks & 3) * 32) >> 4);
          umma_ss(tbase + col_s(t), dq0 + qbuf * kTileDesc + off, dk0 + kst * kTileDesc + off, id_qk,
                  ks > 0 ? 1u : 0u);
        }
      };
      int G = 0;
      bool ok = true;
      for (int it = 0; ok; ++it) {
        if (it > 0 && !all_split) {
          const int pst = (G - 1) & 1;
          for (int t = 0; t < nqt; ++t) {
            ok = mbar_wait(&sm.bar_p_full[t], (G - 1) & 1, &sm.abort, wait_ns);
            if (!ok) break;
            tc_fence_after_sync();
            issue_pv(t, pst, nkv > 1);
            umma_commit(&sm.bar_o_full[t]);
          }
          if (!ok) break;
          umma_commit(&sm.bar_v_empty[pst]);
        }
        Unit w;
        if (!work_of<kSplitAll>(it, ug, w)) break;
        if (w.split) {
          // Split unit (always the CTA's last): tile t takes KV tiles t * half + s from ring
          // entries G + 2 s + t, both against the Q tile in buffer 0. Every K and V tile has
          // one user, so each product frees its own stage; a V tile is waited for right before
          // its P.V product, since the TMA thread loads it only after the previous step's P.V.
          const int half = nkv >> 1, g0 = G;
          // P barriers complete once per warpgroup step: nkv per earlier whole unit, half per
          // earlier split unit
          const int pb = all_split ? it * half : g0;
          for (int s = 0; s < half && ok; ++s) {
            for (int t = 0; t < 2; ++t) {
              const int ring = g0 + 2 * s + t;
              if (s > 0) {
                ok = mbar_wait(&sm.bar_p_full[t], (pb + s - 1) & 1, &sm.abort, wait_ns);
                if (ok) ok = mbar_wait(&sm.bar_v_full[(ring - 2) & 1], ((ring - 2) >> 1) & 1, &sm.abort, wait_ns);
                if (!ok) break;
                tc_fence_after_sync();
                issue_pv(t, (ring - 2) & 1, s > 1);
                umma_commit(&sm.bar_v_empty[(ring - 2) & 1]);
              }
              ok = mbar_wait(&sm.bar_k_full[ring & 1], (ring >> 1) & 1, &sm.abort, wait_ns);
              if (!ok) break;
              tc_fence_after_sync();
              if (s == 0 && t == 0) {
                ok = mbar_wait(&sm.bar_q_full[0], it & 1, &sm.abort, wait_ns);
                if (!ok) break;
                tc_fence_after_sync();
              }
              issue_s(t, 0, ring & 1);
              umma_commit(&sm.bar_s_full[t]);
              umma_commit(&sm.bar_k_empty[ring & 1]);
              if (s == half - 1 && t == 1) umma_commit(&sm.bar_q_empty[0]);
            }
          }
          // the last P.V products of both halves
          for (int t = 0; t < 2 && ok; ++t) {
            const int ring = g0 + 2 * (half - 1) + t;
            ok = mbar_wait(&sm.bar_p_full[t], (pb + half - 1) & 1, &sm.abort, wait_ns);
            if (ok) ok = mbar_wait(&sm.bar_v_full[ring & 1], (ring >> 1) & 1, &sm.abort, wait_ns);
            if (!ok) break;
            tc_fence_after_sync();
            issue_pv(t, ring & 1, half > 1);
            umma_commit(&sm.bar_o_full[t]);
            umma_commit(&sm.bar_v_empty[ring & 1]);
          }
          G = g0 + nkv;
          if (all_split) continue;
          break;
        }
        {
          // step 0: the unit's Q tiles, no P.V yet
          const int st = G & 1;
          for (int t = 0; t < nqt && ok; ++t) {
            if (t == 0) {
              ok = mbar_wait(&sm.bar_k_full[st], (G >> 1) & 1, &sm.abort, wait_ns);
              if (!ok) break;
              tc_fence_after_sync();
            }
            ok = mbar_wait(&sm.bar_q_full[t], it & 1, &sm.abort, wait_ns);
            if (!ok) break;
            tc_fence_after_sync();
            issue_s(t, t, st);
            umma_commit(&sm.bar_s_full[t]);
            if (t == nqt - 1) umma_commit(&sm.bar_k_empty[st]);
            if (nkv == 1) umma_commit(&sm.bar_q_empty[t]);
            if (t == 0) {
              ok = mbar_wait(&sm.bar_v_full[st], (G >> 1) & 1, &sm.abort, wait_ns);
              if (!ok) break;
            }
          }
          ++G;
        }
        // steps 1 .. nkv - 1; the last one also releases the unit's Q tiles
        auto kv_step = [&](int j, bool last) {
          const int st = G & 1, pst = (G - 1) & 1;
          for (int t = 0; t < nqt; ++t) {
            if (!mbar_wait(&sm.bar_p_full[t], (G - 1) & 1, &sm.abort, wait_ns)) return false;
            tc_fence_after_sync();
            issue_pv(t, pst, j > 1);
            if (t == nqt - 1) umma_commit(&sm.bar_v_empty[pst]);
            if (t == 0) {
              if (!mbar_wait(&sm.bar_k_full[st], (G >> 1) & 1, &sm.abort, wait_ns)) return false;
              tc_fence_after_sync();
            }
            issue_s(t, t, st);
            umma_commit(&sm.bar_s_full[t]);
            if (t == nqt - 1) umma_commit(&sm.bar_k_empty[st]);
            if (last) umma_commit(&sm.bar_q_empty[t]);
            // V(j) feeds the P.V products of the next step; it was issued long before
            if (t == 0 && !mbar_wait(&sm.bar_v_full[st], (G >> 1) & 1, &sm.abort, wait_ns)) return false;
          }
          return true;
        };
        for (int j = 1; j + 1 < nkv && ok; ++j, ++G) ok = kv_step(j, false);
        if (ok && nkv > 1) {
          ok = kv_step(nkv - 1, true);
          ++G;
        }
      }
      if (!ok) raise_abort(sm, status, 20);
      // all tensor-core work of this CTA must finish before tensor memory is released
      umma_commit(&sm.bar_drain);
      mbar_wait(&sm.bar_drain, 0, nullptr, wait_ns);
    }
   }
  } else {
    setmaxnreg_inc<kSoftmaxRegs>();
    // ---------------- softmax (warps 0-7) ----------------
    const int qt = warp >> 2;
    // with a single Q tile the second tile's warps sit this launch out, unless its units are split
    if (qt < nqt || all_split) {
      const int r = tid & (kBM - 1);
      const uint32_t trow = tbase + (static_cast<uint32_t>((warp & 3) * 32) << 16);
      const uint32_t s_addr = trow + col_s(qt);
      const uint32_t o_addr = trow + col_o(qt);
      bool ok = true;
      // Only what the KV loop needs stays live across it; the unit's coordinates are
      // recomputed for the epilogue.
      for (int it = 0; ok; ++it) {
        {
          Unit wk;
          if (!work_of<kSplitAll>(it, ug, wk)) break;
        }
        const int sb = it & 1;
        int my_slot;
        int diag_j, diag_c;
        // KV tiles of this warpgroup: all of them, or for a split unit half of them, starting
        // at tile jbase; the tail and diagonal tiles are kept relative to jbase
        int steps, tail_j;
        {
          ok = warp_wait(&sm.bar_slot_full[sb], (it >> 1) & 1, &sm.abort, wait_ns);
          if (!ok) break;
          const Unit w = sm.unit[sb];
          const int grow = tile_row0(w, qt) + r;
          const int jbase = w.split ? qt * (nkv >> 1) : 0;
          steps = w.split ? nkv >> 1 : nkv;
          tail_j = tail_valid < kBN ? nkv - 1 - jbase : -1;   // -1: no ragged tile
          my_slot = sm.slot[sb][qt * kBM + r];
          if (grow >= Lq) my_slot = kNoSlot;
          // the diagonal of a square launch is column r of KV tile row0 / 128 of the row's Q tile;
          // in a window a warp's 32 consecutive rows meet their diagonals in at most two KV tiles
          diag_j = (kWindow ? (q0 + grow) / kBN : tile_row0(w, qt) / kBN) - jbase;
          diag_c = kWindow ? (q0 + grow) % kBN : r;
        }
        const bool is_seed = my_slot != kNoSlot;
        const bool warp_seed = __any_sync(0xffffffffu, is_seed);
        const int dj_lo = kWindow ? __shfl_sync(0xffffffffu, diag_j, 0) : diag_j;
        const int dj_hi = kWindow ? __shfl_sync(0xffffffffu, diag_j, 31) : diag_j;
        const int g0 = it * nkv;   // the CTA's KV steps before this unit
        // this warpgroup's steps before this unit (half a unit's KV tiles each when all are split)
        const int sbase = all_split ? it * (nkv >> 1) : g0;
        float m_run = -INFINITY, l_run = 0.0f;

        for (int j = 0; j < steps && ok; ++j) {
          ok = warp_wait(&sm.bar_s_full[qt], (sbase + j) & 1, &sm.abort, wait_ns);
          if (!ok) break;
          tc_fence_after_sync();
          uint32_t raw[4][32];
#pragma unroll
          for (int c = 0; c < 4; ++c) tmem_ld32(s_addr + 32 * c, raw[c]);
#pragma unroll
          for (int c = 0; c < 4; ++c) tmem_ld_wait(raw[c]);
          float* s = reinterpret_cast<float*>(&raw[0][0]);
          if (j == tail_j) {
            const int valid = Lk - (nkv - 1) * kBN;
#pragma unroll
            for (int c = 0; c < kBN; ++c)
              if (c >= valid) s[c] = -INFINITY;
          }
          if (warp_seed && (j == dj_lo || j == dj_hi)) {
            // exclusion of the cached diagonal term of a seed row
            const bool here = is_seed && j == diag_j;
            if (!kWindow) {
              // square launch: row r's diagonal is column r, element `lane` of 32-column chunk warp & 3
              const uint32_t sel = here ? (1u << lane) : 0u;
              switch (warp & 3) {
                case 0: exclude_in_chunk<0>(s, sel); break;
                case 1: exclude_in_chunk<1>(s, sel); break;
                case 2: exclude_in_chunk<2>(s, sel); break;
                default: exclude_in_chunk<3>(s, sel); break;
              }
            } else {
#pragma unroll
              for (int c = 0; c < kBN; ++c)
                if (here && c == diag_c) s[c] = -INFINITY;
            }
          }
          // row maximum: four independent 3-input max chains
          float mx0 = s[0], mx1 = s[1], mx2 = s[2], mx3 = s[3];
#pragma unroll
          for (int c = 4; c + 8 <= kBN; c += 8) {
            mx0 = fmax3(mx0, s[c], s[c + 1]);
            mx1 = fmax3(mx1, s[c + 2], s[c + 3]);
            mx2 = fmax3(mx2, s[c + 4], s[c + 5]);
            mx3 = fmax3(mx3, s[c + 6], s[c + 7]);
          }
          mx0 = fmax3(mx0, s[kBN - 4], s[kBN - 3]);
          mx1 = fmax3(mx1, s[kBN - 2], s[kBN - 1]);
          const float m_tile = fmax3(mx0, mx1, fmaxf(mx2, mx3)) * scale_log2;
          float alpha = 1.0f;
          bool rescaled = false;
          if (m_tile > m_run + kRescaleThreshold) {
            alpha = (m_run == -INFINITY) ? 0.0f : ex2_approx(m_run - m_tile);
            m_run = m_tile;
            rescaled = true;
          }
          const float m_use = (m_run == -INFINITY) ? 0.0f : m_run;
          // p = 2^(s * scale - m) on pairs; four independent partial row sums
          const uint64_t scale2 = f2_pack(scale_log2, scale_log2);
          const uint64_t negm2 = f2_pack(-m_use, -m_use);
          uint64_t acc2[4] = {0, 0, 0, 0};
          uint32_t packed[64];
#pragma unroll
          for (int c = 0; c < 64; ++c) {
            float t0, t1;
            f2_unpack(f2_fma(f2_pack(s[2 * c], s[2 * c + 1]), scale2, negm2), t0, t1);
            const float p0 = ex2_approx(t0);
            const float p1 = ex2_approx(t1);
            packed[c] = pack_bf16x2(p0, p1);
            acc2[c & 3] = f2_add(acc2[c & 3], f2_pack(p0, p1));
          }
          float rs[8];
          f2_unpack(f2_add(acc2[0], acc2[1]), rs[0], rs[1]);
          f2_unpack(f2_add(acc2[2], acc2[3]), rs[2], rs[3]);
          const float rowsum = (rs[0] + rs[1]) + (rs[2] + rs[3]);
          l_run = l_run * alpha + rowsum;
          tmem_st32(s_addr, *reinterpret_cast<uint32_t(*)[32]>(&packed[0]));
          tmem_st32(s_addr + 32, *reinterpret_cast<uint32_t(*)[32]>(&packed[32]));
          if (j > 0 && __any_sync(0xffffffffu, rescaled)) {
            // O holds the products of tiles < j (complete: they were issued before S(j))
#pragma unroll 1
            for (int c = 0; c < 4; ++c) {
              uint32_t o[32];
              tmem_ld32(o_addr + 32 * c, o);
              tmem_ld_wait(o);
#pragma unroll
              for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
              tmem_st32(o_addr + 32 * c, o);
            }
          }
          tmem_st_wait();
          tc_fence_before_sync();
          mbar_arrive(&sm.bar_p_full[qt]);
        }
        if (ok) ok = warp_wait(&sm.bar_o_full[qt], it & 1, &sm.abort, wait_ns);
        if (!ok) break;
        const Unit w = sm.unit[sb];
        if (w.split) {
          // Split unit: the two warpgroups hold (m, l, O) of the two KV halves of the same rows.
          // They swap (m, l) through shared memory; then each combines O = O0 2^(m0 - m) +
          // O1 2^(m1 - m) for 64 of the 128 columns straight from tensor memory, merges a seed
          // row's self term there, and stages its 64-column box of the rows.
          sm.split_m[qt][r] = m_run;
          sm.split_l[qt][r] = l_run;
          __syncwarp();
          if (lane == 0) mbar_arrive(&sm.bar_split);
          ok = warp_wait(&sm.bar_o_full[qt ^ 1], it & 1, &sm.abort, wait_ns);
          if (ok) ok = warp_wait(&sm.bar_split, all_split ? (it & 1) : 0, &sm.abort, wait_ns);
          if (ok && warp_seed) ok = warp_wait(&sm.bar_sself_full[sb], (it >> 1) & 1, &sm.abort, wait_ns);
          if (!ok) break;
          tc_fence_after_sync();
          const float m0 = sm.split_m[0][r], m1 = sm.split_m[1][r];
          float m = fmaxf(m0, m1);
          const float a0 = (m0 == -INFINITY) ? 0.0f : ex2_approx(m0 - m);
          const float a1 = (m1 == -INFINITY) ? 0.0f : ex2_approx(m1 - m);
          float l = sm.split_l[0][r] * a0 + sm.split_l[1][r] * a1;
          const int cb = qt * 64;   // this warpgroup's columns
          float oh[64];
#pragma unroll
          for (int c = 0; c < 2; ++c) {
            uint32_t x0[32], x1[32];
            tmem_ld32(trow + col_o(0) + cb + 32 * c, x0);
            tmem_ld32(trow + col_o(1) + cb + 32 * c, x1);
            tmem_ld_wait(x0);
            tmem_ld_wait(x1);
#pragma unroll
            for (int e = 0; e < 32; ++e) oh[32 * c + e] = __uint_as_float(x0[e]) * a0 + __uint_as_float(x1[e]) * a1;
          }
          const int grow = tile_row0(w, 0) + r;
          if (is_seed) {
            const float s_self = sm.sself[sb][r];
            const int vi = sm.vidx[sb][r];
            const size_t mrow = ((static_cast<size_t>(w.b) * Hkv + ug.group.div(static_cast<uint32_t>(w.hq))) * n_seeds + my_slot) * kD;
            const uint4* vmv = (vi != kNotStaged ? reinterpret_cast<const uint4*>(sm.vstage[sb][vi])
                                                 : reinterpret_cast<const uint4*>(v_seedmask + mrow)) + cb / 8;
            if (m != -INFINITY && s_self <= m + kSelfInPlace) {
              // (O + p v) / (l + p) with p = 2^(s_self - m): one multiply-add per element
              const float pself = ex2_approx(s_self - m);
              l += pself;
#pragma unroll
              for (int ch = 0; ch < 8; ++ch) {
                const uint4 vv = vmv[ch];
                const __nv_bfloat162* vp = reinterpret_cast<const __nv_bfloat162*>(&vv);
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                  const float2 vf = __bfloat1622float2(vp[e]);
                  oh[ch * 8 + 2 * e] = fmaf(pself, vf.x, oh[ch * 8 + 2 * e]);
                  oh[ch * 8 + 2 * e + 1] = fmaf(pself, vf.y, oh[ch * 8 + 2 * e + 1]);
                }
              }
            } else {
              // a self term far above the row's other scores: rescale (m, l, O) to it
              const float m2 = fmaxf(m, s_self);
              const float a = (m == -INFINITY) ? 0.0f : ex2_approx(m - m2);
              const float pself = ex2_approx(s_self - m2);
              l = l * a + pself;
#pragma unroll
              for (int ch = 0; ch < 8; ++ch) {
                const uint4 vv = vmv[ch];
                const __nv_bfloat162* vp = reinterpret_cast<const __nv_bfloat162*>(&vv);
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                  const float2 vf = __bfloat1622float2(vp[e]);
                  oh[ch * 8 + 2 * e] = oh[ch * 8 + 2 * e] * a + pself * vf.x;
                  oh[ch * 8 + 2 * e + 1] = oh[ch * 8 + 2 * e + 1] * a + pself * vf.y;
                }
              }
              m = m2;
            }
          }
          const int sig = (g0 + nkv - 1) & 1;
          uint8_t* stage = sm.k[sig] + (warp & 3) * (2 * 4096) + qt * 4096;
          const float inv = 1.0f / l;
#pragma unroll
          for (int ch = 0; ch < 8; ++ch) {
            uint4 v;
            v.x = pack_bf16x2(oh[ch * 8 + 0] * inv, oh[ch * 8 + 1] * inv);
            v.y = pack_bf16x2(oh[ch * 8 + 2] * inv, oh[ch * 8 + 3] * inv);
            v.z = pack_bf16x2(oh[ch * 8 + 4] * inv, oh[ch * 8 + 5] * inv);
            v.w = pack_bf16x2(oh[ch * 8 + 6] * inv, oh[ch * 8 + 7] * inv);
            *reinterpret_cast<uint4*>(stage + lane * 128 + ((ch ^ (lane & 7)) << 4)) = v;
          }
          if (qt == 0 && lse != nullptr && grow < Lq)
            lse[(static_cast<size_t>(w.b) * Hq + w.hq) * Lq + grow] = (m + log2f(l)) * 0.6931471805599453f;
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            mbar_arrive(&sm.bar_ostage_full[qt]);
            mbar_arrive(&sm.bar_slot_empty[sb]);
          }
          continue;
        }
        // ---------------- epilogue of the unit ----------------
        // O is read into registers before this warpgroup's next P is published, so the
        // next unit's first P.V product cannot overwrite it early.
        tc_fence_after_sync();
        uint32_t oraw[4][32];
#pragma unroll
        for (int c = 0; c < 4; ++c) tmem_ld32(o_addr + 32 * c, oraw[c]);
#pragma unroll
        for (int c = 0; c < 4; ++c) tmem_ld_wait(oraw[c]);
        float* o = reinterpret_cast<float*>(&oraw[0][0]);
        const int grow = tile_row0(w, qt) + r;
        if (warp_seed) {
          ok = warp_wait(&sm.bar_sself_full[sb], (it >> 1) & 1, &sm.abort, wait_ns);
          if (!ok) break;
        }
        if (is_seed) {
          // merge the masked-input self term (k_i, v_i) of this seed row
          const float s_self = sm.sself[sb][qt * kBM + r];
          const int vi = sm.vidx[sb][qt * kBM + r];
          const size_t mrow = ((static_cast<size_t>(w.b) * Hkv + ug.group.div(static_cast<uint32_t>(w.hq))) * n_seeds + my_slot) * kD;
          // generic loads: shared memory when warp 11 staged the row, else global memory
          const uint4* vmv = vi != kNotStaged ? reinterpret_cast<const uint4*>(sm.vstage[sb][vi])
                                              : reinterpret_cast<const uint4*>(v_seedmask + mrow);
          if (m_run != -INFINITY && s_self <= m_run + kSelfInPlace) {
            // (O + p v) / (l + p) with p = 2^(s_self - m): one multiply-add per element
            const float pself = ex2_approx(s_self - m_run);
            l_run += pself;
#pragma unroll
            for (int ch = 0; ch < 16; ++ch) {
              const uint4 vv = vmv[ch];
              const __nv_bfloat162* vp = reinterpret_cast<const __nv_bfloat162*>(&vv);
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const float2 vf = __bfloat1622float2(vp[e]);
                o[ch * 8 + 2 * e] = fmaf(pself, vf.x, o[ch * 8 + 2 * e]);
                o[ch * 8 + 2 * e + 1] = fmaf(pself, vf.y, o[ch * 8 + 2 * e + 1]);
              }
            }
          } else {
            // a self term far above the row's other scores: rescale (m, l, O) to it
            const float m2 = fmaxf(m_run, s_self);
            const float a = (m_run == -INFINITY) ? 0.0f : ex2_approx(m_run - m2);
            const float pself = ex2_approx(s_self - m2);
            l_run = l_run * a + pself;
#pragma unroll
            for (int ch = 0; ch < 16; ++ch) {
              const uint4 vv = vmv[ch];
              const __nv_bfloat162* vp = reinterpret_cast<const __nv_bfloat162*>(&vv);
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const float2 vf = __bfloat1622float2(vp[e]);
                o[ch * 8 + 2 * e] = o[ch * 8 + 2 * e] * a + pself * vf.x;
                o[ch * 8 + 2 * e + 1] = o[ch * 8 + 2 * e + 1] * a + pself * vf.y;
              }
            }
            m_run = m2;
          }
        }
        // Output: the warp's 32 rows x 128 columns are staged in the shared-memory stage of
        // the unit's last KV tile (K stage for Q tile 0, V stage for Q tile 1: both finished
        // with once O is complete) as two 128-byte-swizzled boxes of 64 columns; the TMA
        // thread writes them out, so the global writes are full lines instead of one 16-byte
        // piece per row, and this warp goes on to the next unit at once.
        {
          const int sig = (g0 + nkv - 1) & 1;
          uint8_t* stage = (qt == 0 ? sm.k[sig] : sm.v[sig]) + (warp & 3) * (2 * 4096);
          const float inv = 1.0f / l_run;
#pragma unroll
          for (int ch = 0; ch < 16; ++ch) {
            uint4 v;
            v.x = pack_bf16x2(o[ch * 8 + 0] * inv, o[ch * 8 + 1] * inv);
            v.y = pack_bf16x2(o[ch * 8 + 2] * inv, o[ch * 8 + 3] * inv);
            v.z = pack_bf16x2(o[ch * 8 + 4] * inv, o[ch * 8 + 5] * inv);
            v.w = pack_bf16x2(o[ch * 8 + 6] * inv, o[ch * 8 + 7] * inv);
            *reinterpret_cast<uint4*>(stage + (ch >> 3) * 4096 + lane * 128 + (((ch & 7) ^ (lane & 7)) << 4)) = v;
          }
          if (lse != nullptr && grow < Lq)
            lse[(static_cast<size_t>(w.b) * Hq + w.hq) * Lq + grow] = (m_run + log2f(l_run)) * 0.6931471805599453f;
          // the staged rows go to the TMA thread, which stores them before it reloads the stage
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) mbar_arrive(&sm.bar_ostage_full[qt]);
        }
        // the unit's routing and self scores are consumed
        __syncwarp();
        if (lane == 0) mbar_arrive(&sm.bar_slot_empty[sb]);
      }
      if (!ok && !sm.abort) raise_abort(sm, status, 30 + qt);
    }
  }

  // ---------------- teardown ----------------
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  // the next kernel of the stream may be scheduled once every CTA is here (it waits for this
  // grid's completion before it reads anything); a trigger right after the prologue measured
  // slower, by 1 % at L=2048 and 1 us a launch at L=512
  griddep_launch_dependents();
  if (warp == kMmaWarp) tmem_dealloc(tbase, 512);
}

// Multiplier and shift of FastDiv for the divisor d >= 1.
FastDiv make_fastdiv(uint32_t d) {
  uint32_t s = 0;
  while ((uint64_t{1} << s) < d) ++s;
  const uint64_t m = ((uint64_t{1} << 32) * ((uint64_t{1} << s) - d)) / d + 1;
  return FastDiv{d, static_cast<uint32_t>(m), s};
}

}  // namespace

int launch_attn_bf16_sm103(const AttnArgs& a, int* status, cudaStream_t stream) {
  CUtensorMap tq, tk, tv, to;
  if (!make_bf16_map_4d(&tq, a.q, kD, a.Lq, a.Hq, a.B, kBM) ||
      !make_bf16_map_4d(&to, a.out, kD, a.Lq, a.Hq, a.B, 32) ||
      !make_bf16_map_4d(&tk, a.k_cached, kD, a.L, a.Hkv, a.B, kBN) ||
      !make_bf16_map_4d(&tv, a.v_cached, kD, a.L, a.Hkv, a.B, kBN))
    return -3;
  const int n_mblk = (a.Lq + kRowsPerCta - 1) / kRowsPerCta;
  const long long n_units = static_cast<long long>(n_mblk) * a.Hq * a.B;
  const int nkv = (a.L + kBN - 1) / kBN;
  const size_t smem = sizeof(AttnSmem) + 1024;
  // per context: the SM count, and the kernels' shared-memory limit set (a function attribute
  // holds only in the context it was set in)
  static ContextCache<int> setup;
  int n_sm = 0;
  const int rc = setup.get(&n_sm, [&](int& v) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v < 1)
      return -3;
    for (auto fn : {attn_bf16_kernel<2, false, false>, attn_bf16_kernel<1, true, false>,
                    attn_bf16_kernel<2, true, false>, attn_bf16_kernel<2, false, true>,
                    attn_bf16_kernel<1, true, true>, attn_bf16_kernel<2, true, true>}) {
      if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem)) != cudaSuccess)
        return -3;
      // the register split inside the kernel assumes exactly kLaunchRegs per thread at launch;
      // any other count could leave setmaxnreg.inc waiting, so refuse to launch
      cudaFuncAttributes fa;
      if (cudaFuncGetAttributes(&fa, fn) != cudaSuccess || fa.numRegs != kLaunchRegs) return -2;
    }
    return 0;
  });
  if (rc != 0) return rc;
  // unit indices advance by the grid size past the last unit: keep them inside int
  if (n_units > 0x7fffffffLL - n_sm) return -2;
  // persistent grid: one CTA per SM (1 CTA/SM fits), each looping over units
  // The last round of units would leave at least half of the SMs idle: split its units
  // (square launches with an even number of KV tiles), two CTAs per unit.
  const long long rounds = n_units / n_sm, n_last = n_units % n_sm;
  const bool window = a.Lq != a.L || a.q0 != 0;
  // A window of at most 128 rows has one Q tile per unit; with an even number of KV tiles every
  // unit is split inside its CTA (both softmax warpgroups on the two halves of the keys).
  const bool split_all = window && a.Lq <= kBM && nkv >= 2 && nkv % 2 == 0;
  const int n_split = split_all ? static_cast<int>(n_units)
                      : (!window && nkv >= 2 && nkv % 2 == 0 && n_last > 0 && 2 * n_last <= n_sm)
                          ? static_cast<int>(n_last) : 0;
  const int n_reg = split_all ? 0 : static_cast<int>(n_units) - n_split;
  const long long grid = split_all ? (rounds > 0 ? n_sm : n_units)
                                   : (rounds > 0 ? n_sm : (n_split > 0 ? 2 * n_split : n_units));
  const float scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(kD));
  const UnitGrid ug{n_reg, n_split, make_fastdiv(static_cast<uint32_t>(n_mblk)),
                    make_fastdiv(static_cast<uint32_t>(a.Hq)), make_fastdiv(static_cast<uint32_t>(a.Hq / a.Hkv))};
  const bool fault = a.fault_cta >= 0 || a.wait_ns > 0;
  auto kernel = !window       ? (fault ? attn_bf16_kernel<2, false, true> : attn_bf16_kernel<2, false, false>)
                : a.Lq <= kBM ? (fault ? attn_bf16_kernel<1, true, true> : attn_bf16_kernel<1, true, false>)
                              : (fault ? attn_bf16_kernel<2, true, true> : attn_bf16_kernel<2, true, false>);
  // programmatic dependent launch: the prologue overlaps the previous kernel's tail
  cudaLaunchAttribute attr[1];
  const cudaLaunchConfig_t cfg = pdl_config(dim3(static_cast<unsigned>(grid)), dim3(kThreads), smem, stream, attr);
  const cudaError_t e = cudaLaunchKernelEx(
      &cfg, kernel, tq, tk, tv, to, static_cast<const __nv_bfloat16*>(a.k_seedmask),
      static_cast<const __nv_bfloat16*>(a.v_seedmask), a.seed_idx, a.n_seeds, a.Hq, a.Hkv, a.Lq, a.L, a.q0, ug,
      scale_log2, static_cast<__nv_bfloat16*>(a.out), a.lse, status,
      Fault{a.fault_cta, a.fault_entry, a.wait_ns > 0 ? a.wait_ns : kWaitLimitNs});
  return e == cudaSuccess && cudaGetLastError() == cudaSuccess ? 0 : -3;
}

}  // namespace cover
