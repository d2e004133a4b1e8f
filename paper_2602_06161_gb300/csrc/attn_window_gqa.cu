// attn_window_gqa.cu - prefix-cache window attention for grouped-query heads: the query heads
// that share a KV head are packed into common Q tiles, and the keys are split over the CTAs of
// a thread-block cluster, which combine their partial results through distributed shared memory.
//
// What it computes: cover_attn_fwd_prefix (Section 6.6, the prefix-cache variant of the override
// attention of Section 5.1 and Appendix B). Query row r of head (b, hq) sits at memory position
// q0 + r and attends over all Lk positions of the overridden memory K', V' of KV head hq / G
// (G = Hq / Hkv query heads per KV head), scale 1/sqrt(d), no causal mask. For a seed row the
// diagonal entry uses the masked-input pair (k_i, v_i): its cached diagonal score is excluded
// (-inf) and the masked self term e^{s_self} v_i is merged into the combined (m, l, O), the
// exclusion form of Appendix B's diagonal correction, as in the square kernel.
//
// Why a kernel of its own: a short window (the active block of a few dozen rows) of a GQA model
// leaves the square kernel one mostly empty Q tile per query head, and each query head walks its
// KV head's whole memory alone, so a launch is a few dozen CTAs each running a long chain of KV
// steps. Here
//   - packed row p = g * Lq + r (0 <= g < G) of KV head (b, hkv) is query row r of head
//     hq = hkv * G + g. Those heads are consecutive in q ([B, Hq, Lq, D]), so the packed rows
//     are one contiguous run of the [B * Hq * Lq, D] view starting at row (b * Hq + hkv * G) * Lq,
//     and one K/V tile serves all G heads at once;
//   - CTA (ks, t, hkv, b) takes Q tile t (packed rows 128 t .. 128 t + 127) against the KV tiles
//     [ks T, min(nkv, ks T + T)) of key split ks; the nsplit CTAs of one (t, hkv, b) form a
//     cluster, so a CTA's chain is T KV steps instead of nkv;
//   - packed row R of the tile is combined by the cluster's CTA R % nsplit: each CTA stages its
//     split (m, l, O) of every row by owner (O as fp16 scaled by the row's largest magnitude)
//     and sends each owner its block with one bulk copy into the owner's shared memory, which
//     completes on the owner's mbarrier; the owner combines from its own shared memory. Reading
//     the partials through distributed shared memory row by row cost several microseconds more
//     on the Dream window (1 x 28 heads / 4 KV heads, 32 rows over 1024 keys); a few large bulk
//     copies of 4 KB each did not measurably add to the launch.
// Roles (160 threads):
//   warps 0-3  routing of the window's positions, the self scores of the seed rows this CTA
//              combines, the softmax of the CTA's KV steps (thread = packed row), the exchange,
//              then the combine of packed rows ks, ks + nsplit, ...
//   warp  4    tensor-memory allocation; lane 0 issues the TMA loads and the tcgen05.mma
// Tensor memory: S (128 fp32 columns; the bf16 probabilities P overwrite its first 64 columns
// and feed P.V from tensor memory) | O (128 fp32 columns). Per KV step j the MMA thread issues
// P.V(j) and then S(j + 1), so the tensor pipe reads P(j) before S(j + 1) overwrites it.
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <math.h>

#include "cluster.cuh"
#include "context.cuh"
#include "kernels.cuh"
#include "ptx.cuh"
#include "route.cuh"
#include "tmap.cuh"

namespace cover {
namespace {

constexpr int kD = 128;
constexpr int kBM = 128;                   // packed rows per Q tile
constexpr int kBN = 128;                   // keys per KV tile
constexpr int kTileBytes = kBM * kD * 2;   // 32 KB
constexpr int kBoxBytes = kTileBytes / 2;  // one 64-column, 128-byte-swizzled box
constexpr int kThreads = 160;
constexpr int kMmaWarp = 4;
constexpr int kMaxSplit = 8;               // portable cluster size
constexpr float kRescaleThreshold = 8.0f;  // log2 units

constexpr int kPartRowBytes = kD * 2;      // a partial row: 128 fp16
constexpr int kStatOff = 36 * 1024;        // (m, l, s) records after at most (128 + 7) partial rows
constexpr int kRecvBytes = kStatOff + (kBM + kMaxSplit) * 16;
static_assert((kBM + kMaxSplit) * kPartRowBytes <= kStatOff && kRecvBytes <= 2 * kTileBytes,
              "the K ring stages the partial blocks and records of every owner");

struct WinSmem {
  uint8_t q[kTileBytes];
  // K and V rings of two stages. Once the CTA's products are complete, the K ring stages its
  // split partials by owner: nsplit blocks of rpo rows of 128 fp16 (part_off), then the
  // (m, l, s) records from kStatOff.
  uint8_t k[2][kTileBytes];
  uint8_t v[2][kTileBytes];
  // the blocks of the rows this CTA combines, one per split, in the same layout
  alignas(16) uint8_t recv[kRecvBytes];
  uint64_t bar_q_full;
  uint64_t bar_k_full[2];
  uint64_t bar_k_empty[2];
  uint64_t bar_v_full[2];
  uint64_t bar_v_empty[2];
  uint64_t bar_s_full;
  uint64_t bar_p_full;
  uint64_t bar_o_full;
  uint64_t bar_drain;
  uint64_t bar_staged;             // the 128 softmax threads have staged their rows' partials
  uint64_t bar_recv;               // the cluster's nsplit blocks of this CTA's rows have arrived
  uint32_t tmem_base;
  int abort;
  float sself[kBM];                // s_self (log2-scaled) of the seed rows this CTA combines
  int slot[kMaxWindowGqaRows];     // seed slot of window position q0 + r, or kNoSlot
};

__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort, uint64_t limit_ns) {
  const bool ok = mbar_wait(bar, parity, abort, limit_ns);
  return __all_sync(0xffffffffu, ok);
}

__device__ __forceinline__ void named_sync_softmax() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

// Byte offset of 16-byte chunk c (eight fp16 columns) of entry qr in a partial block of owner
// `owner`; the chunks are swizzled by (qr + owner) & 7, so the staging writes of eight
// consecutive rows (thread = row, owners R % nsplit) and the reads of one entry (lane = half a
// chunk) spread over all banks.
__device__ __forceinline__ uint32_t part_off(int qr, int owner, int c) {
  return static_cast<uint32_t>(qr * kPartRowBytes + ((c ^ ((qr + owner) & 7)) << 4));
}

// 1/x and log2(x) by the PTX approximations (relative error about 2^-23, absolute error of the
// logarithm about 2^-22 for normal x): one instruction each instead of the correctly rounded
// sequences, whose dependent steps sit on the combine's chain with one warp per scheduler. The
// output is rounded to bf16 (2^-9) and lse is held to 1e-3.
__device__ __forceinline__ float rcp_approx(float x) {
  float y;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float lg2_approx(float x) {
  float y;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack_f16x2(float lo, float hi) {
  const __half2 h = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&h);
}

// kFault: the self-test instance, in which CTA fault_cta leaves out the K load of its first KV
// tile and every bounded wait gives up after wait_ns; the production instance loads every tile.
template <bool kFault>
__global__ void __launch_bounds__(kThreads, 1)
    attn_window_gqa_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                           const __grid_constant__ CUtensorMap tm_v, const __nv_bfloat16* __restrict__ q,
                           const __nv_bfloat16* __restrict__ k_seedmask,
                           const __nv_bfloat16* __restrict__ v_seedmask, const int32_t* __restrict__ seed_idx,
                           int n_seeds, int Hq, int Hkv, int G, int Lq, int Lk, int q0, int n_qt, int nsplit, int T,
                           float scale_log2, __nv_bfloat16* __restrict__ out, float* __restrict__ lse, int* status,
                           uint64_t wait_ns, int fault_cta) {
  extern __shared__ uint8_t smem_raw[];
  WinSmem& sm = *reinterpret_cast<WinSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));

  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;
  // CTA (ks, t, hkv, b); the cluster spans the nsplit key splits of one (t, hkv, b)
  const int ks = static_cast<int>(cluster_ctarank());
  int rest = static_cast<int>(blockIdx.x) / nsplit;
  const int qt = rest % n_qt;
  rest /= n_qt;
  const int hkv = rest % Hkv;
  const int b = rest / Hkv;
  const int nkv = (Lk + kBN - 1) / kBN;
  const int j0 = ks * T;                              // the split's first KV tile
  const int nt = min(nkv, j0 + T) - j0;               // its KV tiles (>= 1)
  const int n_packed = G * Lq;
  const int rowbase = (b * Hq + hkv * G) * Lq;        // packed row 0 in the [B * Hq * Lq, D] view
  const int tail_valid = Lk - (nkv - 1) * kBN;        // valid keys of the memory's last tile
  const int rpo = (kBM + nsplit - 1) / nsplit;        // rows of the tile each CTA combines, at most
  uint8_t* const stage = reinterpret_cast<uint8_t*>(&sm.k);   // the K ring as one 64 KB region
  uint8_t* const recv = sm.recv;

  // ---------------- prologue ----------------
  if (warp == kMmaWarp) {
    if (lane == 0) {
      mbar_init(&sm.bar_q_full, 1);
      for (int s = 0; s < 2; ++s) {
        mbar_init(&sm.bar_k_full[s], 1);
        mbar_init(&sm.bar_k_empty[s], 1);
        mbar_init(&sm.bar_v_full[s], 1);
        mbar_init(&sm.bar_v_empty[s], 1);
      }
      mbar_init(&sm.bar_s_full, 1);
      mbar_init(&sm.bar_p_full, kBM);
      mbar_init(&sm.bar_o_full, 1);
      mbar_init(&sm.bar_drain, 1);
      mbar_init(&sm.bar_staged, kBM);
      mbar_init(&sm.bar_recv, 1);
      sm.abort = 0;
      fence_mbar_init();
      // the blocks of every split: copies of the other CTAs complete bytes on it
      mbar_arrive_expect_tx(&sm.bar_recv, static_cast<uint32_t>(nsplit * rpo * (kPartRowBytes + 16)));
      tma_prefetch_desc(&tm_q);
      tma_prefetch_desc(&tm_k);
      tma_prefetch_desc(&tm_v);
    }
    __syncwarp();
    tmem_alloc(&sm.tmem_base, 256);
    tmem_relinquish();
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  // every CTA of the cluster has initialised its barriers before any copy of another CTA signals
  // them (waited for right before this CTA's first copy, long after every CTA has arrived)
  cluster_arrive();
  const uint32_t tbase = sm.tmem_base;
  // launched as a programmatic dependent of the stream's previous kernel: nothing global is
  // read or written before that kernel's results are complete and visible here
  griddep_wait();
  // The next kernel of the stream may be scheduled now: this grid leaves most SMs free, so its
  // prologue runs beside this launch (it waits for this grid's completion before it reads
  // anything). Measured 0.3 us a call faster than a trigger at the end on the Dream window.
  griddep_launch_dependents();

  if (warp == kMmaWarp) {
    // ---------------- TMA loads and tensor-core products ----------------
    if (lane == 0) {
      int n_loaded = 0;   // KV tiles whose loads were issued
      const bool planted = kFault && static_cast<int>(blockIdx.x) == fault_cta;   // K(0) left out
      auto load_kv = [&](int j) {
        const int st = j & 1;
        if (!(planted && j == 0)) {
          mbar_arrive_expect_tx(&sm.bar_k_full[st], kTileBytes);
          for (int h = 0; h < 2; ++h)
            tma_load_4d(sm.k[st] + h * kBoxBytes, &tm_k, &sm.bar_k_full[st], 64 * h, (j0 + j) * kBN, hkv, b);
        }
        mbar_arrive_expect_tx(&sm.bar_v_full[st], kTileBytes);
        for (int h = 0; h < 2; ++h)
          tma_load_4d(sm.v[st] + h * kBoxBytes, &tm_v, &sm.bar_v_full[st], 64 * h, (j0 + j) * kBN, hkv, b);
        n_loaded = j + 1;
      };
      mbar_arrive_expect_tx(&sm.bar_q_full, kTileBytes);
      for (int h = 0; h < 2; ++h)
        tma_load_4d(sm.q + h * kBoxBytes, &tm_q, &sm.bar_q_full, 64 * h, rowbase + qt * kBM, 0, 0);
      load_kv(0);
      if (nt > 1) load_kv(1);

      constexpr uint32_t id_qk = idesc_bf16_f32(kBM, kBN, false, false);
      constexpr uint32_t id_pv = idesc_bf16_f32(kBM, kD, false, true);
      constexpr uint64_t kTileDesc = kTileBytes >> 4;
      const uint64_t dq = sdesc_sw128(smem_u32(sm.q), 16, 1024);
      const uint64_t dk0 = sdesc_sw128(smem_u32(sm.k[0]), 16, 1024);
      const uint64_t dv0 = sdesc_sw128(smem_u32(sm.v[0]), kBoxBytes, 1024);
      // S = Q . K(stage)^T, both K-major with 128-byte swizzle
      auto issue_s = [&](int st) {
#pragma unroll
        for (int kk = 0; kk < kD / 16; ++kk) {
          const uint64_t off = static_cast<uint64_t>(((kk >> 2) * kBoxBytes + (kk & 3) * 32) >> 4);
          umma_ss(tbase, dq + off, dk0 + st * kTileDesc + off, id_qk, kk > 0 ? 1u : 0u);
        }
      };
      // O (+)= P . V(stage); P from tensor memory, V MN-major from shared memory
      auto issue_pv = [&](int st, bool acc) {
#pragma unroll
        for (int kk = 0; kk < kBN / 16; ++kk)
          umma_ts(tbase + 128, tbase + 8 * kk, dv0 + st * kTileDesc + static_cast<uint64_t>((kk * 2048) >> 4), id_pv,
                  (acc || kk > 0) ? 1u : 0u);
      };
      bool ok = mbar_wait(&sm.bar_q_full, 0, &sm.abort, wait_ns) && mbar_wait(&sm.bar_k_full[0], 0, &sm.abort, wait_ns);
      if (ok) {
        tc_fence_after_sync();
        issue_s(0);
        umma_commit(&sm.bar_s_full);
        umma_commit(&sm.bar_k_empty[0]);
      }
      for (int j = 0; j < nt && ok; ++j) {
        const int st = j & 1;
        ok = mbar_wait(&sm.bar_p_full, j & 1, &sm.abort, wait_ns) &&
             mbar_wait(&sm.bar_v_full[st], (j >> 1) & 1, &sm.abort, wait_ns);
        if (!ok) break;
        tc_fence_after_sync();
        issue_pv(st, j > 0);
        umma_commit(&sm.bar_v_empty[st]);
        if (j + 1 < nt) {
          ok = mbar_wait(&sm.bar_k_full[st ^ 1], ((j + 1) >> 1) & 1, &sm.abort, wait_ns);
          if (!ok) break;
          tc_fence_after_sync();
          issue_s(st ^ 1);
          umma_commit(&sm.bar_s_full);
          umma_commit(&sm.bar_k_empty[st ^ 1]);
        }
        if (j + 2 < nt) {
          // the stage of tile j is free once S(j) and P.V(j) have read it
          ok = mbar_wait(&sm.bar_k_empty[st], (j >> 1) & 1, &sm.abort, wait_ns) &&
               mbar_wait(&sm.bar_v_empty[st], (j >> 1) & 1, &sm.abort, wait_ns);
          if (!ok) break;
          load_kv(j + 2);
        }
      }
      if (ok) {
        umma_commit(&sm.bar_o_full);
      } else {
        report_status(status, kStatusTimeout, 60);
        sm.abort = 1;
        // let every copy already issued land before the CTA's shared memory is released
        mbar_wait(&sm.bar_q_full, 0, nullptr, wait_ns);
        for (int j = max(0, n_loaded - 2); j < n_loaded; ++j) {
          if (!(planted && j == 0)) mbar_wait(&sm.bar_k_full[j & 1], (j >> 1) & 1, nullptr, wait_ns);
          mbar_wait(&sm.bar_v_full[j & 1], (j >> 1) & 1, nullptr, wait_ns);
        }
      }
      // all tensor-core work of this CTA completes before tensor memory is released
      umma_commit(&sm.bar_drain);
      mbar_wait(&sm.bar_drain, 0, nullptr, wait_ns);
    }
    __syncwarp();
  } else {
    // ---------------- routing, self scores, softmax (warps 0-3) ----------------
    const int R = tid;                                // packed row of the Q tile
    const int P = qt * kBM + R;
    const bool valid = P < n_packed;
    const int r = valid ? P - (P / Lq) * Lq : 0;      // its query row (position q0 + r)
    // slot[r] = lowest seed slot naming position q0 + r, else kNoSlot
    route_clear(sm.slot, Lq, tid, kBM);
    named_sync_softmax();
    route_scan(sm.slot, seed_idx + static_cast<size_t>(b) * n_seeds, n_seeds, q0, Lq, Lk, tid, kBM);
    named_sync_softmax();
    const size_t mbase = (static_cast<size_t>(b) * Hkv + hkv) * n_seeds;   // masked rows of this KV head
    const bool is_seed = valid && sm.slot[r] != kNoSlot;
    const bool warp_seed = __any_sync(0xffffffffu, is_seed);
    const int pos = q0 + r;
    const int diag_j = pos / kBN - j0;                // the diagonal's KV step in this split
    const int diag_c = pos - (pos / kBN) * kBN;
    const int tail_j = tail_valid < kBN ? nkv - 1 - j0 : -1;
    const uint32_t trow = tbase + (static_cast<uint32_t>(warp * 32) << 16);
    float m_run = -INFINITY, l_run = 0.0f;
    bool ok = true;
    for (int j = 0; j < nt && ok; ++j) {
      ok = warp_wait(&sm.bar_s_full, j & 1, &sm.abort, wait_ns);
      if (!ok) break;
      tc_fence_after_sync();
      uint32_t raw[4][32];
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld32(trow + 32 * c, raw[c]);
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld_wait(raw[c]);
      float* s = reinterpret_cast<float*>(&raw[0][0]);
      if (j == tail_j) {
#pragma unroll
        for (int c = 0; c < kBN; ++c)
          if (c >= tail_valid) s[c] = -INFINITY;
      }
      if (warp_seed && __any_sync(0xffffffffu, is_seed && j == diag_j)) {
        // exclusion of the cached diagonal term of a seed row
        const bool here = is_seed && j == diag_j;
#pragma unroll
        for (int c = 0; c < kBN; ++c)
          if (here && c == diag_c) s[c] = -INFINITY;
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
      float rs[4];
      f2_unpack(f2_add(acc2[0], acc2[1]), rs[0], rs[1]);
      f2_unpack(f2_add(acc2[2], acc2[3]), rs[2], rs[3]);
      l_run = l_run * alpha + ((rs[0] + rs[1]) + (rs[2] + rs[3]));
      tmem_st32(trow, *reinterpret_cast<uint32_t(*)[32]>(&packed[0]));
      tmem_st32(trow + 32, *reinterpret_cast<uint32_t(*)[32]>(&packed[32]));
      if (j > 0 && __any_sync(0xffffffffu, rescaled)) {
        // O holds the products of steps < j (complete: the S(j) commit came after them)
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
          uint32_t o[32];
          tmem_ld32(trow + 128 + 32 * c, o);
          tmem_ld_wait(o);
#pragma unroll
          for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
          tmem_st32(trow + 128 + 32 * c, o);
        }
      }
      tmem_st_wait();
      tc_fence_before_sync();
      mbar_arrive(&sm.bar_p_full);
    }
    if (ok) ok = warp_wait(&sm.bar_o_full, 0, &sm.abort, wait_ns);
    if (!ok && !sm.abort) {
      report_status(status, kStatusTimeout, 61);
      sm.abort = 1;
    }
    // This split's (m, l, O) of the row, staged in this CTA's K ring (free: every product of the
    // CTA is complete) in the block of the row's owner R % nsplit, as entry qr = R / nsplit. O goes
    // as fp16 of O / s with s the row's largest magnitude (|O / s| <= 1, error at most 2^-12 s
    // per element, below the bf16 rounding of the output), (m, l, s) as one 16-byte record.
    if (ok) {
      tc_fence_after_sync();
      uint32_t o[4][32];
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld32(trow + 128 + 32 * c, o[c]);
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld_wait(o[c]);
      // largest magnitude of the row: four independent max chains
      float am[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
      for (int c = 0; c < 4; ++c)
#pragma unroll
        for (int e = 0; e < 32; e += 2)
          am[c] = fmax3(am[c], fabsf(__uint_as_float(o[c][e])), fabsf(__uint_as_float(o[c][e + 1])));
      const float amax = fmaxf(fmaxf(am[0], am[1]), fmaxf(am[2], am[3]));
      const float sc = amax > 0.0f ? amax : 1.0f;
      const float inv = rcp_approx(sc);
      const int owner = R % nsplit, qr = R / nsplit;
      uint8_t* blk = stage + owner * rpo * kPartRowBytes;
#pragma unroll
      for (int c = 0; c < 4; ++c)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          uint32_t h[4];
#pragma unroll
          for (int x = 0; x < 4; ++x)
            h[x] = pack_f16x2(__uint_as_float(o[c][8 * e + 2 * x]) * inv, __uint_as_float(o[c][8 * e + 2 * x + 1]) * inv);
          *reinterpret_cast<uint4*>(blk + part_off(qr, owner, 4 * c + e)) = make_uint4(h[0], h[1], h[2], h[3]);
        }
      reinterpret_cast<float4*>(stage + kStatOff)[owner * rpo + qr] = make_float4(m_run, l_run, sc, 0.0f);
    }
    // the bulk copies read the staged blocks through the async proxy; warp 4 issues them (and
    // releases tensor memory) once all 128 rows are staged
    fence_proxy_async_smem();
    tc_fence_before_sync();
    mbar_arrive(&sm.bar_staged);
    // While the copies run: s_self = q_i . k_i (log2-scaled) of the seed rows among packed
    // rows ks, ks + nsplit, ... that this warp combines; lane l takes dimensions 4l .. 4l+3, up to
    // four rows in flight
    for (int i0 = warp; ks + i0 * nsplit < kBM; i0 += 16) {
      int row[4];
      uint2 qv[4], kv[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int Rc = ks + (i0 + 4 * u) * nsplit;
        const int Pc = qt * kBM + Rc;
        row[u] = -1;
        if (Rc < kBM && Pc < n_packed) {
          const int s = sm.slot[Pc - (Pc / Lq) * Lq];
          if (s != kNoSlot) {
            row[u] = Rc;
            qv[u] = __ldg(reinterpret_cast<const uint2*>(q + (static_cast<size_t>(rowbase) + Pc) * kD) + lane);
            kv[u] = __ldg(reinterpret_cast<const uint2*>(k_seedmask + (mbase + s) * kD) + lane);
          }
        }
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        if (row[u] < 0) continue;
        const __nv_bfloat162* qp = reinterpret_cast<const __nv_bfloat162*>(&qv[u]);
        const __nv_bfloat162* kp = reinterpret_cast<const __nv_bfloat162*>(&kv[u]);
        const float2 q01 = __bfloat1622float2(qp[0]), q23 = __bfloat1622float2(qp[1]);
        const float2 k01 = __bfloat1622float2(kp[0]), k23 = __bfloat1622float2(kp[1]);
        float dot = fmaf(q01.x, k01.x, q01.y * k01.y) + fmaf(q23.x, k23.x, q23.y * k23.y);
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, o);
        if (lane == 0) sm.sself[row[u]] = dot * scale_log2;
      }
    }
    cluster_wait();   // the prologue's arrival

    // ---------------- combine ----------------
    // the nsplit blocks of this CTA's rows (copied by warp 4 of every CTA of the cluster)
    const bool received = mbar_wait(&sm.bar_recv, 0, nullptr, wait_ns);
    if (!received && !sm.abort) {
      report_status(status, kStatusTimeout, 62);
      sm.abort = 1;
    }
    // Packed row Rc = qr nsplit + ks of the tile is entry qr of every split's block. Warp `warp`
    // takes qr = warp, warp + 4, ..., two rows at a time whose chains interleave; every lane
    // reads the nsplit (m, l, s) records itself (broadcast reads, no shuffles) and holds columns
    // 4 lane .. 4 lane + 3 of the row.
    for (int qa = warp; qa * nsplit + ks < kBM; qa += 8) {
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int qr = qa + 4 * h;
        const int Rc = qr * nsplit + ks;
        const int Pc = qt * kBM + Rc;
        if (Rc >= kBM || Pc >= n_packed) continue;
        float4 st[kMaxSplit];   // (m_j, l_j, s_j) of split j
        uint2 oj[kMaxSplit];    // four fp16 columns of split j's O / s
#pragma unroll
        for (int j = 0; j < kMaxSplit; ++j) {
          if (j < nsplit) {
            st[j] = reinterpret_cast<const float4*>(recv + kStatOff)[j * rpo + qr];
            oj[j] = *reinterpret_cast<const uint2*>(recv + j * rpo * kPartRowBytes + part_off(qr, ks, lane >> 1) +
                                                    ((lane & 1) << 3));
          } else {
            st[j] = make_float4(-INFINITY, 0.0f, 0.0f, 0.0f);
            oj[j] = make_uint2(0u, 0u);
          }
        }
        const int sl = sm.slot[Pc - (Pc / Lq) * Lq];
        const bool seed = sl != kNoSlot;
        uint2 vv = make_uint2(0u, 0u);
        if (seed) vv = __ldg(reinterpret_cast<const uint2*>(v_seedmask + (mbase + sl) * kD) + lane);
        const float s_self = seed ? sm.sself[Rc] : -INFINITY;
        float m = s_self;
#pragma unroll
        for (int j = 0; j < kMaxSplit; ++j) m = fmaxf(m, st[j].x);
        float l = 0.0f;
        float4 acc = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
#pragma unroll
        for (int j = 0; j < kMaxSplit; ++j) {
          const float w = (st[j].x == -INFINITY) ? 0.0f : ex2_approx(st[j].x - m);
          l = fmaf(w, st[j].y, l);
          const float ws = w * st[j].z;
          const float2 a01 = __half22float2(*reinterpret_cast<const __half2*>(&oj[j].x));
          const float2 a23 = __half22float2(*reinterpret_cast<const __half2*>(&oj[j].y));
          acc.x = fmaf(a01.x, ws, acc.x);
          acc.y = fmaf(a01.y, ws, acc.y);
          acc.z = fmaf(a23.x, ws, acc.z);
          acc.w = fmaf(a23.y, ws, acc.w);
        }
        if (seed) {
          // the masked self term of a seed row
          const __nv_bfloat162* vp = reinterpret_cast<const __nv_bfloat162*>(&vv);
          const float2 v01 = __bfloat1622float2(vp[0]), v23 = __bfloat1622float2(vp[1]);
          const float pself = ex2_approx(s_self - m);
          l += pself;
          acc.x = fmaf(pself, v01.x, acc.x);
          acc.y = fmaf(pself, v01.y, acc.y);
          acc.z = fmaf(pself, v23.x, acc.z);
          acc.w = fmaf(pself, v23.y, acc.w);
        }
        const float inv = rcp_approx(l);
        const size_t orow = static_cast<size_t>(rowbase) + Pc;
        uint2 ov;
        ov.x = pack_bf16x2(acc.x * inv, acc.y * inv);
        ov.y = pack_bf16x2(acc.z * inv, acc.w * inv);
        reinterpret_cast<uint2*>(out + orow * kD)[lane] = ov;
        if (lane == 0 && lse != nullptr) lse[orow] = (m + lg2_approx(l)) * 0.6931471805599453f;
      }
    }
    // No CTA leaves while a copy out of its shared memory may still run: an owner arrives once
    // it has received all of its blocks. An owner whose receive wait gave up (a sender of its
    // cluster timed out before its copies) may not have them yet; but every CTA issues its
    // copies before it arrives here, so after the barrier they are all in flight, and that owner
    // waits for them to land before its shared memory is released.
    cluster_sync();
    if (!received) mbar_wait(&sm.bar_recv, 0, nullptr, wait_ns);
  }
  if (warp == kMmaWarp) {
    cluster_wait();   // the prologue's arrival: every CTA of the cluster has its barriers set up
    if (lane == 0) {
      if (!mbar_wait(&sm.bar_staged, 0, nullptr, wait_ns)) {
        report_status(status, kStatusTimeout, 63);
        sm.abort = 1;
      }
      tc_fence_after_sync();
      // the staged blocks to their owners: block o of this CTA becomes block ks of CTA o. Issued
      // whatever happened before, so that every owner's receive barrier completes.
      for (int o = 0; o < nsplit; ++o) {
        const uint32_t bar = cluster_map(smem_u32(&sm.bar_recv), o);
        bulk_copy_cluster(cluster_map(smem_u32(recv + ks * rpo * kPartRowBytes), o),
                          smem_u32(stage + o * rpo * kPartRowBytes), rpo * kPartRowBytes, bar);
        bulk_copy_cluster(cluster_map(smem_u32(recv + kStatOff + ks * rpo * 16), o),
                          smem_u32(stage + kStatOff + o * rpo * 16), rpo * 16, bar);
      }
    }
    __syncwarp();
    tc_fence_after_sync();
    tmem_dealloc(tbase, 256);
    cluster_sync();   // see the softmax warps' last barrier
  }
}

}  // namespace

namespace {

// Launch set-up of one context: the kernel's shared-memory limit set, the SM count, and how many
// clusters of each size (1 .. kMaxSplit CTAs of this kernel) can be resident at once.
struct WinSetup {
  int n_sm;
  int max_clusters[kMaxSplit + 1];
};

// Shape of a packed launch: T KV tiles per CTA, nsplit CTAs per cluster, n_qt Q tiles per KV head.
struct WinShape {
  int G, nkv, T, nsplit, n_qt;
  long long clusters;
};

WinShape win_shape(const AttnArgs& a) {
  WinShape w;
  w.G = a.Hq / a.Hkv;
  w.nkv = (a.L + kBN - 1) / kBN;
  w.T = (w.nkv + kMaxSplit - 1) / kMaxSplit;
  w.nsplit = (w.nkv + w.T - 1) / w.T;   // every split has at least one KV tile
  w.n_qt = (w.G * a.Lq + kBM - 1) / kBM;
  w.clusters = static_cast<long long>(w.n_qt) * a.Hkv * a.B;
  return w;
}

int win_setup(WinSetup* out, size_t smem) {
  static ContextCache<WinSetup> setup;
  return setup.get(out, [&](WinSetup& v) {
    int dev = 0;
    if (cudaFuncSetAttribute(attn_window_gqa_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(smem)) != cudaSuccess ||
        cudaFuncSetAttribute(attn_window_gqa_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(smem)) != cudaSuccess ||
        cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&v.n_sm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return -3;
    v.max_clusters[0] = 0;
    for (int cs = 1; cs <= kMaxSplit; ++cs) {
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3(static_cast<unsigned>(cs));
      cfg.blockDim = dim3(kThreads);
      cfg.dynamicSmemBytes = smem;
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = static_cast<unsigned>(cs);
      attr[0].val.clusterDim.y = 1;
      attr[0].val.clusterDim.z = 1;
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      int n = 0;
      if (cudaOccupancyMaxActiveClusters(&n, attn_window_gqa_kernel<false>, &cfg) != cudaSuccess) {
        cudaGetLastError();
        n = 0;
      }
      v.max_clusters[cs] = n;
    }
    return 0;
  });
}

// Predicted microseconds of one call on each kernel, fitted to calls measured back to back on
// GB300 (Dream-shaped windows of 16 to 128 rows over 1024 keys, batches of 1 to 8, memories of
// 2048 to 8192 keys; within 15 % on every shape measured): a packed CTA takes about 7 us plus
// 1.5 us per KV step, and the clusters beyond those resident at once run in further waves; the
// square kernel's window path takes about 5 us plus 1.7 us per KV step of one softmax warpgroup
// for each round of its persistent grid.
double packed_us(const WinShape& w, const WinSetup& su) {
  const long long waves = (w.clusters + su.max_clusters[w.nsplit] - 1) / su.max_clusters[w.nsplit];
  return static_cast<double>(waves) * (7.0 + 1.5 * w.T);
}

double square_us(const AttnArgs& a, const WinShape& w, const WinSetup& su) {
  const long long units = static_cast<long long>((a.Lq + 255) / 256) * a.Hq * a.B;
  const long long rounds = (units + su.n_sm - 1) / su.n_sm;
  // a window of at most 128 rows with an even number of KV tiles splits each unit's keys over
  // the two softmax warpgroups
  const int steps = (a.Lq <= kBM && w.nkv % 2 == 0) ? w.nkv / 2 : w.nkv;
  return 5.0 + static_cast<double>(rounds) * steps * 1.7;
}

bool packed_supported(const AttnArgs& a) {
  const bool window = a.Lq != a.L || a.q0 != 0;
  const int G = a.Hkv > 0 ? a.Hq / a.Hkv : 0;
  const int nkv = (a.L + kBN - 1) / kBN;
  return window && a.D == kD && G >= 2 && a.Lq <= kMaxWindowGqaRows &&
         G * a.Lq <= kMaxWindowGqaPacked && nkv <= kMaxSplit * kMaxWindowGqaSteps &&
         static_cast<long long>(a.B) * a.Hq * a.Lq + kBM < 0x7fffffffLL;
}

}  // namespace

WindowChoice window_gqa_model(const AttnArgs& a, int n_sm, const int* max_clusters) {
  WindowChoice c{};
  c.supported = packed_supported(a);
  if (!c.supported) return c;
  WinSetup su;
  su.n_sm = n_sm;
  su.max_clusters[0] = 0;
  for (int cs = 1; cs <= kMaxSplit; ++cs) su.max_clusters[cs] = max_clusters[cs - 1];
  const WinShape w = win_shape(a);
  c.T = w.T;
  c.nsplit = w.nsplit;
  c.n_qt = w.n_qt;
  c.clusters = w.clusters;
  // a cluster of nsplit CTAs that cannot be resident leaves only the square kernel
  c.resident = su.max_clusters[w.nsplit] >= 1;
  c.packed_us = c.resident ? packed_us(w, su) : 0.0;
  c.square_us = square_us(a, w, su);
  c.packed = c.resident && c.packed_us < c.square_us;
  return c;
}

int try_launch_attn_window_gqa(const AttnArgs& a, int* status, cudaStream_t stream, bool force) {
  const bool fault = a.fault_cta >= 0 || a.wait_ns > 0;
  // a self-test call of the square kernel never comes here unforced
  if (!packed_supported(a) || (fault && !force)) return kWindowGqaNotTaken;
  const size_t smem = sizeof(WinSmem) + 1024;
  WinSetup su;
  const int rc = win_setup(&su, smem);
  if (rc != 0) return rc;
  const WindowChoice ch = window_gqa_model(a, su.n_sm, su.max_clusters + 1);
  if (!ch.resident || (!force && !ch.packed)) return kWindowGqaNotTaken;
  const WinShape w = win_shape(a);
  const long long grid = w.clusters * w.nsplit;
  if (grid > 0x7fffffffLL) return -2;
  CUtensorMap tq, tk, tv;
  // q as one [B * Hq * Lq, D] matrix; K', V' as [B, Hkv, Lk, D]
  if (!make_bf16_map_4d(&tq, a.q, kD, static_cast<uint64_t>(a.B) * a.Hq * a.Lq, 1, 1, kBM) ||
      !make_bf16_map_4d(&tk, a.k_cached, kD, a.L, a.Hkv, a.B, kBN) ||
      !make_bf16_map_4d(&tv, a.v_cached, kD, a.L, a.Hkv, a.B, kBN))
    return -3;
  const float scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(kD));
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(grid));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = static_cast<unsigned>(w.nsplit);
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  // programmatic dependent launch: the prologue overlaps the previous kernel's tail
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  const cudaError_t e = cudaLaunchKernelEx(
      &cfg, fault ? attn_window_gqa_kernel<true> : attn_window_gqa_kernel<false>, tq, tk, tv,
      static_cast<const __nv_bfloat16*>(a.q),
      static_cast<const __nv_bfloat16*>(a.k_seedmask), static_cast<const __nv_bfloat16*>(a.v_seedmask), a.seed_idx,
      a.n_seeds, a.Hq, a.Hkv, w.G, a.Lq, a.L, a.q0, w.n_qt, w.nsplit, w.T, scale_log2,
      static_cast<__nv_bfloat16*>(a.out), a.lse, status, a.wait_ns > 0 ? a.wait_ns : kWaitLimitNs, a.fault_cta);
  return e == cudaSuccess && cudaGetLastError() == cudaSuccess ? 0 : -3;
}

}  // namespace cover
