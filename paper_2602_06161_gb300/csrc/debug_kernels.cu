// debug_kernels.cu - self-test kernels for the tcgen05/TMA building blocks and
// for the bounded-wait failure path. The paper has no counterpart; see
// include/cover_debug.h.
#include <cuda_bf16.h>

#include "kernels.cuh"
#include "ptx.cuh"
#include "tmap.cuh"

namespace cover {
namespace {

constexpr int kT = 128;                    // tile edge
constexpr int kTileBytes = kT * kT * 2;    // one bf16 tile = two 64-column swizzled boxes
constexpr int kBoxBytes = kTileBytes / 2;

struct UmmaSmem {
  uint8_t a[kTileBytes];
  uint8_t b[kTileBytes];
  uint8_t v[kTileBytes];
  uint64_t bar_load;
  uint64_t bar_mma;
  uint32_t tmem_base;
  int abort;
};

// One CTA of 128 threads (4 warps). Thread t owns row t of every result.
__global__ void __launch_bounds__(128, 1)
    umma_tile_kernel(const __grid_constant__ CUtensorMap map_a, const __grid_constant__ CUtensorMap map_b,
                     const __grid_constant__ CUtensorMap map_v, const uint32_t* __restrict__ p_rows,
                     float* __restrict__ c1, float* __restrict__ c2, int* status) {
  extern __shared__ uint8_t smem_raw[];
  UmmaSmem& sm = *reinterpret_cast<UmmaSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x;
  const int warp = tid / 32;

  if (tid == 0) {
    mbar_init(&sm.bar_load, 1);
    mbar_init(&sm.bar_mma, 1);
    sm.abort = 0;
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(&sm.tmem_base, 512);
    tmem_relinquish();
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tbase = sm.tmem_base;
  const uint32_t c1_col = 0, c2_col = 128, p_col = 256;
  const uint32_t lane_off = static_cast<uint32_t>(warp * 32) << 16;

  if (tid == 0) {
    mbar_arrive_expect_tx(&sm.bar_load, 3 * kTileBytes);
    for (int h = 0; h < 2; ++h) {
      tma_load_4d(sm.a + h * kBoxBytes, &map_a, &sm.bar_load, 64 * h, 0, 0, 0);
      tma_load_4d(sm.b + h * kBoxBytes, &map_b, &sm.bar_load, 64 * h, 0, 0, 0);
      tma_load_4d(sm.v + h * kBoxBytes, &map_v, &sm.bar_load, 64 * h, 0, 0, 0);
    }
  }

  // Stage P (row t = thread t) into tensor memory: 64 columns of bf16 pairs.
  {
    uint32_t r[32];
    for (int h = 0; h < 2; ++h) {
      for (int c = 0; c < 32; ++c) r[c] = p_rows[tid * 64 + h * 32 + c];
      tmem_st32(tbase + lane_off + p_col + h * 32, r);
    }
    tmem_st_wait();
  }
  tc_fence_before_sync();
  __syncthreads();

  bool ok = true;
  if (tid == 0) {
    tc_fence_after_sync();
    ok = mbar_wait(&sm.bar_load, 0, &sm.abort);
    if (ok) {
      const uint32_t a0 = smem_u32(sm.a), b0 = smem_u32(sm.b), v0 = smem_u32(sm.v);
      constexpr uint32_t id_ss = idesc_bf16_f32(128, 128, false, false);
      constexpr uint32_t id_ts = idesc_bf16_f32(128, 128, false, true);
      for (int k = 0; k < 8; ++k) {
        // K-major operands: 16 columns = 32 bytes inside a 128-byte swizzle row
        const uint32_t off = (k / 4) * kBoxBytes + (k % 4) * 32;
        umma_ss(tbase + c1_col, sdesc_sw128(a0 + off, 16, 1024), sdesc_sw128(b0 + off, 16, 1024), id_ss, k > 0);
      }
      for (int k = 0; k < 8; ++k) {
        // MN-major V: 16 rows of 128 bytes per step; the second 64-column box is 16 KB further
        umma_ts(tbase + c2_col, tbase + p_col + 8 * k, sdesc_sw128(v0 + k * 2048, kBoxBytes, 1024), id_ts, k > 0);
      }
      umma_commit(&sm.bar_mma);
    } else {
      report_status(status, kStatusTimeout, 1);
      sm.abort = 1;
    }
  }
  __syncwarp();
  // every thread waits for the MMAs (bounded); thread 0's outcome is shared through abort
  ok = mbar_wait(&sm.bar_mma, 0, &sm.abort);
  if (!ok && tid == 0 && !sm.abort) report_status(status, kStatusTimeout, 2);
  tc_fence_after_sync();
  if (__all_sync(0xffffffffu, ok)) {
    uint32_t r[32];
    for (int h = 0; h < 4; ++h) {
      tmem_ld32(tbase + lane_off + c1_col + h * 32, r);
      tmem_ld_wait(r);
      for (int c = 0; c < 32; ++c) c1[tid * kT + h * 32 + c] = __uint_as_float(r[c]);
      tmem_ld32(tbase + lane_off + c2_col + h * 32, r);
      tmem_ld_wait(r);
      for (int c = 0; c < 32; ++c) c2[tid * kT + h * 32 + c] = __uint_as_float(r[c]);
    }
  }
  tc_fence_before_sync();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tbase, 512);
}

__global__ void wait_timeout_kernel(uint64_t limit_ns, int* status) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    // nothing arrives on this barrier: the wait must give up and report
    if (!mbar_wait(&bar, 0, nullptr, limit_ns)) report_status(status, kStatusTimeout, 100);
  }
}

}  // namespace

int launch_umma_tile(const void* a, const void* b, const void* p, const void* v, float* c1, float* c2, int* status,
                     cudaStream_t stream) {
  CUtensorMap ma, mb, mv;
  if (!make_bf16_map_4d(&ma, a, 128, 128, 1, 1, 128) || !make_bf16_map_4d(&mb, b, 128, 128, 1, 1, 128) ||
      !make_bf16_map_4d(&mv, v, 128, 128, 1, 1, 128))
    return -3;
  // generous allocation: operand reads stay inside the CTA's window even for a misread stride
  const size_t smem = 200 * 1024;
  static_assert(sizeof(UmmaSmem) + 1024 <= 200 * 1024, "self-test tile smem");
  if (cudaFuncSetAttribute(umma_tile_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
    return -3;
  umma_tile_kernel<<<1, 128, smem, stream>>>(ma, mb, mv, static_cast<const uint32_t*>(p), c1, c2, status);
  return cudaGetLastError() == cudaSuccess ? 0 : -3;
}

int launch_wait_timeout(uint64_t limit_ns, int* status, cudaStream_t stream) {
  wait_timeout_kernel<<<1, 32, 0, stream>>>(limit_ns, status);
  return cudaGetLastError() == cudaSuccess ? 0 : -3;
}

}  // namespace cover
