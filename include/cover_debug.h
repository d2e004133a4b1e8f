/*
 * cover_debug.h - self-test entry points of the COVER kernel library.
 *
 * These are not part of the method; the paper has no counterpart. They exist
 * so that tests can check the building blocks of the sm_103a attention kernel
 * (TMA tile loads, tcgen05 shared-memory / tensor-memory operand layouts) and
 * the bounded-wait failure path, in isolation, through the same C ABI.
 * Conventions (device pointers, asynchronous on `stream`, status codes) are
 * those of cover.h.
 */
#ifndef COVER_DEBUG_H_
#define COVER_DEBUG_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/*
 * One 128x128x128 tile of each tensor-core operand form the attention kernel
 * uses, computed by a single CTA with tcgen05.mma (bf16 in, fp32 accumulate):
 *   c1 = a . b^T   a [128,128] bf16 row-major, b [128,128] bf16 row-major
 *                  (both K-major, TMA-loaded with 128-byte swizzle)
 *   c2 = p . v     p [128,128] bf16 row-major, staged in tensor memory;
 *                  v [128,128] bf16 row-major (MN-major operand, TMA-loaded)
 * c1, c2: [128,128] fp32 row-major. All pointers 16-byte aligned.
 */
int cover_debug_umma_tile(const void* a, const void* b, const void* p, const void* v,
                          float* c1, float* c2, void* stream);

/*
 * Launches one CTA that waits on an mbarrier nothing ever arrives on, with a
 * limit of `limit_us` microseconds (1 .. 2000000). The kernel then records
 * COVER_ERR_DEVICE_TIMEOUT in the status word and returns normally; the
 * context stays usable. Read the result with cover_device_status().
 */
int cover_debug_wait_timeout(int limit_us, void* stream);

/*
 * The square bf16 attention kernel (the one cover_attn_fwd runs; windows as in
 * cover_attn_fwd_prefix) with a fault planted on purpose, to drive its own
 * abort path: CTA `fault_cta` of the persistent grid leaves out the K tile load of
 * its KV ring entry `fault_entry` (entries count the CTA's KV tiles over all
 * of its work units, from 0), and every bounded wait of the launch gives up
 * after `limit_us` microseconds (1 .. 2000000) instead of one second.
 * The waits that depend on the missing tile run out: the kernel records
 * COVER_ERR_DEVICE_TIMEOUT with the site of the first wait that gave up, every
 * role of that CTA leaves its loop, lets the copies and tensor-core products
 * it already issued complete, frees its tensor memory and returns; the other
 * CTAs finish their units normally. The failed CTA's output rows are
 * unspecified. An entry the CTA never reaches plants nothing, and
 * fault_cta = -1 gives a clean launch of the same kernel.
 * Arguments, layouts and errors otherwise as cover_attn_fwd_prefix (bf16).
 */
int cover_debug_attn_fault(const void* q, const void* k_cached, const void* v_cached,
                           const void* k_seedmask, const void* v_seedmask,
                           const int32_t* seed_idx, int n_seeds,
                           int B, int Hq, int Hkv, int Lq, int Lk, int q0, int D,
                           void* out, float* lse, int fault_cta, int fault_entry, int limit_us,
                           void* stream);

/*
 * cover_attn_fwd_prefix (bf16) on the packed grouped-query window kernel,
 * whichever kernel the call itself would pick: cover_attn_fwd_prefix runs a
 * window of grouped-query heads on the packed kernel only where a launch-time
 * model predicts it to be faster than the square kernel. For tests of the
 * packed kernel on every shape it supports. With fault_cta >= 0 or
 * limit_us > 0 it runs the kernel's self-test instance instead: CTA fault_cta
 * (grid order: key split fastest, then Q tile, KV head, batch row) leaves out
 * the K load of its first KV tile, and every bounded wait gives up after
 * limit_us microseconds (1 .. 2000000; 0: one second). The first wait that
 * depends on the missing tile to give up records COVER_ERR_DEVICE_TIMEOUT: at
 * site 60 or 61 in that CTA, or at site 62 in a CTA of its cluster waiting for
 * its partial block. Every role leaves its loop, every copy already issued
 * lands before a CTA exits, and the launch completes. The output rows of that
 * CTA's cluster (its Q tile of its KV head) are unspecified, and every other
 * row is the clean result. fault_cta = -1
 * with limit_us = 0 is the normal launch. Arguments, layouts and errors as
 * cover_attn_fwd_prefix, plus COVER_ERR_INVALID_ARG for limit_us outside
 * 0 .. 2000000, and COVER_ERR_UNSUPPORTED where the packed kernel does not
 * apply: Hq / Hkv < 2, Lq > 256, (Hq / Hkv) Lq > 1024, Lk > 8192, Lq == Lk with
 * q0 == 0, or a cluster of its CTAs that cannot be resident.
 */
int cover_debug_attn_prefix_packed(const void* q, const void* k_cached, const void* v_cached,
                                   const void* k_seedmask, const void* v_seedmask,
                                   const int32_t* seed_idx, int n_seeds,
                                   int B, int Hq, int Hkv, int Lq, int Lk, int q0, int D,
                                   void* out, float* lse, int fault_cta, int limit_us, void* stream);

/*
 * The choice cover_attn_fwd_prefix makes for a bf16 window (Lq rows at memory
 * positions q0.., an Lk-long memory, D = 128) between the packed grouped-query
 * kernel and the square kernel, on a GPU with n_sm SMs where max_clusters[c-1]
 * clusters of c CTAs of the packed kernel (c = 1 .. 8) can be resident at once
 * (on the device the call queries both). Host arithmetic only: no device and
 * no stream. Writes choice[6] = {supported, resident, packed, KV tiles per CTA,
 * CTAs per cluster, Q tiles per KV head} (the last three 0 when unsupported)
 * and times[2] = {predicted packed us, predicted square us} (0 when not
 * computed). COVER_ERR_INVALID_ARG for B, Hq, Hkv < 1, Hq % Hkv != 0, an
 * invalid window (as cover_attn_fwd_prefix), n_sm < 1, a negative count or a
 * null pointer.
 */
int cover_debug_window_model(int B, int Hq, int Hkv, int Lq, int Lk, int q0, int n_sm,
                             const int32_t* max_clusters, int32_t* choice, double* times);

/*
 * Like cover_device_status, and also returns where the failure came from:
 * synchronises `stream`, copies the current device's status block to the
 * host array detail[3] = {status code, site id, linear block id} (all 0 when
 * nothing failed), clears it, and returns COVER_OK (COVER_ERR_CUDA if a CUDA
 * call fails). Site ids of the bf16 attention kernel: 10 TMA thread, 20 MMA
 * thread, 30 / 31 softmax warpgroup of Q tile 0 / 1, 40 routing warp,
 * 50 / 51 seed-score warp; of the packed window kernel: 60 TMA / MMA thread,
 * 61 softmax warps, 62 combine (receive barrier), 63 copy issue.
 */
int cover_debug_status_detail(int32_t* detail, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* COVER_DEBUG_H_ */
