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

#ifdef __cplusplus
}
#endif

#endif /* COVER_DEBUG_H_ */
