/*
 * fpo_testing.h -- test-only entry points of libfpo.  Not part of the FPO
 * step; they expose internal building blocks so tests can check them alone.
 */
#ifndef FPO_TESTING_H_
#define FPO_TESTING_H_

#include <stddef.h>
#include <stdint.h>

#include "fpo.h"

#ifdef __cplusplus
extern "C" {
#endif

/*
 * The tensor-core GEMM core of fpo_error_signal / fpo_layer_update with a
 * plain fp32 store epilogue: C[M, N] = sum_k A(m, k) B(n, k), bf16 inputs,
 * fp32 accumulation (the contraction of Eq. (gproj) and Eq. (w3update)).
 *   a_mn = 0: A is [M, K] row-major (K contiguous); a_mn = 1: A is [K, M].
 *   b_mn = 0: B is [N, K] row-major;                 b_mn = 1: B is [K, N].
 * Supported (a_mn, b_mn): (0, 0), (0, 1), (1, 1).  M, N, K > 0; the
 * contiguous extent of each operand must be a multiple of 8.  C is [M, N]
 * fp32 row-major with N a multiple of 8.  workspace holds the device status
 * word (>= 256 bytes).  Returns an fpo_status code.
 */
int32_t fpo_testing_gemm_bf16(int64_t M, int64_t N, int64_t K, int32_t a_mn, int32_t b_mn,
                              const void* A, const void* B, float* C, void* workspace,
                              size_t workspace_bytes, void* stream);

/*
 * Select the tensor-core GEMM kernel every later call uses (process-wide):
 * 0 = one CTA per 128 x 256 output tile, 1 = a CTA pair (tcgen05 cta_group::2)
 * per 256 x 256 tile, 2 = as 1 but 256 x 512 pair tiles for the projection
 * g = E W_U (one accumulator, a quarter less operand traffic; the default).
 * Any other value selects 0.  Returns the previous setting.  All compute the same sums in the same order per
 * output element.
 */
int32_t fpo_testing_set_gemm_variant(int32_t variant);

/*
 * Override the height, in output tiles, of the bands in which GEMM tiles are
 * rasterised for L2 reuse (0 restores the default: bands of 16 tile rows).
 * Tuning hook; results do not depend on it.
 */
void fpo_testing_set_band(int32_t band);

/*
 * Rows of the last token chunk of the most recent fpo_error_signal call on
 * `workspace` (with this `desc`) that the direct algorithm recomputed because
 * S'_t fell outside its anchor window (see FPO_ES_DIRECT).  Synchronizes
 * `stream`.  Returns -1 when desc does not select the direct algorithm, or on
 * a CUDA error.
 */
int64_t fpo_testing_direct_fixup_rows(const fpo_error_signal_desc* desc,
                                      const void* workspace, void* stream);

/*
 * Kernels this library has launched in this process, over every entry point and
 * every thread (a launch the runtime rejected is counted too).  The difference of
 * two readings around a region counts the library's kernels in it.
 */
uint64_t fpo_testing_kernel_launches(void);

/*
 * Failure-detection check of the bounded waits every kernel uses: launches one
 * block that waits on a shared-memory mbarrier nothing ever arrives on, with
 * a limit of `limit_ns` nanoseconds.  The wait gives up, the kernel records
 * FPO_ERR_TIMEOUT in the workspace status word and returns, leaving the CUDA
 * context usable; fpo_get_device_status(workspace, stream) then reports it.
 */
int32_t fpo_testing_wait_timeout(uint64_t limit_ns, void* workspace, size_t workspace_bytes,
                                 void* stream);

#ifdef __cplusplus
}
#endif

#endif /* FPO_TESTING_H_ */
