// error_math.cuh -- the output-layer error of one logit (Sec. 3.1 step 2),
// e = s (softmax(z) - 1_y) with softmax(z)_v = exp(z_v - lse), written once and
// used by every kernel that forms it, so all algorithms give identical bits.
#pragma once

#include <cuda_bf16.h>
#include <stdint.h>

#include "ptx.cuh"

namespace fpo {

constexpr float kLog2e = 1.4426950408889634f;

// bf16 path: 2^(z log2e - lse log2e) on the MUFU unit; lse2 = lse * log2e.
__device__ __forceinline__ float error_value(float z, float lse2, bool is_target, float s) {
    return s * (ex2_approx(fmaf(z, kLog2e, -lse2)) - (is_target ? 1.f : 0.f));
}

// fp32 path: correctly rounded-ish expf for 1e-5 parity.
__device__ __forceinline__ float error_value_f32(float z, float lse, bool is_target, float s) {
    return s * (expf(z - lse) - (is_target ? 1.f : 0.f));
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    __nv_bfloat162 p = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&p);
}

}  // namespace fpo
