// optim_math.cuh -- the per-element optimizer step on the fp32 master (Sec. 3.1: SGD,
// SGD with momentum, AdamW with decoupled weight decay), shared by the stand-alone
// optimizer passes (optimizer.cu) and the fused epilogue of the pseudogradient GEMM
// (EpiOptStep in epilogues.cuh), so that both take the same step.
#pragma once

#include <math.h>

#include "internal.h"

namespace fpo {

// State update and unclipped step for one element (g already scaled by any gradient
// clip): SGD -lr g; momentum s1 <- mu s1 + g, -lr s1; AdamW s1 <- b1 s1 + (1 - b1) g,
// s2 <- b2 s2 + (1 - b2) g^2, -lr (s1 / (1 - b1^t)) / (sqrt(s2 / (1 - b2^t)) + eps)
// - lr wd w.
__device__ __forceinline__ float opt_step(const OptimParams& op, float g, float w, float& s1,
                                          float& s2) {
    if (op.kind == 0) return -op.lr * g;
    if (op.kind == 1) {
        s1 = fmaf(op.momentum, s1, g);
        return -op.lr * s1;
    }
    s1 = fmaf(op.beta1, s1, (1.f - op.beta1) * g);
    s2 = fmaf(op.beta2, s2, (1.f - op.beta2) * g * g);
    const float mhat = s1 * op.inv_bc1;
    const float denom = sqrtf(s2) * op.inv_sqrt_bc2 + op.eps;
    return -op.lr * (mhat / denom + op.weight_decay * w);
}

}  // namespace fpo
