// host_copy.cu -- fpo_h2d_copy: the input stage of a step whose inputs (the final
// residual h, the targets, the cached MLP activations A_l) arrive in host memory.
//
// The copy is done by SM loads of page-locked host memory through its device
// mapping, not by the copy engines: one launch walks a list of buffers, each
// thread keeping two 16-byte loads in flight.  A block needs no shared memory
// beyond the per-block reserve and 256 threads, so one block fits on every SM
// beside a persistent GEMM block that uses the rest of the SM's shared memory,
// and the copy runs concurrently with the step on another stream.  The kernel
// prefers the largest shared-memory carve-out, so an SM that it occupies first
// stays configured for the GEMM blocks that follow.
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/fpo.h"
#include "internal.h"

namespace fpo {
namespace {

constexpr int kCopyThreads = 256;
// 16-byte vectors in flight per thread.  Host loads take microseconds, and every one
// in flight holds a memory request slot of its SM: with four per thread (16 KB per SM)
// the step's kernels beside the copy ran ~9% slower; two (8 KB per SM) still keep the
// host link at its 210 GB/s and leave them within ~1%.
constexpr int kCopyUnroll = 2;

struct CopySeg {
    const uint4* src;          // device mapping of the host buffer
    uint4* dst;
    unsigned long long n16;    // whole 16-byte vectors
    unsigned int tail;         // bytes after them, < 16
};

struct CopyList {
    CopySeg seg[FPO_MAX_COPY_BUFFERS];
    int n;
};

__global__ void __launch_bounds__(kCopyThreads)
    h2d_copy_kernel(const __grid_constant__ CopyList list) {
    const unsigned long long tid =
        static_cast<unsigned long long>(blockIdx.x) * kCopyThreads + threadIdx.x;
    const unsigned long long stride = static_cast<unsigned long long>(gridDim.x) * kCopyThreads;
    for (int s = 0; s < list.n; ++s) {
        const uint4* __restrict__ src = list.seg[s].src;
        uint4* __restrict__ dst = list.seg[s].dst;
        const unsigned long long n16 = list.seg[s].n16;
        unsigned long long i = tid;
        // every index of an iteration is below n16: i + (kCopyUnroll - 1) stride < n16
        for (; i + (kCopyUnroll - 1) * stride < n16; i += kCopyUnroll * stride) {
            uint4 v[kCopyUnroll];
#pragma unroll
            for (int u = 0; u < kCopyUnroll; ++u) v[u] = src[i + u * stride];
#pragma unroll
            for (int u = 0; u < kCopyUnroll; ++u) __stcs(dst + i + u * stride, v[u]);
        }
        for (; i < n16; i += stride) __stcs(dst + i, src[i]);
        if (tid < list.seg[s].tail)
            reinterpret_cast<unsigned char*>(dst + n16)[tid] =
                reinterpret_cast<const unsigned char*>(src + n16)[tid];
    }
}

bool misaligned(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) != 0; }

// Device address of host byte p if p lies in page-locked, device-mapped host memory.
bool mapped_page_locked(const char* p, char** dev) {
    cudaPointerAttributes a;
    if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
        cudaGetLastError();  // the failed lookup is not an error of later calls
        return false;
    }
    if (a.type != cudaMemoryTypeHost || a.devicePointer == nullptr) return false;
    *dev = static_cast<char*>(a.devicePointer);
    return true;
}

}  // namespace
}  // namespace fpo

extern "C" int32_t fpo_h2d_copy(int32_t n, void* const* dst, const void* const* src,
                                const size_t* bytes, void* stream) {
    if (n < 0 || n > FPO_MAX_COPY_BUFFERS) return FPO_ERR_SHAPE;
    if (n == 0) return FPO_OK;
    if (!dst || !src || !bytes) return FPO_ERR_NULL;
    for (int i = 0; i < n; ++i) {
        if (bytes[i] == 0) continue;
        if (!dst[i] || !src[i]) return FPO_ERR_NULL;
        if (fpo::misaligned(dst[i]) || fpo::misaligned(src[i])) return FPO_ERR_ALIGN;
    }
    fpo::DevInfo di;
    if (!fpo::current_device_info(&di)) return FPO_ERR_CUDA;
    if (di.major != 10 || di.minor != 3) return FPO_ERR_ARCH;

    fpo::CopyList list{};
    int m = 0;
    for (int i = 0; i < n; ++i) {
        if (bytes[i] == 0) continue;
        // The first and the last byte must both lie in page-locked host memory that is
        // mapped into the device address space (not pageable memory, which some systems
        // also let a kernel read), with device addresses bytes - 1 apart.
        const char* first = static_cast<const char*>(src[i]);
        char* m0 = nullptr;
        char* m1 = nullptr;
        if (!fpo::mapped_page_locked(first, &m0) ||
            !fpo::mapped_page_locked(first + bytes[i] - 1, &m1) ||
            m1 - m0 != static_cast<ptrdiff_t>(bytes[i] - 1))
            return FPO_ERR_ARG;
        if (fpo::misaligned(m0)) return FPO_ERR_ALIGN;
        list.seg[m].src = reinterpret_cast<const uint4*>(m0);
        list.seg[m].dst = static_cast<uint4*>(dst[i]);
        list.seg[m].n16 = bytes[i] / 16;
        list.seg[m].tail = static_cast<unsigned int>(bytes[i] % 16);
        ++m;
    }
    if (m == 0) return FPO_OK;
    list.n = m;

    if (cudaFuncSetAttribute(fpo::h2d_copy_kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                             cudaSharedmemCarveoutMaxShared) != cudaSuccess)
        return FPO_ERR_CUDA;
    fpo::h2d_copy_kernel<<<di.sm_count, fpo::kCopyThreads, 0, static_cast<cudaStream_t>(stream)>>>(
        list), ::fpo::note_launch();
    return cudaGetLastError() == cudaSuccess ? FPO_OK : FPO_ERR_CUDA;
}
