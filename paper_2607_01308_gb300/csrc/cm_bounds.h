// Bounds-checked builds (compiled with -DCM_DEBUG_BOUNDS: build.py --bounds), a testing
// aid standing in for a device memory checker. Every global access of the kernels that
// carry these checks is tested against the buffer it belongs to; an access outside it is
// counted in the translation unit's violation counter and not made (a load is skipped or
// reads zeros, a store is dropped, a TMA copy is not issued), so a wrong index shows up as
// a count instead of a fault. Without the macro the checks compile to nothing. Not part of
// the public ABI.
#pragma once

#include <cstdint>

#include <cuda_runtime.h>

#ifdef CM_DEBUG_BOUNDS

namespace cm {
namespace {

__device__ unsigned int g_bounds_violations;   // one per translation unit

__device__ __forceinline__ void bounds_fail() { atomicAdd(&g_bounds_violations, 1u); }

// True when [p, p + n) lies in [base, base + size); otherwise counts a violation.
__device__ __forceinline__ bool in_bounds(const void *p, uint64_t n, const void *base,
                                          uint64_t size) {
    const uint64_t a = reinterpret_cast<uint64_t>(p), b = reinterpret_cast<uint64_t>(base);
    const bool ok = a >= b && n <= size && a - b <= size - n;
    if (!ok) bounds_fail();
    return ok;
}

}  // namespace
}  // namespace cm

#define CM_IN_BOUNDS(p, n, base, size) ::cm::in_bounds((p), (n), (base), (size))

// Host side: reads and zeroes this translation unit's counter.
#define CM_DEFINE_BOUNDS_READER(fn)                                                        \
    cudaError_t fn(unsigned int *out) {                                                    \
        const unsigned int zero = 0;                                                       \
        cudaError_t e = cudaMemcpyFromSymbol(out, g_bounds_violations, sizeof(unsigned int)); \
        if (e == cudaSuccess)                                                              \
            e = cudaMemcpyToSymbol(g_bounds_violations, &zero, sizeof(unsigned int));      \
        return e;                                                                          \
    }

#else

#define CM_IN_BOUNDS(p, n, base, size) true

#define CM_DEFINE_BOUNDS_READER(fn)                                                        \
    cudaError_t fn(unsigned int *out) {                                                    \
        *out = 0;                                                                          \
        return cudaSuccess;                                                                \
    }

#endif
