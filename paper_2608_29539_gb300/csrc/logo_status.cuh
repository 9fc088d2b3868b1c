// logo_status.cuh -- the device-side error word of one translation unit.
//
// Kernels never trap: a bounded wait that expires, or a bounds check that
// fails, records a LOGO_ERR_* code here (first error wins) and the kernel
// returns.  Each .cu file gets its own word (the variable is static); the
// host reads and clears all of them through logo_get_device_status().
#pragma once
#include <cuda_runtime.h>

#include "../../include/logo.h"

namespace logo {

static __device__ int g_status_word = 0;

__device__ __forceinline__ void record_status(int code) { atomicCAS(&g_status_word, 0, code); }

// Host side: read (and optionally clear) this translation unit's word.
// Synchronises the device.
static inline int read_tu_status(int clear)
{
    int v = 0;
    if (cudaMemcpyFromSymbol(&v, g_status_word, sizeof(int)) != cudaSuccess) return LOGO_ERR_CUDA;
    if (clear && v != 0) {
        int zero = 0;
        if (cudaMemcpyToSymbol(g_status_word, &zero, sizeof(int)) != cudaSuccess) return LOGO_ERR_CUDA;
    }
    return v;
}

}  // namespace logo
