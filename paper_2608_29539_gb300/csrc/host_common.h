// host_common.h -- host-side helpers shared by the library's translation
// units: argument checks, TMA tensor-map encoding, device properties.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>

#include "../../include/logo.h"

namespace logo {

// Checks common to every attention entry point.
int check_dims(const logo_dims& d);
inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Number of SMs of the current device (cached per device).
int device_sm_count();

// Encode a 4-D bf16 tensor map over a row-major [d3][d2][d1][d0] tensor
// (d0 innermost, contiguous), box {box0, 1, box2, 1}, 128-byte swizzle,
// out-of-bounds elements read as zero.  Returns false on failure.
bool encode_bf16_4d(CUtensorMap* map, const void* base, uint64_t d0, uint64_t d1, uint64_t d2, uint64_t d3,
                    uint32_t box0, uint32_t box2);

// Round up to a multiple of `a`.
inline size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Allow a kernel more than 48 KB of dynamic shared memory (once per kernel).
template <typename K>
inline cudaError_t set_smem_limit(K kernel, int bytes)
{
    return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
}

// Per-translation-unit status readers (each .cu owns one device word).
int select_tu_status(int clear);
int combine_tu_status(int clear);
int attn_fwd_tu_status(int clear);
int attn_bwd_tu_status(int clear);
int decode_tu_status(int clear);
int transform_tu_status(int clear);
int gate_tu_status(int clear);
int selftest_tu_status(int clear);

}  // namespace logo
