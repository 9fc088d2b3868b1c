// host_common.cu -- host helpers: argument checks, tensor-map encoding via
// the driver entry point (no link-time dependency on libcuda), device
// properties, and the library-wide device status query.
#include <mutex>

#include "host_common.h"

namespace logo {

int check_dims(const logo_dims& d)
{
    if (d.B < 1 || d.T < 1 || d.Hq < 1 || d.Hkv < 1 || d.D < 1) return LOGO_ERR_INVALID_ARG;
    if (d.D != 64 && d.D != 128) return LOGO_ERR_UNSUPPORTED;
    if (d.Hq % d.Hkv != 0) return LOGO_ERR_UNSUPPORTED;
    // packed-row indices and element offsets stay within int32 / TMA limits
    if (static_cast<int64_t>(d.B) * d.T > (1ll << 30)) return LOGO_ERR_UNSUPPORTED;
    return LOGO_OK;
}

int device_sm_count()
{
    static std::mutex mu;
    static int cached[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
    std::lock_guard<std::mutex> lock(mu);
    if (cached[dev] == 0) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
        cached[dev] = n;
    }
    return cached[dev];
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn()
{
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    });
    return fn;
}

bool encode_bf16_4d(CUtensorMap* map, const void* base, uint64_t d0, uint64_t d1, uint64_t d2, uint64_t d3,
                    uint32_t box0, uint32_t box2)
{
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[4] = {d0, d1, d2, d3};
    cuuint64_t strides[3] = {d0 * 2, d0 * d1 * 2, d0 * d1 * d2 * 2};
    cuuint32_t box[4] = {box0, 1, box2, 1};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

}  // namespace logo

extern "C" int logo_get_device_status(int* status)
{
    if (!status) return LOGO_ERR_INVALID_ARG;
    int first = LOGO_OK;
    int (*readers[])(int) = {logo::select_tu_status,    logo::combine_tu_status,   logo::attn_fwd_tu_status,
                             logo::attn_bwd_tu_status,  logo::decode_tu_status,    logo::transform_tu_status,
                             logo::gate_tu_status,      logo::selftest_tu_status};
    for (auto rd : readers) {
        int v = rd(1);
        if (v == LOGO_ERR_CUDA) return LOGO_ERR_CUDA;
        if (first == LOGO_OK && v != LOGO_OK) first = v;
    }
    *status = first;
    return LOGO_OK;
}

extern "C" int logo_num_sms(void) { return logo::device_sm_count(); }
