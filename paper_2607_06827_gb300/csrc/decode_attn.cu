// Decode-attention instances -- CUDA-core consumers for fp32 caches,
// tensor-core consumers for bf16 caches with d = 64 -- and the dispatch over
// every compiled decode kernel.  The kernel itself is in decode_attn.cuh; the
// bf16 instances with d = 128 are compiled in decode_attn_mma.cu.
#include "decode_attn.cuh"

namespace speechkv {

bool decode_supported(speechkv_dtype dtype, int d, int group) {
    if (d != 64 && d != 128) return false;
    if (dtype == SPEECHKV_F32) return group == 1 || group == 2 || group == 4;
    return dtype == SPEECHKV_BF16 && group >= 1 && group <= kMmaMaxGroup;
}

int decode_slot_floats(int d, int group) {
    const int f = group * d + 2 * group;  // o [G][d], then m [G] and l [G]
    return (f + 3) & ~3;                  // keep slots 16-byte aligned
}

namespace {

#define SPEECHKV_DECODE_LOCAL_CASES(X)                                                    \
    X(float, 64, 1) X(float, 64, 2) X(float, 64, 4) X(float, 128, 1) X(float, 128, 2)      \
        X(float, 128, 4) X(__nv_bfloat16, 64, 1) X(__nv_bfloat16, 64, 2)                   \
            X(__nv_bfloat16, 64, 3) X(__nv_bfloat16, 64, 4) X(__nv_bfloat16, 64, 5)        \
                X(__nv_bfloat16, 64, 6) X(__nv_bfloat16, 64, 7) X(__nv_bfloat16, 64, 8)

template <typename T>
constexpr speechkv_dtype dtype_of() {
    return sizeof(T) == 4 ? SPEECHKV_F32 : SPEECHKV_BF16;
}

}  // namespace

int decode_ctas_per_sm(speechkv_dtype dtype, int d, int group, int B) {
    if (dtype == SPEECHKV_BF16 && d == 128) return decode_ctas_per_sm_mma128(group, B);
#define X(T, D, G) \
    if (dtype == dtype_of<T>() && d == D && group == G) return occupancy_instance<T, D, G>(B);
    SPEECHKV_DECODE_LOCAL_CASES(X)
#undef X
    return 0;
}

cudaError_t launch_decode(const DecodeArgs &a, int grid, cudaStream_t stream) {
    const int group = a.H_q / a.H_kv;
    const bool append = a.k_new != nullptr;
    // the paged layout comes with the fused append only (speechkv_decode_step_paged)
    if (a.map.table && !append) return cudaErrorInvalidValue;
    if (a.dtype == SPEECHKV_BF16 && a.d == 128) return launch_decode_mma128(a, grid, stream);
#define X(T, D, G)                                                                   \
    if (a.dtype == dtype_of<T>() && a.d == D && group == G)                          \
        return !append ? launch_instance<T, D, G, false, false>(a, grid, stream)     \
               : a.map.table ? launch_instance<T, D, G, true, true>(a, grid, stream) \
                             : launch_instance<T, D, G, true, false>(a, grid, stream);
    SPEECHKV_DECODE_LOCAL_CASES(X)
#undef X
    return cudaErrorInvalidValue;
}

}  // namespace speechkv
