// Decode-attention instances with tensor-core consumers for d = 128: bf16
// caches with 1 to 8 query heads per KV head (the kernel is in
// decode_attn.cuh; compiled apart from the other instances so that the two
// halves build in parallel).
#include "decode_attn.cuh"

namespace speechkv {

#define SPEECHKV_DECODE_MMA128_CASES(X) X(1) X(2) X(3) X(4) X(5) X(6) X(7) X(8)

int decode_ctas_per_sm_mma128(int group, int B) {
#define X(G) \
    if (group == G) return occupancy_instance<__nv_bfloat16, 128, G>(B);
    SPEECHKV_DECODE_MMA128_CASES(X)
#undef X
    return 0;
}

cudaError_t launch_decode_mma128(const DecodeArgs &a, int grid, cudaStream_t stream) {
    using T = __nv_bfloat16;
    const int group = a.H_q / a.H_kv;
    const bool append = a.k_new != nullptr;
#define X(G)                                                                               \
    if (group == G)                                                                        \
        return !append ? launch_instance<T, 128, G, false, false>(a, grid, stream)         \
               : a.map.table ? launch_instance<T, 128, G, true, true>(a, grid, stream)     \
                             : launch_instance<T, 128, G, true, false>(a, grid, stream);
    SPEECHKV_DECODE_MMA128_CASES(X)
#undef X
    return cudaErrorInvalidValue;
}

}  // namespace speechkv
