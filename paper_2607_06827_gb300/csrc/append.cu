// speechkv_append: one decode step's cache update (Sec. III-C: the cache is
// compressed once at prefill; every generated token then adds one
// full-resolution key/value per layer).
//
// One CTA per request: all threads read len[b] first, copy the token's
// [H_kv][d] key and value into row len[b] of every head (a contiguous run or,
// with a block table, the row's page) with 16-byte stores, and after a
// barrier one thread advances len[b].  A full cache (or an invalid block) is
// reported through the error word and left untouched.
#include "common.cuh"
#include "launch.h"

namespace speechkv {
namespace {

template <typename T>
__global__ void __launch_bounds__(256)
    append_kernel(const T *__restrict__ kn, const T *__restrict__ vn, T *__restrict__ kc,
                  T *__restrict__ vc, const int64_t *__restrict__ cache_off,
                  int32_t *__restrict__ len, int H_kv, int D, CacheMap map,
                  int *__restrict__ err) {
    constexpr int kPerVec = 16 / (int)sizeof(T);
    const int b = blockIdx.x;
    const int64_t L = len[b];
    const bool paged = map.table != nullptr;
    const int64_t base = paged ? 0 : cache_off[b];
    const int64_t cap = paged ? ((int64_t)map.max_blocks << map.bs_log2) : cache_off[b + 1] - base;
    if (base < 0 || cap < 0) {
        if (threadIdx.x == 0) report_error(err, SPEECHKV_ERR_INVALID_ARG);
        return;
    }
    if (L < 0 || L >= cap) {
        if (threadIdx.x == 0) report_error(err, SPEECHKV_ERR_CAPACITY);
        return;  // uniform: every thread took the same branch
    }
    // with pages, the row's block must be valid for every head (one table entry)
    if (cache_row(map, b, 0, L, H_kv, D, base, cap) < 0) {
        if (threadIdx.x == 0) report_error(err, SPEECHKV_ERR_INVALID_ARG);
        return;
    }
    const int nvec = H_kv * D / kPerVec;  // 16-byte vectors per tensor
    for (int i = threadIdx.x; i < 2 * nvec; i += blockDim.x) {
        const int tensor = i >= nvec;
        const int e = (i - tensor * nvec) * kPerVec;  // element within [H_kv][d]
        const int h = e / D, c = e - h * D;
        const T *src = (tensor ? vn : kn) + (int64_t)b * H_kv * D + e;
        T *dst = (tensor ? vc : kc) + cache_row(map, b, h, L, H_kv, D, base, cap) + c;
        copy_bytes<16>(dst, src);
    }
    __syncthreads();
    if (threadIdx.x == 0) len[b] = (int32_t)(L + 1);
}

// One thread waits, through the bounded wait every kernel of the library
// uses, for a phase of an mbarrier that no thread ever completes: the wait
// gives up after its time limit, records SPEECHKV_ERR_TIMEOUT and the kernel
// returns normally.
__global__ void selftest_timeout_kernel(int *err) {
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        fence_mbar_init();
        mbar_wait_bounded(&bar, 0, err);  // phase 0 needs one arrival: none comes
    }
}

}  // namespace

cudaError_t launch_selftest_timeout(int *err, cudaStream_t stream) {
    selftest_timeout_kernel<<<1, 32, 0, stream>>>(err);
    return cudaGetLastError();
}

cudaError_t launch_append(const AppendArgs &a, cudaStream_t stream) {
    if (a.dtype == SPEECHKV_F32)
        append_kernel<float><<<a.B, 256, 0, stream>>>(
            static_cast<const float *>(a.k_new), static_cast<const float *>(a.v_new),
            static_cast<float *>(a.k_cache), static_cast<float *>(a.v_cache), a.cache_off, a.len,
            a.H_kv, a.d, a.map, a.err);
    else
        append_kernel<__nv_bfloat16><<<a.B, 256, 0, stream>>>(
            static_cast<const __nv_bfloat16 *>(a.k_new),
            static_cast<const __nv_bfloat16 *>(a.v_new),
            static_cast<__nv_bfloat16 *>(a.k_cache), static_cast<__nv_bfloat16 *>(a.v_cache),
            a.cache_off, a.len, a.H_kv, a.d, a.map, a.err);
    return cudaGetLastError();
}

}  // namespace speechkv
