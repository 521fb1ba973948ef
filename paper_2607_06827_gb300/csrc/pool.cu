// speechkv_pool: Eq. (pool) of the paper (Sec. III-B), run once per request
// and layer at prefill (Sec. III-C) -- writes the compressed cache rows of
// every (request, KV head) from the full-resolution prefill keys/values.
//
// One warp produces one cached row of one (request, KV head).  Task
// tau = r * H_kv + h enumerates (prefill row r, head h); the request b holding
// r is found by binary search over full_off, and t = r - full_off[b] is used
// as the OUTPUT row index, so the first len_b tasks of a request are busy and
// the rest idle.  Consecutive warps handle the heads of one token, which read
// one contiguous token-major prefill row between them.
//
//   t <  P            text before the speech: copy prefill row t
//   t <  P + n        speech window i = t - P: online softmax over the gate
//                     logits u_h . k_j of frames P + i*w .. min(.., P + T) - 1,
//                     weighted sums of keys and values (fp32), one rounding
//   t <  P + n + N    text after the speech: copy prefill row t - n + T
//
// With w_eff = 1 (layers before l0) every row is a bit-exact copy.
#include <math.h>

#include "common.cuh"
#include "launch.h"

namespace speechkv {
namespace {

// Largest b with full_off[b] <= r, for r < full_off[B].
__device__ __forceinline__ int request_of_row(const int64_t *__restrict__ off, int B, int64_t r) {
    int lo = 0, hi = B - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (__ldg(off + mid) <= r)
            lo = mid;
        else
            hi = mid - 1;
    }
    return lo;
}

template <typename T, int D>
__global__ void __launch_bounds__(256)
    pool_kernel(const T *__restrict__ kf, const T *__restrict__ vf,
                const int64_t *__restrict__ full_off, const int32_t *__restrict__ Pa,
                const int32_t *__restrict__ Ta, const int32_t *__restrict__ Na,
                const float *__restrict__ gate, T *__restrict__ kc, T *__restrict__ vc,
                const int64_t *__restrict__ cache_off, int32_t *__restrict__ len, int B,
                int64_t full_rows, int H_kv, int w, int *__restrict__ err) {
    constexpr int kCols = D / 32;  // elements per lane
    const int lane = threadIdx.x & 31;
    const int64_t gwarp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;

    // lengths: the first B threads of the grid
    const int64_t gtid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (gtid < B) {
        const int b = (int)gtid;
        const int64_t S = full_off[b + 1] - full_off[b];
        const int64_t cap = cache_off[b + 1] - cache_off[b];
        const int64_t Pb = Pa[b], Tb = Ta[b], Nb = Na[b];
        const int64_t n = (Tb + w - 1) / w;
        int64_t L = Pb + n + Nb;
        if (Pb < 0 || Tb < 0 || Nb < 0 || S != Pb + Tb + Nb || cap < 0 || full_off[b] < 0 ||
            full_off[b + 1] > full_rows || cache_off[b] < 0) {
            report_error(err, SPEECHKV_ERR_INVALID_ARG);
            L = 0;
        } else if (L > cap) {
            report_error(err, SPEECHKV_ERR_CAPACITY);
            L = cap;
        }
        len[b] = (int32_t)L;
    }

    const int64_t tasks = full_rows * H_kv;
    for (int64_t tau = gwarp; tau < tasks; tau += nwarps) {
        const int64_t r = tau / H_kv;
        const int h = (int)(tau - r * H_kv);
        if (r >= __ldg(full_off + B) || r < __ldg(full_off)) continue;
        const int b = request_of_row(full_off, B, r);
        const int64_t row0 = __ldg(full_off + b);
        const int64_t t = r - row0;
        const int64_t Pb = __ldg(Pa + b), Tb = __ldg(Ta + b), Nb = __ldg(Na + b);
        const int64_t S = __ldg(full_off + b + 1) - row0;
        if (Pb < 0 || Tb < 0 || Nb < 0 || S != Pb + Tb + Nb || row0 < 0 ||
            __ldg(full_off + b + 1) > full_rows || __ldg(cache_off + b) < 0)
            continue;  // reported above
        const int64_t n = (Tb + w - 1) / w;
        if (t >= Pb + n + Nb) continue;  // idle task
        const int64_t cap = __ldg(cache_off + b + 1) - __ldg(cache_off + b);
        if (t >= cap) continue;        // reported above (capacity)
        T *kd = kc + ((__ldg(cache_off + b) * H_kv + (int64_t)h * cap + t) * D) + lane * kCols;
        T *vd = vc + ((__ldg(cache_off + b) * H_kv + (int64_t)h * cap + t) * D) + lane * kCols;
        const int64_t rowstride = (int64_t)H_kv * D;
        const T *kbase = kf + (row0 * H_kv + h) * D + lane * kCols;  // prefill row 0 of b
        const T *vbase = vf + (row0 * H_kv + h) * D + lane * kCols;

        if (t < Pb || t >= Pb + n || w == 1) {
            const int64_t src = (t < Pb || w == 1) ? t : t - n + Tb;
            copy_bytes<kCols * (int)sizeof(T)>(kd, kbase + src * rowstride);
            copy_bytes<kCols * (int)sizeof(T)>(vd, vbase + src * rowstride);
            continue;
        }

        // pooled speech row: frames [j0, j1) of the prefill rows
        const int64_t i = t - Pb;
        const int64_t j0 = Pb + i * w;
        const int64_t j1 = (j0 + w < Pb + Tb) ? j0 + w : Pb + Tb;
        float u[kCols];
#pragma unroll
        for (int c = 0; c < kCols; c++) u[c] = __ldg(gate + h * D + lane * kCols + c);
        float mx = -INFINITY, sum = 0.f, ak[kCols], av[kCols];
#pragma unroll
        for (int c = 0; c < kCols; c++) ak[c] = av[c] = 0.f;
        for (int64_t j = j0; j < j1; j += 4) {
            // four frames in flight, then their logits and the online update
            float kx[4][kCols], vx[4][kCols], z[4];
#pragma unroll
            for (int f = 0; f < 4; f++) {
                if (j + f < j1) {
                    load_vec<T, kCols>(kbase + (j + f) * rowstride, kx[f]);
                    load_vec<T, kCols>(vbase + (j + f) * rowstride, vx[f]);
                }
            }
#pragma unroll
            for (int f = 0; f < 4; f++) {
                float s = 0.f;
                if (j + f < j1) {
#pragma unroll
                    for (int c = 0; c < kCols; c++) s = fmaf(u[c], kx[f][c], s);
                }
                z[f] = warp_sum(s);
            }
#pragma unroll
            for (int f = 0; f < 4; f++) {
                if (j + f >= j1) break;
                const float mnew = fmaxf(mx, z[f]);
                const float corr = expf(mx - mnew);  // 0 on the first frame
                const float e = expf(z[f] - mnew);
                sum = sum * corr + e;
#pragma unroll
                for (int c = 0; c < kCols; c++) {
                    ak[c] = fmaf(e, kx[f][c], ak[c] * corr);
                    av[c] = fmaf(e, vx[f][c], av[c] * corr);
                }
                mx = mnew;
            }
        }
        const float inv = 1.f / sum;
#pragma unroll
        for (int c = 0; c < kCols; c++) {
            ak[c] *= inv;
            av[c] *= inv;
        }
        store_vec<T, kCols>(kd, ak);
        store_vec<T, kCols>(vd, av);
    }
}

template <typename T, int D>
cudaError_t launch_pool_instance(const PoolArgs &a, int num_sms, cudaStream_t stream) {
    const int64_t tasks = a.full_rows * a.H_kv;
    const int64_t warps_per_block = 8;
    int64_t blocks = (tasks + warps_per_block - 1) / warps_per_block;
    const int64_t bmin = (a.B + 255) / 256;  // the length writers
    if (blocks < bmin) blocks = bmin;
    const int64_t cap = (int64_t)num_sms * 16;  // grid-stride beyond this
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    pool_kernel<T, D><<<(unsigned)blocks, 256, 0, stream>>>(
        static_cast<const T *>(a.k_full), static_cast<const T *>(a.v_full), a.full_off, a.P, a.T,
        a.N, a.gate, static_cast<T *>(a.k_cache), static_cast<T *>(a.v_cache), a.cache_off,
        a.len, a.B, a.full_rows, a.H_kv, a.w_eff, a.err);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_pool(const PoolArgs &a, int num_sms, cudaStream_t stream) {
    if (a.dtype == SPEECHKV_F32) {
        if (a.d == 64) return launch_pool_instance<float, 64>(a, num_sms, stream);
        if (a.d == 128) return launch_pool_instance<float, 128>(a, num_sms, stream);
    } else {
        if (a.d == 64) return launch_pool_instance<__nv_bfloat16, 64>(a, num_sms, stream);
        if (a.d == 128) return launch_pool_instance<__nv_bfloat16, 128>(a, num_sms, stream);
    }
    return cudaErrorInvalidValue;
}

}  // namespace speechkv
