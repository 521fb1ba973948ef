// speechkv_pool: Eq. (pool) of the paper (Sec. III-B), run once per request
// and layer at prefill (Sec. III-C) -- writes the compressed cache rows of
// every (request, KV head) from the full-resolution prefill keys/values.
//
// Grid (X, B): the X CTAs of request b share its output rows.  A warp task is
// (output row t, chunk of heads): one chunk is at most 2 KB of a token-major
// prefill row (8 heads of d = 128 in bf16), read with 16-byte loads that
// cover 512 contiguous bytes per warp instruction.  Each 16-byte vector
// belongs to one head, and the vectors of a head sit on consecutive lanes,
// so a head's gate logit u_h . k_j is a shuffle reduction over those lanes
// (deterministic order).
//
//   t <  P            text before the speech: copy prefill row t
//   t <  P + n        speech window i = t - P: online softmax over the gate
//                     logits of frames P + i*w .. min(.., P + T) - 1 (up to 4
//                     frames in flight), weighted sums of keys and values in
//                     fp32, one rounding to the storage type
//   t <  P + n + N    text after the speech: copy prefill row t - n + T
//
// With w_eff = 1 (layers before l0) every row is a bit-exact copy.
#include <math.h>

#include "common.cuh"
#include "launch.h"

namespace speechkv {
namespace {

constexpr int kPoolWarps = 8;
constexpr int kPoolFrames = 4;  // frames of a window loaded at once

template <typename T, int D>
struct PoolCfg {
    static constexpr int kEpv = 16 / (int)sizeof(T);             // elements per 16-byte vector
    static constexpr int kVecPerHead = D * (int)sizeof(T) / 16;  // 8, 16 or 32
    static constexpr int kHeadsPerChunk = 2048 / (D * (int)sizeof(T));
    static constexpr int kVpl = kHeadsPerChunk * kVecPerHead / 32;  // vectors per lane
    static_assert(kVecPerHead <= 32 && 32 % kVecPerHead == 0, "head layout");
    static_assert(kVpl >= 1 && kVpl * 32 * 16 == 2048, "chunk layout");
};

template <typename T, int D>
__global__ void __launch_bounds__(kPoolWarps * 32)
    pool_kernel(const T *__restrict__ kf, const T *__restrict__ vf,
                const int64_t *__restrict__ full_off, const int32_t *__restrict__ Pa,
                const int32_t *__restrict__ Ta, const int32_t *__restrict__ Na,
                const float *__restrict__ gate, T *__restrict__ kc, T *__restrict__ vc,
                const int64_t *__restrict__ cache_off, int32_t *__restrict__ len,
                int64_t full_rows, int H_kv, int w, int *__restrict__ err) {
    using C = PoolCfg<T, D>;
    constexpr int VPL = C::kVpl, EPV = C::kEpv, VH = C::kVecPerHead;
    const int b = blockIdx.y;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    const int64_t row0 = full_off[b], S = full_off[b + 1] - row0;
    const int64_t base = cache_off[b], cap = cache_off[b + 1] - base;
    const int64_t Pb = Pa[b], Tb = Ta[b], Nb = Na[b];
    const int64_t n = (Tb + w - 1) / w;
    const int64_t L = Pb + n + Nb;
    const bool bad = Pb < 0 || Tb < 0 || Nb < 0 || S != Pb + Tb + Nb || cap < 0 || row0 < 0 ||
                     full_off[b + 1] > full_rows || base < 0;
    if (blockIdx.x == 0 && threadIdx.x == 0) {
        if (bad)
            report_error(err, SPEECHKV_ERR_INVALID_ARG);
        else if (L > cap)
            report_error(err, SPEECHKV_ERR_CAPACITY);
        len[b] = (int32_t)(bad ? 0 : (L < cap ? L : cap));
    }
    if (bad) return;
    const int64_t rows_out = L < cap ? L : cap;  // rows beyond the capacity are not written

    const int nchunk = (H_kv + C::kHeadsPerChunk - 1) / C::kHeadsPerChunk;
    const int64_t tasks = rows_out * nchunk;
    const int64_t rowstride = (int64_t)H_kv * D;  // elements per prefill row
    for (int64_t task = (int64_t)blockIdx.x * kPoolWarps + warp; task < tasks;
         task += (int64_t)gridDim.x * kPoolWarps) {
        const int64_t t = task / nchunk;
        const int h0 = (int)(task - t * nchunk) * C::kHeadsPerChunk;
        const int hc = H_kv - h0 < C::kHeadsPerChunk ? H_kv - h0 : C::kHeadsPerChunk;
        const int nv = hc * VH;  // vectors of this chunk
        // the lane's vectors: v = lane + 32 i, of head h0 + v / VH
        bool act[VPL];
        int hv[VPL], cv[VPL];
#pragma unroll
        for (int i = 0; i < VPL; i++) {
            const int v = lane + 32 * i;
            act[i] = v < nv;
            hv[i] = h0 + v / VH;
            cv[i] = (v % VH) * EPV;
        }
        auto dst_of = [&](T *cache, int i) {
            return cache + (base * H_kv + (int64_t)hv[i] * cap + t) * D + cv[i];
        };
        // prefill row 0 of request b, this lane's first vector of the chunk
        const T *kb = kf + row0 * rowstride + (int64_t)h0 * D + lane * EPV;
        const T *vb = vf + row0 * rowstride + (int64_t)h0 * D + lane * EPV;

        if (t < Pb || t >= Pb + n || w == 1) {
            // text row (or no pooling): bit-exact copy
            const int64_t src = (t < Pb || w == 1) ? t : t - n + Tb;
#pragma unroll
            for (int i = 0; i < VPL; i++) {
                if (!act[i]) continue;
                copy_bytes<16>(dst_of(kc, i), kb + src * rowstride + 32 * i * EPV);
                copy_bytes<16>(dst_of(vc, i), vb + src * rowstride + 32 * i * EPV);
            }
            continue;
        }

        // pooled speech row: frames [j0, j1) of the prefill rows
        const int64_t j0 = Pb + (t - Pb) * w;
        const int64_t j1 = (j0 + w < Pb + Tb) ? j0 + w : Pb + Tb;
        float u[VPL][EPV];
#pragma unroll
        for (int i = 0; i < VPL; i++)
#pragma unroll
            for (int e = 0; e < EPV; e++)
                u[i][e] = act[i] ? __ldg(gate + hv[i] * D + cv[i] + e) : 0.f;
        float mx[VPL], sum[VPL], ak[VPL][EPV], av[VPL][EPV];
#pragma unroll
        for (int i = 0; i < VPL; i++) {
            mx[i] = -INFINITY;
            sum[i] = 0.f;
#pragma unroll
            for (int e = 0; e < EPV; e++) ak[i][e] = av[i][e] = 0.f;
        }
        for (int64_t j = j0; j < j1; j += kPoolFrames) {
            float kx[kPoolFrames][VPL][EPV], vx[kPoolFrames][VPL][EPV];
#pragma unroll
            for (int f = 0; f < kPoolFrames; f++)
#pragma unroll
                for (int i = 0; i < VPL; i++) {
                    if (j + f < j1 && act[i]) {
                        load_vec<T, EPV>(kb + (j + f) * rowstride + 32 * i * EPV, kx[f][i]);
                        load_vec<T, EPV>(vb + (j + f) * rowstride + 32 * i * EPV, vx[f][i]);
                    } else {
#pragma unroll
                        for (int e = 0; e < EPV; e++) kx[f][i][e] = vx[f][i][e] = 0.f;
                    }
                }
#pragma unroll
            for (int f = 0; f < kPoolFrames; f++) {
                if (j + f >= j1) break;
#pragma unroll
                for (int i = 0; i < VPL; i++) {
                    // logit of this vector's head: reduce over its VH lanes
                    float z = 0.f;
#pragma unroll
                    for (int e = 0; e < EPV; e++) z = fmaf(u[i][e], kx[f][i][e], z);
#pragma unroll
                    for (int o = 1; o < VH; o <<= 1) z += __shfl_xor_sync(0xffffffffu, z, o);
                    const float mnew = fmaxf(mx[i], z);
                    const float corr = expf(mx[i] - mnew);  // 0 on the first frame
                    const float p = expf(z - mnew);
                    sum[i] = sum[i] * corr + p;
#pragma unroll
                    for (int e = 0; e < EPV; e++) {
                        ak[i][e] = fmaf(p, kx[f][i][e], ak[i][e] * corr);
                        av[i][e] = fmaf(p, vx[f][i][e], av[i][e] * corr);
                    }
                    mx[i] = mnew;
                }
            }
        }
#pragma unroll
        for (int i = 0; i < VPL; i++) {
            if (!act[i]) continue;
            const float inv = 1.f / sum[i];
#pragma unroll
            for (int e = 0; e < EPV; e++) {
                ak[i][e] *= inv;
                av[i][e] *= inv;
            }
            store_vec<T, EPV>(dst_of(kc, i), ak[i]);
            store_vec<T, EPV>(dst_of(vc, i), av[i]);
        }
    }
}

template <typename T, int D>
cudaError_t launch_pool_instance(const PoolArgs &a, int num_sms, cudaStream_t stream) {
    // about four CTAs per SM over the whole batch, at least one per request
    int x = (4 * num_sms + a.B - 1) / a.B;
    if (x < 1) x = 1;
    if (x > 65535) x = 65535;
    const dim3 grid((unsigned)x, (unsigned)a.B);
    pool_kernel<T, D><<<grid, kPoolWarps * 32, 0, stream>>>(
        static_cast<const T *>(a.k_full), static_cast<const T *>(a.v_full), a.full_off, a.P, a.T,
        a.N, a.gate, static_cast<T *>(a.k_cache), static_cast<T *>(a.v_cache), a.cache_off,
        a.len, a.full_rows, a.H_kv, a.w_eff, a.err);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_pool(const PoolArgs &a, int num_sms, cudaStream_t stream) {
    if (a.B > 65535) return cudaErrorInvalidValue;  // grid.y limit
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
