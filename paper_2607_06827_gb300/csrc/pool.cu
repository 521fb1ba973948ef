// speechkv_pool: Eq. (pool) of the paper (Sec. III-B), run once per request
// and layer at prefill (Sec. III-C) -- writes the compressed cache rows of
// every (request, KV head) from the full-resolution prefill keys/values.
//
// Grid (X, B): the X CTAs of request b share its output rows in two phases.
//
//   copy phase    rows kept unchanged -- text before the speech (t < P), text
//                 after it (t >= P + n, prefill row t - n + T), or every row
//                 when w_eff = 1 (layers before l0).  One flat index over
//                 (row, 16-byte vector) for the whole CTA group; each thread
//                 moves several independent vectors of K and V per iteration.
//                 Bit-exact.
//   pooled phase  speech window i (t = P + i): one warp per (window, chunk of
//                 heads), one 16-byte vector of a head per lane, so a chunk is
//                 512 contiguous bytes of a token-major prefill row.  The
//                 gate logit u_h . k_j of a frame is a shuffle reduction over
//                 the lanes of its head (fixed order); up to kPoolFrames
//                 frames are loaded at once, their softmax weights taken in
//                 base 2 against the running maximum, and K and V
//                 accumulated in fp32 pairs (f32x2) with one rounding to the
//                 storage type at the end.
//
// Loaded vectors stay packed (16 bytes in four 32-bit registers) until they
// are used, which keeps the kernel small enough for several CTAs per SM: the
// loads of one warp are few, so the bandwidth comes from many warps in flight.
#include <math.h>

#include "common.cuh"
#include "launch.h"

namespace speechkv {
namespace {

constexpr int kPoolThreads = 256;
constexpr int kPoolWarps = kPoolThreads / 32;
constexpr int kPoolMinCtas = 2;   // CTAs per SM the register budget is set for
constexpr int kPoolFrames = 4;    // frames of a window loaded at once
constexpr int kCopyUnroll = 4;    // (K, V) vector pairs in flight per thread, copy phase

template <typename T, int D>
struct PoolCfg {
    static constexpr int kEpv = 16 / (int)sizeof(T);             // elements per 16-byte vector
    static constexpr int kVecPerHead = D * (int)sizeof(T) / 16;  // 8, 16 or 32
    static constexpr int kHeadsPerWarp = 32 / kVecPerHead;       // heads of one pooled task
    static_assert(kVecPerHead <= 32 && 32 % kVecPerHead == 0, "head layout");
};

// 16 bytes of T, widened to fp32 pairs (element 2k, 2k + 1 in pair k).
template <typename T>
__device__ __forceinline__ void widen2(const uint4 &r, float2 (&f)[8 / sizeof(T)]) {
    if constexpr (sizeof(T) == 4) {
        f[0] = make_float2(__uint_as_float(r.x), __uint_as_float(r.y));
        f[1] = make_float2(__uint_as_float(r.z), __uint_as_float(r.w));
    } else {
        f[0] = bf16x2_to_float2(r.x);
        f[1] = bf16x2_to_float2(r.y);
        f[2] = bf16x2_to_float2(r.z);
        f[3] = bf16x2_to_float2(r.w);
    }
}

// The same widening by byte permutes.  The accumulation pass uses this form
// so that the compiler does not keep the logit pass's widened keys alive
// (twice the registers of the packed words) to reuse them.
template <typename T>
__device__ __forceinline__ void widen2_prmt(const uint4 &r, float2 (&f)[8 / sizeof(T)]) {
    if constexpr (sizeof(T) == 4) {
        widen2<T>(r, f);
    } else {
        const uint32_t w[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
        for (int k = 0; k < 4; k++) {
            uint32_t lo, hi;
            // bytes 4..7 come from the zero operand: lo = w << 16, hi = w & 0xffff0000
            asm("prmt.b32 %0, %1, 0, 0x1054;" : "=r"(lo) : "r"(w[k]));
            asm("prmt.b32 %0, %1, 0, 0x3254;" : "=r"(hi) : "r"(w[k]));
            f[k] = make_float2(__uint_as_float(lo), __uint_as_float(hi));
        }
    }
}

template <typename T, int D>
__global__ void __launch_bounds__(kPoolThreads, kPoolMinCtas)
    pool_kernel(const T *__restrict__ kf, const T *__restrict__ vf,
                const int64_t *__restrict__ full_off, const int32_t *__restrict__ Pa,
                const int32_t *__restrict__ Ta, const int32_t *__restrict__ Na,
                const float *__restrict__ gate, T *__restrict__ kc, T *__restrict__ vc,
                const int64_t *__restrict__ cache_off, int32_t *__restrict__ len,
                int64_t full_rows, int H_kv, int w, CacheMap map, int *__restrict__ err) {
    using C = PoolCfg<T, D>;
    constexpr int EPV = C::kEpv, VH = C::kVecPerHead, HW = C::kHeadsPerWarp, NP = EPV / 2;
    const int b = blockIdx.y;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    const int64_t row0 = full_off[b], S = full_off[b + 1] - row0;
    const bool paged = map.table != nullptr;
    const int64_t base = paged ? 0 : cache_off[b];
    const int64_t cap = paged ? ((int64_t)map.max_blocks << map.bs_log2) : cache_off[b + 1] - base;
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

    const int64_t VR = (int64_t)H_kv * VH;  // 16-byte vectors per prefill row
    const uint4 *kb = reinterpret_cast<const uint4 *>(kf) + row0 * VR;
    const uint4 *vb = reinterpret_cast<const uint4 *>(vf) + row0 * VR;
    // element offset of (row t, vector v); -1 when the row's page is invalid
    auto dst_off = [&](int64_t t, int64_t v) -> int64_t {
        const int h = (int)(v / VH);
        const int64_t r = cache_row(map, b, h, t, H_kv, D, base, cap);
        if (r < 0) {
            report_error(err, SPEECHKV_ERR_INVALID_ARG);
            return -1;
        }
        return r + (v - (int64_t)h * VH) * EPV;
    };

    // ---- copy phase: copy row r is output row r for r < Pc, else the text
    // row after the speech; with w = 1 every row is a copy row.
    const int64_t Pc = w == 1 ? rows_out : (Pb < rows_out ? Pb : rows_out);
    const int64_t after0 = Pb + n;  // first output row after the speech
    const int64_t Ccopy = w == 1 ? rows_out : Pc + (rows_out > after0 ? rows_out - after0 : 0);
    {
        const int64_t g = (int64_t)blockIdx.x * kPoolThreads + threadIdx.x;
        const int64_t Sg = (int64_t)gridDim.x * kPoolThreads;
        int64_t r = g / VR, v = g - r * VR;
        const int64_t dr = Sg / VR, dv = Sg - dr * VR;
        while (r < Ccopy) {
            uint4 kx[kCopyUnroll], vx[kCopyUnroll];
            int64_t o[kCopyUnroll];  // destination element offset, -2 past the end
#pragma unroll
            for (int k = 0; k < kCopyUnroll; k++) {
                o[k] = -2;
                if (r < Ccopy) {
                    const bool before = r < Pc;
                    const int64_t src = before ? r : r - Pc + Pb + Tb;  // prefill row
                    kx[k] = __ldcs(kb + src * VR + v);
                    vx[k] = __ldcs(vb + src * VR + v);
                    o[k] = dst_off(before ? r : r - Pc + after0, v);
                }
                r += dr;
                v += dv;
                if (v >= VR) {
                    v -= VR;
                    r++;
                }
            }
#pragma unroll
            for (int k = 0; k < kCopyUnroll; k++) {
                if (o[k] == -2) break;  // the rows of later k are larger
                if (o[k] < 0) continue;  // invalid page (reported)
                *reinterpret_cast<uint4 *>(kc + o[k]) = kx[k];
                *reinterpret_cast<uint4 *>(vc + o[k]) = vx[k];
            }
        }
    }

    // ---- pooled phase: windows i < npool (those that fit the capacity)
    if (w == 1) return;
    const int64_t room = rows_out - Pb;
    const int64_t npool = room <= 0 ? 0 : (room < n ? room : n);
    const int nchunk = (H_kv + HW - 1) / HW;
    const int64_t tasks = npool * nchunk;
    constexpr float kLog2e = 1.4426950408889634f;
    for (int64_t task = (int64_t)blockIdx.x * kPoolWarps + warp; task < tasks;
         task += (int64_t)gridDim.x * kPoolWarps) {
        const int64_t i = task / nchunk;
        const int64_t vi = (task - i * nchunk) * 32 + lane;  // this lane's vector of the row
        const bool act = vi < VR;
        const int64_t j0 = Pb + i * w;
        const int64_t j1 = (j0 + w < Pb + Tb) ? j0 + w : Pb + Tb;

        // the lane's slice of the gate, scaled by log2(e): the softmax runs
        // in base 2 (2^(log2(e) z) = e^z)
        float2 u[NP];
        if (act) {
            const float4 *gp = reinterpret_cast<const float4 *>(gate + vi * EPV);
#pragma unroll
            for (int k = 0; k < NP; k += 2) {
                const float4 g4 = __ldg(gp + k / 2);
                u[k] = make_float2(g4.x * kLog2e, g4.y * kLog2e);
                u[k + 1] = make_float2(g4.z * kLog2e, g4.w * kLog2e);
            }
        } else {
#pragma unroll
            for (int k = 0; k < NP; k++) u[k] = make_float2(0.f, 0.f);
        }
        float m = -INFINITY, s = 0.f;
        float2 ak[NP], av[NP];
#pragma unroll
        for (int k = 0; k < NP; k++) ak[k] = av[k] = make_float2(0.f, 0.f);

        const uint4 *kp = kb + j0 * VR + vi, *vp = vb + j0 * VR + vi;
        for (int64_t j = j0; j < j1; j += kPoolFrames, kp += kPoolFrames * VR, vp += kPoolFrames * VR) {
            const int nf = j1 - j < kPoolFrames ? (int)(j1 - j) : kPoolFrames;
            uint4 kr[kPoolFrames], vr[kPoolFrames];
#pragma unroll
            for (int f = 0; f < kPoolFrames; f++) {
                if (act && f < nf) {
                    kr[f] = __ldcs(kp + f * VR);
                    vr[f] = __ldcs(vp + f * VR);
                } else {
                    kr[f] = vr[f] = make_uint4(0u, 0u, 0u, 0u);
                }
            }
            // base-2 logits of the frames, reduced over the head's lanes
            float z[kPoolFrames];
            float mb = m;
#pragma unroll
            for (int f = 0; f < kPoolFrames; f++) {
                float2 x[NP];
                widen2<T>(kr[f], x);
                float2 a2 = fmul2(u[0], x[0]);
#pragma unroll
                for (int k = 1; k < NP; k++) a2 = ffma2(u[k], x[k], a2);
                float acc = a2.x + a2.y;
#pragma unroll
                for (int o = 1; o < VH; o <<= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
                z[f] = acc;
                if (f < nf) mb = fmaxf(mb, acc);
            }
            if (j != j0) {  // rescale what the earlier frames of the window left
                const float corr = fast_exp2(m - mb);
                const float2 c2 = make_float2(corr, corr);
                s *= corr;
#pragma unroll
                for (int k = 0; k < NP; k++) {
                    ak[k] = fmul2(ak[k], c2);
                    av[k] = fmul2(av[k], c2);
                }
            }
#pragma unroll
            for (int f = 0; f < kPoolFrames; f++) {
                if (f >= nf) break;
                const float p = fast_exp2(z[f] - mb);
                const float2 p2 = make_float2(p, p);
                s += p;
                float2 xk[NP], xv[NP];
                widen2_prmt<T>(kr[f], xk);
                widen2_prmt<T>(vr[f], xv);
#pragma unroll
                for (int k = 0; k < NP; k++) {
                    ak[k] = ffma2(p2, xk[k], ak[k]);
                    av[k] = ffma2(p2, xv[k], av[k]);
                }
            }
            m = mb;
        }
        if (act) {
            const float inv = 1.f / s;
            float ok[EPV], ov[EPV];
#pragma unroll
            for (int k = 0; k < NP; k++) {
                ok[2 * k] = ak[k].x * inv;
                ok[2 * k + 1] = ak[k].y * inv;
                ov[2 * k] = av[k].x * inv;
                ov[2 * k + 1] = av[k].y * inv;
            }
            const int64_t o = dst_off(Pb + i, vi);
            if (o >= 0) {
                store_vec<T, EPV>(kc + o, ok);
                store_vec<T, EPV>(vc + o, ov);
            }
        }
    }
}

// ---------------------------------------------------------------------------
// Hidden-state pooling (the HS-compression variant): the same operator on
// whole hidden vectors, h^_i = sum_j alpha_j h_j with alpha = softmax over the
// window of gate . h_j.  A CTA of 256 threads handles one output row at a
// time; each thread owns up to kHsVpt 16-byte vectors of the row, the logits
// of up to kPoolFrames frames are reduced across the CTA together.
// ---------------------------------------------------------------------------
constexpr int kHsThreads = 256;
constexpr int kHsVptMax = 4;  // 16-byte vectors per thread: d_model * sizeof(T) <= 16 KB

template <typename T, int kHsVpt>
__global__ void __launch_bounds__(kHsThreads)
    pool_hidden_kernel(const T *__restrict__ hf, const int64_t *__restrict__ full_off,
                       const int32_t *__restrict__ Pa, const int32_t *__restrict__ Ta,
                       const int32_t *__restrict__ Na, const float *__restrict__ gate,
                       T *__restrict__ ho, const int64_t *__restrict__ out_off,
                       int32_t *__restrict__ len, int64_t full_rows, int64_t out_rows, int VR,
                       int w, int *__restrict__ err) {
    constexpr int EPV = 16 / (int)sizeof(T), NP = EPV / 2;
    constexpr int kWarps = kHsThreads / 32;
    __shared__ float red[kPoolFrames][kWarps];
    const int b = blockIdx.y;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    const int64_t row0 = full_off[b], S = full_off[b + 1] - row0;
    const int64_t base = out_off[b], cap = out_off[b + 1] - base;
    const int64_t Pb = Pa[b], Tb = Ta[b], Nb = Na[b];
    const int64_t n = (Tb + w - 1) / w;
    const int64_t L = Pb + n + Nb;
    const bool bad = Pb < 0 || Tb < 0 || Nb < 0 || S != Pb + Tb + Nb || cap < 0 || row0 < 0 ||
                     full_off[b + 1] > full_rows || base < 0 || out_off[b + 1] > out_rows;
    if (blockIdx.x == 0 && tid == 0) {
        if (bad)
            report_error(err, SPEECHKV_ERR_INVALID_ARG);
        else if (L > cap)
            report_error(err, SPEECHKV_ERR_CAPACITY);
        len[b] = (int32_t)(bad ? 0 : (L < cap ? L : cap));
    }
    if (bad) return;
    const int64_t rows_out = L < cap ? L : cap;
    const uint4 *src = reinterpret_cast<const uint4 *>(hf) + row0 * VR;
    uint4 *dst = reinterpret_cast<uint4 *>(ho) + base * VR;

    // the thread's slice of the gate, scaled by log2(e) (softmax in base 2)
    constexpr float kLog2e = 1.4426950408889634f;
    float2 u[kHsVpt][NP];
#pragma unroll
    for (int x = 0; x < kHsVpt; x++) {
        const int v = tid + x * kHsThreads;
#pragma unroll
        for (int k = 0; k < NP; k++) {
            u[x][k] = v < VR ? make_float2(gate[v * EPV + 2 * k] * kLog2e,
                                           gate[v * EPV + 2 * k + 1] * kLog2e)
                             : make_float2(0.f, 0.f);
        }
    }

    for (int64_t t = blockIdx.x; t < rows_out; t += gridDim.x) {
        if (t < Pb || t >= Pb + n || w == 1) {
            // text row (or no pooling): bit-exact copy
            const int64_t s = (t < Pb || w == 1) ? t : t - n + Tb;
#pragma unroll
            for (int x = 0; x < kHsVpt; x++) {
                const int v = tid + x * kHsThreads;
                if (v < VR) dst[t * VR + v] = __ldcs(src + s * VR + v);
            }
            continue;
        }
        const int64_t j0 = Pb + (t - Pb) * w;
        const int64_t j1 = (j0 + w < Pb + Tb) ? j0 + w : Pb + Tb;
        float m = -INFINITY, l = 0.f;
        float2 acc[kHsVpt][NP];
#pragma unroll
        for (int x = 0; x < kHsVpt; x++)
#pragma unroll
            for (int k = 0; k < NP; k++) acc[x][k] = make_float2(0.f, 0.f);
        for (int64_t j = j0; j < j1; j += kPoolFrames) {
            const int nf = j1 - j < kPoolFrames ? (int)(j1 - j) : kPoolFrames;
            uint4 raw[kPoolFrames][kHsVpt];
            float z[kPoolFrames];
#pragma unroll
            for (int f = 0; f < kPoolFrames; f++) {
                float2 a2 = make_float2(0.f, 0.f);
#pragma unroll
                for (int x = 0; x < kHsVpt; x++) {
                    const int v = tid + x * kHsThreads;
                    raw[f][x] = (f < nf && v < VR) ? __ldcs(src + (j + f) * VR + v)
                                                   : make_uint4(0u, 0u, 0u, 0u);
                    float2 e[NP];
                    widen2<T>(raw[f][x], e);
#pragma unroll
                    for (int k = 0; k < NP; k++) a2 = ffma2(u[x][k], e[k], a2);
                }
                z[f] = warp_sum(a2.x + a2.y);
            }
            // CTA-wide sums of the frames' logits (fixed order: deterministic)
            if (lane == 0)
#pragma unroll
                for (int f = 0; f < kPoolFrames; f++) red[f][warp] = z[f];
            __syncthreads();
            float mb = m;
#pragma unroll
            for (int f = 0; f < kPoolFrames; f++) {
                float zz = 0.f;
#pragma unroll
                for (int x = 0; x < kWarps; x++) zz += red[f][x];
                z[f] = zz;
                if (f < nf) mb = fmaxf(mb, zz);
            }
            __syncthreads();  // red[] is rewritten by the next frames
            const float corr = fast_exp2(m - mb);  // 0 on the first frames
            l *= corr;
#pragma unroll
            for (int x = 0; x < kHsVpt; x++)
#pragma unroll
                for (int k = 0; k < NP; k++) acc[x][k] = fmul2(acc[x][k], make_float2(corr, corr));
#pragma unroll
            for (int f = 0; f < kPoolFrames; f++) {
                if (f >= nf) break;
                const float p = fast_exp2(z[f] - mb);
                l += p;
#pragma unroll
                for (int x = 0; x < kHsVpt; x++) {
                    float2 e[NP];
                    widen2_prmt<T>(raw[f][x], e);
#pragma unroll
                    for (int k = 0; k < NP; k++) acc[x][k] = ffma2(make_float2(p, p), e[k], acc[x][k]);
                }
            }
            m = mb;
        }
        const float inv = 1.f / l;
#pragma unroll
        for (int x = 0; x < kHsVpt; x++) {
            const int v = tid + x * kHsThreads;
            if (v >= VR) continue;
            float o[EPV];
#pragma unroll
            for (int k = 0; k < NP; k++) {
                o[2 * k] = acc[x][k].x * inv;
                o[2 * k + 1] = acc[x][k].y * inv;
            }
            store_vec<T, EPV>(reinterpret_cast<T *>(dst + t * VR + v), o);
        }
    }
}

template <typename T, int VPT>
cudaError_t launch_pool_hidden_vpt(const PoolHiddenArgs &a, const dim3 &grid, int VR,
                                   cudaStream_t stream) {
    pool_hidden_kernel<T, VPT><<<grid, kHsThreads, 0, stream>>>(
        static_cast<const T *>(a.h_full), a.full_off, a.P, a.T, a.N, a.gate,
        static_cast<T *>(a.h_out), a.out_off, a.len, a.full_rows, a.out_rows, VR, a.w, a.err);
    return cudaGetLastError();
}

template <typename T>
cudaError_t launch_pool_hidden_instance(const PoolHiddenArgs &a, int num_sms,
                                        cudaStream_t stream) {
    int64_t x = ((int64_t)4 * num_sms + a.B - 1) / a.B;
    if (x < 1) x = 1;
    if (x > 65535) x = 65535;
    const dim3 grid((unsigned)x, (unsigned)a.B);
    const int VR = (int)((int64_t)a.d_model * (int64_t)sizeof(T) / 16);
    const int vpt = (VR + kHsThreads - 1) / kHsThreads;
    if (vpt <= 1) return launch_pool_hidden_vpt<T, 1>(a, grid, VR, stream);
    if (vpt <= 2) return launch_pool_hidden_vpt<T, 2>(a, grid, VR, stream);
    return launch_pool_hidden_vpt<T, kHsVptMax>(a, grid, VR, stream);
}

template <typename T, int D>
cudaError_t launch_pool_instance(const PoolArgs &a, int num_sms, cudaStream_t stream) {
    // enough CTAs over the whole batch to fill every SM once, at least one
    // per request
    static int per_sm = 0;
    if (per_sm == 0) {
        int occ = 0;
        cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, pool_kernel<T, D>,
                                                                      kPoolThreads, 0);
        if (e != cudaSuccess) return e;
        per_sm = occ > 0 ? occ : 1;
    }
    int64_t x = ((int64_t)per_sm * num_sms + a.B - 1) / a.B;
    if (x < 1) x = 1;
    if (x > 65535) x = 65535;
    const dim3 grid((unsigned)x, (unsigned)a.B);
    pool_kernel<T, D><<<grid, kPoolThreads, 0, stream>>>(
        static_cast<const T *>(a.k_full), static_cast<const T *>(a.v_full), a.full_off, a.P, a.T,
        a.N, a.gate, static_cast<T *>(a.k_cache), static_cast<T *>(a.v_cache), a.cache_off,
        a.len, a.full_rows, a.H_kv, a.w_eff, a.map, a.err);
    return cudaGetLastError();
}

}  // namespace

bool pool_hidden_supported(speechkv_dtype dtype, int d_model) {
    const int es = dtype == SPEECHKV_F32 ? 4 : 2;
    return d_model > 0 && (d_model * es) % 16 == 0 && d_model * es <= kHsVptMax * kHsThreads * 16;
}

cudaError_t launch_pool_hidden(const PoolHiddenArgs &a, int num_sms, cudaStream_t stream) {
    if (a.B > 65535) return cudaErrorInvalidValue;  // grid.y limit
    if (a.dtype == SPEECHKV_F32) return launch_pool_hidden_instance<float>(a, num_sms, stream);
    return launch_pool_hidden_instance<__nv_bfloat16>(a, num_sms, stream);
}

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
