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
// window of gate . h_j.
//
// One team of kG warps pools one output row at a time, each lane owning up
// to four 16-byte vectors of the row (a 4 KB bf16 row: four warps), so the
// logits of a window need one shuffle reduction per frame and a two-value
// exchange between the team's warps, no CTA-wide barrier.  The input rows
// stream through shared memory: the team leader copies up to kPoolFrames
// consecutive rows at a time (a window, a part of a long window, or one kept
// text row -- always contiguous in the token-major input) with cp.async.bulk
// into the team's ring of NS stages, completion signalled on an mbarrier per
// stage.  The team moves a landed stage to registers and the leader refills
// it at once, before the logits, the window's softmax (running maximum
// across the parts of a long window, base 2) and the weighted sum in fp32
// pairs are computed, so the copies in flight cover nearly the whole ring.
// The CTA holds NT teams; their rings together take most of the SM's shared
// memory.
// ---------------------------------------------------------------------------
constexpr int kHsMaxWarps = 16;  // 12 for four vectors per lane (registers)
constexpr int kHsMaxTeams = 8;
constexpr int kHsMaxStages = 4;
constexpr int kHsRingBytes = 200 * 1024;  // the teams' rings, one CTA per SM

__device__ __forceinline__ void team_sync(int id, int nthreads) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

// Barrier of a team that also ORs a predicate over its threads.
__device__ __forceinline__ bool team_any(int id, int nthreads, bool pred) {
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.u32 q, %1, 0;\n\t"
        "bar.red.or.pred p, %2, %3, q;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(r)
        : "r"((uint32_t)pred), "r"(id), "r"(nthreads)
        : "memory");
    return r != 0;
}

// Input rows [j, j1) that output row t of a request reads: the window of
// speech frames for a pooled row, the one kept row otherwise.
__device__ __forceinline__ bool hs_row_span(int64_t t, int64_t Pb, int64_t Tb, int64_t n, int w,
                                            int64_t &j, int64_t &j1) {
    if (t < Pb || t >= Pb + n || w == 1) {
        j = (t < Pb || w == 1) ? t : t - n + Tb;
        j1 = j + 1;
        return true;  // kept as is
    }
    j = Pb + (t - Pb) * w;
    j1 = (j + w < Pb + Tb) ? j + w : Pb + Tb;
    return false;
}

template <typename T, int kVpl, int kG>
__global__ void __launch_bounds__(kVpl >= 4 ? 384 : kHsMaxWarps * 32)
    pool_hidden_kernel(const T *__restrict__ hf, const int64_t *__restrict__ full_off,
                       const int32_t *__restrict__ Pa, const int32_t *__restrict__ Ta,
                       const int32_t *__restrict__ Na, const float *__restrict__ gate,
                       T *__restrict__ ho, const int64_t *__restrict__ out_off,
                       int32_t *__restrict__ len, int64_t full_rows, int64_t out_rows, int VR,
                       int w, int NT, int NS, int *__restrict__ err) {
    constexpr int EPV = 16 / (int)sizeof(T), NP = EPV / 2;
    constexpr int kTeamThreads = 32 * kG;
    extern __shared__ __align__(128) unsigned char ring[];
    __shared__ __align__(8) uint64_t full[kHsMaxTeams * kHsMaxStages];
    __shared__ float red[kHsMaxTeams][2][kPoolFrames][kG];
    const int b = blockIdx.y;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int team = warp / kG, tw = warp % kG;

    const int64_t row0 = full_off[b], S = full_off[b + 1] - row0;
    const int64_t base = out_off[b], cap = out_off[b + 1] - base;
    const int64_t Pb = Pa[b], Tb = Ta[b], Nb = Na[b];
    const int64_t n = (Tb + w - 1) / w;
    const int64_t L = Pb + n + Nb;
    const bool bad = Pb < 0 || Tb < 0 || Nb < 0 || S != Pb + Tb + Nb || cap < 0 || row0 < 0 ||
                     full_off[b + 1] > full_rows || base < 0 || out_off[b + 1] > out_rows;
    if (blockIdx.x == 0 && threadIdx.x == 0) {
        if (bad)
            report_error(err, SPEECHKV_ERR_INVALID_ARG);
        else if (L > cap)
            report_error(err, SPEECHKV_ERR_CAPACITY);
        len[b] = (int32_t)(bad ? 0 : (L < cap ? L : cap));
    }
    if (bad) return;  // the whole CTA, before any barrier
    const int64_t rows_out = L < cap ? L : cap;
    const uint32_t row_bytes = (uint32_t)VR * 16u;
    const uint32_t stage_bytes = kPoolFrames * row_bytes;

    if (threadIdx.x == 0) {
        for (int s = 0; s < NT * NS; s++) mbar_init(&full[s], 1);
        fence_mbar_init();
    }
    __syncthreads();
    if (team >= NT) return;

    unsigned char *tring = ring + (size_t)team * NS * stage_bytes;
    uint64_t *tfull = full + team * NS;
    const int bar_id = 1 + team;  // named barrier of the team (kG > 1)
    const bool leader = tw == 0 && lane == 0;
    const int64_t R = (int64_t)gridDim.x * NT;  // teams working on this request
    const int64_t first = (int64_t)blockIdx.x * NT + team;
    const unsigned char *src = reinterpret_cast<const unsigned char *>(hf) + row0 * (int64_t)row_bytes;

    // The leader's copy pointer runs NS chunks ahead of the team.
    int64_t pt = first, pj = 0, pj1 = 0;
    if (pt < rows_out) hs_row_span(pt, Pb, Tb, n, w, pj, pj1);
    int ps = 0;
    auto issue = [&]() {
        if (pt >= rows_out) return;
        const int nf = pj1 - pj < kPoolFrames ? (int)(pj1 - pj) : kPoolFrames;
        mbar_arrive_expect_tx(&tfull[ps], (uint32_t)nf * row_bytes);
        bulk_g2s(tring + (size_t)ps * stage_bytes, src + pj * (int64_t)row_bytes,
                 (uint32_t)nf * row_bytes, &tfull[ps]);
        if (++ps == NS) ps = 0;
        pj += kPoolFrames;
        if (pj >= pj1) {
            pt += R;
            if (pt < rows_out) hs_row_span(pt, Pb, Tb, n, w, pj, pj1);
        }
    };
    int64_t n_issued = 0, n_done = 0;
    if (leader)
        for (int s = 0; s < NS && pt < rows_out; s++) {
            issue();
            n_issued++;
        }

    // the lane's vectors of the row: vec(x) = tw * 32 * kVpl + x * 32 + lane
    const int vbase = tw * 32 * kVpl + lane;
    constexpr float kLog2e = 1.4426950408889634f;
    float2 u[kVpl][NP];
#pragma unroll
    for (int x = 0; x < kVpl; x++) {
        const int v = vbase + x * 32;
#pragma unroll
        for (int k = 0; k < NP; k++)
            u[x][k] = v < VR ? make_float2(gate[v * EPV + 2 * k] * kLog2e,
                                           gate[v * EPV + 2 * k + 1] * kLog2e)
                             : make_float2(0.f, 0.f);
    }
    uint4 *dst = reinterpret_cast<uint4 *>(ho) + base * (int64_t)VR;

    int sc = 0;        // stage of the next chunk
    uint32_t ph = 0;   // its phase parity
    int rb = 0;        // red[] buffer of the next exchange (kG > 1)
    bool stop = false;
    for (int64_t t = first; t < rows_out && !stop; t += R) {
        int64_t j, j1;
        const bool kept = hs_row_span(t, Pb, Tb, n, w, j, j1);
        float m = -INFINITY, l = 0.f;
        float2 acc[kVpl][NP];
#pragma unroll
        for (int x = 0; x < kVpl; x++)
#pragma unroll
            for (int k = 0; k < NP; k++) acc[x][k] = make_float2(0.f, 0.f);
        for (; j < j1; j += kPoolFrames) {
            const int nf = j1 - j < kPoolFrames ? (int)(j1 - j) : kPoolFrames;
            const bool landed = mbar_wait_bounded(&tfull[sc], ph, err);
            const uint4 *st = reinterpret_cast<const uint4 *>(tring + (size_t)sc * stage_bytes);
            uint4 raw[kPoolFrames][kVpl];
#pragma unroll
            for (int f = 0; f < kPoolFrames; f++)
#pragma unroll
                for (int x = 0; x < kVpl; x++) {
                    const int v = vbase + x * 32;
                    raw[f][x] = (landed && f < nf && v < VR) ? st[f * VR + v]
                                                             : make_uint4(0u, 0u, 0u, 0u);
                }
            // one barrier: every thread of the team has its words (the stage
            // may be refilled) and every thread's wait succeeded
            const bool failed = kG > 1 ? team_any(bar_id, kTeamThreads, !landed)
                                       : !__all_sync(0xffffffffu, landed);
            if (failed) {
                stop = true;
                break;
            }
            n_done++;
            if (leader && pt < rows_out) {
                issue();
                n_issued++;
            }
            if (++sc == NS) {
                sc = 0;
                ph ^= 1;
            }
            if (kept) {
                // text row (or no pooling): bit-exact copy
#pragma unroll
                for (int x = 0; x < kVpl; x++) {
                    const int v = vbase + x * 32;
                    if (v < VR) __stcs(dst + t * VR + v, raw[0][x]);
                }
                continue;
            }
            float z[kPoolFrames];
#pragma unroll
            for (int f = 0; f < kPoolFrames; f++) {
                float2 a2 = make_float2(0.f, 0.f);
#pragma unroll
                for (int x = 0; x < kVpl; x++) {
                    float2 e[NP];
                    widen2<T>(raw[f][x], e);
#pragma unroll
                    for (int k = 0; k < NP; k++) a2 = ffma2(u[x][k], e[k], a2);
                }
                z[f] = warp_sum(a2.x + a2.y);
            }
            if (kG > 1) {
                // the team's warps exchange their partial logits (fixed
                // order); red[] alternates between two buffers, so the
                // barriers of the next chunk separate these reads from the
                // next writes of the buffer
                if (lane == 0)
#pragma unroll
                    for (int f = 0; f < kPoolFrames; f++) red[team][rb][f][tw] = z[f];
                team_sync(bar_id, kTeamThreads);
#pragma unroll
                for (int f = 0; f < kPoolFrames; f++) {
                    float zz = 0.f;
#pragma unroll
                    for (int g = 0; g < kG; g++) zz += red[team][rb][f][g];
                    z[f] = zz;
                }
                rb ^= 1;
            }
            float mb = m;
#pragma unroll
            for (int f = 0; f < kPoolFrames; f++)
                if (f < nf) mb = fmaxf(mb, z[f]);
            const float corr = fast_exp2(m - mb);  // 0 on the first frames
            l *= corr;
#pragma unroll
            for (int x = 0; x < kVpl; x++)
#pragma unroll
                for (int k = 0; k < NP; k++) acc[x][k] = fmul2(acc[x][k], make_float2(corr, corr));
#pragma unroll
            for (int f = 0; f < kPoolFrames; f++) {
                if (f < nf) {
                    const float p = fast_exp2(z[f] - mb);
                    l += p;
#pragma unroll
                    for (int x = 0; x < kVpl; x++) {
                        float2 e[NP];
                        widen2_prmt<T>(raw[f][x], e);
#pragma unroll
                        for (int k = 0; k < NP; k++)
                            acc[x][k] = ffma2(make_float2(p, p), e[k], acc[x][k]);
                    }
                }
            }
            m = mb;
        }
        if (stop || kept) continue;
        const float inv = 1.f / l;
#pragma unroll
        for (int x = 0; x < kVpl; x++) {
            const int v = vbase + x * 32;
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
    if (stop && leader) {
        // the copies still in flight land before the CTA's shared memory
        // goes away
        for (int64_t k = n_done; k < n_issued; k++) {
            mbar_wait_bounded(&tfull[sc], ph, err);
            if (++sc == NS) {
                sc = 0;
                ph ^= 1;
            }
        }
    }
}

// Vectors per lane and warps per team for rows of VR 16-byte vectors; the
// teams per CTA and stages per team that fit the ring budget.
struct HsPlan {
    int vpl, g, nt, ns;
};
inline HsPlan hs_plan(int VR) {
    HsPlan p;
    // two vectors per lane up to 4 KB rows (teams of up to four warps, up
    // to 16 warps per CTA), four for wider rows (registers: 12 warps)
    p.vpl = VR <= 32 ? 1 : VR <= 256 ? 2 : 4;
    // warps per team, rounded up to a compiled team size (1, 2, 4 or 8); the
    // lanes past the row's last vector idle
    const int g = (VR + 32 * p.vpl - 1) / (32 * p.vpl);
    p.g = g <= 1 ? 1 : g <= 2 ? 2 : g <= 4 ? 4 : 8;
    const int max_warps = p.vpl >= 4 ? 12 : kHsMaxWarps;
    const int64_t stage = (int64_t)kPoolFrames * VR * 16;
    const int slots = (int)(kHsRingBytes / stage);  // >= 3 for rows of up to 16 KB
    // as many teams as the warp budget allows with two stages each, then
    // the stages that the ring budget leaves for each team
    p.nt = slots / 2;
    if (p.nt > kHsMaxTeams) p.nt = kHsMaxTeams;
    if (p.nt > max_warps / p.g) p.nt = max_warps / p.g;
    if (p.nt < 1) p.nt = 1;
    p.ns = slots / p.nt;
    if (p.ns > kHsMaxStages) p.ns = kHsMaxStages;
    return p;
}

template <typename T, int kVpl, int kG>
cudaError_t launch_pool_hidden_cfg(const PoolHiddenArgs &a, const HsPlan &p, int num_sms, int VR,
                                   cudaStream_t stream) {
    auto kern = pool_hidden_kernel<T, kVpl, kG>;
    static int configured_device_mask = 0;  // devices with the smem attribute set
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (!(dev < 31 && (__atomic_load_n(&configured_device_mask, __ATOMIC_ACQUIRE) & (1 << dev)))) {
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kHsRingBytes);
        if (e != cudaSuccess) return e;
        if (dev < 31) __atomic_fetch_or(&configured_device_mask, 1 << dev, __ATOMIC_ACQ_REL);
    }
    int64_t x = ((int64_t)num_sms + a.B - 1) / a.B;  // one CTA per SM over the batch
    if (x < 1) x = 1;
    if (x > 65535) x = 65535;
    const dim3 grid((unsigned)x, (unsigned)a.B);
    const size_t smem = (size_t)p.nt * p.ns * kPoolFrames * VR * 16;
    kern<<<grid, p.nt * kG * 32, smem, stream>>>(
        static_cast<const T *>(a.h_full), a.full_off, a.P, a.T, a.N, a.gate,
        static_cast<T *>(a.h_out), a.out_off, a.len, a.full_rows, a.out_rows, VR, a.w, p.nt, p.ns,
        a.err);
    return cudaGetLastError();
}

template <typename T>
cudaError_t launch_pool_hidden_instance(const PoolHiddenArgs &a, int num_sms,
                                        cudaStream_t stream) {
    const int VR = (int)((int64_t)a.d_model * (int64_t)sizeof(T) / 16);
    const HsPlan p = hs_plan(VR);
    // (vpl, g): (1, 1) rows of up to 32 vectors; (2, 1 / 2 / 4) up to 256;
    // (4, 4 / 8) up to 1024 -- a team covers 32 * vpl * g >= VR vectors
    if (p.vpl == 4)
        return p.g == 8 ? launch_pool_hidden_cfg<T, 4, 8>(a, p, num_sms, VR, stream)
                        : launch_pool_hidden_cfg<T, 4, 4>(a, p, num_sms, VR, stream);
    if (p.vpl == 2) {
        if (p.g == 4) return launch_pool_hidden_cfg<T, 2, 4>(a, p, num_sms, VR, stream);
        if (p.g == 2) return launch_pool_hidden_cfg<T, 2, 2>(a, p, num_sms, VR, stream);
        return launch_pool_hidden_cfg<T, 2, 1>(a, p, num_sms, VR, stream);
    }
    return launch_pool_hidden_cfg<T, 1, 1>(a, p, num_sms, VR, stream);
}

template <typename T, int D>
cudaError_t launch_pool_instance(const PoolArgs &a, int num_sms, cudaStream_t stream) {
    // enough CTAs over the whole batch to fill every SM once, at least one
    // per request; the occupancy is cached per device (a racing first use
    // stores the same value, atomically)
    constexpr int kDevs = 64;
    static int occ_cache[kDevs] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const bool cacheable = dev >= 0 && dev < kDevs;
    int per_sm = cacheable ? __atomic_load_n(&occ_cache[dev], __ATOMIC_ACQUIRE) : 0;
    if (per_sm == 0) {
        int occ = 0;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, pool_kernel<T, D>, kPoolThreads, 0);
        if (e != cudaSuccess) return e;
        per_sm = occ > 0 ? occ : 1;
        if (cacheable) __atomic_store_n(&occ_cache[dev], per_sm, __ATOMIC_RELEASE);
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
    return d_model > 0 && (d_model * es) % 16 == 0 && d_model * es <= 16 * 1024;  // rows of up to 16 KB
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
