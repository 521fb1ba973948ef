// speechkv_decode_attn: Eq. (attn) of the paper (Sec. III-B) for one decode
// step -- every query head attends over its request's cached (pooled speech
// + text) keys and values, grouped-query style.
//
// Design (GB300, HBM-bound):
//   * Work = sum over requests of len[b] rows times H_kv heads.  A persistent
//     grid cuts this flat range evenly (stream-K): CTA c owns units
//     [U*c/C, U*(c+1)/C).  Its range splits into "pieces", each a run of rows
//     of one (request, KV head).  Every CTA therefore reads the same number of
//     bytes whatever the length mix of the batch.
//   * The cache is head-major per request, so a piece is one contiguous run
//     of rows.  One producer lane streams it HBM -> shared memory with bulk
//     asynchronous copies (TMA, cp.async.bulk) into a ring of stages guarded
//     by mbarriers; eight consumer warps compute on the staged tiles.
//   * All G = H_q/H_kv query heads of the KV head are served from one read of
//     each key/value row.  QK: four lanes per row, each reading a quarter of
//     the row from shared memory in an order that keeps every 8-lane phase on
//     distinct banks, two-step shuffle reduction.  Softmax: online (running
//     max and sum per warp) in base 2, the log2(e)/sqrt(d) factor folded into
//     the query.  PV: each lane owns d/32 output columns of every head.
//   * A piece that covers a whole (request, head) writes the output.  Pieces
//     of a (request, head) split across CTAs write (max, sum, unnormalised o)
//     partials; the CTA that arrives last (atomic ticket, no waiting) merges
//     them with log-sum-exp weights and resets the counter for the next call.
//   * Every mbarrier wait is bounded; on timeout the kernel reports
//     SPEECHKV_ERR_TIMEOUT, stops issuing and computing, lets its copies in
//     flight land and returns.
#include <math.h>

#include "common.cuh"
#include "launch.h"

namespace speechkv {
namespace {

template <typename T, int D, int G>
struct DecodeCfg {
    static constexpr int kWarps = 8;                    // consumer warps
    static constexpr int kThreads = (kWarps + 1) * 32;  // + one producer warp
    static constexpr int kRowBytes = D * (int)sizeof(T);
    static constexpr int kChunks = kRowBytes / 16;      // 16-byte chunks per row
    static constexpr int kChunksPerLane = kChunks / 4;  // QK: 4 lanes per row
    static constexpr int kElemsPerChunk = 16 / (int)sizeof(T);
    static constexpr int kRowsPerGroup = kRowBytes >= 512 ? 1 : 2;
    static constexpr int kRowsPerWarp = 8 * kRowsPerGroup;
    static constexpr int kTileRows = kWarps * kRowsPerWarp;
    static constexpr int kTileBytes = kTileRows * kRowBytes;  // K (or V) of a tile
    static constexpr int kStageBytes = 2 * kTileBytes;
    static constexpr int kColsPerLane = D / 32;               // PV columns per lane
    static constexpr int kMergeBytes = kWarps * G * D * 4 + 2 * kWarps * G * 4;
    static constexpr int kPBytes = kWarps * kRowsPerWarp * G * 4;
    static constexpr int kSmemLimit = 227 * 1024;
    static constexpr int kCumMaxBytes = (SPEECHKV_MAX_BATCH + 1) * 8;
    static constexpr int kFixedMax = kMergeBytes + kPBytes + 2 * 4 * 8 + 16 + kCumMaxBytes;
    static constexpr int kStagesFit = (kSmemLimit - kFixedMax) / kStageBytes;
    static constexpr int kStages = kStagesFit < 4 ? kStagesFit : 4;
    static_assert(kStages >= 2, "shared memory too small for two stages");
    static_assert(kChunksPerLane >= 2, "row too short for the QK lane layout");

    static size_t smem_bytes(int B) {
        return (size_t)kStages * kStageBytes + kMergeBytes + kPBytes + 2 * kStages * 8 + 16 +
               (size_t)(B + 1) * 8;
    }
};

__device__ __forceinline__ void consumer_sync(int nthreads) {
    asm volatile("bar.sync 1, %0;" ::"r"(nthreads) : "memory");
}

// Largest b in [0, B) with H_kv * cum[b] <= u (the request holding unit u).
__device__ __forceinline__ int find_request(const int64_t *cum, int B, int64_t H_kv, int64_t u) {
    int lo = 0, hi = B - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (H_kv * cum[mid] <= u)
            lo = mid;
        else
            hi = mid - 1;
    }
    return lo;
}

struct Piece {
    int b, h;
    int64_t L;       // rows of the (request, head)
    int64_t t0, t1;  // rows [t0, t1) of it handled here
};

__device__ __forceinline__ Piece piece_at(const int64_t *cum, int B, int H_kv, int64_t u,
                                          int64_t u1) {
    Piece p;
    p.b = find_request(cum, B, H_kv, u);
    p.L = cum[p.b + 1] - cum[p.b];
    const int64_t within = u - (int64_t)H_kv * cum[p.b];
    p.h = (int)(within / p.L);
    p.t0 = within - (int64_t)p.h * p.L;
    const int64_t room = u1 - u;
    p.t1 = (p.L - p.t0 < room) ? p.L : p.t0 + room;
    return p;
}

// CTA (of C) whose unit range [U*c/C, U*(c+1)/C) holds unit u.
__device__ __forceinline__ int64_t cta_of(int64_t u, int64_t U, int64_t C) {
    return ((u + 1) * C - 1) / U;
}

template <typename T, int D, int G>
__global__ void __launch_bounds__(DecodeCfg<T, D, G>::kThreads, 1)
    decode_attn_kernel(const T *__restrict__ q, const T *__restrict__ kc,
                       const T *__restrict__ vc, const int64_t *__restrict__ cache_off,
                       const int32_t *__restrict__ len_in, T *__restrict__ out, float qscale,
                       int B, int H_kv, float *__restrict__ partials, int slot_floats,
                       int *__restrict__ counters, int *__restrict__ err) {
    using C = DecodeCfg<T, D, G>;
    constexpr int kConsumers = C::kWarps * 32;
    extern __shared__ __align__(128) unsigned char smem[];
    unsigned char *stages = smem;
    float *mrg_o = reinterpret_cast<float *>(smem + (size_t)C::kStages * C::kStageBytes);
    float *mrg_m = mrg_o + C::kWarps * G * D;
    float *mrg_l = mrg_m + C::kWarps * G;
    float *pbuf = mrg_l + C::kWarps * G;
    uint64_t *full_bar = reinterpret_cast<uint64_t *>(pbuf + C::kWarps * C::kRowsPerWarp * G);
    uint64_t *empty_bar = full_bar + C::kStages;
    volatile int *flags = reinterpret_cast<volatile int *>(empty_bar + C::kStages);
    int64_t *cum = reinterpret_cast<int64_t *>(const_cast<int *>(flags) + 4);

    const int tid = threadIdx.x;
    const int warp = tid >> 5, lane = tid & 31;
    const int H_q = H_kv * G;

    // ---- 1. per-request lengths (clamped to capacity) and their prefix sums
    for (int b = tid; b < B; b += blockDim.x) {
        const int64_t cap = cache_off[b + 1] - cache_off[b];
        int64_t L = len_in[b];
        if (cap < 0 || cache_off[b] < 0) {
            if (blockIdx.x == 0) report_error(err, SPEECHKV_ERR_INVALID_ARG);
            L = 0;
        } else if (L < 0 || L > cap) {
            if (blockIdx.x == 0) report_error(err, SPEECHKV_ERR_CAPACITY);
            L = L < 0 ? 0 : cap;
        }
        cum[b + 1] = L;
    }
    if (tid == 0) {
        cum[0] = 0;
        flags[0] = 0;  // abort
        flags[1] = 0;  // "this CTA merges" ticket result
        flags[2] = 0;  // abort flag as seen by all consumers at a piece's end
        for (int s = 0; s < C::kStages; s++) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], C::kWarps);
        }
        fence_mbar_init();
    }
    __syncthreads();
    if (tid < 32) {
        int64_t carry = 0;
        for (int base = 0; base < B; base += 32) {
            const int i = base + tid;
            int64_t v = i < B ? cum[i + 1] : 0;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int64_t n = __shfl_up_sync(0xffffffffu, v, o);
                if (tid >= o) v += n;
            }
            if (i < B) cum[i + 1] = carry + v;
            carry += __shfl_sync(0xffffffffu, v, 31);
        }
    }
    __syncthreads();

    // ---- 2. empty requests get a zero output (softmax over nothing)
    for (int b = blockIdx.x; b < B; b += gridDim.x) {
        if (cum[b + 1] != cum[b]) continue;
        for (int i = tid; i < H_q * D; i += blockDim.x)
            out[(int64_t)b * H_q * D + i] = from_float<T>(0.f);
    }

    // ---- 3. this CTA's share of the flat (request, head, row) range
    const int64_t U = (int64_t)H_kv * cum[B];
    const int64_t Cn = U < (int64_t)gridDim.x ? U : (int64_t)gridDim.x;
    const int64_t c = blockIdx.x;
    if (c >= Cn) return;
    const int64_t u0 = U * c / Cn, u1 = U * (c + 1) / Cn;

    if (warp == C::kWarps) {
        // ================= producer: one lane issues bulk copies ============
        if (lane != 0) return;
        int stage = 0;
        uint32_t phase = 0;
        int64_t issued = 0;
        bool stop = false;
        for (int64_t u = u0; u < u1 && !stop;) {
            const Piece p = piece_at(cum, B, H_kv, u, u1);
            const int64_t cap = cache_off[p.b + 1] - cache_off[p.b];
            const int64_t base = cache_off[p.b] * H_kv + (int64_t)p.h * cap;
            for (int64_t t = p.t0; t < p.t1; t += C::kTileRows) {
                // (re-check the abort flag after the wait: aborted consumers
                // release stages without waiting for their copies)
                if (flags[0] || !mbar_wait_bounded(&empty_bar[stage], phase ^ 1u, err) ||
                    flags[0]) {
                    flags[0] = 1;
                    stop = true;
                    break;
                }
                const int rows = (int)((p.t1 - t) < C::kTileRows ? (p.t1 - t) : C::kTileRows);
                const uint32_t bytes = (uint32_t)rows * C::kRowBytes;
                unsigned char *dst = stages + (size_t)stage * C::kStageBytes;
                mbar_arrive_expect_tx(&full_bar[stage], 2 * bytes);
                bulk_g2s(dst, kc + (base + t) * D, bytes, &full_bar[stage]);
                bulk_g2s(dst + C::kTileBytes, vc + (base + t) * D, bytes, &full_bar[stage]);
                ++issued;
                if (++stage == C::kStages) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            u += p.t1 - p.t0;
        }
        // Let the copies still in flight land before the CTA may exit.
        const int64_t first = issued > C::kStages ? issued - C::kStages : 0;
        for (int64_t k = first; k < issued; k++)
            if (!mbar_wait_bounded(&full_bar[k % C::kStages], (uint32_t)((k / C::kStages) & 1), err))
                break;
        return;
    }

    // ===================== consumers: 8 warps ==============================
    const int lrow = lane >> 2;  // row of the lane's group within 8 rows
    const int lq = lane & 3;     // quarter of the row the lane reads
    const int ctid = tid;        // 0 .. kConsumers-1
    int ch[C::kChunksPerLane];   // the lane's chunks, rotated by row parity
#pragma unroll
    for (int i = 0; i < C::kChunksPerLane; i++)
        ch[i] = lq + 4 * ((i + (lrow & 1)) % C::kChunksPerLane);
    float *pw = pbuf + warp * C::kRowsPerWarp * G;

    int stage = 0;
    uint32_t phase = 0;
    bool aborted = false;
    for (int64_t u = u0; u < u1;) {
        const Piece p = piece_at(cum, B, H_kv, u, u1);
        const int b = p.b, h = p.h;

        // query fragments of the group's G heads, pre-scaled by log2(e)/sqrt(d)
        float qf[G][C::kChunksPerLane][C::kElemsPerChunk];
#pragma unroll
        for (int g = 0; g < G; g++)
#pragma unroll
            for (int i = 0; i < C::kChunksPerLane; i++) {
                load_vec<T, C::kElemsPerChunk>(
                    q + ((int64_t)b * H_q + h * G + g) * D + ch[i] * C::kElemsPerChunk, qf[g][i]);
#pragma unroll
                for (int e = 0; e < C::kElemsPerChunk; e++) qf[g][i][e] *= qscale;
            }
        float m[G], l[G], o[G][C::kColsPerLane];
#pragma unroll
        for (int g = 0; g < G; g++) {
            m[g] = -INFINITY;
            l[g] = 0.f;
#pragma unroll
            for (int cc = 0; cc < C::kColsPerLane; cc++) o[g][cc] = 0.f;
        }

        for (int64_t t = p.t0; t < p.t1; t += C::kTileRows) {
            const int rows = (int)((p.t1 - t) < C::kTileRows ? (p.t1 - t) : C::kTileRows);
            if (!aborted && (flags[0] || !mbar_wait_bounded(&full_bar[stage], phase, err))) {
                flags[0] = 1;
                aborted = true;
            }
            const unsigned char *ks = stages + (size_t)stage * C::kStageBytes;
            const unsigned char *vs = ks + C::kTileBytes;
            const int r0 = warp * C::kRowsPerWarp;
            int nw = rows - r0;
            nw = nw < 0 ? 0 : (nw > C::kRowsPerWarp ? C::kRowsPerWarp : nw);
            if (nw > 0 && !aborted) {
                // ---- scores s = (q * log2e/sqrt(d)) . k for the warp's rows
                float s[G][C::kRowsPerGroup];
#pragma unroll
                for (int rr = 0; rr < C::kRowsPerGroup; rr++) {
                    const int row = r0 + rr * 8 + lrow;
                    const unsigned char *kr = ks + row * C::kRowBytes;
                    float acc[G][2];
#pragma unroll
                    for (int g = 0; g < G; g++) acc[g][0] = acc[g][1] = 0.f;
#pragma unroll
                    for (int i = 0; i < C::kChunksPerLane; i++) {
                        float kf[C::kElemsPerChunk];
                        load_vec<T, C::kElemsPerChunk>(reinterpret_cast<const T *>(kr + ch[i] * 16), kf);
#pragma unroll
                        for (int e = 0; e < C::kElemsPerChunk; e++)
#pragma unroll
                            for (int g = 0; g < G; g++)
                                acc[g][e & 1] = fmaf(qf[g][i][e], kf[e], acc[g][e & 1]);
                    }
#pragma unroll
                    for (int g = 0; g < G; g++) {
                        float v = acc[g][0] + acc[g][1];
                        v += __shfl_xor_sync(0xffffffffu, v, 1);
                        v += __shfl_xor_sync(0xffffffffu, v, 2);
                        s[g][rr] = (row < rows) ? v : -INFINITY;
                    }
                }
                // ---- online softmax update (warp-wide running max)
#pragma unroll
                for (int g = 0; g < G; g++) {
                    float mt = s[g][0];
#pragma unroll
                    for (int rr = 1; rr < C::kRowsPerGroup; rr++) mt = fmaxf(mt, s[g][rr]);
                    mt = fmaxf(mt, __shfl_xor_sync(0xffffffffu, mt, 4));
                    mt = fmaxf(mt, __shfl_xor_sync(0xffffffffu, mt, 8));
                    mt = fmaxf(mt, __shfl_xor_sync(0xffffffffu, mt, 16));
                    const float mnew = fmaxf(m[g], mt);
                    const float corr = fast_exp2(m[g] - mnew);
                    m[g] = mnew;
                    l[g] *= corr;
#pragma unroll
                    for (int cc = 0; cc < C::kColsPerLane; cc++) o[g][cc] *= corr;
#pragma unroll
                    for (int rr = 0; rr < C::kRowsPerGroup; rr++) {
                        const float pr = fast_exp2(s[g][rr] - mnew);
                        if (lq == 0) pw[(rr * 8 + lrow) * G + g] = pr;
                    }
                }
                __syncwarp();
                // ---- o += p * v over the warp's valid rows
                const T *vrow = reinterpret_cast<const T *>(vs + r0 * C::kRowBytes) +
                                lane * C::kColsPerLane;
#pragma unroll 4
                for (int j = 0; j < nw; j++) {
                    float vf[C::kColsPerLane];
                    load_vec<T, C::kColsPerLane>(vrow + j * D, vf);
#pragma unroll
                    for (int g = 0; g < G; g++) {
                        const float pj = pw[j * G + g];
                        l[g] += pj;
#pragma unroll
                        for (int cc = 0; cc < C::kColsPerLane; cc++)
                            o[g][cc] = fmaf(pj, vf[cc], o[g][cc]);
                    }
                }
                __syncwarp();
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty_bar[stage]);
            if (++stage == C::kStages) {
                stage = 0;
                phase ^= 1u;
            }
        }

        // ---- merge the 8 warps' states of this piece
#pragma unroll
        for (int g = 0; g < G; g++) {
#pragma unroll
            for (int cc = 0; cc < C::kColsPerLane; cc++)
                mrg_o[(warp * G + g) * D + lane * C::kColsPerLane + cc] = o[g][cc];
            if (lane == 0) {
                mrg_m[warp * G + g] = m[g];
                mrg_l[warp * G + g] = l[g];
            }
        }
        consumer_sync(kConsumers);
        if (ctid == 0) flags[2] = flags[0];
        consumer_sync(kConsumers);
        // uniform over the consumers (all branches below that hold a barrier
        // depend only on values every consumer warp agrees on)
        const bool stop = flags[2] != 0;
        const bool whole = (p.t0 == 0 && p.t1 == p.L);
        const int64_t seg = (int64_t)b * H_kv + h;
        if (!stop) {
            for (int idx = ctid; idx < G * D; idx += kConsumers) {
                const int g = idx / D, col = idx - g * D;
                float M = -INFINITY;
#pragma unroll
                for (int w = 0; w < C::kWarps; w++) M = fmaxf(M, mrg_m[w * G + g]);
                float Ls = 0.f, O = 0.f;
#pragma unroll
                for (int w = 0; w < C::kWarps; w++) {
                    const float sc = fast_exp2(mrg_m[w * G + g] - M);
                    Ls = fmaf(mrg_l[w * G + g], sc, Ls);
                    O = fmaf(mrg_o[(w * G + g) * D + col], sc, O);
                }
                if (whole) {
                    out[((int64_t)b * H_q + h * G + g) * D + col] = from_float<T>(O / Ls);
                } else {
                    float *slot = partials + (c + seg) * slot_floats;
                    slot[2 * G + g * D + col] = O;
                    if (col == 0) {
                        slot[g] = M;
                        slot[G + g] = Ls;
                    }
                }
            }
        }
        if (!whole && !stop) {
            // ---- last-arriving CTA of this (request, head) merges the pieces
            __threadfence();
            consumer_sync(kConsumers);
            const int64_t A = (int64_t)H_kv * cum[b] + (int64_t)h * p.L;
            const int64_t cfirst = cta_of(A, U, Cn), clast = cta_of(A + p.L - 1, U, Cn);
            if (ctid == 0) {
                const int old = atomicAdd(&counters[seg], 1);
                flags[1] = (old == (int)(clast - cfirst));
            }
            consumer_sync(kConsumers);
            if (flags[1]) {
                __threadfence();
                for (int idx = ctid; idx < G * D; idx += kConsumers) {
                    const int g = idx / D, col = idx - g * D;
                    float M = -INFINITY;
                    for (int64_t cp = cfirst; cp <= clast; cp++)
                        M = fmaxf(M, __ldcg(partials + (cp + seg) * slot_floats + g));
                    float Ls = 0.f, O = 0.f;
                    for (int64_t cp = cfirst; cp <= clast; cp++) {
                        const float *slot = partials + (cp + seg) * slot_floats;
                        const float sc = fast_exp2(__ldcg(slot + g) - M);
                        Ls = fmaf(__ldcg(slot + G + g), sc, Ls);
                        O = fmaf(__ldcg(slot + 2 * G + g * D + col), sc, O);
                    }
                    out[((int64_t)b * H_q + h * G + g) * D + col] = from_float<T>(O / Ls);
                }
                if (ctid == 0) counters[seg] = 0;
            }
        }
        consumer_sync(kConsumers);  // merge buffers are reused by the next piece
        u += p.t1 - p.t0;
    }
}

template <typename T, int D, int G>
cudaError_t launch_instance(const DecodeArgs &a, int grid, cudaStream_t stream) {
    using C = DecodeCfg<T, D, G>;
    auto kern = decode_attn_kernel<T, D, G>;
    static int configured_device_mask = 0;  // devices with the smem attribute set
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 31 && !(__atomic_load_n(&configured_device_mask, __ATOMIC_ACQUIRE) & (1 << dev))) {
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)C::smem_bytes(SPEECHKV_MAX_BATCH));
        if (e != cudaSuccess) return e;
        __atomic_fetch_or(&configured_device_mask, 1 << dev, __ATOMIC_ACQ_REL);
    } else if (dev >= 31) {
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)C::smem_bytes(SPEECHKV_MAX_BATCH));
        if (e != cudaSuccess) return e;
    }
    const float qscale = a.scale * 1.4426950408889634f;  // log2(e): scores in base 2
    kern<<<grid, C::kThreads, C::smem_bytes(a.B), stream>>>(
        static_cast<const T *>(a.q), static_cast<const T *>(a.k_cache),
        static_cast<const T *>(a.v_cache), a.cache_off, a.len, static_cast<T *>(a.out), qscale,
        a.B, a.H_kv, a.partials, decode_slot_floats(D, G), a.counters, a.err);
    return cudaGetLastError();
}

template <typename T, int D, int G>
int occupancy_instance() {
    using C = DecodeCfg<T, D, G>;
    auto kern = decode_attn_kernel<T, D, G>;
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)C::smem_bytes(SPEECHKV_MAX_BATCH)) != cudaSuccess)
        return 0;
    int n = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kern, C::kThreads,
                                                      C::smem_bytes(SPEECHKV_MAX_BATCH)) !=
        cudaSuccess)
        return 0;
    return n;
}

}  // namespace

bool decode_supported(speechkv_dtype dtype, int d, int group) {
    return (dtype == SPEECHKV_F32 || dtype == SPEECHKV_BF16) && (d == 64 || d == 128) &&
           (group == 1 || group == 2 || group == 4);
}

int decode_slot_floats(int d, int group) {
    const int f = 2 * group + group * d;
    return (f + 3) & ~3;  // keep slots 16-byte aligned
}

#define SPEECHKV_DECODE_CASES(X)                                          \
    X(float, 64, 1) X(float, 64, 2) X(float, 64, 4)                       \
    X(float, 128, 1) X(float, 128, 2) X(float, 128, 4)                    \
    X(__nv_bfloat16, 64, 1) X(__nv_bfloat16, 64, 2) X(__nv_bfloat16, 64, 4) \
    X(__nv_bfloat16, 128, 1) X(__nv_bfloat16, 128, 2) X(__nv_bfloat16, 128, 4)

template <typename T>
constexpr speechkv_dtype dtype_of() {
    return sizeof(T) == 4 ? SPEECHKV_F32 : SPEECHKV_BF16;
}

int decode_ctas_per_sm(speechkv_dtype dtype, int d, int group) {
#define X(T, D, G) \
    if (dtype == dtype_of<T>() && d == D && group == G) return occupancy_instance<T, D, G>();
    SPEECHKV_DECODE_CASES(X)
#undef X
    return 0;
}

cudaError_t launch_decode(const DecodeArgs &a, int grid, cudaStream_t stream) {
    const int group = a.H_q / a.H_kv;
#define X(T, D, G) \
    if (a.dtype == dtype_of<T>() && a.d == D && group == G) return launch_instance<T, D, G>(a, grid, stream);
    SPEECHKV_DECODE_CASES(X)
#undef X
    return cudaErrorInvalidValue;
}

}  // namespace speechkv
