// speechkv_decode_attn: Eq. (attn) of the paper (Sec. III-B) for one decode
// step -- every query head attends over its request's cached (pooled speech
// + text) keys and values, grouped-query style.
//
// Design (GB300, HBM-bound: 2G flop per cached byte, G = H_q / H_kv):
//   * Work = sum over requests of len[b] rows times H_kv heads.  A persistent
//     grid (one CTA per SM: ~217 KB of shared memory each) cuts this flat
//     range evenly (stream-K): CTA c owns units [U*c/C, U*(c+1)/C), whatever
//     the length mix of the batch.  Its range splits into "pieces", each a
//     run of rows of one (request, KV head).
//   * The cache is head-major per request, so a piece is one contiguous run
//     of rows.  The producer warp streams it HBM -> shared memory in tiles of
//     128 rows (64 for 512-byte rows) with bulk asynchronous copies (TMA,
//     cp.async.bulk, plus the piece's queries with its first tile) into a
//     ring of two or three stages guarded by mbarriers.  Eight consumer warps
//     take 16 (8) rows each of every tile.
//   * All G query heads of the KV head are served from one read of each
//     key/value row.
//     bf16 caches -- tensor cores (mma.sync m16n8k16, bf16 operands, fp32
//     accumulators): per warp and tile, S^T (16 keys x 8 heads) = K Q^T and
//     O^T (d x 8 heads) += V^T P^T, the G heads padded to 8.  A tile is laid
//     out as 8 groups of 16 rows, 16 bytes apart modulo 128, so that the
//     ldmatrix loads of K and V (V transposed) are free of bank conflicts;
//     P^T is the score fragment transposed in registers (movmatrix).  One
//     bulk copy per group and tensor, from 16 producer lanes.
//     fp32 caches -- CUDA cores: QK with four lanes per row, each reading a
//     quarter of the row in an order that keeps every 8-lane phase on
//     distinct banks, packed f32x2 FMAs, two-step shuffle reduction; PV with
//     one 16-byte column chunk of a row per lane, f32x2 FMAs.
//     Softmax: online (running max and sum per warp and head) in base 2,
//     log2(e)/sqrt(d) applied to the scores (fp32 path: folded into q).
//   * At the end of a piece the consumer warps deposit their (max, sum, o)
//     states in one of two shared buffers and go on; a merge warp combines
//     them.  A piece covering a whole (request, head) writes the output;
//     otherwise it writes an unnormalised partial, and the CTA that arrives
//     last at that (request, head) (atomic ticket with acquire-release
//     ordering, no waiting) merges the partials with log-sum-exp weights and
//     resets the ticket for the next call.
//   * Every mbarrier wait is bounded; on timeout the kernel reports
//     SPEECHKV_ERR_TIMEOUT, stops issuing and computing, lets its copies in
//     flight land and returns.
#pragma once

#include <math.h>

#include "common.cuh"
#include "launch.h"

namespace speechkv {
namespace {

template <typename T, int D, int G>
struct DecodeCfg {
    static constexpr int kWarps = 8;  // consumer warps
    // + one producer warp (lane 0 issues the bulk copies) + one merge warp
    static constexpr int kThreads = (kWarps + 2) * 32;
    static constexpr int kCtasPerSm = 1;
    static constexpr int kRowBytes = D * (int)sizeof(T);
    static constexpr int kRowsPerWarp = kRowBytes >= 512 ? 8 : 16;
    static constexpr int kTileRows = kWarps * kRowsPerWarp;
    // Tensor-core consumers (bf16 caches): a tile is stored as 8 groups of 16
    // rows, each group 16 bytes further along the banks than the previous one
    // (kGroupStride = 16 rows + 16 bytes), so that the 8 rows an ldmatrix
    // reads -- one from each group -- fall in 8 distinct 16-byte bank groups.
    // CUDA-core consumers (fp32 caches): rows back to back.
    static constexpr bool kMma = sizeof(T) == 2;
    static_assert(!kMma || G <= kMmaMaxGroup, "one 8-column MMA tile of query heads");
    static constexpr int kGroupRows = 16;
    static constexpr int kGroupStride = kGroupRows * kRowBytes + (kMma ? 16 : 0);
    static constexpr int kTileBytes = kTileRows / kGroupRows * kGroupStride;  // keys (or values)
    // byte offset of slot r (0 .. kTileRows - 1) in a tile
    static __device__ __forceinline__ uint32_t row_off(int r) {
        return (uint32_t)(r / kGroupRows) * kGroupStride + (uint32_t)(r % kGroupRows) * kRowBytes;
    }
    // A tile that starts at row t of a (request, head) run puts that row in
    // slot tile_lo(t) and holds tile_rows(t, t1) rows of the run's [t, t1).
    // With kAligned (the grouped layout over a block table), slots follow the
    // row index modulo 16, so that a group is one aligned run of 16 rows -- a
    // whole page with pages of 16 rows or more: one copy per group and
    // tensor, where a tile starting anywhere would split most pages over two
    // groups.  Only the first tile of a piece can then start past slot 0, and
    // it holds fewer rows.  Otherwise every tile starts at slot 0 (fewest
    // tiles).
    template <bool kAligned>
    static __device__ __forceinline__ int tile_lo(int64_t t) {
        return kAligned ? (int)(t & (kGroupRows - 1)) : 0;
    }
    template <bool kAligned>
    static __device__ __forceinline__ int tile_rows(int64_t t, int64_t t1) {
        const int64_t room = kTileRows - tile_lo<kAligned>(t);
        return (int)(t1 - t < room ? t1 - t : room);
    }
    static constexpr int kQBytes = G * kRowBytes;             // the piece's G query rows
    static constexpr int kStageBytes = 2 * kTileBytes + kQBytes;
    // QK layout: 4 lanes per row, 8 rows per pass
    static constexpr int kChunks = kRowBytes / 16;  // 16-byte chunks per row
    static constexpr int kChunksPerLane = kChunks / 4;
    static constexpr int kPairsPerChunk = 16 / (int)sizeof(T) / 2;
    static constexpr int kQkPasses = kRowsPerWarp / 8;
    // PV layout: one 16-byte chunk per lane, kPvRowsPerPass rows per pass
    static constexpr int kPvLanesPerRow = kChunks;
    static constexpr int kPvRowsPerPass = 32 / kPvLanesPerRow;
    // shared memory: stages | barriers | p | 2 merge buffers | flags | cum
    static constexpr int kPPairs = kMma ? 0 : kWarps * kRowsPerWarp * G;  // (p, p) pairs
    static constexpr int kPBytes = kPPairs * 8;
    static constexpr int kMergeFloats = kWarps * G * D + 2 * kWarps * G;
    static constexpr int kMergeBytes = 2 * kMergeFloats * 4;
    static constexpr int kBarBytes = (2 * 3 + 4) * 8;  // full/empty per stage (<= 3), piece/free x2
    // shared memory per CTA: an SM has 228 KB, of which 1 KB per resident CTA
    // is reserved
    static constexpr int kSmemLimit = 228 * 1024 / kCtasPerSm - 1024;
    // per-request tables: prefix sums of rows and cache offsets (int64, B+1
    // each) and the row an appended token takes (int32, B, padded)
    static size_t table_bytes(int B) { return (size_t)(B + 1) * 16 + ((size_t)B * 4 + 15) / 16 * 16; }
    static constexpr int kTableMax =
        (SPEECHKV_MAX_BATCH + 1) * 16 + (SPEECHKV_MAX_BATCH * 4 + 15) / 16 * 16;
    static constexpr int kFixedMax = kBarBytes + kPBytes + kMergeBytes + 16 + kTableMax;
    static constexpr int kStagesFit = (kSmemLimit - kFixedMax) / kStageBytes;
    static constexpr int kStages = kStagesFit < 3 ? kStagesFit : 3;
    static constexpr int kStagesBytes = kStages * kStageBytes;
    static_assert(kStages >= 2, "shared memory too small for two stages");
    static_assert(kStageBytes % 16 == 0 && kTileBytes % 16 == 0, "bulk copy alignment");
    static_assert(kTileRows % kGroupRows == 0, "whole row groups per tile");
    static_assert(!kMma || (kTileRows == 8 * kGroupRows && kWarps == 8 && kRowsPerWarp == 16),
                  "tensor-core consumers: 8 warps x 16 rows over 8 groups of 16 rows");
    static_assert(kChunksPerLane >= 2, "row too short for the QK lane layout");
    static_assert(kPvLanesPerRow <= 32, "row too long for the PV lane layout");

    static size_t smem_bytes(int B) {
        return (size_t)kStagesBytes + kBarBytes + kPBytes + kMergeBytes + 16 + table_bytes(B);
    }
};

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

// The stream-K partition of U units over C CTAs: CTA c owns units
// [U * c / C, U * (c + 1) / C).
struct Partition {
    int64_t U, C;
    __device__ __forceinline__ int64_t lo(int64_t c) const { return U * c / C; }
    // the CTA whose range holds unit u (0 <= u < U)
    __device__ __forceinline__ int64_t cta_of(int64_t u) const { return ((u + 1) * C - 1) / U; }
};
// CTAs used for U units on a grid of `grid`: at least kMinUnitsPerCta units
// each (a small batch spread over every SM would only multiply the partial
// results each (request, head) has to merge), at most the grid.
constexpr int64_t kMinUnitsPerCta = 256;
__device__ __forceinline__ int64_t ctas_for(int64_t U, int64_t grid) {
    const int64_t n = (U + kMinUnitsPerCta - 1) / kMinUnitsPerCta;
    return n < grid ? n : grid;
}

// Tiles a CTA streams into its shared-memory ring before it waits for the
// previous kernel (programmatic dependent launch with
// SPEECHKV_OVERLAP_PRIOR).
#ifndef SPEECHKV_PRE_WAIT_TILES
#define SPEECHKV_PRE_WAIT_TILES 2
#endif
constexpr int kPreWaitTiles = SPEECHKV_PRE_WAIT_TILES;

// kAppend: the decode step fused with the cache update -- each request's new
// key/value (k_new, v_new) is written as cache row len[b], attended to as that
// row (copied straight from k_new/v_new), and len[b] advances by one.
// kPaged: the cache is paged through map's block table (its own instance, so
// that the contiguous kernel carries none of that code).
template <typename T, int D, int G, bool kAppend, bool kPaged>
__global__ void __launch_bounds__(DecodeCfg<T, D, G>::kThreads, DecodeCfg<T, D, G>::kCtasPerSm)
    decode_attn_kernel(const T *__restrict__ q, const T *__restrict__ k_new,
                       const T *__restrict__ v_new, T *__restrict__ kc, T *__restrict__ vc,
                       const int64_t *__restrict__ cache_off, int32_t *__restrict__ len,
                       T *__restrict__ out, float qscale, int B, int H_kv,
                       float *__restrict__ partials, int slot_floats, int *__restrict__ counters,
                       int *__restrict__ done, int *__restrict__ err, int overlap,
                       CacheMap map) {
    using C = DecodeCfg<T, D, G>;
    constexpr int W = C::kWarps, S = C::kStages, TR = C::kTileRows, RW = C::kRowsPerWarp;
    constexpr bool kAligned = C::kMma && kPaged;  // tiles aligned to 16-row groups
    auto tile_lo = [](int64_t t) { return C::template tile_lo<kAligned>(t); };
    auto tile_rows = [](int64_t t, int64_t t1) { return C::template tile_rows<kAligned>(t, t1); };
    extern __shared__ __align__(128) unsigned char smem[];
    unsigned char *stages = smem;
    uint64_t *full_bar = reinterpret_cast<uint64_t *>(smem + C::kStagesBytes);  // [S]
    uint64_t *empty_bar = full_bar + S;                                       // [S]
    uint64_t *piece_bar = full_bar + 2 * S;  // [2]: the consumers deposited a piece
    uint64_t *free_bar = piece_bar + 2;      // [2]: the merge warp released a buffer
    float2 *pbuf = reinterpret_cast<float2 *>(smem + C::kStagesBytes + C::kBarBytes);
    float *mrg = reinterpret_cast<float *>(pbuf + C::kPPairs);  // [2][kMergeFloats]
    volatile int *flags = reinterpret_cast<volatile int *>(mrg + 2 * C::kMergeFloats);
    int64_t *cum = reinterpret_cast<int64_t *>(const_cast<int *>(flags) + 4);  // [B+1]
    int64_t *offs = cum + (B + 1);                                             // [B+1]
    int32_t *newrow = reinterpret_cast<int32_t *>(offs + (B + 1));             // [B]

    const int tid = threadIdx.x;
    const int warp = tid >> 5, lane = tid & 31;
    const int H_q = H_kv * G;

    // Programmatic dependent launch.  Unless the caller declared that the
    // previous kernel on the stream produces at most q, k_new and v_new
    // (overlap != 0), wait for it before touching anything.  With overlap,
    // the prologue and the bulk copies of cached rows run first; every read
    // of q / k_new / v_new and every global write (outputs, cache rows, len,
    // workspace) comes after griddep_wait(), and every warp but the
    // producer's idle lanes waits before it exits (so this grid never
    // completes before the previous one).
    // The next kernel is released (griddep_release) only after this thread's
    // own wait has returned, i.e. once the previous grid has completed.  So
    // when a grid starts, every grid before its immediate predecessor has
    // completed, whatever the grid sizes: the reads done before the wait can
    // only overlap the one kernel the overlap contract speaks of.
    auto griddep_release = [&]() {
        griddep_wait();
        griddep_launch_dependents();
    };
    if (!overlap) griddep_release();

    // ---- 1. per-request lengths (clamped to capacity) and their prefix sums
    // Row count, first cache row and capacity of request b, and the row its
    // new token takes (fused append; -1 if none).
    auto request_row = [&](int b, int64_t o0, int64_t o1, int64_t L) {
        const int64_t cap = o1 - o0;
        int32_t nr = -1;
        if (cap < 0 || o0 < 0) {
            if (blockIdx.x == 0) report_error(err, SPEECHKV_ERR_INVALID_ARG);
            L = 0;
        } else if (L < 0 || L > cap) {
            if (blockIdx.x == 0) report_error(err, SPEECHKV_ERR_CAPACITY);
            L = L < 0 ? 0 : cap;
        } else if (kAppend) {
            if (L < cap) {
                nr = (int32_t)L;  // the new token becomes row L ...
                L += 1;           // ... and is attended to
            } else if (blockIdx.x == 0) {
                report_error(err, SPEECHKV_ERR_CAPACITY);  // full: attend without it
            }
        }
        cum[b + 1] = L;
        offs[b] = o0;
        if (b == B - 1) offs[B] = o1;
        newrow[b] = nr;
    };
    // with pages, every request has the same capacity (max_blocks blocks) and
    // the offsets only carry it
    const int64_t capP = (int64_t)map.max_blocks << map.bs_log2;
    auto off_of = [&](int b) { return kPaged ? (int64_t)b * capP : cache_off[b]; };
    // inclusive prefix sums of cum[1..B] by one warp (lane `ln`)
    auto scan_lengths = [&](int ln) {
        int64_t carry = 0;
        for (int base = 0; base < B; base += 32) {
            const int i = base + ln;
            int64_t v = i < B ? cum[i + 1] : 0;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int64_t n = __shfl_up_sync(0xffffffffu, v, o);
                if (ln >= o) v += n;
            }
            if (i < B) cum[i + 1] = carry + v;
            carry += __shfl_sync(0xffffffffu, v, 31);
        }
    };
    auto init_barriers = [&]() {
        cum[0] = 0;
        flags[0] = 0;  // abort
        for (int s = 0; s < S; s++) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], W);
        }
        for (int x = 0; x < 2; x++) {
            mbar_init(&piece_bar[x], W);
            mbar_init(&free_bar[x], 1);
        }
        fence_mbar_init();
    };
    for (int b = tid; b < B; b += blockDim.x)
        request_row(b, off_of(b), off_of(b + 1), __ldcg(len + b));  // len at L2: another grid wrote it
    if (tid == 0) init_barriers();
    __syncthreads();
    if (tid < 32) scan_lengths(tid);
    __syncthreads();

    // ---- 2. this CTA's share of the flat (request, head, row) range
    const int64_t U = (int64_t)H_kv * cum[B];
    const int64_t Cn = ctas_for(U, gridDim.x);
    Partition part;
    part.U = U;
    part.C = Cn;
    const int64_t c = blockIdx.x;
    // Work that reads what the previous kernel may produce (k_new, v_new) or
    // writes global memory waits for it.  The producer waits after its first
    // copies, the merge warp (idle until the first piece) at once, and the
    // consumers only once the first tile -- whose queries are copied after
    // that wait -- has landed.
    auto merge_warp_prior_part = [&]() {  // merge warp
        griddep_release();
        // empty requests get a zero output (softmax over nothing)
        for (int b = blockIdx.x; b < B; b += gridDim.x) {
            if (cum[b + 1] != cum[b]) continue;
            for (int i = lane; i < H_q * D; i += 32)
                out[(int64_t)b * H_q * D + i] = from_float<T>(0.f);
        }
        if (kAppend) {
            // every CTA has read len[] before its prologue barrier; the last
            // one to get here advances len[] of the requests that took a token
            int last = 0;
            if (lane == 0) last = atomic_add_acq_rel_gpu(done, 1) == (int)gridDim.x - 1;
            last = __shfl_sync(0xffffffffu, last, 0);
            __syncwarp();
            if (last) {
                for (int b = lane; b < B; b += 32)
                    if (newrow[b] >= 0) len[b] = newrow[b] + 1;
                __syncwarp();
                if (lane == 0) *done = 0;
            }
        }
    };
    auto consumer_prior_part = [&]() {  // consumer warps
        griddep_release();
        if (kAppend) {
            // write the new tokens into their cache rows (nothing in this
            // kernel reads those rows from the cache: the attention takes the
            // new row from k_new / v_new)
            constexpr int kVec = 16 / (int)sizeof(T);
            const int nvec = H_kv * D / kVec;  // 16-byte vectors per token
            for (int b = blockIdx.x; b < B; b += gridDim.x) {
                const int32_t nr = newrow[b];
                if (nr < 0) continue;
                const int64_t cap = offs[b + 1] - offs[b];
                for (int i = tid; i < 2 * nvec; i += W * 32) {
                    const int tensor = i >= nvec;
                    const int e = (i - tensor * nvec) * kVec;
                    const int hh = e / D, col = e - hh * D;
                    const T *src = (tensor ? v_new : k_new) + (int64_t)b * H_kv * D + e;
                    const int64_t row =
                        kPaged ? cache_row(map, b, hh, nr, H_kv, D, 0, 0)
                               : (offs[b] * H_kv + (int64_t)hh * cap + nr) * D;
                    if (row < 0) {  // invalid page: reported, not written
                        report_error(err, SPEECHKV_ERR_INVALID_ARG);
                        continue;
                    }
                    copy_bytes<16>((tensor ? vc : kc) + row + col, src);
                }
            }
        }
    };
    if (c >= Cn) {  // no rows for this CTA
        if (warp == W + 1)
            merge_warp_prior_part();
        else if (warp < W)
            consumer_prior_part();
        else
            griddep_release();
        return;
    }
    const int64_t u0 = part.lo(c), u1 = part.lo(c + 1);

    if (warp == W) {
        // ================= producer warp =====================================
        // Lane 0 drives the ring (waits, expected bytes, queries, new rows);
        // with a block table, every lane copies its own page segments of a
        // tile, so small pages cost no more issue time than large ones.  The
        // control flow is warp-uniform (lane 0's decisions are broadcast).
        int stage = 0;
        uint32_t phase = 0;
        int64_t issued = 0;
        bool stop = false;
        // Copies of data the previous kernel may produce (queries, new
        // tokens) wait for it; until then lane 0 queues them here, at most 3
        // per tile.  No more tiles than the ring holds are issued before the
        // wait: the next one would wait for a stage whose queries are queued
        // behind it.
        constexpr int kPre = kPreWaitTiles < S ? kPreWaitTiles : S;
        struct Deferred {
            void *dst;
            const void *src;
            uint32_t bytes;
            uint64_t *bar;
        };
        Deferred deferred[3 * kPre];
        int ndeferred = 0;
        bool waited = !overlap;
        auto copy_prior = [&](void *dst, const void *src, uint32_t bytes, uint64_t *bar) {
            if (lane != 0) return;
            if (waited) {
                bulk_g2s(dst, src, bytes, bar);
            } else {
                // warm L2 meanwhile: a prefetch reads no value, so whatever the
                // previous kernel writes there is what the copy will see
                prefetch_l2(src, bytes);
                deferred[ndeferred++] = Deferred{dst, src, bytes, bar};
            }
        };
        auto flush_deferred = [&]() {
            griddep_release();
            waited = true;
            if (lane == 0)
                for (int i = 0; i < ndeferred; i++)
                    bulk_g2s(deferred[i].dst, deferred[i].src, deferred[i].bytes,
                             deferred[i].bar);
            ndeferred = 0;
        };
        for (int64_t u = u0; u < u1 && !stop;) {
            const Piece p = piece_at(cum, B, H_kv, u, u1);
            const int64_t cap = offs[p.b + 1] - offs[p.b];
            const int64_t base = offs[p.b] * H_kv + (int64_t)p.h * cap;
            // Rows [t_from, t_from + nrows) of this (request, head) into the
            // stage (keys at dst, values kTileBytes further): one bulk copy per
            // tensor for a contiguous run (lane 0), one per page segment with a
            // block table (lane i takes segments i, i + 32, ...).  An invalid
            // page is reported and read from page 0 instead (the stage's byte
            // count must still arrive).
            // With the grouped tile layout of the tensor-core consumers, lane
            // g < 8 copies the rows of group g: rows b16 + 16 g .. b16 + 16 g
            // + 15 of the run (b16: the tile's first row rounded down to a
            // multiple of 16), as far as they belong to [t_from, t_from +
            // nrows).
            auto copy_rows = [&](unsigned char *dst, int64_t t_from, int64_t nrows, uint64_t *bar) {
                if constexpr (C::kMma) {
                    if (lane >= 8) return;
                    const int64_t g0 = t_from - tile_lo(t_from) + (int64_t)C::kGroupRows * lane;
                    const int64_t a = g0 > t_from ? g0 : t_from;
                    const int64_t e = g0 + C::kGroupRows < t_from + nrows ? g0 + C::kGroupRows
                                                                          : t_from + nrows;
                    if (a >= e) return;
                    unsigned char *gd =
                        dst + lane * C::kGroupStride + (uint32_t)(a - g0) * C::kRowBytes;
                    if constexpr (!kPaged) {
                        const uint32_t bytes = (uint32_t)(e - a) * C::kRowBytes;
                        bulk_g2s(gd, kc + (base + a) * D, bytes, bar);
                        bulk_g2s(gd + C::kTileBytes, vc + (base + a) * D, bytes, bar);
                    } else {
                        const int lg = map.bs_log2;
                        for (int64_t pg = a >> lg; pg <= (e - 1) >> lg; pg++) {
                            const int64_t s0 = (pg << lg) > a ? (pg << lg) : a;
                            const int64_t s1 = ((pg + 1) << lg) < e ? ((pg + 1) << lg) : e;
                            int64_t off = cache_row(map, p.b, p.h, s0, H_kv, D, 0, 0);
                            if (off < 0) {
                                report_error(err, SPEECHKV_ERR_INVALID_ARG);
                                off = 0;
                            }
                            const uint32_t at = (uint32_t)(s0 - a) * C::kRowBytes;
                            const uint32_t bytes = (uint32_t)(s1 - s0) * C::kRowBytes;
                            bulk_g2s(gd + at, kc + off, bytes, bar);
                            bulk_g2s(gd + C::kTileBytes + at, vc + off, bytes, bar);
                        }
                    }
                } else if constexpr (!kPaged) {
                    if (lane != 0) return;
                    const uint32_t bytes = (uint32_t)nrows * C::kRowBytes;
                    bulk_g2s(dst, kc + (base + t_from) * D, bytes, bar);
                    bulk_g2s(dst + C::kTileBytes, vc + (base + t_from) * D, bytes, bar);
                } else {
                    const int lg = map.bs_log2;
                    const int64_t t_end = t_from + nrows;
                    for (int64_t pg = (t_from >> lg) + lane; pg <= (t_end - 1) >> lg; pg += 32) {
                        const int64_t s0 = (pg << lg) > t_from ? (pg << lg) : t_from;
                        const int64_t s1 = ((pg + 1) << lg) < t_end ? ((pg + 1) << lg) : t_end;
                        int64_t off = cache_row(map, p.b, p.h, s0, H_kv, D, 0, 0);
                        if (off < 0) {
                            report_error(err, SPEECHKV_ERR_INVALID_ARG);
                            off = 0;
                        }
                        const uint32_t at = (uint32_t)(s0 - t_from) * C::kRowBytes;
                        const uint32_t bytes = (uint32_t)(s1 - s0) * C::kRowBytes;
                        bulk_g2s(dst + at, kc + off, bytes, bar);
                        bulk_g2s(dst + C::kTileBytes + at, vc + off, bytes, bar);
                    }
                }
            };
            // with kAppend, row nr of this (request, head) comes from k_new/v_new
            const int64_t nr = kAppend ? (int64_t)newrow[p.b] : -1;
            for (int64_t t = p.t0; t < p.t1; t += tile_rows(t, p.t1)) {
                // Copies issued before the wait for the previous kernel are
                // limited to kPre tiles (their queries are queued)
                if (!waited && issued == kPre) flush_deferred();
                // (re-check the abort flag after the wait: aborted consumers
                // release stages without waiting for their copies)
                int ok = 1;
                if (lane == 0)
                    ok = !flags[0] && mbar_wait_bounded(&empty_bar[stage], phase ^ 1u, err) &&
                         !flags[0];
                ok = __shfl_sync(0xffffffffu, ok, 0);
                if (!ok) {
                    if (lane == 0) flags[0] = 1;
                    stop = true;
                    break;
                }
                const int rows = tile_rows(t, p.t1);
                const uint32_t bytes = (uint32_t)rows * C::kRowBytes;
                const bool first = (t == p.t0);
                unsigned char *dst = stages + (size_t)stage * C::kStageBytes;
                if (lane == 0)
                    mbar_arrive_expect_tx(&full_bar[stage], 2 * bytes + (first ? C::kQBytes : 0));
                __syncwarp();
                if (kAppend && nr >= t && nr < t + rows) {
                    // the tile ends with the new token: cached rows, then one
                    // row from k_new / v_new (always the last row of the run)
                    if (nr > t) copy_rows(dst, t, nr - t, &full_bar[stage]);
                    const uint32_t at = C::row_off(tile_lo(t) + (int)(nr - t));
                    const int64_t src = ((int64_t)p.b * H_kv + p.h) * D;
                    copy_prior(dst + at, k_new + src, C::kRowBytes, &full_bar[stage]);
                    copy_prior(dst + C::kTileBytes + at, v_new + src, C::kRowBytes,
                               &full_bar[stage]);
                } else {
                    copy_rows(dst, t, rows, &full_bar[stage]);
                }
                if (first)
                    copy_prior(dst + 2 * C::kTileBytes, q + ((int64_t)p.b * H_q + p.h * G) * D,
                               C::kQBytes, &full_bar[stage]);
                ++issued;
                if (++stage == S) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            u += p.t1 - p.t0;
        }
        if (!waited) flush_deferred();
        // Let the copies still in flight land before the CTA may exit.
        if (lane == 0) {
            const int64_t first = issued > S ? issued - S : 0;
            for (int64_t k = first; k < issued; k++)
                if (!mbar_wait_bounded(&full_bar[k % S], (uint32_t)((k / S) & 1), err)) break;
        }
        return;
    }

    if (warp == W + 1) {
        // ======== merge warp: combines the consumers' states of each piece ====
        // lane owns kCols consecutive output columns of every query head
        constexpr int kCols = D / 32;
        // partials fetched per round of the final merge (every query head of
        // a partial in the same round)
        constexpr int kBatch = G >= 8 ? 1 : 8 / G;
        // The merge warp idles until the first piece is deposited: it does
        // its share of the work that waits for the previous kernel now, so
        // that the done-counter round trip is not on the path of a CTA whose
        // only piece ends with the kernel.
        merge_warp_prior_part();
        // Partials of up to kBatch pieces (every query head) as one round of
        // the final merge: slot index c0 + j of this (request, head); this
        // CTA's own piece (index `mine`) is not loaded.
        auto load_round = [&](int64_t c0, int64_t clast, int64_t mine, int64_t seg,
                              float (&bm)[kBatch][G], float (&bl)[kBatch][G],
                              float (&bo)[kBatch][G][kCols]) {
#pragma unroll
            for (int j = 0; j < kBatch; j++) {
                const bool have = c0 + j <= clast && c0 + j != mine;
                const float *sp = partials + (c0 + j + seg) * slot_floats;
#pragma unroll
                for (int g = 0; g < G; g++) {
                    bm[j][g] = have ? __ldcg(sp + G * D + g) : -INFINITY;
                    bl[j][g] = have ? __ldcg(sp + G * D + G + g) : 0.f;
#pragma unroll
                    for (int i = 0; i < kCols; i++)
                        bo[j][g][i] = have ? __ldcg(sp + g * D + lane * kCols + i) : 0.f;
                }
            }
        };
        int64_t k = 0;  // piece index within this CTA
        for (int64_t u = u0; u < u1; k++) {
            const Piece p = piece_at(cum, B, H_kv, u, u1);
            const int x = (int)(k & 1);
            const int64_t seg = (int64_t)p.b * H_kv + p.h;
            const bool whole = (p.t0 == 0 && p.t1 == p.L);
            const int64_t A = (int64_t)H_kv * cum[p.b] + (int64_t)p.h * p.L;
            const int64_t cfirst = whole ? c : part.cta_of(A);
            const int64_t clast = whole ? c : part.cta_of(A + p.L - 1);
            const int others = (int)(clast - cfirst);
            const uint32_t use = (uint32_t)((k >> 1) & 1);
            bool ok = !flags[0] && mbar_wait_bounded(&piece_bar[x], use, err);
            ok = __all_sync(0xffffffffu, ok) && !__shfl_sync(0xffffffffu, flags[0], 0);
            const float *mo = mrg + x * C::kMergeFloats;  // [W][G][D]
            const float *mm = mo + W * G * D;              // [W][G]
            const float *ml = mm + W * G;                  // [W][G]
            // this CTA's state of the piece: the consumer warps' states merged
            float M[G], Ls[G], acc[G][kCols];
            if (ok) {
#pragma unroll
                for (int g = 0; g < G; g++) {
                    M[g] = -INFINITY;
#pragma unroll
                    for (int w = 0; w < W; w++) M[g] = fmaxf(M[g], mm[w * G + g]);
                    Ls[g] = 0.f;
#pragma unroll
                    for (int i = 0; i < kCols; i++) acc[g][i] = 0.f;
#pragma unroll
                    for (int w = 0; w < W; w++) {
                        const float sc = fast_exp2(mm[w * G + g] - M[g]);  // idle warp: 0
                        Ls[g] = fmaf(ml[w * G + g], sc, Ls[g]);
                        const float *src = mo + (w * G + g) * D + lane * kCols;
#pragma unroll
                        for (int i = 0; i < kCols; i++) acc[g][i] = fmaf(src[i], sc, acc[g][i]);
                    }
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&free_bar[x]);  // the buffer may be refilled
            if (ok && !whole) {
                // Split piece: the CTA that finishes last at this (request,
                // head) merges every piece.  Publish this partial, then take a
                // ticket (acquire-release) to find out whether this CTA is the
                // last; the last one merges with its own state from registers.
                // (One L2 round trip for the CTAs that only publish: a CTA's
                // exit frees its SM for the next launch's CTA.)
                float *slot = partials + (c + seg) * slot_floats;  // o [G][D], m [G], l [G]
#pragma unroll
                for (int g = 0; g < G; g++) {
#pragma unroll
                    for (int i = 0; i < kCols; i++) slot[g * D + lane * kCols + i] = acc[g][i];
                    if (lane == 0) {
                        slot[G * D + g] = M[g];
                        slot[G * D + G + g] = Ls[g];
                    }
                }
                __syncwarp();  // the lanes' partial writes precede lane 0's release
                int last = 0;
                if (lane == 0) last = atomic_add_acq_rel_gpu(&counters[seg], 1) == others;
                last = __shfl_sync(0xffffffffu, last, 0);
                __syncwarp();  // lane 0's acquire orders the other lanes' reads too
                if (last) {
                    // online log-sum-exp over the pieces in CTA order (this
                    // CTA's own state taken from registers in its turn), per
                    // query head g, so that the result does not depend on which
                    // CTA came last; kBatch partials (all heads) in flight per
                    // round
                    float Mt[G], Lt[G], at[G][kCols];
#pragma unroll
                    for (int g = 0; g < G; g++) {
                        Mt[g] = -INFINITY;
                        Lt[g] = 0.f;
#pragma unroll
                        for (int i = 0; i < kCols; i++) at[g][i] = 0.f;
                    }
#pragma unroll 1
                    for (int64_t c0 = cfirst; c0 <= clast; c0 += kBatch) {
                        float bm[kBatch][G], bl[kBatch][G], bo[kBatch][G][kCols];
                        load_round(c0, clast, c, seg, bm, bl, bo);
#pragma unroll
                        for (int j = 0; j < kBatch; j++) {  // this CTA's own state
                            if (c0 + j != c) continue;
#pragma unroll
                            for (int g = 0; g < G; g++) {
                                bm[j][g] = M[g];
                                bl[j][g] = Ls[g];
#pragma unroll
                                for (int i = 0; i < kCols; i++) bo[j][g][i] = acc[g][i];
                            }
                        }
#pragma unroll
                        for (int g = 0; g < G; g++) {
                            float Mn = Mt[g];
#pragma unroll
                            for (int j = 0; j < kBatch; j++) Mn = fmaxf(Mn, bm[j][g]);
                            const float r = fast_exp2(Mt[g] - Mn);  // 0 while Mt = -inf
                            Lt[g] *= r;
#pragma unroll
                            for (int i = 0; i < kCols; i++) at[g][i] *= r;
#pragma unroll
                            for (int j = 0; j < kBatch; j++) {
                                const float sc = fast_exp2(bm[j][g] - Mn);  // absent: 0
                                Lt[g] = fmaf(bl[j][g], sc, Lt[g]);
#pragma unroll
                                for (int i = 0; i < kCols; i++)
                                    at[g][i] = fmaf(bo[j][g][i], sc, at[g][i]);
                            }
                            Mt[g] = Mn;
                        }
                    }
#pragma unroll
                    for (int g = 0; g < G; g++) {
                        Ls[g] = Lt[g];
#pragma unroll
                        for (int i = 0; i < kCols; i++) acc[g][i] = at[g][i];
                    }
                    if (lane == 0) counters[seg] = 0;  // ready for the next call
                }
                ok = last;
            }
            if (ok) {  // a whole piece, or the last CTA of a split one
#pragma unroll
                for (int g = 0; g < G; g++) {
                    const float inv = 1.f / Ls[g];
#pragma unroll
                    for (int i = 0; i < kCols; i++) acc[g][i] *= inv;
                    store_vec<T, kCols>(out + ((int64_t)p.b * H_q + p.h * G + g) * D +
                                            lane * kCols,
                                        acc[g]);
                }
            }
            u += p.t1 - p.t0;
        }
        return;
    }

    // ===================== consumers: W warps ==============================
    int stage = 0;
    uint32_t phase = 0;
    bool aborted = false;
    bool prior_part_done = false;
    int64_t k = 0;  // piece index within this CTA
    if constexpr (!C::kMma) {
        const int lrow = lane >> 2;  // row within an 8-row pass
        const int lq = lane & 3;     // quarter of the row
        int ch[C::kChunksPerLane];   // the lane's chunks, rotated by row parity
#pragma unroll
        for (int i = 0; i < C::kChunksPerLane; i++)
            ch[i] = lq + 4 * ((i + (lrow & 1)) % C::kChunksPerLane);
        const int pc = lane % C::kPvLanesPerRow;  // PV: 16-byte column chunk
        const int pr = lane / C::kPvLanesPerRow;  // PV: row within a pass
        float2 *pw = pbuf + warp * RW * G;
        const float2 qs = make_float2(qscale, qscale);

        for (int64_t u = u0; u < u1; k++) {
            const Piece p = piece_at(cum, B, H_kv, u, u1);

            float2 q2[G][C::kChunksPerLane][C::kPairsPerChunk];
            float m[G], l[G];
            float2 o[G][C::kPairsPerChunk];
#pragma unroll
            for (int g = 0; g < G; g++) {
                m[g] = -INFINITY;
                l[g] = 0.f;
#pragma unroll
                for (int e = 0; e < C::kPairsPerChunk; e++) o[g][e] = make_float2(0.f, 0.f);
            }

            for (int64_t t = p.t0; t < p.t1; t += tile_rows(t, p.t1)) {
                const int rows = tile_rows(t, p.t1);
                if (!aborted) {
                    // warp-uniform decision: every lane waits, any failure stops the warp
                    bool fail = flags[0] != 0;
                    if (!fail) fail = !mbar_wait_bounded(&full_bar[stage], phase, err);
                    if (__any_sync(0xffffffffu, fail)) {
                        flags[0] = 1;
                        aborted = true;
                    }
                }
                if (!prior_part_done) {
                    consumer_prior_part();
                    prior_part_done = true;
                }
                const unsigned char *ks = stages + (size_t)stage * C::kStageBytes;
                if (!aborted && t == p.t0) {
                    // the piece's queries came with its first tile; scale them by
                    // log2(e)/sqrt(d) so that scores are in base 2
#pragma unroll
                    for (int g = 0; g < G; g++)
#pragma unroll
                        for (int i = 0; i < C::kChunksPerLane; i++) {
                            load16_pairs<T>(ks + 2 * C::kTileBytes + g * C::kRowBytes + ch[i] * 16,
                                            q2[g][i]);
#pragma unroll
                            for (int e = 0; e < C::kPairsPerChunk; e++)
                                q2[g][i][e] = fmul2(q2[g][i][e], qs);
                        }
                }
                const unsigned char *vs = ks + C::kTileBytes;
                // the warp's rows of the tile are interleaved (tile row warp + W j
                // for its row j), so that a partial tile is shared by every warp
                // and costs in proportion to its rows
                const int nw = rows > warp ? (rows - warp + W - 1) / W : 0;
                if (nw > 0 && !aborted) {
                    // ---- scores (q * log2e/sqrt(d)) . k, two packed partial sums
                    float s[G][C::kQkPasses];
#pragma unroll
                    for (int rr = 0; rr < C::kQkPasses; rr++) {
                        const int row = rr * 8 + lrow;
                        if (rr * 8 >= nw) {  // no row of this pass (warp-uniform)
#pragma unroll
                            for (int g = 0; g < G; g++) s[g][rr] = -INFINITY;
                            continue;
                        }
                        const unsigned char *kr = ks + (warp + W * row) * C::kRowBytes;
                        float2 acc[G];
#pragma unroll
                        for (int g = 0; g < G; g++) acc[g] = make_float2(0.f, 0.f);
#pragma unroll
                        for (int i = 0; i < C::kChunksPerLane; i++) {
                            float2 k2[C::kPairsPerChunk];
                            load16_pairs<T>(kr + ch[i] * 16, k2);
#pragma unroll
                            for (int e = 0; e < C::kPairsPerChunk; e++)
#pragma unroll
                                for (int g = 0; g < G; g++) acc[g] = ffma2(q2[g][i][e], k2[e], acc[g]);
                        }
#pragma unroll
                        for (int g = 0; g < G; g++) {
                            float v = acc[g].x + acc[g].y;
                            v += __shfl_xor_sync(0xffffffffu, v, 1);
                            v += __shfl_xor_sync(0xffffffffu, v, 2);
                            s[g][rr] = (row < nw) ? v : -INFINITY;
                        }
                    }
                    // ---- online softmax update (warp-wide running max and sum)
#pragma unroll
                    for (int g = 0; g < G; g++) {
                        float mt = s[g][0];
#pragma unroll
                        for (int rr = 1; rr < C::kQkPasses; rr++) mt = fmaxf(mt, s[g][rr]);
                        mt = fmaxf(mt, __shfl_xor_sync(0xffffffffu, mt, 4));
                        mt = fmaxf(mt, __shfl_xor_sync(0xffffffffu, mt, 8));
                        mt = fmaxf(mt, __shfl_xor_sync(0xffffffffu, mt, 16));
                        const float mnew = fmaxf(m[g], mt);
                        const float corr = fast_exp2(m[g] - mnew);
                        m[g] = mnew;
                        float ps = 0.f;
#pragma unroll
                        for (int rr = 0; rr < C::kQkPasses; rr++) {
                            const float pv = fast_exp2(s[g][rr] - mnew);
                            ps += pv;
                            if (lq == 0) pw[(rr * 8 + lrow) * G + g] = make_float2(pv, pv);
                        }
                        ps += __shfl_xor_sync(0xffffffffu, ps, 4);
                        ps += __shfl_xor_sync(0xffffffffu, ps, 8);
                        ps += __shfl_xor_sync(0xffffffffu, ps, 16);
                        l[g] = fmaf(l[g], corr, ps);
                        const float2 c2 = make_float2(corr, corr);
#pragma unroll
                        for (int e = 0; e < C::kPairsPerChunk; e++) o[g][e] = fmul2(o[g][e], c2);
                    }
                    __syncwarp();
                    // ---- o += p * v over the warp's valid rows
                    const unsigned char *vw = vs + warp * C::kRowBytes + pc * 16;
#pragma unroll 4
                    for (int j0 = 0; j0 < nw; j0 += C::kPvRowsPerPass) {
                        const int row = j0 + pr;
                        if (row < nw) {
                            float2 v2[C::kPairsPerChunk];
                            load16_pairs<T>(vw + row * (W * C::kRowBytes), v2);
#pragma unroll
                            for (int g = 0; g < G; g++) {
                                const float2 pg = pw[row * G + g];
#pragma unroll
                                for (int e = 0; e < C::kPairsPerChunk; e++)
                                    o[g][e] = ffma2(pg, v2[e], o[g][e]);
                            }
                        }
                    }
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(&empty_bar[stage]);
                if (++stage == S) {
                    stage = 0;
                    phase ^= 1u;
                }
            }

            // ---- deposit this warp's state of the piece for the merge warp
            // (fold the PV row groups onto lanes with pr == 0 first)
#pragma unroll
            for (int g = 0; g < G; g++)
#pragma unroll
                for (int e = 0; e < C::kPairsPerChunk; e++)
#pragma unroll
                    for (int off = C::kPvLanesPerRow; off < 32; off <<= 1) {
                        o[g][e].x += __shfl_xor_sync(0xffffffffu, o[g][e].x, off);
                        o[g][e].y += __shfl_xor_sync(0xffffffffu, o[g][e].y, off);
                    }
            const int x = (int)(k & 1);
            // buffer x was last used by piece k - 2: wait until the merge warp
            // released it (the first use of each buffer passes at once)
            if (!aborted) {
                bool fail = !mbar_wait_bounded(&free_bar[x], (uint32_t)(((k >> 1) & 1) ^ 1), err);
                if (__any_sync(0xffffffffu, fail)) {
                    flags[0] = 1;
                    aborted = true;
                }
            }
            float *mo = mrg + x * C::kMergeFloats;
            if (pr == 0) {
#pragma unroll
                for (int g = 0; g < G; g++)
#pragma unroll
                    for (int e = 0; e < C::kPairsPerChunk; e++) {
                        const int col = pc * (16 / (int)sizeof(T)) + 2 * e;
                        *reinterpret_cast<float2 *>(&mo[(warp * G + g) * D + col]) = o[g][e];
                    }
            }
            if (lane == 0) {
#pragma unroll
                for (int g = 0; g < G; g++) {
                    mo[W * G * D + warp * G + g] = m[g];
                    mo[W * G * D + W * G + warp * G + g] = l[g];
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&piece_bar[x]);
            u += p.t1 - p.t0;
        }
    } else {
        // ---- tensor-core consumers (bf16, 3 to 8 query heads per KV head) --
        // Warp w takes 16 keys of every tile: its key i (0..15) is slot
        // 16 (i % 8) + 2w + i / 8, i.e. rows 2w and 2w + 1 of each 16-row
        // group, so that a ragged tile is shared by the warps and every
        // ldmatrix reads its 8 rows from 8 distinct bank groups.  Per tile,
        // with the G query heads padded to 8 by zero queries:
        //   S^T (16 keys x 8 heads)  = K (16 x d) . Q^T (d x 8)
        //   O^T (d x 8 heads)       += V^T (d x 16 keys) . P^T (16 keys x 8)
        // on mma.sync m16n8k16 (bf16 operands, fp32 accumulators).  Lane
        // 4r + t holds the scores of keys r and r + 8 for heads 2t and 2t + 1,
        // and rows (channels) 16m + r and 16m + r + 8 of O^T for those heads.
        // P^T, the B operand of the second product, is the transpose of the
        // score fragment (movmatrix) after rounding p to bf16; the row sums
        // add the rounded weights, so that the output is a convex combination
        // of the values with exactly the weights the product used.
        constexpr int kSteps = D / 16;  // k-steps of Q.K and m-tiles of O^T
        const int r = lane >> 2, t4 = lane & 3;
        const int h0 = 2 * t4;                    // the lane's heads h0, h0 + 1
        const int mi = lane >> 3, mr = lane & 7;  // ldmatrix: matrix, row of it
        // keys: matrix mi = (keys 0-7 | 8-15 by mi & 1) x (channels by mi >> 1)
        const uint32_t k_lane = (uint32_t)(mr * C::kGroupStride +
                                           (2 * warp + (mi & 1)) * C::kRowBytes + (mi >> 1) * 16);
        // values, transposed: matrix mi = (channels by mi & 1) x (keys by mi >> 1)
        const uint32_t v_lane = (uint32_t)(mr * C::kGroupStride +
                                           (2 * warp + (mi >> 1)) * C::kRowBytes + (mi & 1) * 16);
        // slots of the lane's score keys (r: srow, r + 8: srow + 1) and of
        // its P.V keys (2t: vrow, 2t + 1: vrow + 16, 2t + 8: vrow + 1,
        // 2t + 9: vrow + 17)
        const int srow = 16 * r + 2 * warp;
        const int vrow = 32 * t4 + 2 * warp;
        const uint32_t smem_stages = smem_addr(stages);

        for (int64_t u = u0; u < u1; k++) {
            const Piece p = piece_at(cum, B, H_kv, u, u1);
            uint32_t qf[kSteps][2];  // Q^T fragments: head r, channels 16j + 2t (+1, +8, +9)
            float o[kSteps][4];
            float mx[2] = {-INFINITY, -INFINITY}, ls[2] = {0.f, 0.f};
#pragma unroll
            for (int j = 0; j < kSteps; j++) {
                qf[j][0] = qf[j][1] = 0u;
#pragma unroll
                for (int e = 0; e < 4; e++) o[j][e] = 0.f;
            }

            for (int64_t t = p.t0; t < p.t1; t += tile_rows(t, p.t1)) {
                const int rows = tile_rows(t, p.t1);
                if (!aborted) {
                    // warp-uniform decision: every lane waits, any failure stops the warp
                    bool fail = flags[0] != 0;
                    if (!fail) fail = !mbar_wait_bounded(&full_bar[stage], phase, err);
                    if (__any_sync(0xffffffffu, fail)) {
                        flags[0] = 1;
                        aborted = true;
                    }
                }
                if (!prior_part_done) {
                    consumer_prior_part();
                    prior_part_done = true;
                }
                const uint32_t ks = smem_stages + (uint32_t)stage * C::kStageBytes;
                if (!aborted && t == p.t0 && r < G) {
                    // the piece's queries came with its first tile
                    const unsigned char *qr = stages + (size_t)stage * C::kStageBytes +
                                              2 * C::kTileBytes + r * C::kRowBytes + 4 * t4;
#pragma unroll
                    for (int j = 0; j < kSteps; j++) {
                        qf[j][0] = *reinterpret_cast<const uint32_t *>(qr + 32 * j);
                        qf[j][1] = *reinterpret_cast<const uint32_t *>(qr + 32 * j + 16);
                    }
                }
                // the tile's rows are slots [lo, hi); the warp's first slot at
                // or after lo is 2w, 2w + 1 or 16 + 2w
                const int lo = tile_lo(t), hi = lo + rows;
                const int first = lo <= 2 * warp ? 2 * warp : (lo == 2 * warp + 1 ? lo : 16 + 2 * warp);
                auto in_tile = [&](int x) { return x >= lo && x < hi; };
                if (first < hi && !aborted) {  // the warp has a row of the tile
                    // ---- scores: two accumulator chains over the channels
                    float sa[4] = {0.f, 0.f, 0.f, 0.f}, sb[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                    for (int j = 0; j < kSteps; j += 2) {
                        uint32_t a0[4], a1[4];
                        ldmatrix_x4(a0, ks + k_lane + 32 * j);
                        ldmatrix_x4(a1, ks + k_lane + 32 * (j + 1));
                        mma_bf16_16816(sa, a0, qf[j][0], qf[j][1]);
                        mma_bf16_16816(sb, a1, qf[j + 1][0], qf[j + 1][1]);
                    }
                    float s[4];
#pragma unroll
                    for (int e = 0; e < 4; e++) s[e] = (sa[e] + sb[e]) * qscale;  // base 2
                    if (!in_tile(srow)) s[0] = s[1] = -INFINITY;
                    if (!in_tile(srow + 1)) s[2] = s[3] = -INFINITY;
                    // ---- online softmax over the warp's keys, per head
                    float mt0 = fmaxf(s[0], s[2]), mt1 = fmaxf(s[1], s[3]);
#pragma unroll
                    for (int off = 4; off < 32; off <<= 1) {
                        mt0 = fmaxf(mt0, __shfl_xor_sync(0xffffffffu, mt0, off));
                        mt1 = fmaxf(mt1, __shfl_xor_sync(0xffffffffu, mt1, off));
                    }
                    const float mn0 = fmaxf(mx[0], mt0), mn1 = fmaxf(mx[1], mt1);
                    const float c0 = fast_exp2(mx[0] - mn0), c1 = fast_exp2(mx[1] - mn1);
                    mx[0] = mn0;
                    mx[1] = mn1;
                    const uint32_t pa = pack_bf16x2(fast_exp2(s[0] - mn0), fast_exp2(s[1] - mn1));
                    const uint32_t pb = pack_bf16x2(fast_exp2(s[2] - mn0), fast_exp2(s[3] - mn1));
                    ls[0] = fmaf(ls[0], c0, bf16_lo(pa) + bf16_lo(pb));
                    ls[1] = fmaf(ls[1], c1, bf16_hi(pa) + bf16_hi(pb));
                    const uint32_t b0 = movmatrix_trans(pa), b1 = movmatrix_trans(pb);
                    // slots outside the tile's rows hold stale shared memory
                    // (not necessarily finite); their weights are 0, and so
                    // are their values here
                    uint32_t mk01 = 0xffffffffu, mk89 = 0xffffffffu;
                    if (lo > 0 || hi < TR) {
                        mk01 = (in_tile(vrow) ? 0x0000ffffu : 0u) |
                               (in_tile(vrow + 16) ? 0xffff0000u : 0u);
                        mk89 = (in_tile(vrow + 1) ? 0x0000ffffu : 0u) |
                               (in_tile(vrow + 17) ? 0xffff0000u : 0u);
                    }
                    // ---- o = o * correction + v^T p^T
#pragma unroll
                    for (int m = 0; m < kSteps; m++) {
                        uint32_t a[4];
                        ldmatrix_x4_trans(a, ks + C::kTileBytes + v_lane + 32 * m);
                        a[0] &= mk01;
                        a[1] &= mk01;
                        a[2] &= mk89;
                        a[3] &= mk89;
                        o[m][0] *= c0;
                        o[m][1] *= c1;
                        o[m][2] *= c0;
                        o[m][3] *= c1;
                        mma_bf16_16816(o[m], a, b0, b1);
                    }
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(&empty_bar[stage]);
                if (++stage == S) {
                    stage = 0;
                    phase ^= 1u;
                }
            }

            // ---- deposit this warp's state of the piece for the merge warp
#pragma unroll
            for (int off = 4; off < 32; off <<= 1) {
                ls[0] += __shfl_xor_sync(0xffffffffu, ls[0], off);
                ls[1] += __shfl_xor_sync(0xffffffffu, ls[1], off);
            }
            const int x = (int)(k & 1);
            // buffer x was last used by piece k - 2: wait until the merge warp
            // released it (the first use of each buffer passes at once)
            if (!aborted) {
                bool fail = !mbar_wait_bounded(&free_bar[x], (uint32_t)(((k >> 1) & 1) ^ 1), err);
                if (__any_sync(0xffffffffu, fail)) {
                    flags[0] = 1;
                    aborted = true;
                }
            }
            float *mo = mrg + x * C::kMergeFloats;
#pragma unroll
            for (int hh = 0; hh < 2; hh++) {
                const int g = h0 + hh;
                if (g >= G) continue;
                float *og = mo + (warp * G + g) * D + r;
#pragma unroll
                for (int m = 0; m < kSteps; m++) {
                    og[16 * m] = o[m][hh];
                    og[16 * m + 8] = o[m][2 + hh];
                }
                if (r == 0) {
                    mo[W * G * D + warp * G + g] = mx[hh];
                    mo[W * G * D + W * G + warp * G + g] = ls[hh];
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&piece_bar[x]);
            u += p.t1 - p.t0;
        }
    }
    if (!prior_part_done) consumer_prior_part();  // (only if there was no tile)
    griddep_release();
}

template <typename T, int D, int G, bool kAppend, bool kPaged>
cudaError_t launch_instance(const DecodeArgs &a, int grid, cudaStream_t stream) {
    using C = DecodeCfg<T, D, G>;
    auto kern = decode_attn_kernel<T, D, G, kAppend, kPaged>;
    static int configured_device_mask = 0;  // devices with the smem attributes set
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const bool cached =
        dev < 31 && (__atomic_load_n(&configured_device_mask, __ATOMIC_ACQUIRE) & (1 << dev));
    if (!cached) {
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)C::smem_bytes(SPEECHKV_MAX_BATCH));
        if (e != cudaSuccess) return e;
        // all of the unified L1/shared storage as shared memory
        e = cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
        if (e != cudaSuccess) return e;
        if (dev < 31) __atomic_fetch_or(&configured_device_mask, 1 << dev, __ATOMIC_ACQ_REL);
    }
    const float qscale = a.scale * 1.4426950408889634f;  // log2(e): scores in base 2
    // programmatic dependent launch: may begin while the previous kernel on
    // the stream retires (the kernel orders itself with griddepcontrol)
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3(C::kThreads);
    cfg.dynamicSmemBytes = C::smem_bytes(a.B);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, static_cast<const T *>(a.q),
                              static_cast<const T *>(a.k_new), static_cast<const T *>(a.v_new),
                              static_cast<T *>(a.k_cache), static_cast<T *>(a.v_cache),
                              a.cache_off, a.len, static_cast<T *>(a.out), qscale, a.B, a.H_kv,
                              a.partials, decode_slot_floats(D, G), a.counters, a.done, a.err,
                              a.overlap ? 1 : 0, a.map);
}

// Resident CTAs per SM for a batch of B requests (the per-request tables in
// shared memory grow with B).
template <typename T, int D, int G>
int occupancy_instance(int B) {
    using C = DecodeCfg<T, D, G>;
    auto kern = decode_attn_kernel<T, D, G, false, false>;
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)C::smem_bytes(SPEECHKV_MAX_BATCH)) != cudaSuccess ||
        cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout, 100) !=
            cudaSuccess)
        return 0;
    int n = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kern, C::kThreads, C::smem_bytes(B)) !=
        cudaSuccess)
        return 0;
    return n;
}

}  // namespace

}  // namespace speechkv
