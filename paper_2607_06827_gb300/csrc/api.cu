// C ABI of libspeechkv: argument checks, per-device state and dispatch to the
// kernels (pool.cu, append.cu, decode_attn.cu, prefill_attn.cu).  Declarations
// and the full contract of every entry point are in include/speechkv.h.
#include <math.h>
#include <stdint.h>

#include <mutex>

#include "launch.h"
#include "speechkv.h"

// The per-device error word: kernels record the first device-side error here
// (atomicCAS from 0); speechkv_check_device_error reads and clears it.  A
// module-scope variable, so the library allocates nothing for it.
__device__ int speechkv_error_word;

namespace {

constexpr int kMaxDevices = 64;
constexpr int kDecodeKinds = 32;  // dtype x d x group (1..8)
constexpr int kBatchBuckets = 3;  // occupancy is cached per batch-size bucket
constexpr int kBatchBucketMax[kBatchBuckets] = {128, 512, SPEECHKV_MAX_BATCH};

struct DeviceState {
    int *err = nullptr;  // device address of speechkv_error_word
    int num_sms = 0;
    int decode_ctas_per_sm[kDecodeKinds][kBatchBuckets] = {};
};

std::mutex g_mu;
DeviceState g_dev[kMaxDevices];

speechkv_status current_device(int *dev_out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return SPEECHKV_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices) return SPEECHKV_ERR_UNSUPPORTED;
    *dev_out = dev;
    return SPEECHKV_OK;
}

// Per-device set-up on first use: the error word's device address (which is
// what kernels must be given; the host-side symbol is not a device address)
// and the SM count.
speechkv_status device_state(DeviceState **out) {
    int dev = 0;
    speechkv_status st = current_device(&dev);
    if (st != SPEECHKV_OK) return st;
    std::lock_guard<std::mutex> lock(g_mu);
    DeviceState &s = g_dev[dev];
    if (!s.err) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, speechkv_error_word) != cudaSuccess) return SPEECHKV_ERR_CUDA;
        int sms = 0;
        if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
            sms <= 0)
            return SPEECHKV_ERR_CUDA;
        s.num_sms = sms;
        s.err = static_cast<int *>(p);
    }
    *out = &s;
    return SPEECHKV_OK;
}

bool aligned(const void *p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

bool valid_dtype(speechkv_dtype dt) { return dt == SPEECHKV_F32 || dt == SPEECHKV_BF16; }

// Index of a supported (dtype, d, group) in the per-device occupancy cache.
int decode_kind(speechkv_dtype dt, int d, int group) {
    return (dt == SPEECHKV_BF16 ? 16 : 0) + (d == 128 ? 8 : 0) + (group - 1);
}

// Automatic decode grid: the SM count times the kernel's residency (which
// depends on the batch size through the per-CTA length table), at most
// kAutoCtasPerSmMax.  Workspace sizing uses that upper bound.
constexpr int kAutoCtasPerSmMax = 4;

speechkv_status decode_auto_grid(DeviceState *s, speechkv_dtype dt, int d, int group, int B,
                                 int *grid) {
    const int kind = decode_kind(dt, d, group);
    int bucket = 0;
    while (bucket < kBatchBuckets - 1 && B > kBatchBucketMax[bucket]) bucket++;
    int per_sm;
    {
        std::lock_guard<std::mutex> lock(g_mu);
        per_sm = s->decode_ctas_per_sm[kind][bucket];
    }
    if (per_sm == 0) {
        per_sm = speechkv::decode_ctas_per_sm(dt, d, group, kBatchBucketMax[bucket]);
        if (per_sm <= 0) return SPEECHKV_ERR_CUDA;
        if (per_sm > kAutoCtasPerSmMax) per_sm = kAutoCtasPerSmMax;
        std::lock_guard<std::mutex> lock(g_mu);
        s->decode_ctas_per_sm[kind][bucket] = per_sm;
    }
    *grid = s->num_sms * per_sm;
    return SPEECHKV_OK;
}

size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Workspace layout: counters [B*H_kv] int32 and one more int32 (the fused
// step's CTA count), 256-byte padded, then partial slots
// [grid + B*H_kv][slot_floats] fp32.
size_t counters_bytes(int B, int H_kv) { return round_up(((size_t)B * H_kv + 1) * 4, 256); }

size_t workspace_bytes(int B, int H_q, int H_kv, int d, int grid) {
    const size_t S = (size_t)B * H_kv;
    const size_t slot = (size_t)speechkv::decode_slot_floats(d, H_q / H_kv);
    return counters_bytes(B, H_kv) + ((size_t)grid + S) * slot * 4;
}

// Host checks of a decode call and its launch descriptor; nothing is queued
// on the stream.  *launch stays false when there is nothing to launch
// (B == 0).  Shared by speechkv_decode_attn (k_new == v_new == NULL) and the
// decode steps (both non-NULL).
speechkv_status decode_prepare(const void *q, const void *k_new, const void *v_new,
                               void *k_cache, void *v_cache, const int64_t *cache_off,
                               int32_t *len, void *out, float scale, int32_t B, int32_t H_q,
                               int32_t H_kv, int32_t d, int32_t w, int32_t layer, int32_t l0,
                               int32_t grid_ctas, void *workspace, size_t workspace_bytes_in,
                               speechkv_dtype dtype, uint32_t flags, bool append,
                               const speechkv::CacheMap &map, speechkv::DecodeArgs *out_args,
                               int *out_grid, bool *launch) {
    *launch = false;
    if (B < 0 || H_q < 1 || H_kv < 1 || H_q % H_kv != 0 || w < 1 || layer < 0 || l0 < 0 ||
        grid_ctas < 0 || !valid_dtype(dtype) || isnan(scale) || isinf(scale) ||
        (flags & ~SPEECHKV_OVERLAP_PRIOR))
        return SPEECHKV_ERR_INVALID_ARG;
    if (!speechkv::decode_supported(dtype, d, H_q / H_kv)) return SPEECHKV_ERR_UNSUPPORTED;
    if (B > SPEECHKV_MAX_BATCH) return SPEECHKV_ERR_UNSUPPORTED;
    if (B == 0) return SPEECHKV_OK;
    if (!q || !k_cache || !v_cache || (!cache_off && !map.table) || !len || !out ||
        (append && (!k_new || !v_new)))
        return SPEECHKV_ERR_INVALID_ARG;
    if (!aligned(q, 16) || !aligned(k_cache, 16) || !aligned(v_cache, 16) || !aligned(out, 16) ||
        !aligned(cache_off, 8) || !aligned(len, 4) ||
        (append && (!aligned(k_new, 16) || !aligned(v_new, 16))))
        return SPEECHKV_ERR_INVALID_ARG;
    DeviceState *s = nullptr;
    speechkv_status st = device_state(&s);
    if (st != SPEECHKV_OK) return st;
    int grid = grid_ctas;
    if (grid == 0) {
        st = decode_auto_grid(s, dtype, d, H_q / H_kv, B, &grid);
        if (st != SPEECHKV_OK) return st;
    }
    const size_t need = workspace_bytes(B, H_q, H_kv, d, grid);
    if (!workspace || workspace_bytes_in < need || !aligned(workspace, 16))
        return SPEECHKV_ERR_WORKSPACE;
    speechkv::DecodeArgs a;
    a.q = q;
    a.k_new = append ? k_new : nullptr;
    a.v_new = append ? v_new : nullptr;
    a.k_cache = k_cache;
    a.v_cache = v_cache;
    a.cache_off = cache_off;
    a.len = len;
    a.out = out;
    a.scale = scale > 0.f ? scale : 1.0f / sqrtf((float)d);
    a.B = B;
    a.H_q = H_q;
    a.H_kv = H_kv;
    a.d = d;
    a.dtype = dtype;
    a.counters = static_cast<int *>(workspace);
    a.done = a.counters + (size_t)B * H_kv;
    a.partials = reinterpret_cast<float *>(static_cast<char *>(workspace) +
                                           counters_bytes(B, H_kv));
    a.err = s->err;
    a.overlap = (flags & SPEECHKV_OVERLAP_PRIOR) != 0;
    a.map = map;
    *out_args = a;
    *out_grid = grid;
    *launch = true;
    return SPEECHKV_OK;
}

speechkv_status decode_common(const void *q, const void *k_new, const void *v_new,
                              void *k_cache, void *v_cache, const int64_t *cache_off,
                              int32_t *len, void *out, float scale, int32_t B, int32_t H_q,
                              int32_t H_kv, int32_t d, int32_t w, int32_t layer, int32_t l0,
                              int32_t grid_ctas, void *workspace, size_t workspace_bytes_in,
                              speechkv_dtype dtype, uint32_t flags, cudaStream_t stream,
                              bool append, const speechkv::CacheMap &map = {}) {
    speechkv::DecodeArgs a;
    int grid = 0;
    bool launch = false;
    const speechkv_status st =
        decode_prepare(q, k_new, v_new, k_cache, v_cache, cache_off, len, out, scale, B, H_q,
                       H_kv, d, w, layer, l0, grid_ctas, workspace, workspace_bytes_in, dtype,
                       flags, append, map, &a, &grid, &launch);
    if (st != SPEECHKV_OK || !launch) return st;
    return speechkv::launch_decode(a, grid, stream) == cudaSuccess ? SPEECHKV_OK
                                                                   : SPEECHKV_ERR_CUDA;
}

// Host checks of a block table's description (the table itself is read on
// the device, where a bad entry is reported, not followed).
speechkv_status make_map(const int32_t *block_table, int32_t max_blocks, int32_t block_size,
                         int64_t num_blocks, speechkv::CacheMap *m) {
    if (!block_table || !aligned(block_table, 4) || max_blocks < 1 || num_blocks < 1 ||
        block_size < 1 || (block_size & (block_size - 1)) != 0 || block_size > (1 << 20))
        return SPEECHKV_ERR_INVALID_ARG;
    if ((int64_t)max_blocks * block_size > INT32_MAX) return SPEECHKV_ERR_UNSUPPORTED;
    int lg = 0;
    while ((1 << lg) < block_size) lg++;
    m->table = block_table;
    m->max_blocks = max_blocks;
    m->bs_log2 = lg;
    m->num_blocks = num_blocks;
    return SPEECHKV_OK;
}

speechkv_status pool_impl(const void *k_full, const void *v_full, const int64_t *full_off,
                          const int32_t *P, const int32_t *T, const int32_t *N, const float *gate,
                          void *k_cache, void *v_cache, const int64_t *cache_off, int32_t *len,
                          int32_t B, int64_t full_rows, int32_t H_kv, int32_t d, int32_t w,
                          int32_t layer, int32_t l0, speechkv_dtype dtype, cudaStream_t stream,
                          const speechkv::CacheMap &map);
speechkv_status append_impl(const void *k_new, const void *v_new, void *k_cache, void *v_cache,
                            const int64_t *cache_off, int32_t *len, int32_t B, int32_t H_kv,
                            int32_t d, int32_t w, int32_t layer, int32_t l0,
                            speechkv_dtype dtype, cudaStream_t stream,
                            const speechkv::CacheMap &map);

}  // namespace

extern "C" {

const char *speechkv_status_string(speechkv_status status) {
    switch (status) {
        case SPEECHKV_OK: return "ok";
        case SPEECHKV_ERR_INVALID_ARG: return "invalid argument";
        case SPEECHKV_ERR_UNSUPPORTED: return "unsupported configuration";
        case SPEECHKV_ERR_CUDA: return "CUDA runtime error";
        case SPEECHKV_ERR_CAPACITY: return "cache capacity exceeded";
        case SPEECHKV_ERR_TIMEOUT: return "bounded device wait timed out";
        case SPEECHKV_ERR_WORKSPACE: return "workspace too small";
    }
    return "unknown status";
}

int64_t speechkv_compressed_len(int32_t P, int32_t T, int32_t N, int32_t G, int32_t w,
                                int32_t layer, int32_t l0) {
    if (P < 0 || T < 0 || N < 0 || G < 0 || w < 1 || layer < 0 || l0 < 0) return -1;
    const int64_t we = layer >= l0 ? w : 1;
    return (int64_t)P + ((int64_t)T + we - 1) / we + N + G;
}

speechkv_status speechkv_pool(const void *k_full, const void *v_full, const int64_t *full_off,
                              const int32_t *P, const int32_t *T, const int32_t *N,
                              const float *gate, void *k_cache, void *v_cache,
                              const int64_t *cache_off, int32_t *len, int32_t B,
                              int64_t full_rows, int32_t H_kv, int32_t d, int32_t w,
                              int32_t layer, int32_t l0, speechkv_dtype dtype,
                              cudaStream_t stream) {
    return pool_impl(k_full, v_full, full_off, P, T, N, gate, k_cache, v_cache, cache_off, len, B,
                     full_rows, H_kv, d, w, layer, l0, dtype, stream, {});
}

speechkv_status speechkv_pool_paged(const void *k_full, const void *v_full,
                                    const int64_t *full_off, const int32_t *P, const int32_t *T,
                                    const int32_t *N, const float *gate, void *k_pages,
                                    void *v_pages, const int32_t *block_table,
                                    int32_t max_blocks, int32_t block_size, int64_t num_blocks,
                                    int32_t *len, int32_t B, int64_t full_rows, int32_t H_kv,
                                    int32_t d, int32_t w, int32_t layer, int32_t l0,
                                    speechkv_dtype dtype, cudaStream_t stream) {
    speechkv::CacheMap m;
    if (B == 0) return SPEECHKV_OK;
    const speechkv_status st = make_map(block_table, max_blocks, block_size, num_blocks, &m);
    if (st != SPEECHKV_OK) return st;
    return pool_impl(k_full, v_full, full_off, P, T, N, gate, k_pages, v_pages, nullptr, len, B,
                     full_rows, H_kv, d, w, layer, l0, dtype, stream, m);
}

speechkv_status speechkv_append(const void *k_new, const void *v_new, void *k_cache,
                                void *v_cache, const int64_t *cache_off, int32_t *len,
                                int32_t B, int32_t H_kv, int32_t d, int32_t w, int32_t layer,
                                int32_t l0, speechkv_dtype dtype, cudaStream_t stream) {
    return append_impl(k_new, v_new, k_cache, v_cache, cache_off, len, B, H_kv, d, w, layer, l0,
                       dtype, stream, {});
}

speechkv_status speechkv_append_paged(const void *k_new, const void *v_new, void *k_pages,
                                      void *v_pages, const int32_t *block_table,
                                      int32_t max_blocks, int32_t block_size,
                                      int64_t num_blocks, int32_t *len, int32_t B,
                                      int32_t H_kv, int32_t d, int32_t w, int32_t layer,
                                      int32_t l0, speechkv_dtype dtype, cudaStream_t stream) {
    speechkv::CacheMap m;
    if (B == 0) return SPEECHKV_OK;
    const speechkv_status st = make_map(block_table, max_blocks, block_size, num_blocks, &m);
    if (st != SPEECHKV_OK) return st;
    return append_impl(k_new, v_new, k_pages, v_pages, nullptr, len, B, H_kv, d, w, layer, l0,
                       dtype, stream, m);
}


size_t speechkv_decode_workspace_size(int32_t B, int32_t H_q, int32_t H_kv, int32_t d,
                                      int32_t grid_ctas) {
    if (B < 0 || H_kv < 1 || H_q < 1 || H_q % H_kv != 0 || grid_ctas < 0) return 0;
    if (!speechkv::decode_supported(SPEECHKV_BF16, d, H_q / H_kv)) return 0;
    int grid = grid_ctas;
    if (grid == 0) {
        DeviceState *s = nullptr;
        if (device_state(&s) != SPEECHKV_OK) return 0;
        grid = s->num_sms * kAutoCtasPerSmMax;
    }
    return workspace_bytes(B, H_q, H_kv, d, grid);
}

speechkv_status speechkv_decode_attn(const void *q, const void *k_cache, const void *v_cache,
                                     const int64_t *cache_off, const int32_t *len, void *out,
                                     float scale, int32_t B, int32_t H_q, int32_t H_kv,
                                     int32_t d, int32_t w, int32_t layer, int32_t l0,
                                     int32_t grid_ctas, void *workspace, size_t workspace_bytes_in,
                                     speechkv_dtype dtype, uint32_t flags, cudaStream_t stream) {
    // the caches and len are only read on this path
    return decode_common(q, nullptr, nullptr, const_cast<void *>(k_cache),
                         const_cast<void *>(v_cache), cache_off, const_cast<int32_t *>(len), out,
                         scale, B, H_q, H_kv, d, w, layer, l0, grid_ctas, workspace,
                         workspace_bytes_in, dtype, flags, stream, false);
}

speechkv_status speechkv_decode_step(const void *q, const void *k_new, const void *v_new,
                                     void *k_cache, void *v_cache, const int64_t *cache_off,
                                     int32_t *len, void *out, float scale, int32_t B, int32_t H_q,
                                     int32_t H_kv, int32_t d, int32_t w, int32_t layer, int32_t l0,
                                     int32_t grid_ctas, void *workspace, size_t workspace_bytes_in,
                                     speechkv_dtype dtype, uint32_t flags, cudaStream_t stream) {
    return decode_common(q, k_new, v_new, k_cache, v_cache, cache_off, len, out, scale, B, H_q,
                         H_kv, d, w, layer, l0, grid_ctas, workspace, workspace_bytes_in, dtype,
                         flags, stream, true);
}

speechkv_status speechkv_selftest_timeout(cudaStream_t stream) {
    DeviceState *s = nullptr;
    speechkv_status st = device_state(&s);
    if (st != SPEECHKV_OK) return st;
    return speechkv::launch_selftest_timeout(s->err, stream) == cudaSuccess ? SPEECHKV_OK
                                                                           : SPEECHKV_ERR_CUDA;
}

speechkv_status speechkv_check_device_error(cudaStream_t stream) {
    DeviceState *s = nullptr;
    speechkv_status st = device_state(&s);
    if (st != SPEECHKV_OK) return st;
    if (cudaStreamSynchronize(stream) != cudaSuccess) return SPEECHKV_ERR_CUDA;
    int v = 0;
    if (cudaMemcpyFromSymbol(&v, speechkv_error_word, sizeof(int)) != cudaSuccess)
        return SPEECHKV_ERR_CUDA;
    const int zero = 0;
    if (v != 0 && cudaMemcpyToSymbol(speechkv_error_word, &zero, sizeof(int)) != cudaSuccess)
        return SPEECHKV_ERR_CUDA;
    return static_cast<speechkv_status>(v);
}

speechkv_status speechkv_pool_hidden(const void *h_full, const int64_t *full_off,
                                     const int32_t *P, const int32_t *T, const int32_t *N,
                                     const float *gate, void *h_out, const int64_t *out_off,
                                     int32_t *len, int32_t B, int64_t full_rows,
                                     int64_t out_rows, int32_t d_model, int32_t w,
                                     speechkv_dtype dtype, cudaStream_t stream) {
    if (B < 0 || full_rows < 0 || out_rows < 0 || d_model < 1 || w < 1 || !valid_dtype(dtype))
        return SPEECHKV_ERR_INVALID_ARG;
    if (!speechkv::pool_hidden_supported(dtype, d_model)) return SPEECHKV_ERR_UNSUPPORTED;
    if (B == 0) return SPEECHKV_OK;
    if (!full_off || !P || !T || !N || !gate || !h_out || !out_off || !len ||
        (full_rows > 0 && !h_full))
        return SPEECHKV_ERR_INVALID_ARG;
    if (!aligned(h_full, 16) || !aligned(h_out, 16) || !aligned(full_off, 8) ||
        !aligned(out_off, 8) || !aligned(P, 4) || !aligned(T, 4) || !aligned(N, 4) ||
        !aligned(len, 4) || !aligned(gate, 4))
        return SPEECHKV_ERR_INVALID_ARG;
    DeviceState *s = nullptr;
    speechkv_status st = device_state(&s);
    if (st != SPEECHKV_OK) return st;
    speechkv::PoolHiddenArgs a;
    a.h_full = h_full;
    a.full_off = full_off;
    a.P = P;
    a.T = T;
    a.N = N;
    a.gate = gate;
    a.h_out = h_out;
    a.out_off = out_off;
    a.len = len;
    a.B = B;
    a.full_rows = full_rows;
    a.out_rows = out_rows;
    a.d_model = d_model;
    a.w = w;
    a.dtype = dtype;
    a.err = s->err;
    return speechkv::launch_pool_hidden(a, s->num_sms, stream) == cudaSuccess
               ? SPEECHKV_OK
               : SPEECHKV_ERR_CUDA;
}

// Host checks and launch of speechkv_prefill_attn and its paged form
// (map.table != nullptr: k_cache / v_cache are the page pools).
static speechkv_status prefill_common(const void *q, const int64_t *q_off, int64_t q_rows,
                                      const int32_t *P, const int32_t *T, const int32_t *N,
                                      const void *k_cache, const void *v_cache,
                                      const int64_t *cache_off, int64_t cache_rows, void *out,
                                      float scale, int32_t B, int32_t H_q, int32_t H_kv,
                                      int32_t d, int32_t w, int32_t layer, int32_t l0,
                                      speechkv_dtype dtype, cudaStream_t stream,
                                      const speechkv::CacheMap &map) {
    const bool paged = map.table != nullptr;
    if (B < 0 || B > SPEECHKV_MAX_BATCH || q_rows < 0 || cache_rows < 0 || H_q < 1 ||
        H_kv < 1 || H_q % H_kv != 0 || w < 1 || layer < 0 || l0 < 0 || !valid_dtype(dtype) ||
        isnan(scale) || isinf(scale) || scale < 0.f)
        return SPEECHKV_ERR_INVALID_ARG;
    if (!speechkv::prefill_supported(dtype, d)) return SPEECHKV_ERR_UNSUPPORTED;
    // tensor-copy coordinates are 32-bit; a page is copied as whole 8-row
    // swizzle atoms
    const int64_t kv_rows =
        paged ? map.num_blocks * H_kv * ((int64_t)1 << map.bs_log2) : cache_rows * (int64_t)H_kv;
    if (q_rows >= (1ll << 31) || kv_rows >= (1ll << 31) || H_q > 256 ||
        (paged && map.bs_log2 < 3))
        return SPEECHKV_ERR_UNSUPPORTED;
    if (B == 0 || q_rows == 0) return SPEECHKV_OK;
    if (!q || !q_off || !P || !T || !N || !k_cache || !v_cache || (!paged && !cache_off) ||
        !out || (!paged && cache_rows == 0))
        return SPEECHKV_ERR_INVALID_ARG;
    if (!aligned(q, 16) || !aligned(k_cache, 16) || !aligned(v_cache, 16) || !aligned(out, 16) ||
        !aligned(q_off, 8) || (!paged && !aligned(cache_off, 8)) || !aligned(P, 4) ||
        !aligned(T, 4) || !aligned(N, 4))
        return SPEECHKV_ERR_INVALID_ARG;
    DeviceState *s = nullptr;
    speechkv_status st = device_state(&s);
    if (st != SPEECHKV_OK) return st;
    speechkv::PrefillArgs a;
    a.q = q;
    a.q_off = q_off;
    a.q_rows = q_rows;
    a.P = P;
    a.T = T;
    a.N = N;
    a.k_cache = k_cache;
    a.v_cache = v_cache;
    a.cache_off = paged ? nullptr : cache_off;
    a.cache_rows = paged ? 0 : cache_rows;
    a.out = out;
    a.scale = scale > 0.f ? scale : 1.f / sqrtf((float)d);
    a.B = B;
    a.H_q = H_q;
    a.H_kv = H_kv;
    a.d = d;
    a.w_eff = layer >= l0 ? w : 1;
    a.err = s->err;
    a.map = map;
    return speechkv::launch_prefill(a, s->num_sms, stream) == cudaSuccess ? SPEECHKV_OK
                                                                          : SPEECHKV_ERR_CUDA;
}

speechkv_status speechkv_prefill_attn(const void *q, const int64_t *q_off, int64_t q_rows,
                                      const int32_t *P, const int32_t *T, const int32_t *N,
                                      const void *k_cache, const void *v_cache,
                                      const int64_t *cache_off, int64_t cache_rows, void *out,
                                      float scale, int32_t B, int32_t H_q, int32_t H_kv,
                                      int32_t d, int32_t w, int32_t layer, int32_t l0,
                                      speechkv_dtype dtype, cudaStream_t stream) {
    return prefill_common(q, q_off, q_rows, P, T, N, k_cache, v_cache, cache_off, cache_rows,
                          out, scale, B, H_q, H_kv, d, w, layer, l0, dtype, stream,
                          speechkv::CacheMap{});
}

speechkv_status speechkv_prefill_attn_paged(
    const void *q, const int64_t *q_off, int64_t q_rows, const int32_t *P, const int32_t *T,
    const int32_t *N, const void *k_pages, const void *v_pages, const int32_t *block_table,
    int32_t max_blocks, int32_t block_size, int64_t num_blocks, void *out, float scale,
    int32_t B, int32_t H_q, int32_t H_kv, int32_t d, int32_t w, int32_t layer, int32_t l0,
    speechkv_dtype dtype, cudaStream_t stream) {
    speechkv::CacheMap m;
    if (B == 0 || q_rows == 0) return SPEECHKV_OK;
    const speechkv_status st = make_map(block_table, max_blocks, block_size, num_blocks, &m);
    if (st != SPEECHKV_OK) return st;
    return prefill_common(q, q_off, q_rows, P, T, N, k_pages, v_pages, nullptr, 0, out, scale,
                          B, H_q, H_kv, d, w, layer, l0, dtype, stream, m);
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Allocation-free variant of speechkv_decode_step (no counterpart in the
// paper).  Its split-K scratch lives in a fixed-size array in device memory
// that belongs to the library itself, so the caller passes no workspace.
// ---------------------------------------------------------------------------

// Every GPU that loads this library holds this array until the process exits.
static __device__ __align__(256) unsigned char speechkv_noalloc_scratch[SPEECHKV_NOALLOC_SCRATCH_BYTES];

namespace {

void *g_noalloc_scratch[kMaxDevices];  // the array's device address, per device

// In host code `speechkv_noalloc_scratch` names a host-side stand-in, not the
// device memory; kernels must be given the address cudaGetSymbolAddress
// returns for the current device.  Done once per device, on first use.
speechkv_status noalloc_scratch(void **out) {
    int dev = 0;
    speechkv_status st = current_device(&dev);
    if (st != SPEECHKV_OK) return st;
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_noalloc_scratch[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, speechkv_noalloc_scratch) != cudaSuccess || !p)
            return SPEECHKV_ERR_CUDA;
        g_noalloc_scratch[dev] = p;
    }
    *out = g_noalloc_scratch[dev];
    return SPEECHKV_OK;
}

}  // namespace

extern "C" speechkv_status speechkv_decode_step_noalloc(
    const void *q, const void *k_new, const void *v_new, void *k_cache, void *v_cache,
    const int64_t *cache_off, int32_t *len, void *out, float scale, int32_t B, int32_t H_q,
    int32_t H_kv, int32_t d, int32_t w, int32_t layer, int32_t l0, int32_t grid_ctas,
    speechkv_dtype dtype, uint32_t flags, cudaStream_t stream) {
    if (B < 0 || H_q < 1 || H_kv < 1 || H_q % H_kv != 0 || grid_ctas < 0)
        return SPEECHKV_ERR_INVALID_ARG;
    if (!speechkv::decode_supported(dtype, d, H_q / H_kv)) return SPEECHKV_ERR_UNSUPPORTED;
    if (B > SPEECHKV_MAX_BATCH) return SPEECHKV_ERR_UNSUPPORTED;
    if (B == 0) return SPEECHKV_OK;
    DeviceState *s = nullptr;
    speechkv_status st = device_state(&s);
    if (st != SPEECHKV_OK) return st;
    void *scratch = nullptr;
    st = noalloc_scratch(&scratch);
    if (st != SPEECHKV_OK) return st;
    int grid = grid_ctas;
    if (grid == 0) {
        st = decode_auto_grid(s, dtype, d, H_q / H_kv, B, &grid);
        if (st != SPEECHKV_OK) return st;
    }
    // a batch whose scratch would not fit is refused before anything runs
    if (workspace_bytes(B, H_q, H_kv, d, grid) > (size_t)SPEECHKV_NOALLOC_SCRATCH_BYTES)
        return SPEECHKV_ERR_WORKSPACE;
    // every other argument is checked before anything is queued on the stream
    speechkv::DecodeArgs a;
    bool launch = false;
    st = decode_prepare(q, k_new, v_new, k_cache, v_cache, cache_off, len, out, scale, B, H_q,
                        H_kv, d, w, layer, l0, grid, scratch, SPEECHKV_NOALLOC_SCRATCH_BYTES,
                        dtype, flags, true, {}, &a, &grid, &launch);
    if (st != SPEECHKV_OK || !launch) return st;
    // the counters must start at zero; the array keeps the previous call's data
    if (cudaMemsetAsync(scratch, 0, counters_bytes(B, H_kv), stream) != cudaSuccess)
        return SPEECHKV_ERR_CUDA;
    return speechkv::launch_decode(a, grid, stream) == cudaSuccess ? SPEECHKV_OK
                                                                   : SPEECHKV_ERR_CUDA;
}

extern "C" speechkv_status speechkv_decode_step_paged(
    const void *q, const void *k_new, const void *v_new, void *k_pages, void *v_pages,
    const int32_t *block_table, int32_t max_blocks, int32_t block_size, int64_t num_blocks,
    int32_t *len, void *out, float scale, int32_t B, int32_t H_q, int32_t H_kv, int32_t d,
    int32_t w, int32_t layer, int32_t l0, int32_t grid_ctas, void *workspace,
    size_t workspace_bytes_in, speechkv_dtype dtype, uint32_t flags, cudaStream_t stream) {
    speechkv::CacheMap m;
    if (B == 0) return SPEECHKV_OK;
    const speechkv_status st = make_map(block_table, max_blocks, block_size, num_blocks, &m);
    if (st != SPEECHKV_OK) return st;
    return decode_common(q, k_new, v_new, k_pages, v_pages, nullptr, len, out, scale, B, H_q,
                         H_kv, d, w, layer, l0, grid_ctas, workspace, workspace_bytes_in, dtype,
                         flags, stream, true, m);
}

namespace {

speechkv_status pool_impl(const void *k_full, const void *v_full, const int64_t *full_off,
                              const int32_t *P, const int32_t *T, const int32_t *N,
                              const float *gate, void *k_cache, void *v_cache,
                              const int64_t *cache_off, int32_t *len, int32_t B,
                              int64_t full_rows, int32_t H_kv, int32_t d, int32_t w,
                              int32_t layer, int32_t l0, speechkv_dtype dtype,
                              cudaStream_t stream, const speechkv::CacheMap &map) {
    if (B < 0 || full_rows < 0 || H_kv < 1 || w < 1 || layer < 0 || l0 < 0 || !valid_dtype(dtype))
        return SPEECHKV_ERR_INVALID_ARG;
    if (d != 64 && d != 128) return SPEECHKV_ERR_UNSUPPORTED;
    if (B == 0) return SPEECHKV_OK;
    if (!full_off || !P || !T || !N || !gate || !k_cache || !v_cache ||
        (!cache_off && !map.table) || !len ||
        (full_rows > 0 && (!k_full || !v_full)))
        return SPEECHKV_ERR_INVALID_ARG;
    if (!aligned(k_full, 16) || !aligned(v_full, 16) || !aligned(k_cache, 16) ||
        !aligned(v_cache, 16) || !aligned(full_off, 8) || !aligned(cache_off, 8) ||
        !aligned(P, 4) || !aligned(T, 4) || !aligned(N, 4) || !aligned(len, 4) ||
        !aligned(gate, 16))
        return SPEECHKV_ERR_INVALID_ARG;
    DeviceState *s = nullptr;
    speechkv_status st = device_state(&s);
    if (st != SPEECHKV_OK) return st;
    speechkv::PoolArgs a;
    a.k_full = k_full;
    a.v_full = v_full;
    a.full_off = full_off;
    a.P = P;
    a.T = T;
    a.N = N;
    a.gate = gate;
    a.k_cache = k_cache;
    a.v_cache = v_cache;
    a.cache_off = cache_off;
    a.len = len;
    a.B = B;
    a.full_rows = full_rows;
    a.H_kv = H_kv;
    a.d = d;
    a.w_eff = layer >= l0 ? w : 1;
    a.dtype = dtype;
    a.err = s->err;
    a.map = map;
    return speechkv::launch_pool(a, s->num_sms, stream) == cudaSuccess ? SPEECHKV_OK
                                                                       : SPEECHKV_ERR_CUDA;
}




speechkv_status append_impl(const void *k_new, const void *v_new, void *k_cache,
                                void *v_cache, const int64_t *cache_off, int32_t *len,
                                int32_t B, int32_t H_kv, int32_t d, int32_t w, int32_t layer,
                                int32_t l0, speechkv_dtype dtype, cudaStream_t stream,
                            const speechkv::CacheMap &map) {
    if (B < 0 || H_kv < 1 || w < 1 || layer < 0 || l0 < 0 || !valid_dtype(dtype))
        return SPEECHKV_ERR_INVALID_ARG;
    if (d != 64 && d != 128) return SPEECHKV_ERR_UNSUPPORTED;
    if (B == 0) return SPEECHKV_OK;
    if (!k_new || !v_new || !k_cache || !v_cache || (!cache_off && !map.table) || !len)
        return SPEECHKV_ERR_INVALID_ARG;
    if (!aligned(k_new, 16) || !aligned(v_new, 16) || !aligned(k_cache, 16) ||
        !aligned(v_cache, 16) || !aligned(cache_off, 8) || !aligned(len, 4))
        return SPEECHKV_ERR_INVALID_ARG;
    DeviceState *s = nullptr;
    speechkv_status st = device_state(&s);
    if (st != SPEECHKV_OK) return st;
    speechkv::AppendArgs a;
    a.k_new = k_new;
    a.v_new = v_new;
    a.k_cache = k_cache;
    a.v_cache = v_cache;
    a.cache_off = cache_off;
    a.len = len;
    a.B = B;
    a.H_kv = H_kv;
    a.d = d;
    a.dtype = dtype;
    a.err = s->err;
    a.map = map;
    return speechkv::launch_append(a, stream) == cudaSuccess ? SPEECHKV_OK : SPEECHKV_ERR_CUDA;
}

}  // namespace
