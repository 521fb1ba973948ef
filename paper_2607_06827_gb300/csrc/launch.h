// Host-side launchers of the SpeechKV kernels (internal to libspeechkv).
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "speechkv.h"

namespace speechkv {

// Where a layer's cached rows live.  Contiguous (table == nullptr): request
// b owns rows [cache_off[b], cache_off[b+1]) of every KV head's run, head h
// of request b starting at row cache_off[b] * H_kv + h * cap_b.  Paged:
// logical block t >> bs_log2 of request b is physical block
// table[b * max_blocks + (t >> bs_log2)] of pages [num_blocks][H_kv]
// [1 << bs_log2][d]; a request's capacity is max_blocks << bs_log2 rows.
struct CacheMap {
    const int32_t *table = nullptr;
    int32_t max_blocks = 0, bs_log2 = 0;
    int64_t num_blocks = 0;
};

struct PoolArgs {
    const void *k_full, *v_full;
    const int64_t *full_off;
    const int32_t *P, *T, *N;
    const float *gate;
    void *k_cache, *v_cache;
    const int64_t *cache_off;
    int32_t *len;
    int32_t B;
    int64_t full_rows;
    int32_t H_kv, d, w_eff;
    speechkv_dtype dtype;
    int *err;
    CacheMap map;  // paged layout when map.table != nullptr (cache_off unused)
};
cudaError_t launch_pool(const PoolArgs &a, int num_sms, cudaStream_t stream);

struct PoolHiddenArgs {
    const void *h_full;  // [full_rows][d_model]
    const int64_t *full_off;
    const int32_t *P, *T, *N;
    const float *gate;   // [d_model]
    void *h_out;         // [out_rows][d_model]
    const int64_t *out_off;
    int32_t *len;
    int32_t B;
    int64_t full_rows, out_rows;
    int32_t d_model, w;
    speechkv_dtype dtype;
    int *err;
};
// Whether (dtype, d_model) is supported by the hidden-state pooling kernel.
bool pool_hidden_supported(speechkv_dtype dtype, int d_model);
cudaError_t launch_pool_hidden(const PoolHiddenArgs &a, int num_sms, cudaStream_t stream);

struct AppendArgs {
    const void *k_new, *v_new;
    void *k_cache, *v_cache;
    const int64_t *cache_off;
    int32_t *len;
    int32_t B, H_kv, d;
    speechkv_dtype dtype;
    int *err;
    CacheMap map;  // paged layout when map.table != nullptr (cache_off unused)
};
cudaError_t launch_append(const AppendArgs &a, cudaStream_t stream);
// A bounded wait that runs out (see speechkv_selftest_timeout).
cudaError_t launch_selftest_timeout(int *err, cudaStream_t stream);

struct DecodeArgs {
    const void *q;
    const void *k_new, *v_new;  // non-null: fused append (speechkv_decode_step)
    void *k_cache, *v_cache;
    const int64_t *cache_off;
    int32_t *len;  // read; with a fused append also advanced
    void *out;
    float scale;  // > 0
    int32_t B, H_q, H_kv, d;
    speechkv_dtype dtype;
    float *partials;   // [grid + B*H_kv][slot_floats]
    int *counters;     // [B*H_kv]
    int *done;         // CTAs past the prologue (fused append only)
    int *err;
    bool overlap;      // SPEECHKV_OVERLAP_PRIOR: start before the previous kernel ends
    CacheMap map;      // paged layout when map.table != nullptr (cache_off unused)
};

// Whether (dtype, d, group) has a compiled decode kernel.
bool decode_supported(speechkv_dtype dtype, int d, int group);
// Most query heads per KV head of the bf16 decode instances (tensor-core
// consumers: the heads of a group are padded to one 8-column MMA tile).
constexpr int kMmaMaxGroup = 8;
// The bf16, d = 128 instances (decode_attn_mma.cu).
int decode_ctas_per_sm_mma128(int group, int B);
cudaError_t launch_decode_mma128(const DecodeArgs &a, int grid, cudaStream_t stream);
// Resident CTAs per SM of that kernel on the current device for a batch of
// B requests (0 on error).
int decode_ctas_per_sm(speechkv_dtype dtype, int d, int group, int B);
// Floats per partial-result slot (m, l and o for every query head of a group).
int decode_slot_floats(int d, int group);
cudaError_t launch_decode(const DecodeArgs &a, int grid, cudaStream_t stream);

struct PrefillArgs {
    const void *q;  // [q_rows][H_q][d]
    const int64_t *q_off;
    int64_t q_rows;
    const int32_t *P, *T, *N;
    const void *k_cache, *v_cache;
    const int64_t *cache_off;
    int64_t cache_rows;  // rows per KV head block extent: buffers hold cache_rows * H_kv * d
    void *out;           // [q_rows][H_q][d]
    float scale;         // > 0
    int32_t B, H_q, H_kv, d, w_eff;
    int *err;
    CacheMap map;  // paged layout when map.table != nullptr (cache_off, cache_rows unused)
};
// Whether (dtype, d) has a compiled prefill kernel.
bool prefill_supported(speechkv_dtype dtype, int d);
cudaError_t launch_prefill(const PrefillArgs &a, int num_sms, cudaStream_t stream);

}  // namespace speechkv
