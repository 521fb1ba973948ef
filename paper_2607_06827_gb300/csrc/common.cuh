// Device-side helpers shared by the SpeechKV kernels (sm_103a).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "speechkv.h"

namespace speechkv {

// Host-visible launch descriptors live in launch.h; this header is device-side.

// Upper bound of every device-side wait, in nanoseconds of %globaltimer.
constexpr unsigned long long kWaitLimitNs = 1000ull * 1000ull * 1000ull;  // 1 s

__device__ __forceinline__ void report_error(int *err, int code) {
    atomicCAS(err, 0, code);  // first error wins
}

__device__ __forceinline__ unsigned long long global_timer_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// ---------------------------------------------------------------------------
// cache addressing (contiguous runs or pages; see CacheMap in launch.h)
// ---------------------------------------------------------------------------
// Element offset of row t of (request b, KV head h): contiguous runs start
// at row off_b * H_kv + h * cap_b; pages at ((block * H_kv + h) << bs_log2).
// -1 when the request's block-table entry for t is not a valid block.
template <typename Map>
__device__ __forceinline__ int64_t cache_row(const Map &m, int b, int h, int64_t t, int H_kv,
                                             int D, int64_t off_b, int64_t cap_b) {
    if (!m.table) return (off_b * H_kv + (int64_t)h * cap_b + t) * D;
    const int32_t blk = __ldg(m.table + (int64_t)b * m.max_blocks + (t >> m.bs_log2));
    if (blk < 0 || blk >= m.num_blocks) return -1;
    const int64_t in_blk = t & ((1ll << m.bs_log2) - 1);
    return ((((int64_t)blk * H_kv + h) << m.bs_log2) + in_blk) * D;
}

// ---------------------------------------------------------------------------
// element conversions
// ---------------------------------------------------------------------------
// bf16 pair packed in a 32-bit word (element 2k in the low half).
__device__ __forceinline__ float bf16_lo(uint32_t x) { return __uint_as_float(x << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t x) { return __uint_as_float(x & 0xffff0000u); }

template <typename T>
__device__ __forceinline__ T from_float(float x);
template <>
__device__ __forceinline__ float from_float<float>(float x) { return x; }
template <>
__device__ __forceinline__ __nv_bfloat16 from_float<__nv_bfloat16>(float x) {
    return __float2bfloat16_rn(x);
}

template <typename T>
__device__ __forceinline__ float to_float(T x);
template <>
__device__ __forceinline__ float to_float<float>(float x) { return x; }
template <>
__device__ __forceinline__ float to_float<__nv_bfloat16>(__nv_bfloat16 x) {
    return __bfloat162float(x);
}

// Load N consecutive elements (N * sizeof(T) in {4, 8, 16} bytes, aligned)
// and widen to fp32.
template <typename T, int N>
__device__ __forceinline__ void load_vec(const T *p, float (&f)[N]) {
    constexpr int BYTES = N * (int)sizeof(T);
    static_assert(BYTES == 4 || BYTES == 8 || BYTES == 16, "vector width");
    if constexpr (sizeof(T) == 4) {
        if constexpr (N == 1) {
            f[0] = *reinterpret_cast<const float *>(p);
        } else if constexpr (N == 2) {
            float2 v = *reinterpret_cast<const float2 *>(p);
            f[0] = v.x; f[1] = v.y;
        } else {
            float4 v = *reinterpret_cast<const float4 *>(p);
            f[0] = v.x; f[1] = v.y; f[2] = v.z; f[3] = v.w;
        }
    } else {
        if constexpr (N == 2) {
            uint32_t v = *reinterpret_cast<const uint32_t *>(p);
            f[0] = bf16_lo(v); f[1] = bf16_hi(v);
        } else if constexpr (N == 4) {
            uint2 v = *reinterpret_cast<const uint2 *>(p);
            f[0] = bf16_lo(v.x); f[1] = bf16_hi(v.x);
            f[2] = bf16_lo(v.y); f[3] = bf16_hi(v.y);
        } else {
            uint4 v = *reinterpret_cast<const uint4 *>(p);
            f[0] = bf16_lo(v.x); f[1] = bf16_hi(v.x);
            f[2] = bf16_lo(v.y); f[3] = bf16_hi(v.y);
            f[4] = bf16_lo(v.z); f[5] = bf16_hi(v.z);
            f[6] = bf16_lo(v.w); f[7] = bf16_hi(v.w);
        }
    }
}

// Round N fp32 values to T and store them (N * sizeof(T) in {4, 8, 16}).
template <typename T, int N>
__device__ __forceinline__ void store_vec(T *p, const float (&f)[N]) {
    if constexpr (sizeof(T) == 4) {
        if constexpr (N == 2) {
            *reinterpret_cast<float2 *>(p) = make_float2(f[0], f[1]);
        } else {
            static_assert(N == 4, "vector width");
            *reinterpret_cast<float4 *>(p) = make_float4(f[0], f[1], f[2], f[3]);
        }
    } else {
        uint32_t w[N / 2];
#pragma unroll
        for (int i = 0; i < N / 2; i++) {
            __nv_bfloat162 h = __floats2bfloat162_rn(f[2 * i], f[2 * i + 1]);
            w[i] = *reinterpret_cast<uint32_t *>(&h);
        }
        if constexpr (N == 2) {
            *reinterpret_cast<uint32_t *>(p) = w[0];
        } else if constexpr (N == 4) {
            *reinterpret_cast<uint2 *>(p) = make_uint2(w[0], w[1]);
        } else {
            static_assert(N == 8, "vector width");
            *reinterpret_cast<uint4 *>(p) = make_uint4(w[0], w[1], w[2], w[3]);
        }
    }
}

// Raw copy of BYTES (4, 8 or 16) bytes.
template <int BYTES>
__device__ __forceinline__ void copy_bytes(void *dst, const void *src) {
    if constexpr (BYTES == 16) {
        *reinterpret_cast<uint4 *>(dst) = *reinterpret_cast<const uint4 *>(src);
    } else if constexpr (BYTES == 8) {
        *reinterpret_cast<uint2 *>(dst) = *reinterpret_cast<const uint2 *>(src);
    } else {
        static_assert(BYTES == 4, "copy width");
        *reinterpret_cast<uint32_t *>(dst) = *reinterpret_cast<const uint32_t *>(src);
    }
}

__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

// 2^x on the special-function unit (ex2.approx; 2^-inf = +0).
__device__ __forceinline__ float fast_exp2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// ---------------------------------------------------------------------------
// packed fp32 pairs (sm_100+ f32x2 arithmetic: two lanes of math per issue)
// ---------------------------------------------------------------------------
__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) {
    float2 d;
    asm("{\n\t.reg .b64 ra, rb, rc, rd;\n\t"
        "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\tmov.b64 rc, {%6, %7};\n\t"
        "fma.rn.f32x2 rd, ra, rb, rc;\n\tmov.b64 {%0, %1}, rd;\n\t}"
        : "=f"(d.x), "=f"(d.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
    return d;
}

__device__ __forceinline__ float2 fmul2(float2 a, float2 b) {
    float2 d;
    asm("{\n\t.reg .b64 ra, rb, rd;\n\t"
        "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
        "mul.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd;\n\t}"
        : "=f"(d.x), "=f"(d.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return d;
}

// The two bf16 of a packed 32-bit word as an fp32 pair (exact).
__device__ __forceinline__ float2 bf16x2_to_float2(uint32_t x) {
    return make_float2(bf16_lo(x), bf16_hi(x));
}

// 16 bytes of T as fp32 pairs: 4 pairs for bf16, 2 for fp32.
template <typename T>
__device__ __forceinline__ void load16_pairs(const void *p, float2 (&f)[16 / sizeof(T) / 2]) {
    if constexpr (sizeof(T) == 2) {
        const uint4 v = *reinterpret_cast<const uint4 *>(p);
        f[0] = bf16x2_to_float2(v.x);
        f[1] = bf16x2_to_float2(v.y);
        f[2] = bf16x2_to_float2(v.z);
        f[3] = bf16x2_to_float2(v.w);
    } else {
        const float4 v = *reinterpret_cast<const float4 *>(p);
        f[0] = make_float2(v.x, v.y);
        f[1] = make_float2(v.z, v.w);
    }
}

// ---------------------------------------------------------------------------
// warp-level tensor-core operations (mma.sync / ldmatrix / movmatrix, PTX ISA
// "Warp-level matrix instructions"); fragment layouts are those of the
// m16n8k16 shape: lane = 4 r + t holds rows r and r + 8, columns (or k
// indices) 2t and 2t + 1 (+ 8)
// ---------------------------------------------------------------------------
// d += a (16 x 16, row-major fragments) * b (16 x 8, column-major), bf16 in,
// fp32 accumulate.
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                               uint32_t b1) {
    asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, "
        "{%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Four 8x8 b16 matrices from shared memory; lanes 8i .. 8i + 7 give the row
// addresses (16 bytes each) of matrix i.  Lane 4r + t receives row r,
// elements 2t and 2t + 1 of each (transposed: row 2t and 2t + 1, element r).
__device__ __forceinline__ void ldmatrix_x4(uint32_t (&r)[4], uint32_t addr) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr)
                 : "memory");
}
__device__ __forceinline__ void ldmatrix_x4_trans(uint32_t (&r)[4], uint32_t addr) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr)
                 : "memory");
}

// Transpose of an 8x8 b16 matrix held one row pair per lane (lane 4r + t:
// row r, elements 2t, 2t + 1) into the same layout.
__device__ __forceinline__ uint32_t movmatrix_trans(uint32_t x) {
    uint32_t y;
    asm("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(y) : "r"(x));
    return y;
}

// Two floats rounded to bf16 (to nearest even) in one word: lo in the low half.
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}

// Atomic add with acquire-release semantics at GPU scope (publishes the
// CTA's earlier writes, ordered before it by a barrier, to the acquirer).
__device__ __forceinline__ int atomic_add_acq_rel_gpu(int *p, int v) {
    int old;
    asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v)
                 : "memory");
    return old;
}

// Hint: bring `bytes` (a multiple of 16, 16-byte aligned) of global memory
// into L2.  No value is read; later reads see whatever the memory holds then.
__device__ __forceinline__ void prefetch_l2(const void *p, uint32_t bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

// Orders this thread's earlier generic-proxy shared-memory accesses before
// later async-proxy (TMA) accesses of the same shared memory.
__device__ __forceinline__ void fence_proxy_async_shared() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// ---------------------------------------------------------------------------
// programmatic dependent launch (kernels launched with the PDL attribute)
// ---------------------------------------------------------------------------
// Let the next kernel on the stream (if it was launched with the attribute)
// be scheduled as this grid's CTAs retire.
__device__ __forceinline__ void griddep_launch_dependents() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
// Block until the grids this one depends on have completed and their memory
// operations are visible (a no-op when launched without the attribute).
__device__ __forceinline__ void griddep_wait() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
}

// ---------------------------------------------------------------------------
// mbarrier + bulk asynchronous copy (TMA, non-tensor form)
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_addr(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count)
                 : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)),
                 "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_addr(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

// Wait until the phase with the given parity has completed, for at most
// kWaitLimitNs.  Returns false (and reports SPEECHKV_ERR_TIMEOUT) on timeout.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t *bar, uint32_t parity, int *err) {
    if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long t0 = global_timer_ns();
    for (;;) {
        for (int i = 0; i < 64; i++)
            if (mbar_try_wait(bar, parity)) return true;
        if (global_timer_ns() - t0 > kWaitLimitNs) {
            report_error(err, SPEECHKV_ERR_TIMEOUT);
            return false;
        }
    }
}

// Bulk copy global -> shared of `bytes` (multiple of 16, both ends 16-byte
// aligned); completion is signalled on `bar` as transaction bytes.
__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes,
                                         uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
            "r"(smem_addr(dst)),
        "l"(src), "r"(bytes), "r"(smem_addr(bar))
        : "memory");
}

}  // namespace speechkv
