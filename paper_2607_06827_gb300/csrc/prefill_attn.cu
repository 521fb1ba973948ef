// speechkv_prefill_attn: Eq. (attn) at prefill (Sec. III-B) -- every
// full-resolution prompt query attends over the compressed cache rows that
// precede it.  A query at prompt position t sits at compressed position
//   pi(t) = t                     text before the speech   (t < P)
//         = P + (t - P) / w_eff   speech frame (its own window)
//         = t - T + n             text after the speech
// and sees rows 0 .. pi(t) (causality over the compressed sequence).
//
// Blackwell tensor-core flash attention, bf16 in, fp32 accumulate, d = 128:
//   * persistent: one CTA per SM walks work items (request, KV head, 128-row
//     query tile, pair of query heads of that KV head) ordered by (request,
//     KV head), so that the CTAs running together read the same keys and
//     values (from L2); the two query tiles of an item ("slots") share every
//     key and value tile, which halves the L2 -> SM traffic per FLOP (at one
//     query tile per CTA the loads, not the tensor cores, set the pace);
//   * warp 0 lane 0: TMA tensor copies (128-byte swizzle) of the two query
//     tiles and of 128-row key tiles (three stages) and value tiles (two
//     stages), keys one tile ahead of values;
//   * warp 1: tcgen05.mma issue, the warp converged and one elected lane
//     issuing (a lone issuing thread was slowed more by the softmax warps'
//     instruction issue on its sub-partition) -- per key tile and slot x,
//     O_x += P_x V then S_x = Q_x K^T of the next key tile, into 128-column
//     TMEM buffers (S_0, S_1, O_0, O_1: all 512 columns); P_x is stored over
//     the first half of S_x and read as the A operand from TMEM, so a slot's
//     next Q K^T waits for its P V while the other slot's products keep the
//     tensor pipe busy;
//   * warps 2-5 (slot 0) and 6-9 (slot 1): softmax, one query row per thread
//     (= TMEM lane): the S row read from TMEM in one load, masked keys set to
//     -inf once per masked tile, row maximum, base-2 exponentials with
//     log2(e)/sqrt(d) folded in, P stored as bf16 pairs, O rescaled in TMEM
//     only when a row's maximum rose by more than 2^8 (lazy rescaling), and
//     the epilogue O / l to global memory.
// Cache rows past a request's compressed length are zeroed in the value
// stage (their contents are unspecified and the MMA would multiply them by
// zero weights: 0 x NaN is NaN).  Every wait is bounded; on a timeout the CTA
// stops, lets its copies and MMAs finish and reports SPEECHKV_ERR_TIMEOUT.
#include <cuda.h>
#include <math.h>

#include <mutex>

#include "common.cuh"
#include "launch.h"

namespace speechkv {
namespace {

constexpr int kBM = 128;  // query rows per tile = TMEM lanes
constexpr int kBN = 128;  // keys per tile
constexpr int kSlots = 2;    // query tiles per CTA (two query heads of one KV head)
constexpr int kThreads = 64 + kSlots * 128;  // TMA warp, MMA warp, a softmax warpgroup per slot
constexpr int kBlockBytes = kBM * 128;    // a 64-column block of a tile (128-byte rows)
constexpr uint32_t kTmemCols = 512;       // S_x: 128 x, O_x: 256 + D x; P_x over S_x's first 64

// Per head dimension D (64 or 128): a tile of 128 rows x D is D / 64 blocks;
// shared memory (offsets from a 1024-byte aligned base) holds the two query
// tiles and the key and value rings, then the barriers.
template <int D>
struct PfCfg {
    static constexpr int kTile = kBM * D * 2;
    static constexpr int kBlocks = D / 64;
    static constexpr int kKStages = D == 64 ? 5 : 3;  // key ring
    static constexpr int kVStages = D == 64 ? 4 : 2;  // value ring
    static constexpr int kOffQ = 0;
    static constexpr int kOffK = kOffQ + kSlots * kTile;
    static constexpr int kOffV = kOffK + kKStages * kTile;
    static constexpr int kOffBar = kOffV + kVStages * kTile;
    // barriers
    static constexpr int kQFull = 0, kQEmpty = kQFull + kSlots, kKFull = kQEmpty + kSlots,
                         kKEmpty = kKFull + kKStages, kVFull = kKEmpty + kKStages,
                         kVEmpty = kVFull + kVStages,
                         kSFull = kVEmpty + kVStages,  // [slot]: S_x = Q_x K^T is in TMEM
                         kPFull = kSFull + kSlots,  // [slot]: P_x is in TMEM (the slot's 128 threads)
                         kODone = kPFull + kSlots,  // [slot]: O_x += P_x V is done
                         kDrain = kODone + kSlots, kNumBars = kDrain + 1;
    static constexpr int kOffMisc = kOffBar + kNumBars * 8;  // tmem address, abort flag, tile count
    static constexpr size_t kSmemBytes = (size_t)kOffMisc + 16 + 1024;  // + alignment of the base
    static_assert(kSmemBytes <= 227 * 1024, "shared memory of one CTA");
    static_assert(D == 64 || D == 128, "head dimension");
};

struct Req {         // one request's geometry, from the argument arrays
    int64_t q0;      // first query row
    int64_t kv0;     // cache_off[b]
    int64_t cap;     // capacity (rows)
    int32_t P, T, N, n, S, tiles;
};


// Request b's table entry, read from the argument arrays (cached in L1);
// tiles = 0 marks a request that is skipped.  *bad: 1 inconsistent, 2 the
// compressed rows exceed the capacity.  A paged cache (kPaged; no cache_off)
// gives every request capP rows.
template <bool kPaged>
struct ReqSrc {
    const int64_t *q_off, *cache_off;
    const int32_t *P, *T, *N;
    int64_t q_rows, cache_rows;
    int w;
    int64_t capP;
    __device__ __forceinline__ Req operator()(int b, int *bad = nullptr) const {
        Req q;
        q.q0 = q_off[b];
        const int64_t q1 = q_off[b + 1];
        q.kv0 = kPaged ? 0 : cache_off[b];
        const int64_t kv1 = kPaged ? capP : cache_off[b + 1];
        q.cap = kv1 - q.kv0;
        q.P = P[b];
        q.T = T[b];
        q.N = N[b];
        q.n = q.T >= 0 ? (int32_t)(((int64_t)q.T + w - 1) / w) : 0;
        const int64_t S = (int64_t)q.P + q.T + q.N;
        const int64_t c = (int64_t)q.P + q.n + q.N;
        q.S = (int32_t)S;
        const bool ok = q.P >= 0 && q.T >= 0 && q.N >= 0 && q.q0 >= 0 && q1 - q.q0 == S &&
                        q1 <= q_rows && q.kv0 >= 0 && (kPaged || kv1 <= cache_rows) &&
                        S < (1ll << 31);
        const int why = !ok ? 1 : (c > q.cap ? 2 : 0);
        if (bad) *bad = why;
        q.tiles = why == 0 ? (int32_t)((S + kBM - 1) / kBM) : 0;
        return q;
    }
};

__device__ __forceinline__ int64_t pi_of(const Req &q, int64_t t, int w) {
    if (t < q.P) return t;
    if (t < (int64_t)q.P + q.T) return q.P + (t - q.P) / w;
    return t - q.T + q.n;
}

// packed fp32 pair addition (sm_100+ f32x2) and a three-input maximum
__device__ __forceinline__ float2 fadd2(float2 a, float2 b) {
    float2 d;
    asm("{\n\t.reg .b64 ra, rb, rd;\n\t"
        "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
        "add.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd;\n\t}"
        : "=f"(d.x), "=f"(d.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return d;
}

// Largest of three floats in one instruction (sm_100+).
__device__ __forceinline__ float fmax3(float a, float b, float c) {
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}

// ---------------------------------------------------------------- tcgen05 --
// Shared-memory matrix descriptor, 128-byte swizzle: start address, leading
// and stride byte offsets (16-byte units), descriptor version 1.
__device__ __forceinline__ uint64_t smem_desc(uint32_t addr, uint32_t lbo, uint32_t sbo) {
    return (uint64_t)((addr & 0x3FFFFu) >> 4) | ((uint64_t)((lbo >> 4) & 0x3FFFu) << 16) |
           ((uint64_t)((sbo >> 4) & 0x3FFFu) << 32) | (1ull << 46) | (2ull << 61);
}
// Instruction descriptor, kind::f16: fp32 accumulator, bf16 A and B, A
// K-major, B K-major or MN-major, M = 128, N = n.
__device__ __forceinline__ uint32_t instr_desc(bool b_mn_major, int n) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((b_mn_major ? 1u : 0u) << 16) |
           ((uint32_t)(n >> 3) << 17) | ((uint32_t)(kBM >> 4) << 24);
}
// tcgen05.mma (A and B in shared memory), issued by one elected lane of a
// converged warp: the whole warp runs the issue loop, so the descriptors and
// counters are warp-uniform values.
__device__ __forceinline__ void umma(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t id,
                                     uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p, e;\n\telect.sync _|e, 0xffffffff;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "@e tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(id), "r"(accumulate));
}
// The same with the A operand in TMEM: row m in lane m, two bf16 per 32-bit
// column (the even element in the low half), 8 columns per 16-element K step.
__device__ __forceinline__ void umma_tmem_a(uint32_t d_tmem, uint32_t a_tmem, uint64_t b,
                                            uint32_t id, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p, e;\n\telect.sync _|e, 0xffffffff;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "@e tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
        "r"(a_tmem), "l"(b), "r"(id), "r"(accumulate));
}
// Arrive on `bar` (one elected lane) once every tcgen05 operation issued so
// far by this warp has completed.
__device__ __forceinline__ void umma_commit(uint64_t *bar) {
    asm volatile(
        "{\n\t.reg .pred e;\n\telect.sync _|e, 0xffffffff;\n\t"
        "@e tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n\t}" ::"r"(
            smem_addr(bar))
        : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// All 128 fp32 columns of this thread's TMEM lane in one load.
__device__ __forceinline__ void tmem_ld128(uint32_t taddr, uint32_t (&r)[128]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x128.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32,%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,%45,%46,%47,%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63,%64,%65,%66,%67,%68,%69,%70,%71,%72,%73,%74,%75,%76,%77,%78,%79,%80,%81,%82,%83,%84,%85,%86,%87,%88,%89,%90,%91,%92,%93,%94,%95,%96,%97,%98,%99,%100,%101,%102,%103,%104,%105,%106,%107,%108,%109,%110,%111,%112,%113,%114,%115,%116,%117,%118,%119,%120,%121,%122,%123,%124,%125,%126,%127}, [%128];"
        : "=r"(r[0]),"=r"(r[1]),"=r"(r[2]),"=r"(r[3]),"=r"(r[4]),"=r"(r[5]),"=r"(r[6]),"=r"(r[7]),"=r"(r[8]),"=r"(r[9]),"=r"(r[10]),"=r"(r[11]),"=r"(r[12]),"=r"(r[13]),"=r"(r[14]),"=r"(r[15]),"=r"(r[16]),"=r"(r[17]),"=r"(r[18]),"=r"(r[19]),"=r"(r[20]),"=r"(r[21]),"=r"(r[22]),"=r"(r[23]),"=r"(r[24]),"=r"(r[25]),"=r"(r[26]),"=r"(r[27]),"=r"(r[28]),"=r"(r[29]),"=r"(r[30]),"=r"(r[31]),"=r"(r[32]),"=r"(r[33]),"=r"(r[34]),"=r"(r[35]),"=r"(r[36]),"=r"(r[37]),"=r"(r[38]),"=r"(r[39]),"=r"(r[40]),"=r"(r[41]),"=r"(r[42]),"=r"(r[43]),"=r"(r[44]),"=r"(r[45]),"=r"(r[46]),"=r"(r[47]),"=r"(r[48]),"=r"(r[49]),"=r"(r[50]),"=r"(r[51]),"=r"(r[52]),"=r"(r[53]),"=r"(r[54]),"=r"(r[55]),"=r"(r[56]),"=r"(r[57]),"=r"(r[58]),"=r"(r[59]),"=r"(r[60]),"=r"(r[61]),"=r"(r[62]),"=r"(r[63]),"=r"(r[64]),"=r"(r[65]),"=r"(r[66]),"=r"(r[67]),"=r"(r[68]),"=r"(r[69]),"=r"(r[70]),"=r"(r[71]),"=r"(r[72]),"=r"(r[73]),"=r"(r[74]),"=r"(r[75]),"=r"(r[76]),"=r"(r[77]),"=r"(r[78]),"=r"(r[79]),"=r"(r[80]),"=r"(r[81]),"=r"(r[82]),"=r"(r[83]),"=r"(r[84]),"=r"(r[85]),"=r"(r[86]),"=r"(r[87]),"=r"(r[88]),"=r"(r[89]),"=r"(r[90]),"=r"(r[91]),"=r"(r[92]),"=r"(r[93]),"=r"(r[94]),"=r"(r[95]),"=r"(r[96]),"=r"(r[97]),"=r"(r[98]),"=r"(r[99]),"=r"(r[100]),"=r"(r[101]),"=r"(r[102]),"=r"(r[103]),"=r"(r[104]),"=r"(r[105]),"=r"(r[106]),"=r"(r[107]),"=r"(r[108]),"=r"(r[109]),"=r"(r[110]),"=r"(r[111]),"=r"(r[112]),"=r"(r[113]),"=r"(r[114]),"=r"(r[115]),"=r"(r[116]),"=r"(r[117]),"=r"(r[118]),"=r"(r[119]),"=r"(r[120]),"=r"(r[121]),"=r"(r[122]),"=r"(r[123]),"=r"(r[124]),"=r"(r[125]),"=r"(r[126]),"=r"(r[127])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_st128(uint32_t taddr, const uint32_t (&r)[128]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x128.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32,%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,%45,%46,%47,%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63,%64,%65,%66,%67,%68,%69,%70,%71,%72,%73,%74,%75,%76,%77,%78,%79,%80,%81,%82,%83,%84,%85,%86,%87,%88,%89,%90,%91,%92,%93,%94,%95,%96,%97,%98,%99,%100,%101,%102,%103,%104,%105,%106,%107,%108,%109,%110,%111,%112,%113,%114,%115,%116,%117,%118,%119,%120,%121,%122,%123,%124,%125,%126,%127,%128};"
        :: "r"(taddr), "r"(r[0]),"r"(r[1]),"r"(r[2]),"r"(r[3]),"r"(r[4]),"r"(r[5]),"r"(r[6]),"r"(r[7]),"r"(r[8]),"r"(r[9]),"r"(r[10]),"r"(r[11]),"r"(r[12]),"r"(r[13]),"r"(r[14]),"r"(r[15]),"r"(r[16]),"r"(r[17]),"r"(r[18]),"r"(r[19]),"r"(r[20]),"r"(r[21]),"r"(r[22]),"r"(r[23]),"r"(r[24]),"r"(r[25]),"r"(r[26]),"r"(r[27]),"r"(r[28]),"r"(r[29]),"r"(r[30]),"r"(r[31]),"r"(r[32]),"r"(r[33]),"r"(r[34]),"r"(r[35]),"r"(r[36]),"r"(r[37]),"r"(r[38]),"r"(r[39]),"r"(r[40]),"r"(r[41]),"r"(r[42]),"r"(r[43]),"r"(r[44]),"r"(r[45]),"r"(r[46]),"r"(r[47]),"r"(r[48]),"r"(r[49]),"r"(r[50]),"r"(r[51]),"r"(r[52]),"r"(r[53]),"r"(r[54]),"r"(r[55]),"r"(r[56]),"r"(r[57]),"r"(r[58]),"r"(r[59]),"r"(r[60]),"r"(r[61]),"r"(r[62]),"r"(r[63]),"r"(r[64]),"r"(r[65]),"r"(r[66]),"r"(r[67]),"r"(r[68]),"r"(r[69]),"r"(r[70]),"r"(r[71]),"r"(r[72]),"r"(r[73]),"r"(r[74]),"r"(r[75]),"r"(r[76]),"r"(r[77]),"r"(r[78]),"r"(r[79]),"r"(r[80]),"r"(r[81]),"r"(r[82]),"r"(r[83]),"r"(r[84]),"r"(r[85]),"r"(r[86]),"r"(r[87]),"r"(r[88]),"r"(r[89]),"r"(r[90]),"r"(r[91]),"r"(r[92]),"r"(r[93]),"r"(r[94]),"r"(r[95]),"r"(r[96]),"r"(r[97]),"r"(r[98]),"r"(r[99]),"r"(r[100]),"r"(r[101]),"r"(r[102]),"r"(r[103]),"r"(r[104]),"r"(r[105]),"r"(r[106]),"r"(r[107]),"r"(r[108]),"r"(r[109]),"r"(r[110]),"r"(r[111]),"r"(r[112]),"r"(r[113]),"r"(r[114]),"r"(r[115]),"r"(r[116]),"r"(r[117]),"r"(r[118]),"r"(r[119]),"r"(r[120]),"r"(r[121]),"r"(r[122]),"r"(r[123]),"r"(r[124]),"r"(r[125]),"r"(r[126]),"r"(r[127])
        : "memory");
}
// 64 32-bit columns of this thread's TMEM lane (then waits for the store).
__device__ __forceinline__ void tmem_st64(uint32_t taddr, const uint32_t (&r)[64]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x64.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32,%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,%45,%46,%47,%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63,%64};"
        :: "r"(taddr), "r"(r[0]),"r"(r[1]),"r"(r[2]),"r"(r[3]),"r"(r[4]),"r"(r[5]),"r"(r[6]),"r"(r[7]),"r"(r[8]),"r"(r[9]),"r"(r[10]),"r"(r[11]),"r"(r[12]),"r"(r[13]),"r"(r[14]),"r"(r[15]),"r"(r[16]),"r"(r[17]),"r"(r[18]),"r"(r[19]),"r"(r[20]),"r"(r[21]),"r"(r[22]),"r"(r[23]),"r"(r[24]),"r"(r[25]),"r"(r[26]),"r"(r[27]),"r"(r[28]),"r"(r[29]),"r"(r[30]),"r"(r[31]),"r"(r[32]),"r"(r[33]),"r"(r[34]),"r"(r[35]),"r"(r[36]),"r"(r[37]),"r"(r[38]),"r"(r[39]),"r"(r[40]),"r"(r[41]),"r"(r[42]),"r"(r[43]),"r"(r[44]),"r"(r[45]),"r"(r[46]),"r"(r[47]),"r"(r[48]),"r"(r[49]),"r"(r[50]),"r"(r[51]),"r"(r[52]),"r"(r[53]),"r"(r[54]),"r"(r[55]),"r"(r[56]),"r"(r[57]),"r"(r[58]),"r"(r[59]),"r"(r[60]),"r"(r[61]),"r"(r[62]),"r"(r[63])
        : "memory");
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// 64 fp32 columns of this thread's TMEM lane in one load.
__device__ __forceinline__ void tmem_ld64(uint32_t taddr, uint32_t (&r)[64]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x64.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32,%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,%45,%46,%47,%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63}, [%64];"
        : "=r"(r[0]),"=r"(r[1]),"=r"(r[2]),"=r"(r[3]),"=r"(r[4]),"=r"(r[5]),"=r"(r[6]),"=r"(r[7]),"=r"(r[8]),"=r"(r[9]),"=r"(r[10]),"=r"(r[11]),"=r"(r[12]),"=r"(r[13]),"=r"(r[14]),"=r"(r[15]),"=r"(r[16]),"=r"(r[17]),"=r"(r[18]),"=r"(r[19]),"=r"(r[20]),"=r"(r[21]),"=r"(r[22]),"=r"(r[23]),"=r"(r[24]),"=r"(r[25]),"=r"(r[26]),"=r"(r[27]),"=r"(r[28]),"=r"(r[29]),"=r"(r[30]),"=r"(r[31]),"=r"(r[32]),"=r"(r[33]),"=r"(r[34]),"=r"(r[35]),"=r"(r[36]),"=r"(r[37]),"=r"(r[38]),"=r"(r[39]),"=r"(r[40]),"=r"(r[41]),"=r"(r[42]),"=r"(r[43]),"=r"(r[44]),"=r"(r[45]),"=r"(r[46]),"=r"(r[47]),"=r"(r[48]),"=r"(r[49]),"=r"(r[50]),"=r"(r[51]),"=r"(r[52]),"=r"(r[53]),"=r"(r[54]),"=r"(r[55]),"=r"(r[56]),"=r"(r[57]),"=r"(r[58]),"=r"(r[59]),"=r"(r[60]),"=r"(r[61]),"=r"(r[62]),"=r"(r[63])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}
// D fp32 columns (64 or 128) of this thread's TMEM lane: load, store.
template <int N>
__device__ __forceinline__ void tmem_ld_cols(uint32_t taddr, uint32_t (&r)[N]) {
    if constexpr (N == 128) tmem_ld128(taddr, r); else tmem_ld64(taddr, r);
}
template <int N>
__device__ __forceinline__ void tmem_st_cols(uint32_t taddr, const uint32_t (&r)[N]) {
    if constexpr (N == 128) {
        tmem_st128(taddr, r);
        asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
    } else {
        tmem_st64(taddr, r);  // (waits for the store)
    }
}

// TMA tensor copies global -> shared (completion as transaction bytes on bar)
__device__ __forceinline__ void tma_2d(void *dst, const CUtensorMap *map, int x, int y,
                                       uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, "
        "{%3, %4}], [%2];" ::"r"(smem_addr(dst)),
        "l"(reinterpret_cast<unsigned long long>(map)), "r"(smem_addr(bar)), "r"(x), "r"(y)
        : "memory");
}
__device__ __forceinline__ void tma_3d(void *dst, const CUtensorMap *map, int x, int y, int z,
                                       uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, "
        "{%3, %4, %5}], [%2];" ::"r"(smem_addr(dst)),
        "l"(reinterpret_cast<unsigned long long>(map)), "r"(smem_addr(bar)), "r"(x), "r"(y),
        "r"(z)
        : "memory");
}

// Bounded wait that also gives up once another role has aborted.
__device__ __forceinline__ bool wait_bar(uint64_t *bar, uint32_t parity, volatile int *abort,
                                         int *err) {
    if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long t0 = global_timer_ns();
    for (;;) {
        for (int i = 0; i < 64; i++)
            if (mbar_try_wait(bar, parity)) return true;
        if (*abort) return false;
        if (global_timer_ns() - t0 > kWaitLimitNs) {
            report_error(err, SPEECHKV_ERR_TIMEOUT);
            *abort = 1;
            return false;
        }
    }
}

// Work item k of the CTA-independent order: (request, KV head) outermost,
// then query tiles from the last down, then groups of up to kSlots query
// heads of the KV head's group (they share every key and value tile).  CTAs
// working at the same time share one (request, KV head)'s keys and values.
struct Item {
    int b, hq0, n, i;  // request, first query head, heads (slots used), query tile
    bool valid;
};
template <bool kPaged>
__device__ __forceinline__ Item item_at(int64_t k, int tiles_max, int H_q, int H_kv,
                                        const ReqSrc<kPaged> &tab, Req &q) {
    Item it;
    const int G = H_q / H_kv;
    const int ng = (G + kSlots - 1) / kSlots;    // head groups of a KV head
    const int64_t per = (int64_t)tiles_max * ng;  // items of one (request, KV head)
    const int bh = (int)(k / per);
    const int rem = (int)(k - (int64_t)bh * per);
    it.b = bh / H_kv;
    const int grp = rem % ng;
    it.hq0 = (bh - it.b * H_kv) * G + grp * kSlots;
    it.n = min(kSlots, G - grp * kSlots);
    it.i = tiles_max - 1 - rem / ng;
    q = tab(it.b);
    it.valid = it.i < q.tiles;
    return it;
}

// kPaged: the cache is paged through map's block table (its own instance, so
// that the contiguous kernel carries none of that code).
template <int D, bool kPaged>
__global__ void __launch_bounds__(kThreads, 1)
    prefill_attn_kernel(const __grid_constant__ CUtensorMap tm_q,
                        const __grid_constant__ CUtensorMap tm_k,
                        const __grid_constant__ CUtensorMap tm_v,
                        const int64_t *__restrict__ q_off, const int32_t *__restrict__ Pa,
                        const int32_t *__restrict__ Ta, const int32_t *__restrict__ Na,
                        const int64_t *__restrict__ cache_off, __nv_bfloat16 *__restrict__ out,
                        int64_t q_rows, int64_t cache_rows, float sl2, int B, int H_q,
                        int H_kv, int w, int *__restrict__ err, CacheMap map) {
    using C = PfCfg<D>;
    extern __shared__ unsigned char smem_raw[];
    unsigned char *sm = reinterpret_cast<unsigned char *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint64_t *bar = reinterpret_cast<uint64_t *>(sm + C::kOffBar);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(sm + C::kOffMisc);
    volatile int *abort = reinterpret_cast<volatile int *>(sm + C::kOffMisc + 4);
    int *tiles_max_s = reinterpret_cast<int *>(sm + C::kOffMisc + 8);
    const ReqSrc<kPaged> tab{q_off,      cache_off, Pa, Ta, Na, q_rows,
                             cache_rows, w,         (int64_t)map.max_blocks << map.bs_log2};
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int G = H_q / H_kv;

    // ---- prologue: barriers, TMEM, largest tile count
    if (tid == 0) {
        for (int x = 0; x < kSlots; x++) {
            mbar_init(&bar[C::kQFull + x], 1);
            mbar_init(&bar[C::kQEmpty + x], 1);
            mbar_init(&bar[C::kSFull + x], 1);
            mbar_init(&bar[C::kPFull + x], kBM);
            mbar_init(&bar[C::kODone + x], 1);
        }
        for (int s = 0; s < C::kKStages; s++) {
            mbar_init(&bar[C::kKFull + s], 1);
            mbar_init(&bar[C::kKEmpty + s], 1);
        }
        for (int s = 0; s < C::kVStages; s++) {
            mbar_init(&bar[C::kVFull + s], 1);
            mbar_init(&bar[C::kVEmpty + s], 1);
        }
        mbar_init(&bar[C::kDrain], 1);
        fence_mbar_init();
        *abort = 0;
    }
    if (warp == 1) {
        asm volatile(
            "tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                smem_addr(tmem_slot)),
            "r"(kTmemCols)
            : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    if (warp == 0) {
        // largest tile count over the batch; CTA 0 reports the skipped requests
        int mx = 0;
        for (int b = lane; b < B; b += 32) {
            int bad = 0;
            mx = max(mx, tab(b, &bad).tiles);
            if (bad && blockIdx.x == 0)
                report_error(err, bad == 1 ? SPEECHKV_ERR_INVALID_ARG : SPEECHKV_ERR_CAPACITY);
        }
        for (int o = 16; o > 0; o >>= 1) mx = max(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        if (lane == 0) *tiles_max_s = mx;
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    const int tiles_max = *tiles_max_s;
    const int ng = (G + kSlots - 1) / kSlots;
    const int64_t total = (int64_t)tiles_max * B * H_kv * ng;
    unsigned char *sQ = sm + C::kOffQ, *sK = sm + C::kOffK, *sV = sm + C::kOffV;

    if (warp == 0) {
        // ===================== TMA producer =====================
        // One stream of copies over the CTA's items: the query tiles of an
        // item (one buffer per slot), then its key and value tiles with the
        // keys one tile ahead of the values (a value tile waits for an older
        // P V than the key tile issued before it).
        if constexpr (!kPaged) {
            if (lane == 0) {
                int64_t uq[kSlots] = {}, gk = 0, gv = 0;  // query (per slot), key, value tiles issued
                int pend_y = -1;                          // cache row of the value tile still to issue
                bool stop = false;
                auto issue_v = [&](int y) -> bool {
                    const int s = (int)(gv % C::kVStages);
                    const int64_t u = gv / C::kVStages;
                    if (gv >= C::kVStages && !wait_bar(&bar[C::kVEmpty + s], (uint32_t)((u - 1) & 1), abort, err))
                        return false;
                    mbar_arrive_expect_tx(&bar[C::kVFull + s], C::kTile);
#pragma unroll
                    for (int blk = 0; blk < C::kBlocks; blk++)
                        tma_2d(sV + s * C::kTile + blk * kBlockBytes, &tm_v, 64 * blk, y,
                               &bar[C::kVFull + s]);
                    ++gv;
                    return true;
                };
                for (int64_t k = blockIdx.x; k < total && !stop && !*abort; k += gridDim.x) {
                    Req q;
                    const Item item = item_at(k, tiles_max, H_q, H_kv, tab, q);
                    if (!item.valid) continue;
                    const int64_t t0 = (int64_t)item.i * kBM;
                    const int64_t tl = min(t0 + kBM, (int64_t)q.S) - 1;
                    const int n_kt = (int)(pi_of(q, tl, w) / kBN) + 1;
                    const int64_t kvrow = q.kv0 * H_kv + (int64_t)(item.hq0 / G) * q.cap;
                    for (int x = 0; x < item.n && !stop; x++) {
                        // slot x's query buffer is free once its last Q K^T is done
                        if (uq[x] > 0 &&
                            !wait_bar(&bar[C::kQEmpty + x], (uint32_t)((uq[x] - 1) & 1), abort, err)) {
                            stop = true;
                            break;
                        }
                        unsigned char *sQx = sQ + x * C::kTile;
                        mbar_arrive_expect_tx(&bar[C::kQFull + x], C::kTile);
#pragma unroll
                        for (int blk = 0; blk < C::kBlocks; blk++)
                            tma_3d(sQx + blk * kBlockBytes, &tm_q, 64 * blk, item.hq0 + x,
                                   (int)(q.q0 + t0), &bar[C::kQFull + x]);
                        ++uq[x];
                    }
                    for (int j = 0; j < n_kt && !stop; j++) {
                        // keys are free once their Q K^T is done, values once their P V is
                        const int y = (int)(kvrow + (int64_t)j * kBN);
                        const int s = (int)(gk % C::kKStages);
                        const int64_t u = gk / C::kKStages;
                        if (gk >= C::kKStages &&
                            !wait_bar(&bar[C::kKEmpty + s], (uint32_t)((u - 1) & 1), abort, err)) {
                            stop = true;
                            break;
                        }
                        mbar_arrive_expect_tx(&bar[C::kKFull + s], C::kTile);
#pragma unroll
                        for (int blk = 0; blk < C::kBlocks; blk++)
                            tma_2d(sK + s * C::kTile + blk * kBlockBytes, &tm_k, 64 * blk, y,
                                   &bar[C::kKFull + s]);
                        ++gk;
                        if (pend_y >= 0 && !issue_v(pend_y)) {
                            stop = true;
                            break;
                        }
                        pend_y = y;
                    }
                    // the item's last value tile now, not behind the next item's
                    // query-buffer wait (its P V would stall on the load)
                    if (!stop && pend_y >= 0) stop = !issue_v(pend_y);
                    pend_y = -1;
                }
                // let every copy issued land before the CTA may exit
                for (int x = 0; x < kSlots; x++)
                    if (uq[x] > 0)
                        mbar_wait_bounded(&bar[C::kQFull + x], (uint32_t)((uq[x] - 1) & 1), err);
                for (int64_t x = gk - C::kKStages; x < gk; x++)
                    if (x >= 0)
                        mbar_wait_bounded(&bar[C::kKFull + (int)(x % C::kKStages)], (uint32_t)((x / C::kKStages) & 1),
                                          err);
                for (int64_t x = gv - C::kVStages; x < gv; x++)
                    if (x >= 0)
                        mbar_wait_bounded(&bar[C::kVFull + (int)(x % C::kVStages)], (uint32_t)((x / C::kVStages) & 1),
                                          err);
            }
        } else {
            // Paged: every lane walks the same items and tiles; lane 0 waits
            // for the stages, sets the expected bytes and copies the queries,
            // and lane p copies page p of a key or value tile (pages of 8
            // rows or more: at most 16 per 128-row tile), so that the small
            // copies are issued in parallel.  Each lane reads its block-table
            // entry one key tile ahead of the copies that need it (a cold
            // entry read in front of every tile's copies set the producer's
            // pace).  Pages past the compressed rows are not read (their rows
            // are masked, and the values zeroed, by the softmax warps).
            int64_t uq[kSlots] = {}, gk = 0, gv = 0;  // query (per slot), key, value tiles issued
            bool stop = false;
            const int lg = map.bs_log2;
            const int lgr = lg < 7 ? lg : 7;  // rows per copy (the maps' box): 1 << lgr
            const int rows = 1 << lgr;
            auto wait0 = [&](uint64_t *b, uint32_t parity) -> bool {  // lane 0 waits for all
                int ok = 1;
                if (lane == 0) ok = wait_bar(b, parity, abort, err);
                return __shfl_sync(0xffffffffu, ok, 0) != 0;
            };
            for (int64_t k = blockIdx.x; k < total && !stop; k += gridDim.x) {
                if (__shfl_sync(0xffffffffu, lane == 0 ? (int)*abort : 0, 0)) break;
                Req q;
                const Item item = item_at(k, tiles_max, H_q, H_kv, tab, q);
                if (!item.valid) continue;
                const int64_t t0 = (int64_t)item.i * kBM;
                const int64_t tl = min(t0 + kBM, (int64_t)q.S) - 1;
                const int n_kt = (int)(pi_of(q, tl, w) / kBN) + 1;
                const int hk = item.hq0 / G;                      // the KV head
                const int64_t crows = (int64_t)q.P + q.n + q.N;  // compressed rows
                const int32_t *row_table = map.table + (int64_t)item.b * map.max_blocks;
                // Lane p's page of key tile kt (its copies are issued only
                // where ncopy(kt) > p); read one tile ahead of its copies.
                auto entry = [&](int kt) -> int32_t {
                    const int64_t r = (int64_t)kt * kBN + ((int64_t)lane << lgr);
                    return kt < n_kt && r < crows ? __ldg(row_table + (r >> lg)) : 0;
                };
                auto ncopy_of = [&](int kt) -> int {  // segments of tile kt that hold rows
                    const int64_t left = crows - (int64_t)kt * kBN;
                    if (left <= 0) return 0;
                    const int64_t c = (left + rows - 1) >> lgr;
                    return c < kBN / rows ? (int)c : kBN / rows;
                };
                auto copy_tile = [&](unsigned char *dst, const CUtensorMap *tm, int kt, int32_t blk_id,
                                     uint64_t *fb) {
                    const int ncopy = ncopy_of(kt);
                    if (lane == 0) mbar_arrive_expect_tx(fb, (uint32_t)(ncopy * rows * 128 * C::kBlocks));
                    __syncwarp();
                    if (lane < ncopy) {
                        const int64_t r = (int64_t)kt * kBN + ((int64_t)lane << lgr);
                        if (blk_id < 0 || blk_id >= map.num_blocks) {
                            report_error(err, SPEECHKV_ERR_INVALID_ARG);  // read page 0 instead
                            blk_id = 0;
                        }
                        const int y = (int)((((int64_t)blk_id * H_kv + hk) << lg) +
                                            (r & ((1ll << lg) - 1)));
#pragma unroll
                        for (int blk = 0; blk < C::kBlocks; blk++)
                            tma_2d(dst + blk * kBlockBytes + lane * rows * 128, tm, 64 * blk, y,
                                   fb);
                    }
                };
                auto issue_v = [&](int kt, int32_t blk_id) -> bool {
                    const int s = (int)(gv % C::kVStages);
                    const int64_t u = gv / C::kVStages;
                    if (gv >= C::kVStages && !wait0(&bar[C::kVEmpty + s], (uint32_t)((u - 1) & 1)))
                        return false;
                    copy_tile(sV + s * C::kTile, &tm_v, kt, blk_id, &bar[C::kVFull + s]);
                    ++gv;
                    return true;
                };
                for (int x = 0; x < item.n && !stop; x++) {
                    // slot x's query buffer is free once its last Q K^T is done
                    if (uq[x] > 0 && !wait0(&bar[C::kQEmpty + x], (uint32_t)((uq[x] - 1) & 1))) {
                        stop = true;
                        break;
                    }
                    if (lane == 0) {
                        unsigned char *sQx = sQ + x * C::kTile;
                        mbar_arrive_expect_tx(&bar[C::kQFull + x], C::kTile);
#pragma unroll
                        for (int blk = 0; blk < C::kBlocks; blk++)
                            tma_3d(sQx + blk * kBlockBytes, &tm_q, 64 * blk, item.hq0 + x,
                                   (int)(q.q0 + t0), &bar[C::kQFull + x]);
                    }
                    ++uq[x];
                }
                int32_t e_cur = entry(0), e_prev = 0;  // this lane's page of tiles j and j - 1
                for (int j = 0; j < n_kt && !stop; j++) {
                    const int32_t e_next = entry(j + 1);  // in flight during this tile's waits
                    // keys are free once their Q K^T is done, values once their P V is
                    const int s = (int)(gk % C::kKStages);
                    const int64_t u = gk / C::kKStages;
                    if (gk >= C::kKStages && !wait0(&bar[C::kKEmpty + s], (uint32_t)((u - 1) & 1))) {
                        stop = true;
                        break;
                    }
                    copy_tile(sK + s * C::kTile, &tm_k, j, e_cur, &bar[C::kKFull + s]);
                    ++gk;
                    if (j > 0 && !issue_v(j - 1, e_prev)) {
                        stop = true;
                        break;
                    }
                    e_prev = e_cur;
                    e_cur = e_next;
                }
                // the item's last value tile now, not behind the next item's
                // query-buffer wait (its P V would stall on the load)
                if (!stop) stop = !issue_v(n_kt - 1, e_prev);
            }
            // let every copy issued land before the CTA may exit
            if (lane == 0) {
                for (int x = 0; x < kSlots; x++)
                    if (uq[x] > 0)
                        mbar_wait_bounded(&bar[C::kQFull + x], (uint32_t)((uq[x] - 1) & 1), err);
                for (int64_t x = gk - C::kKStages; x < gk; x++)
                    if (x >= 0)
                        mbar_wait_bounded(&bar[C::kKFull + (int)(x % C::kKStages)],
                                          (uint32_t)((x / C::kKStages) & 1), err);
                for (int64_t x = gv - C::kVStages; x < gv; x++)
                    if (x >= 0)
                        mbar_wait_bounded(&bar[C::kVFull + (int)(x % C::kVStages)],
                                          (uint32_t)((x / C::kVStages) & 1), err);
            }
        }
    } else if (warp == 1) {
        // ===================== MMA issue =====================
        // Per key/value tile j of an item, for each slot x in turn:
        //   O_x += P_x V (j), then S_x = Q_x K^T (j + 1).
        // P_x lives in the first half of S_x's columns, so slot x's next
        // Q K^T waits for its P V to complete; the other slot's products keep
        // the tensor pipe busy meanwhile, and each slot's softmax overlaps
        // the other slot's products.  The whole warp runs this loop (its
        // waits agree through a vote) and one elected lane issues.
        {
            auto wb = [&](uint64_t *bb, uint32_t par) -> bool {
                return __all_sync(0xffffffffu, wait_bar(bb, par, abort, err));
            };
            const uint32_t id_qk = instr_desc(false, kBN), id_pv = instr_desc(true, D);
            const uint32_t aQ = smem_addr(sQ), aK = smem_addr(sK), aV = smem_addr(sV);
            // Descriptors are built once per buffer; a K step or a stage only
            // moves the start address, whose field (address / 16, 14 bits)
            // cannot carry over inside shared memory.
            const uint64_t dQ = smem_desc(aQ, 16, 1024);
            const uint64_t dK = smem_desc(aK, 16, 1024), dV = smem_desc(aV, kBlockBytes, 1024);
            constexpr uint64_t kStageD = C::kTile >> 4;
            int64_t g = 0;                       // key/value tiles
            int64_t ut[kSlots] = {}, uq[kSlots] = {};  // per slot: tiles (P V issued), items
            bool issued = false, stop = false;
            auto qk = [&](int x, int64_t gg) -> bool {  // S_x = Q_x K^T of key tile gg
                const int s = (int)(gg % C::kKStages);
                if (x == 0 && !wb(&bar[C::kKFull + s], (uint32_t)((gg / C::kKStages) & 1)))
                    return false;
                // P V of slot x's previous tile has read P_x (inside S_x)
                if (ut[x] > 0 && !wb(&bar[C::kODone + x], (uint32_t)((ut[x] - 1) & 1)))
                    return false;
                tc_fence_after();
                const uint64_t dQx = dQ + (uint64_t)x * kStageD, dKs = dK + (uint64_t)s * kStageD;
#pragma unroll
                for (int kk = 0; kk < D / 16; kk++) {
                    const uint64_t ko = (uint64_t)(((kk >> 2) * kBlockBytes + (kk & 3) * 32) >> 4);
                    umma(tmem + x * kBN, dQx + ko, dKs + ko, id_qk, kk > 0 ? 1u : 0u);
                }
                umma_commit(&bar[C::kSFull + x]);
                issued = true;
                return true;
            };
            for (int64_t k = blockIdx.x;
                 k < total && !stop && !__shfl_sync(0xffffffffu, (int)*abort, 0); k += gridDim.x) {
                Req q;
                const Item item = item_at(k, tiles_max, H_q, H_kv, tab, q);
                if (!item.valid) continue;
                const int n = item.n;
                const int64_t t0 = (int64_t)item.i * kBM;
                const int64_t tl = min(t0 + kBM, (int64_t)q.S) - 1;
                const int n_kt = (int)(pi_of(q, tl, w) / kBN) + 1;
                for (int x = 0; x < n && !stop; x++)
                    stop = !wb(&bar[C::kQFull + x], (uint32_t)(uq[x] & 1));
                for (int x = 0; x < n && !stop; x++) stop = !qk(x, g);
                if (stop) break;
                umma_commit(&bar[C::kKEmpty + (int)(g % C::kKStages)]);
                if (n_kt == 1)
                    for (int x = 0; x < n; x++) umma_commit(&bar[C::kQEmpty + x]);
                for (int j = 0; j < n_kt && !stop; j++, g++) {
                    const int sv = (int)(g % C::kVStages);
                    for (int x = 0; x < n; x++) {
                        if (!wb(&bar[C::kPFull + x], (uint32_t)(ut[x] & 1)) ||
                            (x == 0 &&
                             !wb(&bar[C::kVFull + sv], (uint32_t)((g / C::kVStages) & 1)))) {
                            stop = true;
                            break;
                        }
                        tc_fence_after();
                        const uint64_t dVs = dV + (uint64_t)sv * kStageD;
#pragma unroll
                        for (int kk = 0; kk < kBN / 16; kk++) {
                            const uint64_t vo = (uint64_t)((kk * 16 * 128) >> 4);  // 16 keys further
                            umma_tmem_a(tmem + 2 * kBN + x * D, tmem + x * kBN + kk * 8, dVs + vo,
                                        id_pv, (j == 0 && kk == 0) ? 0u : 1u);
                        }
                        umma_commit(&bar[C::kODone + x]);
                        ++ut[x];
                        if (x == n - 1) umma_commit(&bar[C::kVEmpty + sv]);  // values of tile j are read
                        if (j + 1 < n_kt) {
                            if (!qk(x, g + 1)) {
                                stop = true;
                                break;
                            }
                            if (x == n - 1) {
                                umma_commit(&bar[C::kKEmpty + (int)((g + 1) % C::kKStages)]);
                                // the query tiles are free once the item's last Q K^T is done
                                if (j + 2 == n_kt)
                                    for (int y = 0; y < n; y++) umma_commit(&bar[C::kQEmpty + y]);
                            }
                        }
                    }
                }
                for (int x = 0; x < n; x++) ++uq[x];
            }
            if (issued) {  // every MMA issued has completed before TMEM is freed
                umma_commit(&bar[C::kDrain]);
                mbar_wait_bounded(&bar[C::kDrain], 0, err);
            }
        }
    } else {
        // ===================== softmax: a warpgroup per slot ==========
        const int x = (warp - 2) >> 2;        // slot
        const int quarter = warp & 3;         // TMEM lanes 32*quarter .. +31
        const int r = quarter * 32 + lane;    // the row of the tile
        const uint32_t lanes = (uint32_t)(quarter * 32) << 16;
        const uint32_t tS = tmem + lanes + x * kBN, tO = tmem + lanes + 2 * kBN + x * D;
        int64_t ut = 0, g = 0;  // this slot's tiles; key/value tiles of the CTA
        bool stop = false;
        for (int64_t k = blockIdx.x; k < total && !stop; k += gridDim.x) {
            Req q;
            const Item item = item_at(k, tiles_max, H_q, H_kv, tab, q);
            if (!item.valid) continue;
            const int64_t t0 = (int64_t)item.i * kBM;
            const int64_t tl = min(t0 + kBM, (int64_t)q.S) - 1;
            const int n_kt = (int)(pi_of(q, tl, w) / kBN) + 1;
            if (x >= item.n) {  // this slot idles for the item
                g += n_kt;
                continue;
            }
            const int n_full = (int)((pi_of(q, t0, w) + 1) / kBN);  // tiles no row masks
            const int64_t c = (int64_t)q.P + q.n + q.N;
            const int64_t t = t0 + r;
            const int64_t lim = pi_of(q, t < q.S ? t : (int64_t)q.S - 1, w);
            float m = -INFINITY, l = 0.f;
            for (int j = 0; j < n_kt; j++, g++, ut++) {
                if (!__all_sync(0xffffffffu, wait_bar(&bar[C::kSFull + x], (uint32_t)(ut & 1), abort, err))) {
                    stop = true;
                    break;
                }
                tc_fence_after();
                const bool masked = j >= n_full;
                const int64_t e0 = (int64_t)j * kBN;
                // keys e0 + i, i <= vis, are visible to this row
                int64_t vis64 = lim - e0;
                vis64 = vis64 > kBN - 1 ? kBN - 1 : (vis64 < -1 ? -1 : vis64);
                const int vis = masked ? (int)vis64 : kBN - 1;
                uint32_t v[128];
                tmem_ld128(tS, v);
                if (masked) {
                    // keys past this row's last visible one weigh 0 (scale > 0)
#pragma unroll
                    for (int i = 0; i < kBN; i++)
                        if (i > vis) v[i] = __float_as_uint(-INFINITY);
                }
                // row maximum: four chains of three-input maxima
                float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
                for (int i = 0; i < kBN; i += 2)
                    m4[(i >> 1) & 3] = fmax3(m4[(i >> 1) & 3], __uint_as_float(v[i]),
                                             __uint_as_float(v[i + 1]));
                float mx = fmax3(m4[0], m4[1], fmaxf(m4[2], m4[3]));
                mx *= sl2;
                // Lazy rescaling: the weights keep using the running maximum
                // unless the tile's exceeds it by more than 8 (weights then
                // stay below 2^8); O / l is the same either way.
                const bool bump = mx > m + 8.f;  // always on the first tile (m = -inf)
                const float mu = bump ? mx : m;
                const float corr = fast_exp2(m - mu);  // 1 without a bump, 0 on the first tile
                // exponent arguments and row sums on column pairs (f32x2)
                const float2 sc2 = make_float2(sl2, sl2), nm2 = make_float2(-mu, -mu);
                float2 sums[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
                uint32_t pk[64];
#pragma unroll
                for (int i = 0; i < kBN; i += 2) {
                    const float2 e = ffma2(make_float2(__uint_as_float(v[i]), __uint_as_float(v[i + 1])),
                                           sc2, nm2);
                    const float p0 = fast_exp2(e.x), p1 = fast_exp2(e.y);
                    sums[(i >> 1) & 1] = fadd2(sums[(i >> 1) & 1], make_float2(p0, p1));
                    pk[i / 2] = pack_bf16x2(p0, p1);
                }
                // P over the first half of S's columns (S is in registers; the
                // P V that read the previous P completed before this Q K^T)
                tmem_st64(tS, pk);
                if (j > 0 && __any_sync(0xffffffffu, bump)) {
                    // rescale O (the earlier tiles' sum: their P V completed
                    // before this tile's Q K^T was issued)
                    uint32_t o[D];
                    tmem_ld_cols<D>(tO, o);
#pragma unroll
                    for (int i = 0; i < D; i++)
                        o[i] = __float_as_uint(__uint_as_float(o[i]) * corr);
                    tmem_st_cols<D>(tO, o);
                }
                l = l * corr + ((sums[0].x + sums[1].x) + (sums[0].y + sums[1].y));
                m = mu;
                if (x == 0 && e0 + kBN > c) {
                    // value rows at or past the compressed length: zero them
                    // (slot 0's P V reads the stage first)
                    const int s = (int)(g % C::kVStages);
                    if (!__all_sync(0xffffffffu, wait_bar(&bar[C::kVFull + s],
                                                          (uint32_t)((g / C::kVStages) & 1), abort,
                                                          err))) {
                        stop = true;
                        break;
                    }
                    if (e0 + r >= c) {
                        unsigned char *row = sV + s * C::kTile + r * 128;
#pragma unroll
                        for (int blk = 0; blk < C::kBlocks; blk++)
#pragma unroll
                            for (int y = 0; y < 8; y++)
                                *reinterpret_cast<uint4 *>(row + blk * kBlockBytes + y * 16) =
                                    make_uint4(0, 0, 0, 0);
                    }
                    fence_proxy_async_shared();  // the MMA reads these rows
                }
                tc_fence_before();
                mbar_arrive(&bar[C::kPFull + x]);
            }
            if (stop) break;
            // epilogue: O / l once the last P V is done
            if (!__all_sync(0xffffffffu, wait_bar(&bar[C::kODone + x], (uint32_t)((ut - 1) & 1), abort,
                                                  err)))
                break;
            tc_fence_after();
            const float inv = 1.f / l;
            __nv_bfloat16 *dst = out + ((q.q0 + t) * H_q + item.hq0 + x) * D;
            uint32_t o[D];
            tmem_ld_cols<D>(tO, o);
            if (t < q.S) {
#pragma unroll
                for (int y = 0; y < D / 8; y++) {
                    uint32_t wv[4];
#pragma unroll
                    for (int z = 0; z < 4; z++) {
                        __nv_bfloat162 h = __floats2bfloat162_rn(__uint_as_float(o[8 * y + 2 * z]) * inv,
                                                                 __uint_as_float(o[8 * y + 2 * z + 1]) * inv);
                        wv[z] = *reinterpret_cast<uint32_t *>(&h);
                    }
                    *reinterpret_cast<uint4 *>(dst + y * 8) = make_uint4(wv[0], wv[1], wv[2], wv[3]);
                }
            }
            tc_fence_before();
        }
    }

    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                     "r"(kTmemCols)
                     : "memory");
    }
}

// ------------------------------------------------------------------- host --
typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                  const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                  const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static std::once_flag once;
    static EncodeTiledFn fn = nullptr;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    });
    return fn;
}

bool encode(CUtensorMap *m, const void *base, int rank, const cuuint64_t *dims,
            const cuuint64_t *strides, const cuuint32_t *box) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    const cuuint32_t es[3] = {1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, (cuuint32_t)rank, const_cast<void *>(base), dims,
              strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

namespace {

template <int D>
cudaError_t launch_prefill_d(const PrefillArgs &a, int num_sms, cudaStream_t stream) {
    using C = PfCfg<D>;
    CUtensorMap tq, tk, tv;
    {
        const cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)a.H_q, (cuuint64_t)a.q_rows};
        const cuuint64_t strides[2] = {(cuuint64_t)D * 2, (cuuint64_t)a.H_q * D * 2};
        const cuuint32_t box[3] = {64, 1, kBM};
        if (!encode(&tq, a.q, 3, dims, strides, box)) return cudaErrorInvalidValue;
    }
    const bool paged = a.map.table != nullptr;
    {
        // the cache rows as one 2-D array: contiguous caches cache_rows x
        // H_kv rows, tiles of 128 rows; pages num_blocks x H_kv x block_size
        // rows, one box per page (at most 128 rows)
        const int64_t bs = (int64_t)1 << a.map.bs_log2;
        const cuuint64_t rows = paged ? (cuuint64_t)(a.map.num_blocks * a.H_kv * bs)
                                      : (cuuint64_t)(a.cache_rows * a.H_kv);
        const cuuint64_t dims[2] = {(cuuint64_t)D, rows};
        const cuuint64_t strides[1] = {(cuuint64_t)D * 2};
        const cuuint32_t box[2] = {64, (cuuint32_t)(paged && bs < kBN ? bs : kBN)};
        if (!encode(&tk, a.k_cache, 2, dims, strides, box)) return cudaErrorInvalidValue;
        if (!encode(&tv, a.v_cache, 2, dims, strides, box)) return cudaErrorInvalidValue;
    }
    auto kern = paged ? prefill_attn_kernel<D, true> : prefill_attn_kernel<D, false>;
    // the shared-memory opt-in is per device: set it once on each
    static int configured_device_mask = 0;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (!(dev < 31 && (__atomic_load_n(&configured_device_mask, __ATOMIC_ACQUIRE) & (1 << dev)))) {
        for (auto kk : {prefill_attn_kernel<D, false>, prefill_attn_kernel<D, true>}) {
            e = cudaFuncSetAttribute(kk, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)C::kSmemBytes);
            if (e != cudaSuccess) return e;
        }
        if (dev < 31) __atomic_fetch_or(&configured_device_mask, 1 << dev, __ATOMIC_ACQ_REL);
    }
    const float sl2 = a.scale * 1.4426950408889634f;
    kern<<<num_sms, kThreads, C::kSmemBytes, stream>>>(
        tq, tk, tv, a.q_off, a.P, a.T, a.N, a.cache_off, static_cast<__nv_bfloat16 *>(a.out),
        a.q_rows, a.cache_rows, sl2, a.B, a.H_q, a.H_kv, a.w_eff, a.err, a.map);
    return cudaGetLastError();
}

}  // namespace

bool prefill_supported(speechkv_dtype dtype, int d) {
    return dtype == SPEECHKV_BF16 && (d == 64 || d == 128);
}

cudaError_t launch_prefill(const PrefillArgs &a, int num_sms, cudaStream_t stream) {
    if (a.d == 128) return launch_prefill_d<128>(a, num_sms, stream);
    if (a.d == 64) return launch_prefill_d<64>(a, num_sms, stream);
    return cudaErrorInvalidValue;
}

}  // namespace speechkv
