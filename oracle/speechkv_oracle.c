/*
 * SpeechKV CPU oracle -- TEST INFRASTRUCTURE, not part of the product.
 *
 * Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline /
 * reference leg may load or call this library.  The CUDA path never links,
 * includes or calls it, and this file shares no code with the CUDA path.
 *
 * What it computes (paper "Compress the Cache, Not the Speech Embedding",
 * Sec. III-B "SpeechKV", Eq. (pool) and Eq. (attn); Sec. III-C):
 *
 *   Pooling P_R at layers l >= l0: the T speech positions of a request are cut
 *   into non-overlapping windows of R (= w) consecutive frames; text positions
 *   are kept as they are.  In a window, a linear gate g(k) = u . k gives one
 *   logit per key; a softmax over the window turns the logits into weights
 *   alpha_j; the pooled key and value are sum_j alpha_j k_j and
 *   sum_j alpha_j v_j (the value uses the key's weights).
 *
 *   Decode attention: at every layer the full-resolution query attends over
 *   the (compressed) cache, softmax(q K^T / sqrt(d_h)) V, grouped-query style.
 *
 *   Prefill attention (Sec. III-B, Eq. (attn) with the adjusted causal mask):
 *   every full-resolution prompt query attends over the compressed rows that
 *   precede it.  Reading of "causality over the compressed sequence": a
 *   query at prompt position t is placed at the compressed position pi(t)
 *   of the row that holds it (t for the text prefix, P + floor((t - P) / w)
 *   for a speech frame -- its own window --, t - T + n for the text after
 *   the speech) and sees compressed rows 0 .. pi(t).
 *
 * Everything is plain loops in fp64 written straight from those
 * definitions.  No blocking, no fusion, no online softmax.  Readings of
 * points the paper leaves open (see the design notes of the repository):
 *   - one gate vector u[h] in R^{d_h} per (layer, KV head); no bias (a bias
 *     is constant over a window and cancels in the softmax);
 *   - the last window may hold fewer than w frames; n = ceil(T / w) and the
 *     softmax runs over the frames present;
 *   - layers are 0-indexed: layer l is pooled iff l >= l0, else w_eff = 1;
 *   - query head hq uses KV head floor(hq / (H_q / H_kv));
 *   - cached row order of a request: [text prefix P; pooled speech n;
 *     text suffix N; generated tokens];
 *   - attention over an empty cache returns zeros (the softmax is undefined
 *     there; decode always appends before it attends, so it never arises in
 *     the method itself).
 *
 * Storage rounding: `storage` 0 leaves results exact (fp64), 1 rounds each
 * produced value once to fp32 (round to nearest even), 2 rounds it once to
 * bf16 (8 significant bits, round to nearest even).
 *
 * Layouts used here are the plain ones: a request's keys are [rows][H_kv][d]
 * (token-major), queries and outputs are [H_q][d].
 */
#include <math.h>
#include <stdint.h>
#include <string.h>
#include <stdlib.h>

#define ORACLE_STORE_EXACT 0
#define ORACLE_STORE_F32 1
#define ORACLE_STORE_BF16 2

/* Round to the nearest value with `bits` significant bits (ties to even),
 * with the exponent range of IEEE binary32 (bf16 shares it).  Written from
 * the definition of round-to-nearest-even: scale so that the quantum is 1,
 * round to an integer with nearbyint (default rounding mode is nearest-even),
 * scale back. */
static double round_sig_bits(double x, int bits, double max_finite)
{
    if (!isfinite(x) || x == 0.0)
        return x;
    int e;
    (void)frexp(x, &e);              /* x = m * 2^e, 0.5 <= |m| < 1 */
    int q = e - bits;                /* exponent of the last kept bit */
    const int min_q = -126 - (bits - 1); /* quantum of the subnormal range */
    if (q < min_q)
        q = min_q;
    double r = ldexp(nearbyint(ldexp(x, -q)), q);
    if (fabs(r) > max_finite)
        return x > 0 ? INFINITY : -INFINITY;
    return r;
}

/* bf16: 8 significant bits; largest finite value (2 - 2^-7) * 2^127. */
double oracle_round_bf16(double x)
{
    return round_sig_bits(x, 8, ldexp(2.0 - ldexp(1.0, -7), 127));
}

/* fp32: the C conversion double -> float rounds to nearest even. */
double oracle_round_f32(double x)
{
    return (double)(float)x;
}

static double store(double x, int32_t storage)
{
    if (storage == ORACLE_STORE_F32)
        return oracle_round_f32(x);
    if (storage == ORACLE_STORE_BF16)
        return oracle_round_bf16(x);
    return x;
}

/* Effective window: pooling applies only at layers l >= l0 (Sec. III-B). */
int32_t oracle_effective_window(int32_t w, int32_t layer, int32_t l0)
{
    return layer >= l0 ? w : 1;
}

/* Number of cached rows of one request at one layer:
 * P + ceil(T / w_eff) + N + G  (text kept, speech pooled per window). */
int64_t oracle_compressed_len(int32_t P, int32_t T, int32_t N, int32_t G,
                              int32_t w, int32_t layer, int32_t l0)
{
    if (P < 0 || T < 0 || N < 0 || G < 0 || w < 1 || layer < 0 || l0 < 0)
        return -1;
    int64_t we = oracle_effective_window(w, layer, l0);
    int64_t n = 0;
    while (n * we < (int64_t)T) /* smallest n with n * w_eff >= T */
        n++;
    return (int64_t)P + n + (int64_t)N + (int64_t)G;
}

/* Eq. (pool) for one request at one layer.
 * K, V: [P + T + N][H_kv][d]; gate: [H_kv][d] (the vector u of g(k) = u.k).
 * Writes rows [P + n + N][H_kv][d] to K_out / V_out; returns that row count
 * (-1 on bad arguments).  alpha (optional, may be NULL): receives the
 * softmax weight of every speech frame, [T][H_kv]. */
int64_t oracle_pool_request(const double *K, const double *V,
                            int32_t P, int32_t T, int32_t N,
                            int32_t H_kv, int32_t d, const double *gate,
                            int32_t w, int32_t layer, int32_t l0,
                            int32_t storage, double *K_out, double *V_out,
                            double *alpha)
{
    if (P < 0 || T < 0 || N < 0 || H_kv < 1 || d < 1 || w < 1)
        return -1;
    const int64_t row = (int64_t)H_kv * d; /* elements per token row */
    const int32_t we = oracle_effective_window(w, layer, l0);
    const int64_t n = oracle_compressed_len(0, T, 0, 0, w, layer, l0);
    double *z = (double *)malloc(sizeof(double) * (size_t)(we > 0 ? we : 1));
    if (!z)
        return -1;

    /* text prefix: rows 0..P-1 unchanged */
    for (int64_t t = 0; t < P; t++)
        for (int64_t e = 0; e < row; e++) {
            K_out[t * row + e] = store(K[t * row + e], storage);
            V_out[t * row + e] = store(V[t * row + e], storage);
        }

    /* speech: window i covers frames P + i*we .. P + min((i+1)*we, T) - 1 */
    for (int64_t i = 0; i < n; i++) {
        const int64_t j0 = (int64_t)P + i * we;
        int64_t j1 = (int64_t)P + (i + 1) * we;
        if (j1 > (int64_t)P + T)
            j1 = (int64_t)P + T;
        for (int32_t h = 0; h < H_kv; h++) {
            /* logits g(k_j) = u_h . k_j */
            for (int64_t j = j0; j < j1; j++) {
                double s = 0.0;
                for (int32_t c = 0; c < d; c++)
                    s += gate[(int64_t)h * d + c] * K[j * row + (int64_t)h * d + c];
                z[j - j0] = s;
            }
            /* softmax over the window (max-subtracted) */
            double m = z[0];
            for (int64_t j = j0; j < j1; j++)
                if (z[j - j0] > m)
                    m = z[j - j0];
            double sum = 0.0;
            for (int64_t j = j0; j < j1; j++) {
                z[j - j0] = exp(z[j - j0] - m);
                sum += z[j - j0];
            }
            for (int64_t j = j0; j < j1; j++) {
                z[j - j0] /= sum;
                if (alpha)
                    alpha[(j - P) * H_kv + h] = z[j - j0];
            }
            /* weighted sums; V takes the weights computed from K */
            const int64_t o = ((int64_t)P + i) * row + (int64_t)h * d;
            for (int32_t c = 0; c < d; c++) {
                double ks = 0.0, vs = 0.0;
                for (int64_t j = j0; j < j1; j++) {
                    ks += z[j - j0] * K[j * row + (int64_t)h * d + c];
                    vs += z[j - j0] * V[j * row + (int64_t)h * d + c];
                }
                K_out[o + c] = store(ks, storage);
                V_out[o + c] = store(vs, storage);
            }
        }
    }

    /* text after the speech: source rows P+T .. P+T+N-1 go to P+n .. */
    for (int64_t t = 0; t < N; t++) {
        const int64_t src = ((int64_t)P + T + t) * row;
        const int64_t dst = ((int64_t)P + n + t) * row;
        for (int64_t e = 0; e < row; e++) {
            K_out[dst + e] = store(K[src + e], storage);
            V_out[dst + e] = store(V[src + e], storage);
        }
    }
    free(z);
    return (int64_t)P + n + N;
}

/* Append one decoded token's key and value ([H_kv][d]) as row `n` of a
 * request's cache of capacity `cap` rows.  Returns the new row count, or -1
 * when the cache is full (nothing written). */
int64_t oracle_append_request(double *K_cache, double *V_cache, int64_t n,
                              int64_t cap, const double *k_new,
                              const double *v_new, int32_t H_kv, int32_t d)
{
    if (n < 0 || n >= cap)
        return -1;
    const int64_t row = (int64_t)H_kv * d;
    memcpy(K_cache + n * row, k_new, sizeof(double) * (size_t)row);
    memcpy(V_cache + n * row, v_new, sizeof(double) * (size_t)row);
    return n + 1;
}

/* Eq. (attn) for one decode query of one request.
 * q: [H_q][d]; K, V: [n][H_kv][d]; out: [H_q][d].  scale <= 0 means
 * 1 / sqrt(d).  probs (optional, may be NULL): receives the softmax weights,
 * [H_q][n]. */
int32_t oracle_decode_attn_request(const double *q, const double *K,
                                   const double *V, int64_t n, int32_t H_q,
                                   int32_t H_kv, int32_t d, double scale,
                                   int32_t storage, double *out, double *probs)
{
    if (H_q < 1 || H_kv < 1 || d < 1 || H_q % H_kv != 0 || n < 0)
        return -1;
    if (!(scale > 0.0))
        scale = 1.0 / sqrt((double)d);
    const int32_t group = H_q / H_kv;
    const int64_t row = (int64_t)H_kv * d;
    double *p = (double *)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
    if (!p)
        return -1;
    for (int32_t hq = 0; hq < H_q; hq++) {
        const int32_t h = hq / group;
        if (n == 0) {
            for (int32_t c = 0; c < d; c++)
                out[(int64_t)hq * d + c] = 0.0;
            continue;
        }
        for (int64_t j = 0; j < n; j++) {
            double s = 0.0;
            for (int32_t c = 0; c < d; c++)
                s += q[(int64_t)hq * d + c] * K[j * row + (int64_t)h * d + c];
            p[j] = s * scale;
        }
        double m = p[0];
        for (int64_t j = 1; j < n; j++)
            if (p[j] > m)
                m = p[j];
        double sum = 0.0;
        for (int64_t j = 0; j < n; j++) {
            p[j] = exp(p[j] - m);
            sum += p[j];
        }
        for (int64_t j = 0; j < n; j++) {
            p[j] /= sum;
            if (probs)
                probs[(int64_t)hq * n + j] = p[j];
        }
        for (int32_t c = 0; c < d; c++) {
            double acc = 0.0;
            for (int64_t j = 0; j < n; j++)
                acc += p[j] * V[j * row + (int64_t)h * d + c];
            out[(int64_t)hq * d + c] = store(acc, storage);
        }
    }
    free(p);
    return 0;
}

/* Compressed position of prompt position t (0 <= t < P + T + N) at window
 * w_eff: the row of the compressed cache that holds position t.  -1 on bad
 * arguments. */
int64_t oracle_prefill_position(int32_t P, int32_t T, int32_t N, int32_t w_eff,
                                int64_t t)
{
    if (P < 0 || T < 0 || N < 0 || w_eff < 1 || t < 0 ||
        t >= (int64_t)P + T + N)
        return -1;
    int64_t n = 0;
    while (n * w_eff < T)
        n++;
    if (t < P)
        return t;
    if (t < (int64_t)P + T)
        return P + (t - P) / w_eff;
    return t - T + n;
}

/* Eq. (attn) at prefill for one request: Q [S][H_q][d] (S = P + T + N
 * prompt positions), compressed K, V [c][H_kv][d] (c = P + n + N rows, as
 * the pooling writes them), out [S][H_q][d].  Query t, head hq attends over
 * rows 0 .. pi(t) of KV head hq / (H_q / H_kv) with weights
 * softmax(q . k / sqrt(d)) (scale <= 0 means 1 / sqrt(d)). */
int32_t oracle_prefill_attn_request(const double *Q, const double *K,
                                    const double *V, int32_t P, int32_t T,
                                    int32_t N, int32_t w_eff, int32_t H_q,
                                    int32_t H_kv, int32_t d, double scale,
                                    int32_t storage, double *out)
{
    if (H_q < 1 || H_kv < 1 || d < 1 || H_q % H_kv != 0 || P < 0 || T < 0 ||
        N < 0 || w_eff < 1)
        return -1;
    if (!(scale > 0.0))
        scale = 1.0 / sqrt((double)d);
    const int64_t S = (int64_t)P + T + N;
    int64_t n = 0;
    while (n * w_eff < T)
        n++;
    const int64_t c = P + n + N;
    const int32_t group = H_q / H_kv;
    const int64_t qrow = (int64_t)H_q * d, krow = (int64_t)H_kv * d;
    double *p = (double *)malloc(sizeof(double) * (size_t)(c > 0 ? c : 1));
    if (!p)
        return -1;
    for (int64_t t = 0; t < S; t++) {
        const int64_t last = oracle_prefill_position(P, T, N, w_eff, t);
        for (int32_t hq = 0; hq < H_q; hq++) {
            const int32_t h = hq / group;
            const double *q = Q + t * qrow + (int64_t)hq * d;
            for (int64_t e = 0; e <= last; e++) {
                double s = 0.0;
                for (int32_t k = 0; k < d; k++)
                    s += q[k] * K[e * krow + (int64_t)h * d + k];
                p[e] = s * scale;
            }
            double m = p[0];
            for (int64_t e = 1; e <= last; e++)
                if (p[e] > m)
                    m = p[e];
            double sum = 0.0;
            for (int64_t e = 0; e <= last; e++) {
                p[e] = exp(p[e] - m);
                sum += p[e];
            }
            for (int32_t k = 0; k < d; k++) {
                double acc = 0.0;
                for (int64_t e = 0; e <= last; e++)
                    acc += p[e] * V[e * krow + (int64_t)h * d + k];
                out[t * qrow + (int64_t)hq * d + k] = store(acc / sum, storage);
            }
        }
    }
    free(p);
    return 0;
}
