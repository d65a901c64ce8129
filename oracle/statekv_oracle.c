/*
 * StateKV per-frame cache-builder step: plain CPU oracle (fp64).
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the slow, obviously-correct
 * statement of what the GPU path computes.  Only the test-suite, the smoke
 * check and the CPU-baseline leg of the benchmark may load it.  It shares no
 * code, header, table or helper with the CUDA library, and it never calls it.
 *
 * What it follows (Eyzaguirre, Wu, Niebles, "Linear Scaling Video VLMs for
 * Long Video Understanding"):
 *   - Sec. 3.3, Eq. 5: the frame's queries attend to [state ; frame] keys with
 *     softmax(Q [Kbar;K]^T / sqrt(d_h) + M_n) [Vbar;V]; M_n lets every query see
 *     every state (memory) token and is causal in stream order inside the frame.
 *   - Sec. 3.1, Eq. 1 and Sec. 3.3 (score of a candidate): the importance of a
 *     pool token is the attention it receives from the frame's queries, summed
 *     over the queries (the 1/T mean does not change the ranking) and over the
 *     query heads that share its KV head (App. A: sinks are kept per layer and
 *     per KV head).  App. B.1 recovers each weight as exp(score - LSE_query).
 *   - Sec. 3.3, Eq. 6: the candidate pool is the current state plus the frame's
 *     tokens; the B best-scoring candidates become the next state.
 *   - Sec. 3.2 (detailed state) / Sec. 3.3: the frame's K and V are appended to
 *     the per-frame decode cache; the virtual length L_n advances by T.
 *
 * Readings where the paper is silent:
 *   - ties in the score are broken by position: the older token wins;
 *   - while the pool holds no more than B tokens, every token is kept;
 *   - B = 0 leaves no cross-frame context;
 *   - the state is a set: its entries are kept here in ascending position.
 *
 * Inputs are bf16 bit patterns; every bf16 value is exactly representable in
 * a double, so all arithmetic below is fp64.  The oracle is pinned by the CPU
 * tests (brute-force full attention, closed forms at Q = 0, a hand-worked
 * example, invariants, brute-force subset selection).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

static double bf16_to_double(uint16_t bits)
{
    uint32_t u = ((uint32_t)bits) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* One candidate of the pool of Sec. 3.3: an old state entry or a frame token. */
typedef struct {
    double score;
    int64_t pos;
    int from_frame; /* 0: state entry `index`, 1: frame token `index` */
    int index;
} candidate;

/* Order of Eq. 6's TopK: higher score first; equal scores keep the older token. */
static int candidate_cmp(const void* pa, const void* pb)
{
    const candidate* a = (const candidate*)pa;
    const candidate* b = (const candidate*)pb;
    if (a->score > b->score) return -1;
    if (a->score < b->score) return 1;
    if (a->pos < b->pos) return -1;
    if (a->pos > b->pos) return 1;
    return 0;
}

static int pos_cmp(const void* pa, const void* pb)
{
    const candidate* a = (const candidate*)pa;
    const candidate* b = (const candidate*)pb;
    return (a->pos > b->pos) - (a->pos < b->pos);
}

/*
 * One frame of one (stream, layer).
 *
 *   n_q, n_kv, d      query heads, KV heads (n_q % n_kv == 0), head dim
 *   T, B              tokens per frame, state capacity
 *   causal            1: key t of the frame is visible to query i iff t <= i
 *   scale             softmax scale (1/sqrt(d) in the paper)
 *   virtual_len       L_{n-1}: tokens seen before this frame; token t of the
 *                     frame sits at position virtual_len + t
 *   q                 [T][n_q][d] bf16 bits
 *   k, v              [T][n_kv][d] bf16 bits
 *   count             [n_kv] in/out: valid state entries per KV head
 *   pos               [n_kv][B] in/out: their positions, ascending
 *   sk, sv            [n_kv][B][d] in/out: their K and V (bf16 bits)
 *   out               [T][n_q][d] attention output
 *   imp               [n_kv][B+T]: column c < B is state entry c (0 when
 *                     c >= count), column B + t is frame token t
 *   kept              optional [n_kv][B+T] 0/1 flags, same columns as imp
 * Returns 0, or -1 on bad arguments or allocation failure.
 */
int oracle_prefill_frame_policy(int n_q, int n_kv, int d, int T, int B, int causal, double scale,
                                int64_t virtual_len, const uint16_t* q, const uint16_t* k,
                                const uint16_t* v, int32_t* count, int64_t* pos, uint16_t* sk,
                                uint16_t* sv, double* out, double* imp, int32_t* kept, int policy);

int oracle_prefill_frame(int n_q, int n_kv, int d, int T, int B, int causal, double scale,
                         int64_t virtual_len, const uint16_t* q, const uint16_t* k,
                         const uint16_t* v, int32_t* count, int64_t* pos, uint16_t* sk,
                         uint16_t* sv, double* out, double* imp, int32_t* kept)
{
    return oracle_prefill_frame_policy(n_q, n_kv, d, T, B, causal, scale, virtual_len, q, k, v,
                                       count, pos, sk, sv, out, imp, kept, 0);
}

/*
 * The same frame step with a choice of which B pool tokens the state keeps:
 *   policy 0  the method (Eq. 6): the B highest importances, ties to the
 *             older token;
 *   policy 1  the recency window of the ReKV-style baseline the paper compares
 *             with (Sec. 2, Sec. 4): the B most recent positions;
 *   policy 2  layer-level selection: one ranking per layer by the attention
 *             summed over all heads (the score of Sec. 3.3 aggregated over
 *             heads, and the layer-level score of App. A.1), applied to every
 *             KV head, which therefore all hold the same positions.  The
 *             states given must already agree across heads (-1 otherwise).
 * The attention and the per-KV-head importance are computed the same way for
 * all three.
 */
int oracle_prefill_frame_policy(int n_q, int n_kv, int d, int T, int B, int causal, double scale,
                                int64_t virtual_len, const uint16_t* q, const uint16_t* k,
                                const uint16_t* v, int32_t* count, int64_t* pos, uint16_t* sk,
                                uint16_t* sv, double* out, double* imp, int32_t* kept, int policy)
{
    if (policy < 0 || policy > 2) return -1;
    if (n_q <= 0 || n_kv <= 0 || n_q % n_kv != 0 || d <= 0 || T <= 0 || B < 0) return -1;
    const int G = n_q / n_kv;
    const int P = B + T;

    double* z = (double*)malloc(sizeof(double) * (size_t)P);
    double* qd = (double*)malloc(sizeof(double) * (size_t)d);
    candidate* pool = (candidate*)malloc(sizeof(candidate) * (size_t)P);
    uint16_t* nk = (uint16_t*)malloc(sizeof(uint16_t) * (size_t)(B > 0 ? B : 1) * (size_t)d);
    uint16_t* nv = (uint16_t*)malloc(sizeof(uint16_t) * (size_t)(B > 0 ? B : 1) * (size_t)d);
    double* shared = (double*)calloc((size_t)P, sizeof(double));
    if (!z || !qd || !pool || !nk || !nv || !shared) {
        free(z); free(qd); free(pool); free(nk); free(nv); free(shared);
        return -1;
    }
    for (int h = 0; h < n_kv; ++h)
        if (count[h] < 0 || count[h] > B) {
            free(z); free(qd); free(pool); free(nk); free(nv); free(shared);
            return -1;
        }
    if (policy == 2)
        for (int h = 1; h < n_kv; ++h) {
            int same = count[h] == count[0];
            for (int c = 0; same && c < count[0]; ++c)
                same = pos[(size_t)h * B + c] == pos[c];
            if (!same) { free(z); free(qd); free(pool); free(nk); free(nv); free(shared); return -1; }
        }

    /* Attention and importance of every KV head. */
    for (int h = 0; h < n_kv; ++h) {
        const int b = count[h];
        const uint16_t* hk = sk + (size_t)h * B * d;
        const uint16_t* hv = sv + (size_t)h * B * d;
        double* himp = imp + (size_t)h * P;
        for (int c = 0; c < P; ++c) himp[c] = 0.0;

        /* Eq. 5 for every query head g of this KV head and every query i. */
        for (int g = 0; g < G; ++g) {
            const int hq = h * G + g;
            for (int i = 0; i < T; ++i) {
                for (int e = 0; e < d; ++e)
                    qd[e] = bf16_to_double(q[((size_t)i * n_q + hq) * d + e]);
                /* Visible keys: all b state entries, then frame tokens t <= i. */
                const int nf = causal ? i + 1 : T;
                double m = -INFINITY;
                for (int c = 0; c < b; ++c) {
                    double acc = 0.0;
                    for (int e = 0; e < d; ++e)
                        acc += qd[e] * bf16_to_double(hk[(size_t)c * d + e]);
                    z[c] = scale * acc;
                    if (z[c] > m) m = z[c];
                }
                for (int t = 0; t < nf; ++t) {
                    double acc = 0.0;
                    for (int e = 0; e < d; ++e)
                        acc += qd[e] * bf16_to_double(k[((size_t)t * n_kv + h) * d + e]);
                    z[b + t] = scale * acc;
                    if (z[b + t] > m) m = z[b + t];
                }
                double s = 0.0;
                for (int c = 0; c < b + nf; ++c) s += exp(z[c] - m);
                const double lse = m + log(s);

                double* o = out + ((size_t)i * n_q + hq) * d;
                for (int e = 0; e < d; ++e) o[e] = 0.0;
                for (int c = 0; c < b + nf; ++c) {
                    const double a = exp(z[c] - lse); /* App. B.1: exp(score - LSE) */
                    const uint16_t* vrow = (c < b) ? hv + (size_t)c * d
                                                   : v + ((size_t)(c - b) * n_kv + h) * d;
                    for (int e = 0; e < d; ++e) o[e] += a * bf16_to_double(vrow[e]);
                    /* Eq. 1: the weight counts toward the key's importance. */
                    if (c < b) himp[c] += a;
                    else himp[B + (c - b)] += a;
                }
            }
        }
    }
    /* Layer-level score: the importance summed over the KV heads (each already
     * a sum over its query heads), column by column; the columns name the
     * same positions in every head. */
    if (policy == 2)
        for (int h = 0; h < n_kv; ++h)
            for (int c = 0; c < P; ++c) shared[c] += imp[(size_t)h * P + c];

    /* Selection and gather, per KV head. */
    for (int h = 0; h < n_kv; ++h) {
        const int b = count[h];
        const uint16_t* hk = sk + (size_t)h * B * d;
        const uint16_t* hv = sv + (size_t)h * B * d;
        const double* himp = policy == 2 ? shared : imp + (size_t)h * P;

        /* Eq. 6: pool = state entries + frame tokens; keep the B best. */
        int np = 0;
        for (int c = 0; c < b; ++c) {
            pool[np].score = himp[c];
            pool[np].pos = pos[(size_t)h * B + c];
            pool[np].from_frame = 0;
            pool[np].index = c;
            ++np;
        }
        for (int t = 0; t < T; ++t) {
            pool[np].score = himp[B + t];
            pool[np].pos = virtual_len + t;
            pool[np].from_frame = 1;
            pool[np].index = t;
            ++np;
        }
        int nkeep = np;
        if (np > B) {
            if (policy == 1)  /* most recent first: rank by position */
                for (int c = 0; c < np; ++c) pool[c].score = (double)pool[c].pos;
            qsort(pool, (size_t)np, sizeof(candidate), candidate_cmp);
            nkeep = B;
        }
        qsort(pool, (size_t)nkeep, sizeof(candidate), pos_cmp);

        if (kept) {
            int32_t* hkept = kept + (size_t)h * P;
            for (int c = 0; c < P; ++c) hkept[c] = 0;
            for (int c = 0; c < nkeep; ++c)
                hkept[pool[c].from_frame ? B + pool[c].index : pool[c].index] = 1;
        }

        /* Gather: the new state holds bit copies of the kept rows. */
        for (int c = 0; c < nkeep; ++c) {
            const uint16_t* srck;
            const uint16_t* srcv;
            if (pool[c].from_frame) {
                srck = k + ((size_t)pool[c].index * n_kv + h) * d;
                srcv = v + ((size_t)pool[c].index * n_kv + h) * d;
            } else {
                srck = hk + (size_t)pool[c].index * d;
                srcv = hv + (size_t)pool[c].index * d;
            }
            memcpy(nk + (size_t)c * d, srck, sizeof(uint16_t) * (size_t)d);
            memcpy(nv + (size_t)c * d, srcv, sizeof(uint16_t) * (size_t)d);
        }
        for (int c = 0; c < nkeep; ++c) pos[(size_t)h * B + c] = pool[c].pos;
        for (int c = nkeep; c < B; ++c) pos[(size_t)h * B + c] = -1;
        if (nkeep > 0) {
            memcpy(sk + (size_t)h * B * d, nk, sizeof(uint16_t) * (size_t)nkeep * d);
            memcpy(sv + (size_t)h * B * d, nv, sizeof(uint16_t) * (size_t)nkeep * d);
        }
        count[h] = nkeep;
    }

    free(z); free(qd); free(pool); free(nk); free(nv); free(shared);
    return 0;
}

/*
 * Detailed state (Sec. 3.2, Sec. 3.3): D_n = D_{n-1} with the frame's
 * (K_n, V_n) appended at rows virtual_len .. virtual_len + T - 1.
 *   k, v     [T][n_kv][d] bf16 bits
 *   dk, dv   [n_kv][capacity][d] bf16 bits
 * Returns -1 if the cache would overflow.
 */
int oracle_append_cache(int n_kv, int d, int T, int64_t virtual_len, int64_t capacity,
                        const uint16_t* k, const uint16_t* v, uint16_t* dk, uint16_t* dv)
{
    if (virtual_len < 0 || virtual_len + T > capacity) return -1;
    for (int h = 0; h < n_kv; ++h)
        for (int t = 0; t < T; ++t) {
            const size_t src = ((size_t)t * n_kv + h) * d;
            const size_t dst = ((size_t)h * capacity + (size_t)(virtual_len + t)) * d;
            memcpy(dk + dst, k + src, sizeof(uint16_t) * (size_t)d);
            memcpy(dv + dst, v + src, sizeof(uint16_t) * (size_t)d);
        }
    return 0;
}
