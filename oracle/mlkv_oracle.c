/*
 * MLKV decode- and prefill-attention oracle, and the KV-weight merge of the model conversion.
 *
 * TEST INFRASTRUCTURE ONLY.  This file states, in plain double-precision C, what the MLKV decode
 * path computes, so that the CUDA library can be checked against it.  Only the test suite,
 * __graft_entry__.smoke() and bench.py's CPU-baseline / reference legs may load it.  It shares no
 * code, header, table or constant with the CUDA library, and the library never calls it.
 *
 * Source: Zuhri, Adilazuarda, Purwarianti, Aji, "MLKV: Multi-Layer Key-Value Heads for Memory
 * Efficient Transformer Decoding" (arXiv 2406.09297).  Every function names the section / equation
 * it follows.  The paper counts layers and heads from 1; this file counts from 0 and converts
 * explicitly where an equation is restated.
 *
 * Readings taken where the paper is silent or ambiguous (all recorded in the design notes):
 *  - K/V of a block are produced once by its bottom layer and cached; the other layers of the block
 *    only read them (Sec. 3 cache size 2bsmgd_k, Fig. 2 caption, Sec. 4.2).
 *  - The new token attends to itself: positions [0, L) are visible, L counts the new token.
 *  - The softmax scale is 1/sqrt(d_k) with d_k the head dimension (Eq. 2).
 *  - An explicit layer -> owner map with owner[n] <= n and owner[owner[n]] == owner[n] generalises
 *    the contiguous blocks of Eq. 18; h must be divisible by g.
 *
 * Parity is pinned (tests/test_oracle_pins.py) by the paper's Table 1 ratios and Table 2 head
 * totals, torch's scaled_dot_product_attention for the MHA / GQA special cases, the equality of
 * MLKV with MHA on explicitly duplicated K/V, closed forms and a high-precision brute force.
 *
 * Build: gcc -O2 -ffp-contract=off -fPIC -shared (no FMA contraction, so x86 and Arm agree).
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_OK 0
#define ORACLE_ERR_ARG (-1)
#define ORACLE_ERR_MAP (-2)
#define ORACLE_ERR_RANGE (-3)
#define ORACLE_ERR_OOM (-4)

/* ------------------------------------------------------------------------------------------- */
/* Maps                                                                                          */
/* ------------------------------------------------------------------------------------------- */

/* Eq. 18 (Sec. 3): layer n (1-based) belongs to block k = floor((n-1)/(l/m)) + 1.  The block's
 * KV heads come from its bottom layer (Fig. 2 caption: "the one key-value head from the bottom
 * layer"; Sec. 4.2: later layers "do not have KV heads of their own").  Writes owner[] 0-based. */
int oracle_block_owner_map(int l, int m, int *owner)
{
    if (l <= 0 || m <= 0 || m > l || (l % m) != 0 || owner == NULL)
        return ORACLE_ERR_ARG;
    int per_block = l / m;                          /* l/m layers share one KV set */
    for (int n = 1; n <= l; ++n) {
        int k = (n - 1) / per_block + 1;            /* block of layer n, 1-based */
        int bottom = (k - 1) * per_block + 1;       /* first (bottom) layer of block k, 1-based */
        owner[n - 1] = bottom - 1;
    }
    return ORACLE_OK;
}

/* Eq. 12 (Sec. 2.3), repeated in Eq. 15: query head i (1-based) reads KV head
 * j = floor((i-1)/(h/g)) + 1.  Takes and returns 0-based indices. */
int oracle_kv_head_of(int h, int g, int i0)
{
    int i = i0 + 1;
    int j = (i - 1) / (h / g) + 1;
    return j - 1;
}

/* Checks a layer -> owner map and the head counts.  An owner must be an earlier (or the same)
 * layer that owns itself; g must divide h (Sec. 2.3 forms h/g groups). */
int oracle_validate(int l, const int *owner, int h, int g, int d)
{
    if (l <= 0 || h <= 0 || g <= 0 || d <= 0 || owner == NULL)
        return ORACLE_ERR_ARG;
    if (g > h || (h % g) != 0)
        return ORACLE_ERR_MAP;
    for (int n = 0; n < l; ++n) {
        int o = owner[n];
        if (o < 0 || o > n)
            return ORACLE_ERR_MAP;
        if (owner[o] != o)
            return ORACLE_ERR_MAP;
    }
    return ORACLE_OK;
}

/* Sec. 3: m is the number of layers that have KV heads of their own.  slot[n] is the position of
 * owner[n] among those layers in increasing layer order.  Returns m, or an error code. */
int oracle_slots(int l, const int *owner, int *slot)
{
    int m = 0;
    for (int n = 0; n < l; ++n) {
        if (owner[n] == n) {
            /* n is an owner; it is the m-th one met so far */
            for (int q = 0; q < l; ++q)
                if (owner[q] == n)
                    slot[q] = m;
            ++m;
        }
    }
    return m;
}

/* Sec. 2.5 and Sec. 3 / Table 1: the cache holds 2*b*s*m*g*d_k elements (K and V, b sequences of
 * s positions, m owner layers of g KV heads of width d_k).  MHA is m=l, g=h; MQA m=l, g=1. */
long long oracle_cache_elements(long long b, long long s, long long m, long long g, long long dk)
{
    return 2LL * b * s * m * g * dk;
}

/* ------------------------------------------------------------------------------------------- */
/* Attention                                                                                     */
/* ------------------------------------------------------------------------------------------- */

/* Eqs. 2-3 for one query vector: alpha = softmax(q K^T / sqrt(d_k)), o = alpha V, over the L
 * visible positions.  Subtracting the largest score before exp() leaves the softmax unchanged
 * (the factor cancels between numerator and denominator) and keeps exp() finite.
 * work must hold L doubles. */
static void attention_one_query(const double *q, const double *K, const double *V, int L, int d,
                                double *work, double *o)
{
    double inv_sqrt_dk = 1.0 / sqrt((double)d);
    double smax = -INFINITY;
    for (int t = 0; t < L; ++t) {
        double dot = 0.0;
        for (int e = 0; e < d; ++e)
            dot += q[e] * K[(size_t)t * d + e];
        work[t] = dot * inv_sqrt_dk;                  /* q k_t^T / sqrt(d_k) */
        if (work[t] > smax)
            smax = work[t];
    }
    double Z = 0.0;
    for (int t = 0; t < L; ++t) {
        work[t] = exp(work[t] - smax);
        Z += work[t];
    }
    for (int t = 0; t < L; ++t)
        work[t] = work[t] / Z;                        /* alpha_t */
    for (int e = 0; e < d; ++e) {
        double acc = 0.0;
        for (int t = 0; t < L; ++t)
            acc += work[t] * V[(size_t)t * d + e];    /* sum_t alpha_t v_t */
        o[e] = acc;
    }
}

typedef struct {
    int layer, h, g, d, b, max_seq;
    const int *owner;
    const int *seq_lens;
    const double *Q;
    const double *const *Kc;
    const double *const *Vc;
    double *out;
    int beta_lo, beta_hi;
    int status;
} layer_job;

static void *run_layer_job(void *arg)
{
    layer_job *jb = (layer_job *)arg;
    int h = jb->h, g = jb->g, d = jb->d;
    /* Eqs. 13-18: the layer's query heads read the KV heads of the layer that owns its block. */
    int k_owner = jb->owner[jb->layer];
    const double *Kown = jb->Kc[k_owner];
    const double *Vown = jb->Vc[k_owner];
    double *work = (double *)malloc(sizeof(double) * (size_t)(jb->max_seq > 0 ? jb->max_seq : 1));
    if (work == NULL) {
        jb->status = ORACLE_ERR_OOM;
        return NULL;
    }
    for (int beta = jb->beta_lo; beta < jb->beta_hi; ++beta) {
        int L = jb->seq_lens[beta];
        for (int i = 0; i < h; ++i) {
            int j = oracle_kv_head_of(h, g, i);                        /* Eq. 15 */
            const double *q = jb->Q + ((size_t)beta * h + i) * d;
            size_t kv_row = ((size_t)beta * g + j) * (size_t)jb->max_seq * d;
            double *o = jb->out + ((size_t)beta * h + i) * d;
            attention_one_query(q, Kown + kv_row, Vown + kv_row, L, d, work, o);
        }
    }
    free(work);
    jb->status = ORACLE_OK;
    return NULL;
}

/* One decode step of one layer (Sec. 3, Eqs. 13-18): every query head i of layer `layer` attends
 * over positions [0, seq_lens[beta]) of KV head j(i) held by the layer's owner.
 *   Q    [b][h][d]                 queries of this layer
 *   Kc,Vc  arrays indexed by layer; Kc[n] is layer n's own cache [b][g][max_seq][d] when n owns
 *          itself (other entries are never read)
 *   out  [b][h][d]
 * nthreads > 1 splits the batch across POSIX threads; the arithmetic per output is unchanged. */
int oracle_decode_layer(int layer, int l, const int *owner, int h, int g, int d, int b,
                        const int *seq_lens, int max_seq, const double *Q,
                        const double *const *Kc, const double *const *Vc, double *out,
                        int nthreads)
{
    int rc = oracle_validate(l, owner, h, g, d);
    if (rc != ORACLE_OK)
        return rc;
    if (layer < 0 || layer >= l || b < 0 || max_seq <= 0 || Q == NULL || out == NULL)
        return ORACLE_ERR_ARG;
    if (Kc == NULL || Vc == NULL || Kc[owner[layer]] == NULL || Vc[owner[layer]] == NULL)
        return ORACLE_ERR_ARG;
    for (int beta = 0; beta < b; ++beta)
        if (seq_lens[beta] < 1 || seq_lens[beta] > max_seq)
            return ORACLE_ERR_RANGE;
    if (nthreads < 1)
        nthreads = 1;
    if (nthreads > b)
        nthreads = b > 0 ? b : 1;

    layer_job *jobs = (layer_job *)calloc((size_t)nthreads, sizeof(layer_job));
    pthread_t *tids = (pthread_t *)calloc((size_t)nthreads, sizeof(pthread_t));
    if (jobs == NULL || tids == NULL) {
        free(jobs);
        free(tids);
        return ORACLE_ERR_OOM;
    }
    for (int w = 0; w < nthreads; ++w) {
        layer_job *jb = &jobs[w];
        jb->layer = layer; jb->h = h; jb->g = g; jb->d = d; jb->b = b; jb->max_seq = max_seq;
        jb->owner = owner; jb->seq_lens = seq_lens; jb->Q = Q; jb->Kc = Kc; jb->Vc = Vc;
        jb->out = out;
        jb->beta_lo = (int)((long long)b * w / nthreads);
        jb->beta_hi = (int)((long long)b * (w + 1) / nthreads);
        jb->status = ORACLE_ERR_ARG;
    }
    int started = 0;
    for (int w = 1; w < nthreads; ++w) {
        if (pthread_create(&tids[w], NULL, run_layer_job, &jobs[w]) != 0)
            break;
        started = w;
    }
    run_layer_job(&jobs[0]);
    for (int w = 1; w <= started; ++w)
        pthread_join(tids[w], NULL);
    /* any job whose thread could not be started runs here */
    for (int w = started + 1; w < nthreads; ++w)
        run_layer_job(&jobs[w]);
    rc = ORACLE_OK;
    for (int w = 0; w < nthreads; ++w)
        if (jobs[w].status != ORACLE_OK)
            rc = jobs[w].status;
    free(jobs);
    free(tids);
    return rc;
}

typedef struct {
    int layer, h, g, d, max_seq, s_max;
    const int *owner;
    const int *prompt_lens;
    const double *Q;
    const double *const *Kc;
    const double *const *Vc;
    double *out;
    int beta_lo, beta_hi;
    int status;
} prefill_job;

static void *run_prefill_job(void *arg)
{
    prefill_job *jb = (prefill_job *)arg;
    int h = jb->h, g = jb->g, d = jb->d;
    int k_owner = jb->owner[jb->layer];                                /* Eqs. 13-18 */
    const double *Kown = jb->Kc[k_owner];
    const double *Vown = jb->Vc[k_owner];
    double *work = (double *)malloc(sizeof(double) * (size_t)(jb->s_max > 0 ? jb->s_max : 1));
    if (work == NULL) {
        jb->status = ORACLE_ERR_OOM;
        return NULL;
    }
    for (int beta = jb->beta_lo; beta < jb->beta_hi; ++beta) {
        int S = jb->prompt_lens[beta];
        for (int t = 0; t < S; ++t) {
            int L = t + 1;                     /* position t sees positions 0 .. t */
            for (int i = 0; i < h; ++i) {
                int j = oracle_kv_head_of(h, g, i);                    /* Eq. 15 */
                const double *q = jb->Q + (((size_t)beta * jb->s_max + t) * h + i) * d;
                size_t kv_row = ((size_t)beta * g + j) * (size_t)jb->max_seq * d;
                double *o = jb->out + (((size_t)beta * jb->s_max + t) * h + i) * d;
                attention_one_query(q, Kown + kv_row, Vown + kv_row, L, d, work, o);
            }
        }
    }
    free(work);
    jb->status = ORACLE_OK;
    return NULL;
}

/* Prefill of one layer: the prompt processed at once.  A decoder-only model (Sec. 2.1; the
 * autoregressive order of Sec. 4.5) lets prompt position t attend to positions 0 .. t only, so
 * every row is Eqs. 2-3 over the owner's KV head j(i) (Eqs. 13-18) at visible length t + 1 --
 * the decode of Sec. 3 at that length.
 *   Q    [b][s_max][h][d]   the prompt's queries, position-major
 *   Kc,Vc as for oracle_decode_layer (the owner's cache holds the prompt's K/V)
 *   out  [b][s_max][h][d]   rows t >= prompt_lens[beta] are left untouched
 * nthreads > 1 splits the batch across POSIX threads. */
int oracle_prefill_layer(int layer, int l, const int *owner, int h, int g, int d, int b,
                         const int *prompt_lens, int s_max, int max_seq, const double *Q,
                         const double *const *Kc, const double *const *Vc, double *out,
                         int nthreads)
{
    int rc = oracle_validate(l, owner, h, g, d);
    if (rc != ORACLE_OK)
        return rc;
    if (layer < 0 || layer >= l || b < 0 || s_max <= 0 || s_max > max_seq || Q == NULL ||
        out == NULL)
        return ORACLE_ERR_ARG;
    if (Kc == NULL || Vc == NULL || Kc[owner[layer]] == NULL || Vc[owner[layer]] == NULL)
        return ORACLE_ERR_ARG;
    for (int beta = 0; beta < b; ++beta)
        if (prompt_lens[beta] < 1 || prompt_lens[beta] > s_max)
            return ORACLE_ERR_RANGE;
    if (nthreads < 1)
        nthreads = 1;
    if (nthreads > b)
        nthreads = b > 0 ? b : 1;
    prefill_job *jobs = (prefill_job *)calloc((size_t)nthreads, sizeof(prefill_job));
    pthread_t *tids = (pthread_t *)calloc((size_t)nthreads, sizeof(pthread_t));
    if (jobs == NULL || tids == NULL) {
        free(jobs);
        free(tids);
        return ORACLE_ERR_OOM;
    }
    for (int w = 0; w < nthreads; ++w) {
        prefill_job *jb = &jobs[w];
        jb->layer = layer; jb->h = h; jb->g = g; jb->d = d; jb->max_seq = max_seq;
        jb->s_max = s_max; jb->owner = owner; jb->prompt_lens = prompt_lens; jb->Q = Q;
        jb->Kc = Kc; jb->Vc = Vc; jb->out = out;
        jb->beta_lo = (int)((long long)b * w / nthreads);
        jb->beta_hi = (int)((long long)b * (w + 1) / nthreads);
        jb->status = ORACLE_ERR_ARG;
    }
    int started = 0;
    for (int w = 1; w < nthreads; ++w) {
        if (pthread_create(&tids[w], NULL, run_prefill_job, &jobs[w]) != 0)
            break;
        started = w;
    }
    run_prefill_job(&jobs[0]);
    for (int w = 1; w <= started; ++w)
        pthread_join(tids[w], NULL);
    for (int w = started + 1; w < nthreads; ++w)
        run_prefill_job(&jobs[w]);
    rc = ORACLE_OK;
    for (int w = 0; w < nthreads; ++w)
        if (jobs[w].status != ORACLE_OK)
            rc = jobs[w].status;
    free(jobs);
    free(tids);
    return rc;
}

/* Sec. 2.4 and Sec. 3: during decoding only a layer that owns KV heads projects and stores the
 * new token's keys and values (Eq. 13 exists for owner layers only); for any other layer the
 * append stores nothing.  K_new, V_new: [b][g][d]; the token goes to position seq_lens[beta]-1.
 * Returns 1 when something was written, 0 for a non-owner layer, or an error code. */
int oracle_append(int layer, int l, const int *owner, int g, int d, int b, const int *seq_lens,
                  int max_seq, const double *K_new, const double *V_new, double *const *Kc,
                  double *const *Vc)
{
    if (layer < 0 || layer >= l || owner == NULL)
        return ORACLE_ERR_ARG;
    if (owner[layer] != layer)
        return 0;
    if (Kc == NULL || Vc == NULL || Kc[layer] == NULL || Vc[layer] == NULL)
        return ORACLE_ERR_ARG;
    for (int beta = 0; beta < b; ++beta) {
        int L = seq_lens[beta];
        if (L < 1 || L > max_seq)
            return ORACLE_ERR_RANGE;
        for (int j = 0; j < g; ++j) {
            size_t dst = (((size_t)beta * g + j) * (size_t)max_seq + (size_t)(L - 1)) * d;
            size_t src = ((size_t)beta * g + j) * d;
            memcpy(Kc[layer] + dst, K_new + src, sizeof(double) * (size_t)d);
            memcpy(Vc[layer] + dst, V_new + src, sizeof(double) * (size_t)d);
        }
    }
    return 1;
}

/* ------------------------------------------------------------------------------------------- */
/* KV-weight merging (Sec. 4.2)                                                                  */
/* ------------------------------------------------------------------------------------------- */

/* Sec. 4.2: the variants are converted from the MHA baseline by merging KV-head weights by
 * averaging (the method the GQA paper found best): the heads of one group of a layer, and the
 * heads of the later layers of a block, which have no KV heads of their own, become one KV head.
 * Merged head j of owner layer o = the mean, over every layer n with owner[n] == o and every head
 * i of group j (Eq. 12: i / (h/g) == j, 0-based), of W[n][i][:].
 * W: [l][h][row] (per head, one projection's rows: head_dim x d_model, or head_dim for a bias);
 * out: [m][g][row], owners in increasing layer order (the slots of oracle_slots).  The sum is
 * taken in double precision in member order, then divided by the member count. */
int oracle_merge_kv(int l, const int *owner, int h, int g, long long row, const double *W,
                    double *out)
{
    if (row <= 0 || W == NULL || out == NULL)
        return ORACLE_ERR_ARG;
    int rc = oracle_validate(l, owner, h, g, 1);
    if (rc != ORACLE_OK)
        return rc;
    const int G = h / g;
    int s = 0;   /* slot of the current owner */
    for (int o = 0; o < l; ++o) {
        if (owner[o] != o)
            continue;
        for (int j = 0; j < g; ++j) {
            double *dst = out + ((size_t)s * g + j) * (size_t)row;
            for (long long r = 0; r < row; ++r) {
                double sum = 0.0;
                long long count = 0;
                for (int n = 0; n < l; ++n) {
                    if (owner[n] != o)
                        continue;
                    for (int i = j * G; i < (j + 1) * G; ++i) {
                        sum += W[((size_t)n * h + i) * (size_t)row + (size_t)r];
                        ++count;
                    }
                }
                dst[r] = sum / (double)count;
            }
        }
        ++s;
    }
    return ORACLE_OK;
}

/* bfloat16 (1 sign, 8 exponent, 7 stored significand bits) nearest to x, ties to the even
 * significand; beyond the largest finite value by half a unit in the last place or more,
 * infinity.  Written from the definition: scale |x| by its quantum (2^(e-7) for |x| in [2^e,
 * 2^(e+1)), at least 2^-133, the subnormal quantum), round to an integer half-to-even (rint in the
 * default rounding mode), scale back.  Returns the 16-bit pattern. */
unsigned oracle_bf16_rne(double x)
{
    const unsigned sign = signbit(x) ? 0x8000u : 0u;
    if (isnan(x))
        return sign | 0x7FC0u;
    const double a = fabs(x);
    if (a == 0.0)
        return sign;
    int e;
    (void)frexp(a, &e);            /* a = f 2^e, f in [0.5, 1): a in [2^(e-1), 2^e) */
    int q = (e - 1) - 7;           /* 8 significant bits */
    if (q < -133)
        q = -133;
    const double k = rint(ldexp(a, -q));   /* exact scaling, then half-to-even */
    const double v = ldexp(k, q);
    if (v > 0x1.FEp127)            /* largest finite bfloat16: (2 - 2^-7) 2^127 */
        return sign | 0x7F80u;
    const float f = (float)v;      /* exact: at most 8 significant bits, inside float's range */
    uint32_t bits;
    memcpy(&bits, &f, sizeof bits);
    return sign | ((bits >> 16) & 0x7FFFu);
}

void oracle_bf16_rne_array(const double *x, long long n, uint16_t *out)
{
    for (long long k = 0; k < n; ++k)
        out[k] = (uint16_t)oracle_bf16_rne(x[k]);
}
