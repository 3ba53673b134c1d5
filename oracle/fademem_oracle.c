/*
 * fademem_oracle.c -- plain, slow, fp64 CPU oracle of FadeMem
 * (arxiv 2606.10671, "FadeMem: Distance-Aware Memory Consolidation for
 * Autoregressive Video Diffusion").
 *
 * TEST INFRASTRUCTURE ONLY.  The test-suite, the smoke check and the CPU
 * baseline leg of the benchmark load this library; the CUDA library never
 * includes, links or calls it, and this file includes nothing of the CUDA
 * library.  Every result here is computed in IEEE double precision.
 *
 * What it computes
 *   1. The online memory update of Algorithm S1 (supplementary Sec. S1), one
 *      generation unit (one latent frame, Sec. S4) per call:
 *        - append (K_t, V_t, mu = t, s = 1)                (Sec. 3.3, "insertion")
 *        - if more than M entries, score every adjacent pair except the one
 *          holding the newest entry by g_i = |u(t-mu_{i+1}) - u(t-mu_i)|,
 *          u(d) = d^beta                     (Sec. 3.3, "distance-aware scheduling")
 *        - j = argmin_i g_i
 *        - s_new = s_j + s_{j+1}; if the pair holds the first-frame anchor the
 *          result keeps the anchor's K/V and mu = 0 (Sec. 3.3, "boundary
 *          handling"; Algorithm S1), otherwise mu_new is the span-weighted
 *          centre and the K/V blocks are merged by the operator (Sec. 3.3,
 *          "consolidation operator", square-root span weights by default;
 *          Table 2 for the alternatives)
 *        - the result replaces the pair.
 *   2. Attention of query tokens over every token of every memory entry,
 *      per head: out = softmax(scale * q K^T) V (the backbone attention whose
 *      context the memory supplies, Sec. 3.3 last paragraph, Sec. 4.1).
 *
 * Readings where the paper is silent:
 *   - frames are numbered from t = 0, so the anchor's own centre is mu = 0;
 *   - ties in the argmin go to the lowest pair index (the oldest pair);
 *   - the anchor is entry 0; its pair is j == 0;
 *   - storage slots: the paper has none.  To check a device slot table the
 *     oracle also keeps one: the merged entry keeps the slot of m_j, and the
 *     new entry takes the slot freed by m_{j+1} (or slot count-1 when no
 *     merge happens).  This never changes what is computed.
 *   - "Select Nearest" keeps the block of the entry nearer to the current step
 *     (m_{j+1}, the smaller distance d).
 *   - Temporal RoPE (Sec. 3.3, "Boundary and positional handling"; optional,
 *     oracle_set_rope): the temporal band is the first P complex pairs
 *     (dims 2k, 2k+1 for k < P) of each head's key, with the standard RoPE
 *     frequencies omega_k = theta^(-k/P) (Su et al., the RoFormer paper the
 *     section cites) and the rotation (x, y) -> (x cos a - y sin a,
 *     x sin a + y cos a) by a = position * omega_k.  Keys arrive rotated to
 *     their frame's position t; they are stored with that phase removed
 *     (rotated by -t * omega_k).  At attention time entry i of the count
 *     entries (temporal order) is re-indexed to position
 *     tau_i = t_next - count + i: consecutive positions ending right before
 *     the current chunk (frame t_next), so the exposed temporal range is
 *     bounded by the budget M.  With no merges this gives every frame its
 *     own position back.  Values are never rotated.
 *
 * Layout of a K or V block: elems_per_block doubles, in the caller's order.
 * For attention the order must be [token][head][dim] (tokens x heads x dim).
 * Merges are elementwise, so a caller may also pass any subset of coordinates
 * (e.g. a fixed sample), and the oracle's values at those coordinates are
 * exactly those of the full computation.
 */
#include <math.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

enum { OP_WEIGHTED = 0, OP_AVERAGE = 1, OP_SELECT_NEAREST = 2, OP_MAX_POOL = 3 };

struct entry {
    int slot;           /* storage slot (reading: slot policy above) */
    long long first;    /* first generation unit summarised */
    long long span;     /* s: number of units summarised */
    double mu;          /* temporal centre */
    double *K, *V;      /* representative blocks */
};

typedef struct oracle_memory {
    int M;               /* entry budget */
    double beta;         /* warp exponent, 0 < beta <= 1 */
    int anchor;          /* first-frame global anchor on/off */
    int op;              /* consolidation operator */
    long long elems;     /* doubles per K (or V) block */
    long long t_next;    /* index of the next generation unit */
    int count;           /* |M_t| */
    struct entry *e;     /* e[0..count-1], temporal order; room for M+1 */
    /* record of the latest update, for tests */
    int last_j;          /* merged pair index, -1 if none */
    double last_margin;  /* (g_second - g_min) / g_second, +inf if < 2 pairs */
    double last_gmin;
    /* temporal RoPE (0 pairs: off) */
    int rope_pairs, rope_tokens, rope_H, rope_D;
    double rope_theta;
} oracle_memory;

oracle_memory *oracle_create(int M, double beta, int anchor, int op, long long elems)
{
    if (M < 2 || !(beta > 0.0 && beta <= 1.0) || op < 0 || op > 3 || elems < 0) return NULL;
    oracle_memory *m = (oracle_memory *)calloc(1, sizeof(*m));
    if (!m) return NULL;
    m->M = M; m->beta = beta; m->anchor = anchor ? 1 : 0; m->op = op; m->elems = elems;
    m->e = (struct entry *)calloc((size_t)M + 1, sizeof(struct entry));
    if (!m->e) { free(m); return NULL; }
    m->last_j = -1;
    return m;
}

void oracle_destroy(oracle_memory *m)
{
    if (!m) return;
    for (int i = 0; i < m->count; ++i) { free(m->e[i].K); free(m->e[i].V); }
    free(m->e);
    free(m);
}

static double warp_u(double d, double beta) { return pow(d, beta); }   /* u(d) = d^beta */

/* Enable temporal RoPE handling for blocks laid out [tokens][H][D]
 * (tokens * H * D == elems), with `pairs` complex pairs (1 <= pairs <= D/2)
 * and base theta > 1.  Call before the first insert.  Returns 0, or -1 if
 * the arguments do not fit the memory. */
int oracle_set_rope(oracle_memory *m, int pairs, double theta, int tokens, int H, int D)
{
    if (m->t_next != 0 || pairs < 1 || 2 * pairs > D || !(theta > 1.0) || tokens < 1 || H < 1 ||
        (long long)tokens * H * D != m->elems)
        return -1;
    m->rope_pairs = pairs; m->rope_theta = theta;
    m->rope_tokens = tokens; m->rope_H = H; m->rope_D = D;
    return 0;
}

/* Rotate the temporal band of every (token, head) row of a key block by
 * position * omega_k, in place. */
static void rope_rotate(const oracle_memory *m, double *K, double position)
{
    const int P = m->rope_pairs;
    for (int k = 0; k < P; ++k) {
        const double a = position * pow(m->rope_theta, -(double)k / (double)P);
        const double c = cos(a), sn = sin(a);
        for (long long r = 0; r < (long long)m->rope_tokens * m->rope_H; ++r) {
            double *x = K + r * m->rope_D + 2 * k;
            const double x0 = x[0], x1 = x[1];
            x[0] = x0 * c - x1 * sn;
            x[1] = x0 * sn + x1 * c;
        }
    }
}

/* Keys of every entry as attention sees them: the stored (phase-free) keys
 * rotated to the re-indexed positions tau_i = t_next - count + i.  Returns a
 * malloc'd array of count * elems doubles, or NULL without RoPE (use the
 * stored keys) or on allocation failure (*failed set). */
static double *rope_attention_keys(const oracle_memory *m, int *failed)
{
    if (m->rope_pairs == 0 || m->count == 0) return NULL;
    double *K = (double *)malloc((size_t)m->count * m->elems * sizeof(double));
    if (!K) { *failed = 1; return NULL; }
    for (int i = 0; i < m->count; ++i) {
        double *Ki = K + (size_t)i * m->elems;
        memcpy(Ki, m->e[i].K, (size_t)m->elems * sizeof(double));
        rope_rotate(m, Ki, (double)(m->t_next - m->count + i));
    }
    return K;
}

/* One update of Algorithm S1.  K_t, V_t: the new unit's blocks (elems doubles
 * each; may be NULL when elems == 0, i.e. schedule-only runs).  Returns 0. */
int oracle_insert(oracle_memory *m, const double *K_t, const double *V_t)
{
    const long long t = m->t_next++;
    const size_t bytes = (size_t)m->elems * sizeof(double);

    /* Append (K_t, V_t, t, 1). */
    struct entry *nw = &m->e[m->count];
    nw->first = t; nw->span = 1; nw->mu = (double)t;
    nw->K = (double *)malloc(bytes ? bytes : 1);
    nw->V = (double *)malloc(bytes ? bytes : 1);
    if (bytes) { memcpy(nw->K, K_t, bytes); memcpy(nw->V, V_t, bytes); }
    if (bytes && m->rope_pairs) rope_rotate(m, nw->K, -(double)t);   /* store without the frame's phase */
    m->count += 1;
    m->last_j = -1; m->last_margin = INFINITY; m->last_gmin = NAN;

    /* |M_t| <= M: simply appended; it takes the next free slot. */
    if (m->count <= m->M) { nw->slot = m->count - 1; return 0; }

    /* Score every adjacent pair (i, i+1) except the pair holding the newest
     * entry, which is (count-2, count-1). */
    const int npairs = m->count - 2;
    int j = 0;
    double gmin = INFINITY, gsecond = INFINITY;
    for (int i = 0; i < npairs; ++i) {
        const double d_i = (double)t - m->e[i].mu;
        const double d_i1 = (double)t - m->e[i + 1].mu;
        const double g = fabs(warp_u(d_i1, m->beta) - warp_u(d_i, m->beta));
        if (g < gmin) { gsecond = gmin; gmin = g; j = i; }       /* strict: lowest index wins ties */
        else if (g < gsecond) { gsecond = g; }
    }
    m->last_j = j; m->last_gmin = gmin;
    m->last_margin = (npairs >= 2) ? (gsecond - gmin) / gsecond : INFINITY;

    struct entry *a = &m->e[j], *b = &m->e[j + 1];
    const long long s_j = a->span, s_j1 = b->span;
    const long long s_new = s_j + s_j1;
    double mu_new;

    if (m->anchor && j == 0) {
        /* Pair holds the first-frame anchor: keep its blocks, mu = 0. */
        mu_new = 0.0;
    } else {
        mu_new = ((double)s_j * a->mu + (double)s_j1 * b->mu) / (double)s_new;
        double w_j, w_j1;
        switch (m->op) {
        case OP_AVERAGE:        w_j = 0.5; w_j1 = 0.5; break;
        case OP_SELECT_NEAREST: w_j = 0.0; w_j1 = 1.0; break;
        default:                w_j = sqrt((double)s_j) / (sqrt((double)s_j) + sqrt((double)s_j1));
                                w_j1 = 1.0 - w_j; break;
        }
        for (long long k = 0; k < m->elems; ++k) {
            if (m->op == OP_MAX_POOL) {
                a->K[k] = fmax(a->K[k], b->K[k]);
                a->V[k] = fmax(a->V[k], b->V[k]);
            } else {
                a->K[k] = w_j * a->K[k] + w_j1 * b->K[k];
                a->V[k] = w_j * a->V[k] + w_j1 * b->V[k];
            }
        }
    }
    a->span = s_new;
    a->mu = mu_new;
    /* a->first and a->slot are kept (the result keeps m_j's slot). */

    /* Remove m_{j+1}; the newest entry takes its slot. */
    const int freed_slot = b->slot;
    free(b->K); free(b->V);
    for (int i = j + 1; i < m->count - 1; ++i) m->e[i] = m->e[i + 1];
    m->count -= 1;
    m->e[m->count - 1].slot = freed_slot;
    return 0;
}

int oracle_count(const oracle_memory *m) { return m->count; }
long long oracle_frames(const oracle_memory *m) { return m->t_next; }
int oracle_last_pair(const oracle_memory *m) { return m->last_j; }
double oracle_last_margin(const oracle_memory *m) { return m->last_margin; }
double oracle_last_gmin(const oracle_memory *m) { return m->last_gmin; }

void oracle_entries(const oracle_memory *m, int *slot, long long *first, long long *span, double *mu)
{
    for (int i = 0; i < m->count; ++i) {
        if (slot) slot[i] = m->e[i].slot;
        if (first) first[i] = m->e[i].first;
        if (span) span[i] = m->e[i].span;
        if (mu) mu[i] = m->e[i].mu;
    }
}

/* Copy entry i's K and V blocks out (elems doubles each). */
int oracle_entry_kv(const oracle_memory *m, int i, double *K, double *V)
{
    if (i < 0 || i >= m->count) return -1;
    const size_t bytes = (size_t)m->elems * sizeof(double);
    if (K) memcpy(K, m->e[i].K, bytes);
    if (V) memcpy(V, m->e[i].V, bytes);
    return 0;
}

/* Attention of Lq query tokens over every token of every entry.
 * Q, out: [Lq][H][D].  Entry blocks: [tokens][H][D] with tokens*H*D == elems.
 * For each query row and head: logits l_k = scale * <q, k_k> over all
 * count*tokens keys, p = softmax(l) (max-subtracted), out = sum_k p_k v_k. */
int oracle_attend(const oracle_memory *m, int tokens, int H, int D,
                  const double *Q, long long Lq, double scale, double *out)
{
    if ((long long)tokens * H * D != m->elems || m->count == 0) return -1;
    const long long Lk = (long long)m->count * tokens;
    int failed = 0;
    double *Krope = rope_attention_keys(m, &failed);
    if (failed) return -2;
#pragma omp parallel
    {
        double *logit = (double *)malloc((size_t)Lk * sizeof(double));
        if (!logit) {
#pragma omp atomic write
            failed = 1;
        }
#pragma omp for collapse(2) schedule(dynamic, 4)
        for (long long q = 0; q < Lq; ++q) {
            for (int h = 0; h < H; ++h) {
                if (!logit) continue;
                const double *qv = Q + ((size_t)q * H + h) * D;
                double mx = -INFINITY;
                long long k = 0;
                for (int e = 0; e < m->count; ++e) {
                    for (int n = 0; n < tokens; ++n, ++k) {
                        const double *kv = (Krope ? Krope + (size_t)e * m->elems : m->e[e].K) +
                                           ((size_t)n * H + h) * D;
                        double dot = 0.0;
                        for (int d = 0; d < D; ++d) dot += qv[d] * kv[d];
                        logit[k] = scale * dot;
                        if (logit[k] > mx) mx = logit[k];
                    }
                }
                double Z = 0.0;
                for (k = 0; k < Lk; ++k) { logit[k] = exp(logit[k] - mx); Z += logit[k]; }
                double *o = out + ((size_t)q * H + h) * D;
                for (int d = 0; d < D; ++d) o[d] = 0.0;
                k = 0;
                for (int e = 0; e < m->count; ++e) {
                    for (int n = 0; n < tokens; ++n, ++k) {
                        const double *vv = m->e[e].V + ((size_t)n * H + h) * D;
                        const double p = logit[k] / Z;
                        for (int d = 0; d < D; ++d) o[d] += p * vv[d];
                    }
                }
            }
        }
        free(logit);
    }
    free(Krope);
    return failed ? -2 : 0;
}

int oracle_num_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* Attention over the memory plus the current chunk's own keys and values (the
 * paper's attention sees the cached entries and the frames of the chunk being
 * generated, Sec. 4.1 / Sec. S4): the key set is every token of every entry,
 * followed by the ncur tokens of Kcur/Vcur ([ncur][H][D]).  With ncur = 0 this
 * is oracle_attend; with an empty memory it is attention over the chunk alone. */
int oracle_attend_ext(const oracle_memory *m, int tokens, int H, int D, const double *Kcur, const double *Vcur,
                      long long ncur, const double *Q, long long Lq, double scale, double *out)
{
    if ((long long)tokens * H * D != m->elems || (m->count == 0 && ncur == 0) || ncur < 0) return -1;
    const long long Lmem = (long long)m->count * tokens;
    const long long Lk = Lmem + ncur;
    int failed = 0;
    double *Krope = rope_attention_keys(m, &failed);
    if (failed) return -2;
#pragma omp parallel
    {
        double *logit = (double *)malloc((size_t)Lk * sizeof(double));
        if (!logit) {
#pragma omp atomic write
            failed = 1;
        }
#pragma omp for collapse(2) schedule(dynamic, 4)
        for (long long q = 0; q < Lq; ++q) {
            for (int h = 0; h < H; ++h) {
                if (!logit) continue;
                const double *qv = Q + ((size_t)q * H + h) * D;
                double mx = -INFINITY;
                for (long long k = 0; k < Lk; ++k) {
                    const double *kv;
                    if (k < Lmem)
                        kv = (Krope ? Krope + (size_t)(k / tokens) * m->elems : m->e[k / tokens].K) +
                             ((size_t)(k % tokens) * H + h) * D;
                    else
                        kv = Kcur + ((size_t)(k - Lmem) * H + h) * D;
                    double dot = 0.0;
                    for (int d = 0; d < D; ++d) dot += qv[d] * kv[d];
                    logit[k] = scale * dot;
                    if (logit[k] > mx) mx = logit[k];
                }
                double Z = 0.0;
                for (long long k = 0; k < Lk; ++k) { logit[k] = exp(logit[k] - mx); Z += logit[k]; }
                double *o = out + ((size_t)q * H + h) * D;
                for (int d = 0; d < D; ++d) o[d] = 0.0;
                for (long long k = 0; k < Lk; ++k) {
                    const double *vv = k < Lmem ? m->e[k / tokens].V + ((size_t)(k % tokens) * H + h) * D
                                                : Vcur + ((size_t)(k - Lmem) * H + h) * D;
                    const double p = logit[k] / Z;
                    for (int d = 0; d < D; ++d) o[d] += p * vv[d];
                }
            }
        }
        free(logit);
    }
    free(Krope);
    return failed ? -2 : 0;
}
