/*
 * mk_oracle.c -- plain fp64 CPU oracle for the attention forward pass, its
 * backward pass (gradients of q, k, v), one paged decode step and one latent
 * (MLA) decode step.
 *
 * TEST INFRASTRUCTURE.  Only tests/, __graft_entry__.smoke() and bench.py's
 * cpu_baseline / reference legs may load this file's library.  The product
 * path (the CUDA library and its Python binding) never calls it and shares
 * no code with it.
 *
 * What it computes.  The paper's problem statement (Section 2.1, the Testing
 * and Verification Agents; Section 3.1, correctness against the unoptimized
 * reference implementation) fixes the contract: a kernel takes the same input
 * arrays as the reference operation and must return the same outputs.  The
 * reference operation for the Flash Attention and GQA Attention rows of
 * Table 2 is the plain definition of scaled dot-product attention, which this
 * file writes out directly, with no tiling, no online softmax and no
 * reordering:
 *
 *   for each sequence b, query head h (key/value head g = h / (Hq / Hkv)),
 *   and query position i of that sequence:
 *     K_i  = { j : 0 <= j < L_b  and  (not causal  or  j <= i) }
 *     s_j  = scale * sum_d q[b,i,h,d] * k[b,j,g,d]          (j in K_i)
 *     m    = max_j s_j
 *     l    = sum_j exp(s_j - m)
 *     o[d] = sum_j exp(s_j - m) * v[b,j,g,d] / l
 *     lse  = m + ln(l)                                        (natural log)
 *
 * Subtracting m is the textbook overflow guard; it cancels exactly in o and
 * is added back in lse, so the result is the definition itself.
 *
 * Inputs are bf16 bit patterns (uint16); they are widened exactly to fp64.
 * All arithmetic is fp64.  Layouts:
 *   fixed length (cu_seqlens == NULL): q/o [B,S,Hq,D], k/v [B,S,Hkv,D],
 *                                      lse [B,Hq,S]
 *   packed varlen (cu_seqlens != NULL): q/o [T,Hq,D], k/v [T,Hkv,D],
 *                                      lse [Hq,T], T = S = cu_seqlens[B]
 * Readings where the paper is silent: contiguous query-head groups
 * (g = h / (Hq/Hkv)); causal alignment with Sq == Sk, so row i sees keys
 * 0..i; the log-sum-exp includes the scale and uses the natural log.
 * A row with no visible key (cannot happen for valid inputs) gets o = 0,
 * lse = -inf.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define MK_ORACLE_OK 0
#define MK_ORACLE_BAD_ARG (-1)
#define MK_ORACLE_NO_MEM (-2)

static double bf16_bits_to_f64(uint16_t bits)
{
    uint32_t u = ((uint32_t)bits) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

typedef struct {
    const uint16_t *q, *k, *v;
    int B, Hq, Hkv, S, D, causal;
    double scale;
    const int32_t *cu;
} problem_t;

/* Token offset and length of sequence b. */
static void seq_bounds(const problem_t *p, int b, int64_t *tok0, int *len)
{
    if (p->cu) {
        *tok0 = p->cu[b];
        *len = p->cu[b + 1] - p->cu[b];
    } else {
        *tok0 = (int64_t)b * p->S;
        *len = p->S;
    }
}

/* One output row: the definition above for (sequence b, head h, position i).
 * s_buf must hold at least L_b doubles. */
static void attention_row(const problem_t *p, int b, int h, int i, double *s_buf,
                          double *o_row, double *lse_out)
{
    const int D = p->D;
    const int group = p->Hq / p->Hkv;
    const int g = h / group;
    int64_t tok0;
    int L;
    seq_bounds(p, b, &tok0, &L);

    const uint16_t *qi = p->q + ((tok0 + i) * p->Hq + h) * (int64_t)D;
    int n_keys = p->causal ? (i + 1 < L ? i + 1 : L) : L; /* |K_i| */

    double m = -INFINITY;
    for (int j = 0; j < n_keys; ++j) {
        const uint16_t *kj = p->k + ((tok0 + j) * p->Hkv + g) * (int64_t)D;
        double dot = 0.0;
        for (int d = 0; d < D; ++d)
            dot += bf16_bits_to_f64(qi[d]) * bf16_bits_to_f64(kj[d]);
        double s = p->scale * dot;
        s_buf[j] = s;
        if (s > m)
            m = s;
    }

    for (int d = 0; d < D; ++d)
        o_row[d] = 0.0;
    if (n_keys == 0) {
        *lse_out = -INFINITY;
        return;
    }

    double l = 0.0;
    for (int j = 0; j < n_keys; ++j) {
        const uint16_t *vj = p->v + ((tok0 + j) * p->Hkv + g) * (int64_t)D;
        double w = exp(s_buf[j] - m);
        l += w;
        for (int d = 0; d < D; ++d)
            o_row[d] += w * bf16_bits_to_f64(vj[d]);
    }
    for (int d = 0; d < D; ++d)
        o_row[d] /= l;
    *lse_out = m + log(l);
}

static int check_problem(const problem_t *p)
{
    if (!p->q || !p->k || !p->v)
        return MK_ORACLE_BAD_ARG;
    if (p->B < 1 || p->Hq < 1 || p->Hkv < 1 || p->S < 0 || p->D < 1)
        return MK_ORACLE_BAD_ARG;
    if (p->Hq % p->Hkv != 0)
        return MK_ORACLE_BAD_ARG;
    if (p->cu) {
        if (p->cu[0] != 0 || p->cu[p->B] != p->S)
            return MK_ORACLE_BAD_ARG;
        for (int b = 0; b < p->B; ++b)
            if (p->cu[b + 1] < p->cu[b])
                return MK_ORACLE_BAD_ARG;
    }
    return MK_ORACLE_OK;
}

static int max_seq_len(const problem_t *p)
{
    int mx = 0;
    for (int b = 0; b < p->B; ++b) {
        int64_t t0;
        int L;
        seq_bounds(p, b, &t0, &L);
        if (L > mx)
            mx = L;
    }
    return mx;
}

/* ---------------------------------------------------------------- full pass */

typedef struct {
    const problem_t *p;
    double *o, *lse;
    int64_t n_tasks;   /* (b, h) pairs */
    int64_t *next;     /* shared task counter */
    int max_len;
    int status;
} full_job_t;

static void *full_worker(void *arg)
{
    full_job_t *job = (full_job_t *)arg;
    const problem_t *p = job->p;
    double *s_buf = (double *)malloc(sizeof(double) * (size_t)(job->max_len > 0 ? job->max_len : 1));
    if (!s_buf) {
        job->status = MK_ORACLE_NO_MEM;
        return NULL;
    }
    for (;;) {
        int64_t t = __atomic_fetch_add(job->next, 1, __ATOMIC_RELAXED);
        if (t >= job->n_tasks)
            break;
        int b = (int)(t / p->Hq), h = (int)(t % p->Hq);
        int64_t tok0;
        int L;
        seq_bounds(p, b, &tok0, &L);
        for (int i = 0; i < L; ++i) {
            double *o_row = job->o + ((tok0 + i) * p->Hq + h) * (int64_t)p->D;
            int64_t lse_idx = p->cu ? (int64_t)h * p->S + tok0 + i
                                    : ((int64_t)b * p->Hq + h) * p->S + i;
            attention_row(p, b, h, i, s_buf, o_row, &job->lse[lse_idx]);
        }
    }
    free(s_buf);
    return NULL;
}

/* Runs `worker` on n_threads threads, each given its own copy of *job
 * (the copies share the task counter). */
static int run_threads(void *(*worker)(void *), void *job, size_t job_size, int n_threads)
{
    if (n_threads < 1)
        n_threads = 1;
    pthread_t *tids = (pthread_t *)calloc((size_t)n_threads, sizeof(pthread_t));
    char *jobs = (char *)malloc(job_size * (size_t)n_threads);
    if (!tids || !jobs) {
        free(tids);
        free(jobs);
        return MK_ORACLE_NO_MEM;
    }
    int started = 0;
    for (int t = 0; t < n_threads; ++t) {
        memcpy(jobs + job_size * t, job, job_size);
        if (pthread_create(&tids[t], NULL, worker, jobs + job_size * t) != 0)
            break;
        ++started;
    }
    if (started == 0) /* no thread could start: do the work here */
        worker(jobs);
    for (int t = 0; t < started; ++t)
        pthread_join(tids[t], NULL);
    free(tids);
    free(jobs);
    return MK_ORACLE_OK;
}

/*
 * Full forward pass.  o has the layout of q; lse as described above.
 * Returns 0, or a negative code for invalid arguments / allocation failure.
 */
int mk_oracle_attn_fwd_f64(const uint16_t *q, const uint16_t *k, const uint16_t *v,
                           double *o, double *lse, int B, int Hq, int Hkv, int S, int D,
                           int causal, double scale, const int32_t *cu_seqlens,
                           int n_threads)
{
    problem_t p = {q, k, v, B, Hq, Hkv, S, D, causal != 0, scale, cu_seqlens};
    int st = check_problem(&p);
    if (st != MK_ORACLE_OK)
        return st;
    if (!o || !lse)
        return MK_ORACLE_BAD_ARG;
    int64_t next = 0;
    full_job_t job = {&p, o, lse, (int64_t)B * Hq, &next, max_seq_len(&p), MK_ORACLE_OK};
    st = run_threads(full_worker, &job, sizeof job, n_threads);
    return st;
}

/* ------------------------------------------------------------ sampled rows */

typedef struct {
    const problem_t *p;
    const int64_t *rows; /* n_rows x 3: (b, h, i) */
    double *o_rows;      /* n_rows x D */
    double *lse_rows;    /* n_rows */
    int64_t n_rows;
    int64_t *next;
    int max_len;
} rows_job_t;

static void *rows_worker(void *arg)
{
    rows_job_t *job = (rows_job_t *)arg;
    const problem_t *p = job->p;
    double *s_buf = (double *)malloc(sizeof(double) * (size_t)(job->max_len > 0 ? job->max_len : 1));
    if (!s_buf)
        return NULL;
    for (;;) {
        int64_t r = __atomic_fetch_add(job->next, 1, __ATOMIC_RELAXED);
        if (r >= job->n_rows)
            break;
        int b = (int)job->rows[3 * r], h = (int)job->rows[3 * r + 1], i = (int)job->rows[3 * r + 2];
        attention_row(p, b, h, i, s_buf, job->o_rows + r * (int64_t)p->D, &job->lse_rows[r]);
    }
    free(s_buf);
    return NULL;
}

/*
 * The same definition evaluated only on selected rows (b, h, i), for inputs
 * too large to evaluate in full.  Each row is independent of the others, so a
 * sampled row equals the corresponding row of mk_oracle_attn_fwd_f64.
 */
int mk_oracle_attn_rows_f64(const uint16_t *q, const uint16_t *k, const uint16_t *v,
                            int B, int Hq, int Hkv, int S, int D, int causal, double scale,
                            const int32_t *cu_seqlens, const int64_t *rows, int64_t n_rows,
                            double *o_rows, double *lse_rows, int n_threads)
{
    problem_t p = {q, k, v, B, Hq, Hkv, S, D, causal != 0, scale, cu_seqlens};
    int st = check_problem(&p);
    if (st != MK_ORACLE_OK)
        return st;
    if (n_rows < 0 || (n_rows > 0 && (!rows || !o_rows || !lse_rows)))
        return MK_ORACLE_BAD_ARG;
    for (int64_t r = 0; r < n_rows; ++r) {
        int b = (int)rows[3 * r], h = (int)rows[3 * r + 1], i = (int)rows[3 * r + 2];
        if (b < 0 || b >= B || h < 0 || h >= Hq || i < 0)
            return MK_ORACLE_BAD_ARG;
        int64_t t0;
        int L;
        seq_bounds(&p, b, &t0, &L);
        if (i >= L)
            return MK_ORACLE_BAD_ARG;
    }
    int64_t next = 0;
    rows_job_t job = {&p, rows, o_rows, lse_rows, n_rows, &next, max_seq_len(&p)};
    return run_threads(rows_worker, &job, sizeof job, n_threads);
}

/* ------------------------------------------------------ paged decode step */

/*
 * One decode step against a paged key/value cache: for each sequence b, its
 * newest query q[b,h,:] attends to the L_b = seq_lens[b] cached positions
 * 0..L_b-1 of that sequence (all of them: the new token is the last
 * position, so no causal mask applies).  Position j lives in physical page
 * page_table[b * max_pages + j / page_size], slot j % page_size:
 *
 *   k_j  = k_cache[page, slot, g, :],  v_j = v_cache[page, slot, g, :]
 *   s_j  = scale * sum_d q[b,h,d] * k_j[d]          (g = h / (Hq / Hkv))
 *   o[d] = sum_j exp(s_j - m) v_j[d] / sum_j exp(s_j - m),  m = max_j s_j
 *   lse  = m + ln(sum_j exp(s_j - m))
 *
 * This is the attention definition above, for a single query row whose key
 * set is gathered through a page table (the Paged Attention row of Table 2).
 * Layouts: q, o [B, Hq, D]; k_cache, v_cache [num_pages, page_size, Hkv, D];
 * page_table int32 [B, max_pages]; seq_lens int32 [B]; lse [B, Hq].
 * L_b = 0 gives o = 0 and lse = -inf.  Returns MK_ORACLE_BAD_ARG for sizes
 * out of range, a length above max_pages * page_size, or a page index
 * outside [0, num_pages).
 */
typedef struct {
    const uint16_t *q, *kc, *vc;
    const int32_t *page_table, *seq_lens;
    double *o, *lse;
    int B, Hq, Hkv, D, page_size, max_pages;
    double scale;
    int64_t *next;
    int max_len;
} decode_job_t;

static void *decode_worker(void *arg)
{
    decode_job_t *job = (decode_job_t *)arg;
    const int G = job->Hq / job->Hkv, D = job->D;
    double *s_buf = (double *)malloc(sizeof(double) * (size_t)(job->max_len > 0 ? job->max_len : 1));
    if (!s_buf)
        return NULL;
    for (;;) {
        int64_t t = __atomic_fetch_add(job->next, 1, __ATOMIC_RELAXED);
        if (t >= (int64_t)job->B * job->Hq)
            break;
        const int b = (int)(t / job->Hq), h = (int)(t % job->Hq), g = h / G;
        const int L = job->seq_lens[b];
        const uint16_t *qr = job->q + ((int64_t)b * job->Hq + h) * D;
        double *orow = job->o + ((int64_t)b * job->Hq + h) * D;
        for (int d = 0; d < D; ++d)
            orow[d] = 0.0;
        if (L == 0) {
            job->lse[t] = -INFINITY;
            continue;
        }
        double m = -INFINITY;
        for (int j = 0; j < L; ++j) {
            const int64_t page = job->page_table[(int64_t)b * job->max_pages + j / job->page_size];
            const int64_t row = (page * job->page_size + j % job->page_size) * job->Hkv + g;
            const uint16_t *kr = job->kc + row * D;
            double acc = 0.0;
            for (int d = 0; d < D; ++d)
                acc += bf16_bits_to_f64(qr[d]) * bf16_bits_to_f64(kr[d]);
            s_buf[j] = job->scale * acc;
            if (s_buf[j] > m)
                m = s_buf[j];
        }
        double l = 0.0;
        for (int j = 0; j < L; ++j) {
            const double e = exp(s_buf[j] - m);
            l += e;
            const int64_t page = job->page_table[(int64_t)b * job->max_pages + j / job->page_size];
            const int64_t row = (page * job->page_size + j % job->page_size) * job->Hkv + g;
            const uint16_t *vr = job->vc + row * D;
            for (int d = 0; d < D; ++d)
                orow[d] += e * bf16_bits_to_f64(vr[d]);
        }
        for (int d = 0; d < D; ++d)
            orow[d] /= l;
        job->lse[t] = m + log(l);
    }
    free(s_buf);
    return NULL;
}

int mk_oracle_decode_paged_f64(const uint16_t *q, const uint16_t *k_cache,
                               const uint16_t *v_cache, const int32_t *page_table,
                               const int32_t *seq_lens, double *o, double *lse, int B, int Hq,
                               int Hkv, int D, int page_size, int max_pages, int num_pages,
                               double scale, int n_threads)
{
    if (!q || !k_cache || !v_cache || !page_table || !seq_lens || !o || !lse)
        return MK_ORACLE_BAD_ARG;
    if (B < 1 || Hq < 1 || Hkv < 1 || Hq % Hkv != 0 || D < 1 || page_size < 1 ||
        max_pages < 1 || num_pages < 1)
        return MK_ORACLE_BAD_ARG;
    int max_len = 0;
    for (int b = 0; b < B; ++b) {
        const int L = seq_lens[b];
        if (L < 0 || (int64_t)L > (int64_t)max_pages * page_size)
            return MK_ORACLE_BAD_ARG;
        for (int j = 0; j * page_size < L; ++j) {
            const int32_t pg = page_table[(int64_t)b * max_pages + j];
            if (pg < 0 || pg >= num_pages)
                return MK_ORACLE_BAD_ARG;
        }
        if (L > max_len)
            max_len = L;
    }
    int64_t next = 0;
    decode_job_t job = {q, k_cache, v_cache, page_table, seq_lens, o, lse, B, Hq, Hkv, D,
                        page_size, max_pages, scale, &next, max_len};
    return run_threads(decode_worker, &job, sizeof job, n_threads);
}

/* ------------------------------------------------------------ backward pass */

/*
 * Gradients of the forward definition with respect to q, k and v, given dO,
 * the gradient of a loss with respect to o (the training step's backward
 * pass of the same reference operation).  Reverse-mode chain rule through
 * the definition, written out for every sequence b, key/value head g, query
 * head h of g's group and query position i:
 *
 *   P_ij    = exp(s_ij - lse_i)                       j in K_i (0 elsewhere)
 *   dP_ij   = sum_d dO[i,h,d] * v[j,g,d]              (dL/dP_ij, since o_i = sum_j P_ij v_j)
 *   Delta_i = sum_{j in K_i} P_ij * dP_ij
 *   dS_ij   = P_ij * (dP_ij - Delta_i)                (dL/ds_ij through the softmax)
 *   dq[i,h] = scale * sum_{j in K_i} dS_ij * k[j,g]   (s_ij = scale * q_i . k_j)
 *   dk[j,g] = scale * sum_{h in group g} sum_{i : j in K_i} dS_ij * q[i,h]
 *   dv[j,g] =         sum_{h in group g} sum_{i : j in K_i} P_ij * dO[i,h]
 *
 * s_ij and lse_i are recomputed here in fp64 from the bf16 inputs (the
 * forward definition above), and Delta_i is the sum over P_ij dP_ij itself,
 * not a product with a rounded o.  dq has the layout of q, dk and dv that of
 * k and v; dO that of q.  A key that no query sees gets dk = dv = 0.
 */
typedef struct {
    const problem_t *p;
    const uint16_t *dO;
    double *dq, *dk, *dv;
    int64_t n_tasks; /* (b, g) pairs */
    int64_t *next;
    int max_len;
} bwd_job_t;

/* Row statistics of (b, h, i): s_buf[j] = s_ij for j < n_keys, returns lse_i
 * (-inf for an empty row). */
static double row_scores(const problem_t *p, int64_t tok0, int g, int h, int i, int n_keys,
                         double *s_buf)
{
    const int D = p->D;
    const uint16_t *qi = p->q + ((tok0 + i) * p->Hq + h) * (int64_t)D;
    double m = -INFINITY;
    for (int j = 0; j < n_keys; ++j) {
        const uint16_t *kj = p->k + ((tok0 + j) * p->Hkv + g) * (int64_t)D;
        double dot = 0.0;
        for (int d = 0; d < D; ++d)
            dot += bf16_bits_to_f64(qi[d]) * bf16_bits_to_f64(kj[d]);
        s_buf[j] = p->scale * dot;
        if (s_buf[j] > m)
            m = s_buf[j];
    }
    if (n_keys == 0)
        return -INFINITY;
    double l = 0.0;
    for (int j = 0; j < n_keys; ++j)
        l += exp(s_buf[j] - m);
    return m + log(l);
}

/* P_ij into s_buf and dP_ij into dp_buf for j < n_keys; returns Delta_i. */
static double row_probs(const problem_t *p, const uint16_t *dO, int64_t tok0, int g, int h,
                        int i, int n_keys, double *s_buf, double *dp_buf)
{
    const int D = p->D;
    const double lse = row_scores(p, tok0, g, h, i, n_keys, s_buf);
    const uint16_t *doi = dO + ((tok0 + i) * p->Hq + h) * (int64_t)D;
    double delta = 0.0;
    for (int j = 0; j < n_keys; ++j) {
        const uint16_t *vj = p->v + ((tok0 + j) * p->Hkv + g) * (int64_t)D;
        double dp = 0.0;
        for (int d = 0; d < D; ++d)
            dp += bf16_bits_to_f64(doi[d]) * bf16_bits_to_f64(vj[d]);
        s_buf[j] = exp(s_buf[j] - lse);
        dp_buf[j] = dp;
        delta += s_buf[j] * dp;
    }
    return delta;
}

static int keys_of_row(const problem_t *p, int i, int L)
{
    return p->causal ? (i + 1 < L ? i + 1 : L) : L; /* |K_i| */
}

static void *bwd_worker(void *arg)
{
    bwd_job_t *job = (bwd_job_t *)arg;
    const problem_t *p = job->p;
    const int D = p->D, group = p->Hq / p->Hkv;
    const size_t n = (size_t)(job->max_len > 0 ? job->max_len : 1);
    double *s_buf = (double *)malloc(sizeof(double) * n);
    double *dp_buf = (double *)malloc(sizeof(double) * n);
    if (!s_buf || !dp_buf) {
        free(s_buf);
        free(dp_buf);
        return NULL;
    }
    for (;;) {
        int64_t t = __atomic_fetch_add(job->next, 1, __ATOMIC_RELAXED);
        if (t >= job->n_tasks)
            break;
        const int b = (int)(t / p->Hkv), g = (int)(t % p->Hkv);
        int64_t tok0;
        int L;
        seq_bounds(p, b, &tok0, &L);
        for (int j = 0; j < L; ++j)
            for (int d = 0; d < D; ++d) {
                job->dk[((tok0 + j) * p->Hkv + g) * (int64_t)D + d] = 0.0;
                job->dv[((tok0 + j) * p->Hkv + g) * (int64_t)D + d] = 0.0;
            }
        for (int h = g * group; h < (g + 1) * group; ++h) {
            for (int i = 0; i < L; ++i) {
                const int n_keys = keys_of_row(p, i, L);
                double *dqi = job->dq + ((tok0 + i) * p->Hq + h) * (int64_t)D;
                for (int d = 0; d < D; ++d)
                    dqi[d] = 0.0;
                if (n_keys == 0)
                    continue;
                const double delta = row_probs(p, job->dO, tok0, g, h, i, n_keys, s_buf, dp_buf);
                const uint16_t *qi = p->q + ((tok0 + i) * p->Hq + h) * (int64_t)D;
                const uint16_t *doi = job->dO + ((tok0 + i) * p->Hq + h) * (int64_t)D;
                for (int j = 0; j < n_keys; ++j) {
                    const double P = s_buf[j];
                    const double dS = P * (dp_buf[j] - delta);
                    const uint16_t *kj = p->k + ((tok0 + j) * p->Hkv + g) * (int64_t)D;
                    double *dkj = job->dk + ((tok0 + j) * p->Hkv + g) * (int64_t)D;
                    double *dvj = job->dv + ((tok0 + j) * p->Hkv + g) * (int64_t)D;
                    for (int d = 0; d < D; ++d) {
                        dqi[d] += p->scale * dS * bf16_bits_to_f64(kj[d]);
                        dkj[d] += p->scale * dS * bf16_bits_to_f64(qi[d]);
                        dvj[d] += P * bf16_bits_to_f64(doi[d]);
                    }
                }
            }
        }
    }
    free(s_buf);
    free(dp_buf);
    return NULL;
}

/*
 * Full backward pass.  Tasks are (sequence, key/value head) pairs: one thread
 * owns the dk, dv rows of its head and the dq rows of the head's query group,
 * so no two threads write the same element.
 */
int mk_oracle_attn_bwd_f64(const uint16_t *q, const uint16_t *k, const uint16_t *v,
                           const uint16_t *dO, double *dq, double *dk, double *dv, int B,
                           int Hq, int Hkv, int S, int D, int causal, double scale,
                           const int32_t *cu_seqlens, int n_threads)
{
    problem_t p = {q, k, v, B, Hq, Hkv, S, D, causal != 0, scale, cu_seqlens};
    int st = check_problem(&p);
    if (st != MK_ORACLE_OK)
        return st;
    if (!dO || !dq || !dk || !dv)
        return MK_ORACLE_BAD_ARG;
    int64_t next = 0;
    bwd_job_t job = {&p, dO, dq, dk, dv, (int64_t)B * Hkv, &next, max_seq_len(&p)};
    return run_threads(bwd_worker, &job, sizeof job, n_threads);
}

/* ---------------------------------------------------- sampled backward parts */

typedef struct {
    const problem_t *p;
    const uint16_t *dO;
    const int64_t *items; /* dq rows: (b, h, i); dk/dv ranges: (b, g, j0, j1) */
    double *out0, *out1;  /* dq rows; or dk, dv rows of the ranges, in order */
    const int64_t *out_off; /* ranges: first output row of each range */
    int64_t n_items;
    int64_t *next;
    int max_len;
} bwd_sample_job_t;

static void *dq_rows_worker(void *arg)
{
    bwd_sample_job_t *job = (bwd_sample_job_t *)arg;
    const problem_t *p = job->p;
    const int D = p->D, group = p->Hq / p->Hkv;
    const size_t n = (size_t)(job->max_len > 0 ? job->max_len : 1);
    double *s_buf = (double *)malloc(sizeof(double) * n);
    double *dp_buf = (double *)malloc(sizeof(double) * n);
    if (!s_buf || !dp_buf) {
        free(s_buf);
        free(dp_buf);
        return NULL;
    }
    for (;;) {
        int64_t r = __atomic_fetch_add(job->next, 1, __ATOMIC_RELAXED);
        if (r >= job->n_items)
            break;
        const int b = (int)job->items[3 * r], h = (int)job->items[3 * r + 1];
        const int i = (int)job->items[3 * r + 2], g = h / group;
        int64_t tok0;
        int L;
        seq_bounds(p, b, &tok0, &L);
        const int n_keys = keys_of_row(p, i, L);
        double *dqi = job->out0 + r * (int64_t)D;
        for (int d = 0; d < D; ++d)
            dqi[d] = 0.0;
        if (n_keys == 0)
            continue;
        const double delta = row_probs(p, job->dO, tok0, g, h, i, n_keys, s_buf, dp_buf);
        for (int j = 0; j < n_keys; ++j) {
            const double dS = s_buf[j] * (dp_buf[j] - delta);
            const uint16_t *kj = p->k + ((tok0 + j) * p->Hkv + g) * (int64_t)D;
            for (int d = 0; d < D; ++d)
                dqi[d] += p->scale * dS * bf16_bits_to_f64(kj[d]);
        }
    }
    free(s_buf);
    free(dp_buf);
    return NULL;
}

/*
 * dq on selected rows (b, h, i) only.  dq of a row depends on that row's
 * scores alone, so a sampled row equals the row of mk_oracle_attn_bwd_f64.
 */
int mk_oracle_attn_bwd_dq_rows_f64(const uint16_t *q, const uint16_t *k, const uint16_t *v,
                                   const uint16_t *dO, int B, int Hq, int Hkv, int S, int D,
                                   int causal, double scale, const int32_t *cu_seqlens,
                                   const int64_t *rows, int64_t n_rows, double *dq_rows,
                                   int n_threads)
{
    problem_t p = {q, k, v, B, Hq, Hkv, S, D, causal != 0, scale, cu_seqlens};
    int st = check_problem(&p);
    if (st != MK_ORACLE_OK)
        return st;
    if (!dO || n_rows < 0 || (n_rows > 0 && (!rows || !dq_rows)))
        return MK_ORACLE_BAD_ARG;
    for (int64_t r = 0; r < n_rows; ++r) {
        int b = (int)rows[3 * r], h = (int)rows[3 * r + 1], i = (int)rows[3 * r + 2];
        if (b < 0 || b >= B || h < 0 || h >= Hq || i < 0)
            return MK_ORACLE_BAD_ARG;
        int64_t t0;
        int L;
        seq_bounds(&p, b, &t0, &L);
        if (i >= L)
            return MK_ORACLE_BAD_ARG;
    }
    int64_t next = 0;
    bwd_sample_job_t job = {&p, dO, rows, dq_rows, NULL, NULL, n_rows, &next, max_seq_len(&p)};
    return run_threads(dq_rows_worker, &job, sizeof job, n_threads);
}

static void *dkv_range_worker(void *arg)
{
    bwd_sample_job_t *job = (bwd_sample_job_t *)arg;
    const problem_t *p = job->p;
    const int D = p->D, group = p->Hq / p->Hkv;
    const size_t n = (size_t)(job->max_len > 0 ? job->max_len : 1);
    double *s_buf = (double *)malloc(sizeof(double) * n);
    double *dp_buf = (double *)malloc(sizeof(double) * n);
    if (!s_buf || !dp_buf) {
        free(s_buf);
        free(dp_buf);
        return NULL;
    }
    for (;;) {
        int64_t r = __atomic_fetch_add(job->next, 1, __ATOMIC_RELAXED);
        if (r >= job->n_items)
            break;
        const int b = (int)job->items[4 * r], g = (int)job->items[4 * r + 1];
        const int j0 = (int)job->items[4 * r + 2], j1 = (int)job->items[4 * r + 3];
        int64_t tok0;
        int L;
        seq_bounds(p, b, &tok0, &L);
        double *dk = job->out0 + job->out_off[r] * (int64_t)D;
        double *dv = job->out1 + job->out_off[r] * (int64_t)D;
        for (int64_t e = 0; e < (int64_t)(j1 - j0) * D; ++e)
            dk[e] = dv[e] = 0.0;
        /* Every query row that sees a key of [j0, j1): all rows, or rows
         * i >= j0 when causal. */
        for (int h = g * group; h < (g + 1) * group; ++h) {
            for (int i = p->causal ? j0 : 0; i < L; ++i) {
                const int n_keys = keys_of_row(p, i, L);
                if (n_keys <= j0)
                    continue;
                const double delta = row_probs(p, job->dO, tok0, g, h, i, n_keys, s_buf, dp_buf);
                const uint16_t *qi = p->q + ((tok0 + i) * p->Hq + h) * (int64_t)D;
                const uint16_t *doi = job->dO + ((tok0 + i) * p->Hq + h) * (int64_t)D;
                for (int j = j0; j < j1 && j < n_keys; ++j) {
                    const double P = s_buf[j];
                    const double dS = P * (dp_buf[j] - delta);
                    for (int d = 0; d < D; ++d) {
                        dk[(int64_t)(j - j0) * D + d] += p->scale * dS * bf16_bits_to_f64(qi[d]);
                        dv[(int64_t)(j - j0) * D + d] += P * bf16_bits_to_f64(doi[d]);
                    }
                }
            }
        }
    }
    free(s_buf);
    free(dp_buf);
    return NULL;
}

/*
 * dk and dv for key ranges [j0, j1) of (sequence b, key/value head g), given
 * as n_ranges x 4 int64 (b, g, j0, j1); the ranges' rows are written one
 * after the other into dk_rows and dv_rows (sum of (j1 - j0) rows of D).
 * Each range visits every query row that sees one of its keys, so it equals
 * the same rows of mk_oracle_attn_bwd_f64.
 */
int mk_oracle_attn_bwd_dkv_ranges_f64(const uint16_t *q, const uint16_t *k, const uint16_t *v,
                                      const uint16_t *dO, int B, int Hq, int Hkv, int S, int D,
                                      int causal, double scale, const int32_t *cu_seqlens,
                                      const int64_t *ranges, int64_t n_ranges, double *dk_rows,
                                      double *dv_rows, int n_threads)
{
    problem_t p = {q, k, v, B, Hq, Hkv, S, D, causal != 0, scale, cu_seqlens};
    int st = check_problem(&p);
    if (st != MK_ORACLE_OK)
        return st;
    if (!dO || n_ranges < 0 || (n_ranges > 0 && (!ranges || !dk_rows || !dv_rows)))
        return MK_ORACLE_BAD_ARG;
    int64_t *off = (int64_t *)malloc(sizeof(int64_t) * (size_t)(n_ranges > 0 ? n_ranges : 1));
    if (!off)
        return MK_ORACLE_NO_MEM;
    int64_t rows = 0;
    for (int64_t r = 0; r < n_ranges; ++r) {
        const int64_t b = ranges[4 * r], g = ranges[4 * r + 1];
        const int64_t j0 = ranges[4 * r + 2], j1 = ranges[4 * r + 3];
        int64_t t0;
        int L = 0;
        if (b >= 0 && b < B)
            seq_bounds(&p, (int)b, &t0, &L);
        if (b < 0 || b >= B || g < 0 || g >= Hkv || j0 < 0 || j1 < j0 || j1 > L) {
            free(off);
            return MK_ORACLE_BAD_ARG;
        }
        off[r] = rows;
        rows += j1 - j0;
    }
    int64_t next = 0;
    bwd_sample_job_t job = {&p, dO, ranges, dk_rows, dv_rows, off, n_ranges, &next, max_seq_len(&p)};
    st = run_threads(dkv_range_worker, &job, sizeof job, n_threads);
    free(off);
    return st;
}

/* ------------------------------------------------- latent (MLA) decode step */

/*
 * One decode step of multi-head latent attention in its absorbed form: every
 * query head attends to one shared latent cache (a single key/value head),
 * whose rows serve as keys in full and as values through their first Dv
 * components (the paper's MLA Attention row, Table 2 and Table 3).  For
 * sequence b and query head h, with c_j the cached latent row of position j
 * (slot j % page_size of page page_table[b, j / page_size]):
 *
 *   s_j  = scale * sum_{d < Dqk} q[b,h,d] * c_j[d]
 *   o[d] = sum_j exp(s_j - m) c_j[d] / sum_j exp(s_j - m),  d < Dv,  m = max_j s_j
 *   lse  = m + ln(sum_j exp(s_j - m))
 *
 * Layouts: q [B, Hq, Dqk]; cache [num_pages, page_size, Dqk]; o [B, Hq, Dv];
 * lse [B, Hq]; page_table int32 [B, max_pages]; seq_lens int32 [B].
 * L_b = 0 gives o = 0 and lse = -inf.  Returns MK_ORACLE_BAD_ARG for sizes out
 * of range (Dv > Dqk included), a length above max_pages * page_size, or a
 * page index outside [0, num_pages).
 */
typedef struct {
    const uint16_t *q, *cache;
    const int32_t *page_table, *seq_lens;
    double *o, *lse;
    int B, Hq, Dqk, Dv, page_size, max_pages;
    double scale;
    int64_t *next;
    int max_len;
} mla_job_t;

static const uint16_t *mla_row(const mla_job_t *job, int b, int j)
{
    const int64_t page = job->page_table[(int64_t)b * job->max_pages + j / job->page_size];
    return job->cache + (page * job->page_size + j % job->page_size) * (int64_t)job->Dqk;
}

static void *mla_worker(void *arg)
{
    mla_job_t *job = (mla_job_t *)arg;
    double *s_buf = (double *)malloc(sizeof(double) * (size_t)(job->max_len > 0 ? job->max_len : 1));
    if (!s_buf)
        return NULL;
    for (;;) {
        int64_t t = __atomic_fetch_add(job->next, 1, __ATOMIC_RELAXED);
        if (t >= (int64_t)job->B * job->Hq)
            break;
        const int b = (int)(t / job->Hq);
        const int L = job->seq_lens[b];
        const uint16_t *qr = job->q + t * (int64_t)job->Dqk;
        double *orow = job->o + t * (int64_t)job->Dv;
        for (int d = 0; d < job->Dv; ++d)
            orow[d] = 0.0;
        if (L == 0) {
            job->lse[t] = -INFINITY;
            continue;
        }
        double m = -INFINITY;
        for (int j = 0; j < L; ++j) {
            const uint16_t *cj = mla_row(job, b, j);
            double acc = 0.0;
            for (int d = 0; d < job->Dqk; ++d)
                acc += bf16_bits_to_f64(qr[d]) * bf16_bits_to_f64(cj[d]);
            s_buf[j] = job->scale * acc;
            if (s_buf[j] > m)
                m = s_buf[j];
        }
        double l = 0.0;
        for (int j = 0; j < L; ++j) {
            const double e = exp(s_buf[j] - m);
            const uint16_t *cj = mla_row(job, b, j);
            l += e;
            for (int d = 0; d < job->Dv; ++d)
                orow[d] += e * bf16_bits_to_f64(cj[d]);
        }
        for (int d = 0; d < job->Dv; ++d)
            orow[d] /= l;
        job->lse[t] = m + log(l);
    }
    free(s_buf);
    return NULL;
}

int mk_oracle_mla_decode_f64(const uint16_t *q, const uint16_t *cache, const int32_t *page_table,
                             const int32_t *seq_lens, double *o, double *lse, int B, int Hq,
                             int Dqk, int Dv, int page_size, int max_pages, int num_pages,
                             double scale, int n_threads)
{
    if (!q || !cache || !page_table || !seq_lens || !o || !lse)
        return MK_ORACLE_BAD_ARG;
    if (B < 1 || Hq < 1 || Dqk < 1 || Dv < 1 || Dv > Dqk || page_size < 1 || max_pages < 1 ||
        num_pages < 1)
        return MK_ORACLE_BAD_ARG;
    int max_len = 0;
    for (int b = 0; b < B; ++b) {
        const int L = seq_lens[b];
        if (L < 0 || (int64_t)L > (int64_t)max_pages * page_size)
            return MK_ORACLE_BAD_ARG;
        for (int j = 0; j * page_size < L; ++j) {
            const int32_t pg = page_table[(int64_t)b * max_pages + j];
            if (pg < 0 || pg >= num_pages)
                return MK_ORACLE_BAD_ARG;
        }
        if (L > max_len)
            max_len = L;
    }
    int64_t next = 0;
    mla_job_t job = {q, cache, page_table, seq_lens, o, lse, B, Hq, Dqk, Dv, page_size, max_pages,
                     scale, &next, max_len};
    return run_threads(mla_worker, &job, sizeof job, n_threads);
}
