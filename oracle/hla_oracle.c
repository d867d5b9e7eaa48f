/*
 * hla_oracle.c -- plain, slow, fp64 CPU oracle for Higher-order Linear
 * Attention (Zhang, Qin, Wang, Gu, "Higher-order Linear Attention").
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the reference that the CUDA path is
 * checked against.  It shares no code, header, table or helper with the CUDA
 * library; only the test suite, the smoke check and the CPU-baseline leg of
 * the benchmark load it.  The product path never calls it.
 *
 * Everything is written the obvious way, in the paper's notation and in the
 * order the paper states it.  No blocking, no fusion, no symmetry tricks.
 *
 * Data layout (all double precision, row-major, heads outermost):
 *   q, k : [BH][n][d]      v, out : [BH][n][dv]      den : [BH][n]
 * Second-order state tuple per head (Sec. "Causal masking via extended
 * summaries", Fig. 1(A)):
 *   [ S (d*d) | C (d*dv) | m (d) | G (d*dv) | h (d) ]
 * Third-order state tuple per head (Sec. "Streaming form of Causal HLA",
 * Theorem 3):
 *   [ SK (d*d) | SQ (d*d) | P (d*dv) | mK (d) |
 *     G1 (d*dv) | G2 (d*dv) | G3 (d*dv) | h1 (d) | h2 (d) | h3 (d) ]
 *
 * Functions and the passages they follow:
 *   hla2_serial_f64    online updates after Theorem 1, outputs of Theorem 1
 *                      (masked) or Eq. hla-unnorm / Eq. hla-row (unmasked)
 *   hla2_combine_f64   the masked semidirect product, Eq. semidirect
 *                      (unmasked: the additive monoid of Sec. 4.1)
 *   hla2_chunked_f64   Theorem 2 / Remark on scan modes: exclusive Blelloch
 *                      scan within chunks and across chunk summaries, then
 *                      local inclusion of the token segment
 *   hla3_serial_f64    Algorithm 3 at gamma = 1 (masked); the unmasked
 *                      factorisation q^T S^K S^Q P^KV (Sec. 7.1)
 *   hla3_chunked_f64   Theorem 4 / Algorithm 4: exclusive scans under the
 *                      third-order concatenation (Eqs. hla3-base-concat and
 *                      hla3-corrected-concat), segment maps applied by
 *                      contraction
 *   hla2_state_to_sde_f64  the masked tuple folded to (S, D = S C - G,
 *                      e = S m - h), what Theorem 1's num and den read
 *   ahla_serial_f64    AHLA online updates (Theorem AHLA, Algorithm
 *                      AHLA-stream at gamma = 1); state [P | m | E | n]
 *   ahla_combine_f64   Eq. AHLA-semidirect on summaries [R | P | m | E | n]
 *   ahla_chunked_f64   AHLA scan equivalence: exclusive Blelloch scans under
 *                      the AHLA product within and across chunks
 *   hla2_backward_f64  gradients of L = sum_t dout_t . o_t: the reverse sweep
 *                      over the online updates after Theorem 1, with the
 *                      forward states checkpointed at tile boundaries and
 *                      recomputed within a tile (Sec. "Chunk-parallel
 *                      training via associative scans")
 *
 * Threads: the serial functions spread the BH heads over nthreads POSIX
 * threads (heads are independent); each head is computed by one thread in
 * exactly the same order, so results do not depend on nthreads.
 */
#include <pthread.h>
#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------------ */
/* small dense helpers (plain loops)                                         */
/* ------------------------------------------------------------------------ */

static double *zalloc(size_t count)
{
    double *p = (double *)calloc(count ? count : 1, sizeof(double));
    return p;
}

/* y[c] = sum_r x[r] * M[r][c]   (row vector times matrix, M is R x Cc) */
static void rowvec_mat(const double *x, const double *M, int R, int Cc, double *y)
{
    for (int c = 0; c < Cc; ++c) {
        double s = 0.0;
        for (int r = 0; r < R; ++r) s += x[r] * M[(size_t)r * Cc + c];
        y[c] = s;
    }
}

/* y[r] = sum_c M[r][c] * x[c]   (matrix times column vector) */
static void mat_vec(const double *M, const double *x, int R, int Cc, double *y)
{
    for (int r = 0; r < R; ++r) {
        double s = 0.0;
        for (int c = 0; c < Cc; ++c) s += M[(size_t)r * Cc + c] * x[c];
        y[r] = s;
    }
}

/* Z = X * Y with X: R x K, Y: K x Cc */
static void mat_mul(const double *X, const double *Y, int R, int K, int Cc, double *Z)
{
    for (int r = 0; r < R; ++r)
        for (int c = 0; c < Cc; ++c) {
            double s = 0.0;
            for (int t = 0; t < K; ++t) s += X[(size_t)r * K + t] * Y[(size_t)t * Cc + c];
            Z[(size_t)r * Cc + c] = s;
        }
}

static double dot(const double *a, const double *b, int len)
{
    double s = 0.0;
    for (int i = 0; i < len; ++i) s += a[i] * b[i];
    return s;
}

/* ------------------------------------------------------------------------ */
/* head-parallel driver                                                      */
/* ------------------------------------------------------------------------ */

typedef void (*head_fn)(void *args, int head);

typedef struct {
    head_fn fn;
    void *args;
    int first, stride, count;
} worker_t;

static void *worker_main(void *p)
{
    worker_t *w = (worker_t *)p;
    for (int hd = w->first; hd < w->count; hd += w->stride) w->fn(w->args, hd);
    return NULL;
}

static void run_heads(head_fn fn, void *args, int BH, int nthreads)
{
    if (nthreads < 1) nthreads = 1;
    if (nthreads > BH) nthreads = BH;
    if (nthreads <= 1) {
        for (int hd = 0; hd < BH; ++hd) fn(args, hd);
        return;
    }
    pthread_t *tid = (pthread_t *)malloc(sizeof(pthread_t) * (size_t)nthreads);
    worker_t *w = (worker_t *)malloc(sizeof(worker_t) * (size_t)nthreads);
    for (int i = 0; i < nthreads; ++i) {
        w[i].fn = fn; w[i].args = args; w[i].first = i; w[i].stride = nthreads; w[i].count = BH;
        pthread_create(&tid[i], NULL, worker_main, &w[i]);
    }
    for (int i = 0; i < nthreads; ++i) pthread_join(tid[i], NULL);
    free(tid);
    free(w);
}

/* ======================================================================== */
/* Second order                                                              */
/* ======================================================================== */

size_t hla2_state_len_f64(int d, int dv)
{
    return (size_t)d * d + 2 * (size_t)d * dv + 2 * (size_t)d;
}

typedef struct {
    const double *q, *k, *v;
    double *out, *den;
    int n, d, dv, masked, normalized;
    double eps;
    const double *state_in;
    double *state_out;
} hla2_args;

/*
 * One head of the serial recurrence.  For t = 1..n:
 *   masked:  G_t = G_{t-1} + k_t (k_t^T C_{t-1}),  h_t = h_{t-1} + k_t (k_t^T m_{t-1})
 *            (the cross-summaries use the PREVIOUS C and m; online updates)
 *   S_t = S_{t-1} + k_t k_t^T,  C_t = C_{t-1} + q_t v_t^T,  m_t = m_{t-1} + q_t
 *   masked:   num = q_t^T (S_t C_t - G_t),  den = q_t^T (S_t m_t - h_t)     (Theorem 1)
 *   unmasked: num = q_t^T S_t C_t,          den = q_t^T S_t m_t             (Eq. hla-unnorm)
 *   out = num (default) or num / (den + eps) (Eq. masked / Eq. hla-row)
 * The products are evaluated as u = q^T S first and then u C, which is the
 * order the implementation notes give.
 */
static void hla2_serial_head(void *pargs, int hd)
{
    const hla2_args *a = (const hla2_args *)pargs;
    const int n = a->n, d = a->d, dv = a->dv;
    const double *q = a->q + (size_t)hd * n * d;
    const double *k = a->k + (size_t)hd * n * d;
    const double *v = a->v + (size_t)hd * n * dv;
    double *out = a->out ? a->out + (size_t)hd * n * dv : NULL;
    double *den_out = a->den ? a->den + (size_t)hd * n : NULL;

    double *S = zalloc((size_t)d * d), *C = zalloc((size_t)d * dv), *m = zalloc(d);
    double *G = zalloc((size_t)d * dv), *h = zalloc(d);
    double *kC = zalloc(dv), *u = zalloc(d), *uC = zalloc(dv), *qG = zalloc(dv);

    if (a->state_in) {
        const double *st = a->state_in + (size_t)hd * hla2_state_len_f64(d, dv);
        memcpy(S, st, sizeof(double) * (size_t)d * d);
        memcpy(C, st + (size_t)d * d, sizeof(double) * (size_t)d * dv);
        memcpy(m, st + (size_t)d * d + (size_t)d * dv, sizeof(double) * d);
        if (a->masked) {
            memcpy(G, st + (size_t)d * d + (size_t)d * dv + d, sizeof(double) * (size_t)d * dv);
            memcpy(h, st + (size_t)d * d + 2 * (size_t)d * dv + d, sizeof(double) * d);
        }
    }

    for (int t = 0; t < n; ++t) {
        const double *qt = q + (size_t)t * d, *kt = k + (size_t)t * d, *vt = v + (size_t)t * dv;

        if (a->masked) {
            /* k_t^T C_{t-1} and k_t^T m_{t-1}, with the state before this token */
            rowvec_mat(kt, C, d, dv, kC);
            double km = dot(kt, m, d);
            for (int r = 0; r < d; ++r) {
                for (int c = 0; c < dv; ++c) G[(size_t)r * dv + c] += kt[r] * kC[c];
                h[r] += kt[r] * km;
            }
        }
        for (int r = 0; r < d; ++r) {
            for (int c = 0; c < d; ++c) S[(size_t)r * d + c] += kt[r] * kt[c];
            for (int c = 0; c < dv; ++c) C[(size_t)r * dv + c] += qt[r] * vt[c];
            m[r] += qt[r];
        }

        rowvec_mat(qt, S, d, d, u);          /* u = q_t^T S_t       */
        rowvec_mat(u, C, d, dv, uC);         /* u C_t               */
        double den = dot(u, m, d);           /* u m_t               */
        if (a->masked) {
            rowvec_mat(qt, G, d, dv, qG);    /* q_t^T G_t           */
            den -= dot(qt, h, d);            /* - q_t^T h_t         */
        }
        if (out) {
            for (int c = 0; c < dv; ++c) {
                double num = uC[c] - (a->masked ? qG[c] : 0.0);
                out[(size_t)t * dv + c] = a->normalized ? num / (den + a->eps) : num;
            }
        }
        if (den_out) den_out[t] = den;
    }

    if (a->state_out) {
        double *st = a->state_out + (size_t)hd * hla2_state_len_f64(d, dv);
        memcpy(st, S, sizeof(double) * (size_t)d * d);
        memcpy(st + (size_t)d * d, C, sizeof(double) * (size_t)d * dv);
        memcpy(st + (size_t)d * d + (size_t)d * dv, m, sizeof(double) * d);
        if (!a->masked) { memset(G, 0, sizeof(double) * (size_t)d * dv); memset(h, 0, sizeof(double) * d); }
        memcpy(st + (size_t)d * d + (size_t)d * dv + d, G, sizeof(double) * (size_t)d * dv);
        memcpy(st + (size_t)d * d + 2 * (size_t)d * dv + d, h, sizeof(double) * d);
    }
    free(S); free(C); free(m); free(G); free(h); free(kC); free(u); free(uC); free(qG);
}

int hla2_serial_f64(const double *q, const double *k, const double *v, double *out, double *den,
                    int BH, int n, int d, int dv, int masked, int normalized, double eps,
                    const double *state_in, double *state_out, int nthreads)
{
    if (BH < 0 || n < 0 || d < 1 || dv < 1) return 1;
    hla2_args a = {q, k, v, out, den, n, d, dv, masked, normalized, eps, state_in, state_out};
    run_heads(hla2_serial_head, &a, BH, nthreads);
    return 0;
}

/* ------------------------------------------------------------------------ */
/* The associative operator on state tuples                                  */
/* ------------------------------------------------------------------------ */

/*
 * out = A (+) B for adjacent segments, A first (Eq. semidirect):
 *   S = S_A + S_B,  C = C_A + C_B,  m = m_A + m_B,
 *   G = G_A + G_B + S_B C_A,  h = h_A + h_B + S_B m_A.
 * Unmasked (Sec. 4.1): the same without the cross terms (G, h stay as given,
 * summed).  out may alias neither A nor B.
 */
void hla2_combine_f64(const double *A, const double *B, double *out, int d, int dv, int masked)
{
    const size_t oS = 0, oC = (size_t)d * d, om = oC + (size_t)d * dv, oG = om + d, oh = oG + (size_t)d * dv;
    size_t len = hla2_state_len_f64(d, dv);
    for (size_t i = 0; i < len; ++i) out[i] = A[i] + B[i];
    if (masked) {
        double *SC = zalloc((size_t)d * dv), *Sm = zalloc(d);
        mat_mul(B + oS, A + oC, d, d, dv, SC);  /* S_B C_A */
        mat_vec(B + oS, A + om, d, d, Sm);      /* S_B m_A */
        for (size_t i = 0; i < (size_t)d * dv; ++i) out[oG + i] += SC[i];
        for (int i = 0; i < d; ++i) out[oh + i] += Sm[i];
        free(SC); free(Sm);
    }
}

/* Elementary segment of one token: (k k^T, q v^T, q, 0, 0).  A single-token
 * segment has G = h = 0 (Sec. 4.2). */
static void hla2_token_segment(const double *qt, const double *kt, const double *vt, int d, int dv, double *T)
{
    const size_t oC = (size_t)d * d, om = oC + (size_t)d * dv;
    memset(T, 0, sizeof(double) * hla2_state_len_f64(d, dv));
    for (int r = 0; r < d; ++r) {
        for (int c = 0; c < d; ++c) T[(size_t)r * d + c] = kt[r] * kt[c];
        for (int c = 0; c < dv; ++c) T[oC + (size_t)r * dv + c] = qt[r] * vt[c];
        T[om + r] = qt[r];
    }
}

/* Outputs from an inclusive state (Theorem 1 / Eq. hla-unnorm). */
static void hla2_read_out(const double *st, const double *qt, int d, int dv, int masked, int normalized,
                          double eps, double *out_t, double *den_t)
{
    const size_t oC = (size_t)d * d, om = oC + (size_t)d * dv, oG = om + d, oh = oG + (size_t)d * dv;
    double *u = zalloc(d), *uC = zalloc(dv), *qG = zalloc(dv);
    rowvec_mat(qt, st, d, d, u);
    rowvec_mat(u, st + oC, d, dv, uC);
    double den = dot(u, st + om, d);
    if (masked) {
        rowvec_mat(qt, st + oG, d, dv, qG);
        den -= dot(qt, st + oh, d);
    }
    for (int c = 0; c < dv; ++c) {
        double num = uC[c] - (masked ? qG[c] : 0.0);
        out_t[c] = normalized ? num / (den + eps) : num;
    }
    if (den_t) *den_t = den;
    free(u); free(uC); free(qG);
}

/*
 * Exclusive Blelloch scan (up-sweep then down-sweep) of `count` tuples under
 * the operator above, in place: afterwards x[i] = x[0] (+) ... (+) x[i-1], and
 * x[0] = identity (all zeros).  `count` is padded to a power of two with
 * identity elements.  Ordering of the operands is kept (left before right),
 * which is what an associative, non-commutative operator needs.
 */
static void hla2_blelloch_exclusive(double *x, int count, int d, int dv, int masked)
{
    const size_t len = hla2_state_len_f64(d, dv);
    int p2 = 1;
    while (p2 < count) p2 <<= 1;
    double *buf = zalloc(len * (size_t)p2);
    memcpy(buf, x, sizeof(double) * len * (size_t)count);
    double *tmp = zalloc(len);
    /* up-sweep: buf[r] <- buf[l] (+) buf[r] */
    for (int stride = 1; stride < p2; stride <<= 1)
        for (int i = 2 * stride - 1; i < p2; i += 2 * stride) {
            double *l = buf + len * (size_t)(i - stride), *r = buf + len * (size_t)i;
            hla2_combine_f64(l, r, tmp, d, dv, masked);
            memcpy(r, tmp, sizeof(double) * len);
        }
    /* down-sweep */
    memset(buf + len * (size_t)(p2 - 1), 0, sizeof(double) * len);
    double *old_left = zalloc(len);
    for (int stride = p2 >> 1; stride >= 1; stride >>= 1)
        for (int i = 2 * stride - 1; i < p2; i += 2 * stride) {
            double *l = buf + len * (size_t)(i - stride), *r = buf + len * (size_t)i;
            memcpy(old_left, l, sizeof(double) * len);
            memcpy(l, r, sizeof(double) * len);          /* left  <- prefix before the pair  */
            hla2_combine_f64(r, old_left, tmp, d, dv, masked);
            memcpy(r, tmp, sizeof(double) * len);        /* right <- prefix (+) left         */
        }
    memcpy(x, buf, sizeof(double) * len * (size_t)count);
    free(buf); free(tmp); free(old_left);
}

typedef struct {
    hla2_args base;
    int chunk;
} hla2_chunk_args;

/*
 * Theorem 2 and the Remark on inclusive vs exclusive scans, per head:
 *  1. token segments T_t;
 *  2. within each chunk, exclusive Blelloch scan -> local prefixes P_t, and
 *     the chunk summary S^(c) = (+) of all T_t in the chunk;
 *  3. exclusive Blelloch scan across the chunk summaries -> carry-in P^(c)
 *     (the optional initial state is a segment placed before everything);
 *  4. inclusive state I_t = P^(c) (+) P_t (+) T_t, and outputs from I_t.
 */
static void hla2_chunked_head(void *pargs, int hd)
{
    const hla2_chunk_args *ca = (const hla2_chunk_args *)pargs;
    const hla2_args *a = &ca->base;
    const int n = a->n, d = a->d, dv = a->dv, W = ca->chunk;
    const size_t len = hla2_state_len_f64(d, dv);
    const double *q = a->q + (size_t)hd * n * d;
    const double *k = a->k + (size_t)hd * n * d;
    const double *v = a->v + (size_t)hd * n * dv;
    const int nchunks = (n + W - 1) / W;

    double *tok = zalloc(len * (size_t)(n ? n : 1));      /* T_t, then P_t after the local scans */
    double *tok_seg = zalloc(len * (size_t)(n ? n : 1));  /* T_t kept */
    double *summ = zalloc(len * (size_t)(nchunks + 1));   /* chunk summaries, slot 0 = initial state */
    double *tmp = zalloc(len), *tmp2 = zalloc(len);

    for (int t = 0; t < n; ++t) {
        hla2_token_segment(q + (size_t)t * d, k + (size_t)t * d, v + (size_t)t * dv, d, dv, tok + len * (size_t)t);
        memcpy(tok_seg + len * (size_t)t, tok + len * (size_t)t, sizeof(double) * len);
    }
    if (a->state_in) {
        memcpy(summ, a->state_in + (size_t)hd * len, sizeof(double) * len);
        /* unmasked: G and h are not part of the state */
        if (!a->masked) memset(summ + (size_t)d * d + (size_t)d * dv + d, 0, sizeof(double) * ((size_t)d * dv + d));
    }
    for (int c = 0; c < nchunks; ++c) {
        int t0 = c * W, t1 = t0 + W < n ? t0 + W : n;
        /* chunk summary: P_last (+) T_last after the exclusive scan */
        hla2_blelloch_exclusive(tok + len * (size_t)t0, t1 - t0, d, dv, a->masked);
        hla2_combine_f64(tok + len * (size_t)(t1 - 1), tok_seg + len * (size_t)(t1 - 1), summ + len * (size_t)(c + 1),
                         d, dv, a->masked);
    }
    /* carry-in of chunk c = initial (+) S^(1) (+) ... (+) S^(c-1): exclusive scan over
       [initial, S^(1), ..., S^(M)] gives slot c+1 = initial (+) S^(1..c); we want the
       prefix INCLUDING the initial state, i.e. the exclusive prefix of slot c+1. */
    hla2_blelloch_exclusive(summ, nchunks + 1, d, dv, a->masked);
    double *out = a->out ? a->out + (size_t)hd * n * dv : NULL;
    double *den_out = a->den ? a->den + (size_t)hd * n : NULL;
    for (int c = 0; c < nchunks; ++c) {
        int t0 = c * W, t1 = t0 + W < n ? t0 + W : n;
        const double *carry = summ + len * (size_t)(c + 1);
        for (int t = t0; t < t1; ++t) {
            hla2_combine_f64(carry, tok + len * (size_t)t, tmp, d, dv, a->masked);
            hla2_combine_f64(tmp, tok_seg + len * (size_t)t, tmp2, d, dv, a->masked);
            double dn;
            hla2_read_out(tmp2, q + (size_t)t * d, d, dv, a->masked, a->normalized, a->eps,
                          out ? out + (size_t)t * dv : tmp /* scratch */, &dn);
            if (den_out) den_out[t] = dn;
            if (t == n - 1 && a->state_out) memcpy(a->state_out + (size_t)hd * len, tmp2, sizeof(double) * len);
        }
    }
    if (n == 0 && a->state_out) memcpy(a->state_out + (size_t)hd * len, summ, sizeof(double) * len);
    free(tok); free(tok_seg); free(summ); free(tmp); free(tmp2);
}

int hla2_chunked_f64(const double *q, const double *k, const double *v, double *out, double *den,
                     int BH, int n, int d, int dv, int masked, int normalized, double eps, int chunk,
                     const double *state_in, double *state_out, int nthreads)
{
    if (BH < 0 || n < 0 || d < 1 || dv < 1 || chunk < 1) return 1;
    hla2_chunk_args a = {{q, k, v, out, den, n, d, dv, masked, normalized, eps, state_in, state_out}, chunk};
    run_heads(hla2_chunked_head, &a, BH, nthreads);
    return 0;
}

/* ======================================================================== */
/* Third order                                                               */
/* ======================================================================== */

size_t hla3_state_len_f64(int d, int dv)
{
    return 2 * (size_t)d * d + 4 * (size_t)d * dv + 4 * (size_t)d;
}

typedef struct {
    const double *q, *k, *v;
    double *out, *den;
    int n, d, dv, masked, normalized;
    double eps;
    const double *state_in;
    double *state_out;
} hla3_args;

/*
 * Algorithm 3 (masked third-order streaming kernel) at gamma = 1, one head.
 * Unmasked: o_t = q_t^T S^K_t S^Q_t P^KV_t, den = q_t^T S^K_t S^Q_t m^K_t.
 */
static void hla3_serial_head(void *pargs, int hd)
{
    const hla3_args *a = (const hla3_args *)pargs;
    const int n = a->n, d = a->d, dv = a->dv;
    const size_t dd = (size_t)d * d, ddv = (size_t)d * dv;
    const double *q = a->q + (size_t)hd * n * d;
    const double *k = a->k + (size_t)hd * n * d;
    const double *v = a->v + (size_t)hd * n * dv;
    double *out = a->out ? a->out + (size_t)hd * n * dv : NULL;
    double *den_out = a->den ? a->den + (size_t)hd * n : NULL;

    double *SK = zalloc(dd), *SQ = zalloc(dd), *P = zalloc(ddv), *mK = zalloc(d);
    double *G1 = zalloc(ddv), *G2 = zalloc(ddv), *G3 = zalloc(ddv), *h1 = zalloc(d), *h2 = zalloc(d), *h3 = zalloc(d);
    double *SKp = zalloc(dd), *SQp = zalloc(dd), *Pp = zalloc(ddv), *mp = zalloc(d);
    double *u1 = zalloc(d), *a2 = zalloc(d), *u3 = zalloc(d), *a3 = zalloc(d);
    double *rowP = zalloc(dv), *r1 = zalloc(d), *r2 = zalloc(d), *termA = zalloc(dv), *tB = zalloc(dv);
    double *sqm = zalloc(d), *denvec = zalloc(d);

    if (a->state_in) {
        const double *st = a->state_in + (size_t)hd * hla3_state_len_f64(d, dv);
        size_t o = 0;
        memcpy(SK, st + o, sizeof(double) * dd); o += dd;
        memcpy(SQ, st + o, sizeof(double) * dd); o += dd;
        memcpy(P, st + o, sizeof(double) * ddv); o += ddv;
        memcpy(mK, st + o, sizeof(double) * d); o += d;
        if (a->masked) {
            memcpy(G1, st + o, sizeof(double) * ddv); o += ddv;
            memcpy(G2, st + o, sizeof(double) * ddv); o += ddv;
            memcpy(G3, st + o, sizeof(double) * ddv); o += ddv;
            memcpy(h1, st + o, sizeof(double) * d); o += d;
            memcpy(h2, st + o, sizeof(double) * d); o += d;
            memcpy(h3, st + o, sizeof(double) * d);
        }
    }

    for (int t = 0; t < n; ++t) {
        const double *qt = q + (size_t)t * d, *kt = k + (size_t)t * d, *vt = v + (size_t)t * dv;
        /* keep the previous first-order state */
        memcpy(SKp, SK, sizeof(double) * dd);
        memcpy(SQp, SQ, sizeof(double) * dd);
        memcpy(Pp, P, sizeof(double) * ddv);
        memcpy(mp, mK, sizeof(double) * d);
        /* inclusive first-order updates */
        for (int r = 0; r < d; ++r) {
            for (int c = 0; c < d; ++c) {
                SK[(size_t)r * d + c] += kt[r] * kt[c];
                SQ[(size_t)r * d + c] += qt[r] * qt[c];
            }
            for (int c = 0; c < dv; ++c) P[(size_t)r * dv + c] += kt[r] * vt[c];
            mK[r] += kt[r];
        }
        if (a->masked) {
            /* G1 += k_t (u1^T P_prev), h1 += k_t (u1^T m_prev), u1 = S^Q_prev k_t */
            mat_vec(SQp, kt, d, d, u1);
            rowvec_mat(u1, Pp, d, dv, rowP);
            double s1 = dot(u1, mp, d);
            for (int r = 0; r < d; ++r) {
                for (int c = 0; c < dv; ++c) G1[(size_t)r * dv + c] += kt[r] * rowP[c];
                h1[r] += kt[r] * s1;
            }
            /* G2 += a2 (q_t^T P_prev), h2 += a2 (q_t^T m_prev), a2 = S^K_prev q_t */
            mat_vec(SKp, qt, d, d, a2);
            rowvec_mat(qt, Pp, d, dv, rowP);
            double s2 = dot(qt, mp, d);
            for (int r = 0; r < d; ++r) {
                for (int c = 0; c < dv; ++c) G2[(size_t)r * dv + c] += a2[r] * rowP[c];
                h2[r] += a2[r] * s2;
            }
            /* G3 += a3 v_t^T, h3 += a3, a3 = S^K_prev (S^Q_prev k_t) */
            mat_vec(SQp, kt, d, d, u3);
            mat_vec(SKp, u3, d, d, a3);
            for (int r = 0; r < d; ++r) {
                for (int c = 0; c < dv; ++c) G3[(size_t)r * dv + c] += a3[r] * vt[c];
                h3[r] += a3[r];
            }
        }
        /* termA = q_t^T S^K S^Q P^KV (row-vector products left to right) */
        rowvec_mat(qt, SK, d, d, r1);
        rowvec_mat(r1, SQ, d, d, r2);
        rowvec_mat(r2, P, d, dv, termA);
        /* den = q_t^T S^K S^Q m^K  [- q_t^T (h1 + h2 + h3)] */
        double den = dot(r2, mK, d);
        if (a->masked) {
            for (int r = 0; r < d; ++r) denvec[r] = h1[r] + h2[r] + h3[r];
            den -= dot(qt, denvec, d);
        }
        if (out) {
            for (int c = 0; c < dv; ++c) tB[c] = 0.0;
            if (a->masked) {
                for (int c = 0; c < dv; ++c) {
                    double s = 0.0;
                    for (int r = 0; r < d; ++r)
                        s += qt[r] * (G1[(size_t)r * dv + c] + G2[(size_t)r * dv + c] + G3[(size_t)r * dv + c]);
                    tB[c] = s;
                }
            }
            for (int c = 0; c < dv; ++c) {
                double num = termA[c] - tB[c];
                out[(size_t)t * dv + c] = a->normalized ? num / (den + a->eps) : num;
            }
        }
        if (den_out) den_out[t] = den;
    }
    if (a->state_out) {
        double *st = a->state_out + (size_t)hd * hla3_state_len_f64(d, dv);
        size_t o = 0;
        if (!a->masked) {
            memset(G1, 0, sizeof(double) * ddv); memset(G2, 0, sizeof(double) * ddv); memset(G3, 0, sizeof(double) * ddv);
            memset(h1, 0, sizeof(double) * d); memset(h2, 0, sizeof(double) * d); memset(h3, 0, sizeof(double) * d);
        }
        memcpy(st + o, SK, sizeof(double) * dd); o += dd;
        memcpy(st + o, SQ, sizeof(double) * dd); o += dd;
        memcpy(st + o, P, sizeof(double) * ddv); o += ddv;
        memcpy(st + o, mK, sizeof(double) * d); o += d;
        memcpy(st + o, G1, sizeof(double) * ddv); o += ddv;
        memcpy(st + o, G2, sizeof(double) * ddv); o += ddv;
        memcpy(st + o, G3, sizeof(double) * ddv); o += ddv;
        memcpy(st + o, h1, sizeof(double) * d); o += d;
        memcpy(st + o, h2, sizeof(double) * d); o += d;
        memcpy(st + o, h3, sizeof(double) * d);
    }
    free(SK); free(SQ); free(P); free(mK); free(G1); free(G2); free(G3); free(h1); free(h2); free(h3);
    free(SKp); free(SQp); free(Pp); free(mp); free(u1); free(a2); free(u3); free(a3);
    free(rowP); free(r1); free(r2); free(termA); free(tB); free(sqm); free(denvec);
}

int hla3_serial_f64(const double *q, const double *k, const double *v, double *out, double *den,
                    int BH, int n, int d, int dv, int masked, int normalized, double eps,
                    const double *state_in, double *state_out, int nthreads)
{
    if (BH < 0 || n < 0 || d < 1 || dv < 1) return 1;
    hla3_args a = {q, k, v, out, den, n, d, dv, masked, normalized, eps, state_in, state_out};
    run_heads(hla3_serial_head, &a, BH, nthreads);
    return 0;
}

/* ------------------------------------------------------------------------ */
/* Third-order scan state and concatenation (Sec. 7.3)                       */
/* ------------------------------------------------------------------------ */

/*
 * Segment scan state for a contiguous token range [t0, t1) of one head:
 *   SK, SQ (d x d), P (d x dv), mK (d), F (d x dv), eta (d),
 *   R^QP (d x dv), r^Qm (d), U^KQ (d x d),
 * and the maps M^KQP, M^KQm, which are linear in Z and are represented by
 * the token range itself and applied by contraction:
 *   M^KQP_X[Z] = sum_{t in X} k_t k_t^T Z k_t v_t^T,
 *   M^KQm_X[Z] = sum_{t in X} k_t k_t^T Z k_t.
 * Concatenation of ranges is concatenation of the sums, so the map of A (x) B
 * is the map of the merged range; segments in a scan are always adjacent.
 */
typedef struct {
    double *SK, *SQ, *P, *mK, *F, *eta, *R, *r, *U;
    int t0, t1; /* token range of the maps; t0 == t1 is the empty map */
} seg3;

static void seg3_alloc(seg3 *s, int d, int dv)
{
    s->SK = zalloc((size_t)d * d); s->SQ = zalloc((size_t)d * d); s->P = zalloc((size_t)d * dv);
    s->mK = zalloc(d); s->F = zalloc((size_t)d * dv); s->eta = zalloc(d);
    s->R = zalloc((size_t)d * dv); s->r = zalloc(d); s->U = zalloc((size_t)d * d);
    s->t0 = s->t1 = 0;
}

static void seg3_free(seg3 *s)
{
    free(s->SK); free(s->SQ); free(s->P); free(s->mK); free(s->F); free(s->eta); free(s->R); free(s->r); free(s->U);
}

static void seg3_zero(seg3 *s, int d, int dv)
{
    memset(s->SK, 0, sizeof(double) * (size_t)d * d); memset(s->SQ, 0, sizeof(double) * (size_t)d * d);
    memset(s->P, 0, sizeof(double) * (size_t)d * dv); memset(s->mK, 0, sizeof(double) * d);
    memset(s->F, 0, sizeof(double) * (size_t)d * dv); memset(s->eta, 0, sizeof(double) * d);
    memset(s->R, 0, sizeof(double) * (size_t)d * dv); memset(s->r, 0, sizeof(double) * d);
    memset(s->U, 0, sizeof(double) * (size_t)d * d);
    s->t0 = s->t1 = 0;
}

static void seg3_copy(seg3 *dst, const seg3 *src, int d, int dv)
{
    memcpy(dst->SK, src->SK, sizeof(double) * (size_t)d * d); memcpy(dst->SQ, src->SQ, sizeof(double) * (size_t)d * d);
    memcpy(dst->P, src->P, sizeof(double) * (size_t)d * dv); memcpy(dst->mK, src->mK, sizeof(double) * d);
    memcpy(dst->F, src->F, sizeof(double) * (size_t)d * dv); memcpy(dst->eta, src->eta, sizeof(double) * d);
    memcpy(dst->R, src->R, sizeof(double) * (size_t)d * dv); memcpy(dst->r, src->r, sizeof(double) * d);
    memcpy(dst->U, src->U, sizeof(double) * (size_t)d * d);
    dst->t0 = src->t0; dst->t1 = src->t1;
}

/* Single-token segment T_t (Algorithm 4, initialisation of the token segment):
 *   D^K = k k^T, D^Q = q q^T, D^P = k v^T, d^m = k,
 *   F = D^K D^Q D^P, eta = D^K D^Q d^m, R = D^Q D^P, r = D^Q d^m, U = D^K D^Q. */
static void seg3_token(seg3 *s, const double *qt, const double *kt, const double *vt, int t, int d, int dv)
{
    double *DK = zalloc((size_t)d * d), *DQ = zalloc((size_t)d * d), *DP = zalloc((size_t)d * dv);
    double *tmp = zalloc((size_t)d * d);
    for (int r = 0; r < d; ++r) {
        for (int c = 0; c < d; ++c) { DK[(size_t)r * d + c] = kt[r] * kt[c]; DQ[(size_t)r * d + c] = qt[r] * qt[c]; }
        for (int c = 0; c < dv; ++c) DP[(size_t)r * dv + c] = kt[r] * vt[c];
    }
    memcpy(s->SK, DK, sizeof(double) * (size_t)d * d);
    memcpy(s->SQ, DQ, sizeof(double) * (size_t)d * d);
    memcpy(s->P, DP, sizeof(double) * (size_t)d * dv);
    memcpy(s->mK, kt, sizeof(double) * d);
    mat_mul(DK, DQ, d, d, d, s->U);         /* U = D^K D^Q          */
    mat_mul(s->U, DP, d, d, dv, s->F);      /* F = D^K D^Q D^P      */
    mat_vec(s->U, kt, d, d, s->eta);        /* eta = D^K D^Q d^m    */
    mat_mul(DQ, DP, d, d, dv, s->R);        /* R = D^Q D^P          */
    mat_vec(DQ, kt, d, d, s->r);            /* r = D^Q d^m          */
    s->t0 = t; s->t1 = t + 1;
    free(DK); free(DQ); free(DP); free(tmp);
}

typedef struct {
    const double *k, *v; /* this head's tokens */
    int d, dv;
} tokens3;

/* M^KQP_X[Z] and M^KQm_X[Z] by contraction over the tokens of X. */
static void seg3_apply_maps(const tokens3 *tk, int t0, int t1, const double *Z, double *outP, double *outm)
{
    const int d = tk->d, dv = tk->dv;
    double *Zk = zalloc(d);
    memset(outP, 0, sizeof(double) * (size_t)d * dv);
    memset(outm, 0, sizeof(double) * d);
    for (int t = t0; t < t1; ++t) {
        const double *kt = tk->k + (size_t)t * d, *vt = tk->v + (size_t)t * dv;
        mat_vec(Z, kt, d, d, Zk);
        double s = dot(kt, Zk, d); /* k_t^T Z k_t */
        for (int r = 0; r < d; ++r) {
            for (int c = 0; c < dv; ++c) outP[(size_t)r * dv + c] += kt[r] * s * vt[c];
            outm[r] += kt[r] * s;
        }
    }
    free(Zk);
}

/*
 * out = A (x)_3 B, A before B (Eqs. hla3-base-concat and hla3-corrected-concat):
 *   additive parts summed;
 *   F   = F_A + F_B + S^K_A R^QP_B + M^KQP_B[S^Q_A] + U^KQ_B P^KV_A
 *   eta = eta_A + eta_B + S^K_A r^Qm_B + M^KQm_B[S^Q_A] + U^KQ_B m^K_A
 */
static void seg3_combine(const tokens3 *tk, const seg3 *A, const seg3 *B, seg3 *out)
{
    const int d = tk->d, dv = tk->dv;
    const size_t dd = (size_t)d * d, ddv = (size_t)d * dv;
    double *t1 = zalloc(ddv), *t2 = zalloc(ddv), *t3 = zalloc(ddv), *e1 = zalloc(d), *e2 = zalloc(d), *e3 = zalloc(d);
    mat_mul(A->SK, B->R, d, d, dv, t1);
    mat_vec(A->SK, B->r, d, d, e1);
    seg3_apply_maps(tk, B->t0, B->t1, A->SQ, t2, e2);
    mat_mul(B->U, A->P, d, d, dv, t3);
    mat_vec(B->U, A->mK, d, d, e3);
    for (size_t i = 0; i < dd; ++i) { out->SK[i] = A->SK[i] + B->SK[i]; out->SQ[i] = A->SQ[i] + B->SQ[i]; out->U[i] = A->U[i] + B->U[i]; }
    for (size_t i = 0; i < ddv; ++i) {
        out->P[i] = A->P[i] + B->P[i];
        out->R[i] = A->R[i] + B->R[i];
        out->F[i] = A->F[i] + B->F[i] + t1[i] + t2[i] + t3[i];
    }
    for (int i = 0; i < d; ++i) {
        out->mK[i] = A->mK[i] + B->mK[i];
        out->r[i] = A->r[i] + B->r[i];
        out->eta[i] = A->eta[i] + B->eta[i] + e1[i] + e2[i] + e3[i];
    }
    /* merged token range of the maps (empty maps are the identity) */
    if (A->t0 == A->t1) { out->t0 = B->t0; out->t1 = B->t1; }
    else if (B->t0 == B->t1) { out->t0 = A->t0; out->t1 = A->t1; }
    else { out->t0 = A->t0; out->t1 = B->t1; }
    free(t1); free(t2); free(t3); free(e1); free(e2); free(e3);
}

/* exclusive Blelloch scan over `count` segments (see hla2_blelloch_exclusive) */
static void seg3_blelloch_exclusive(const tokens3 *tk, seg3 *x, int count)
{
    const int d = tk->d, dv = tk->dv;
    int p2 = 1;
    while (p2 < count) p2 <<= 1;
    seg3 *buf = (seg3 *)calloc((size_t)p2, sizeof(seg3));
    for (int i = 0; i < p2; ++i) {
        seg3_alloc(&buf[i], d, dv);
        if (i < count) seg3_copy(&buf[i], &x[i], d, dv);
    }
    seg3 tmp, old_left;
    seg3_alloc(&tmp, d, dv);
    seg3_alloc(&old_left, d, dv);
    for (int stride = 1; stride < p2; stride <<= 1)
        for (int i = 2 * stride - 1; i < p2; i += 2 * stride) {
            seg3_combine(tk, &buf[i - stride], &buf[i], &tmp);
            seg3_copy(&buf[i], &tmp, d, dv);
        }
    seg3_zero(&buf[p2 - 1], d, dv);
    for (int stride = p2 >> 1; stride >= 1; stride >>= 1)
        for (int i = 2 * stride - 1; i < p2; i += 2 * stride) {
            seg3_copy(&old_left, &buf[i - stride], d, dv);
            seg3_copy(&buf[i - stride], &buf[i], d, dv);
            seg3_combine(tk, &buf[i], &old_left, &tmp);
            seg3_copy(&buf[i], &tmp, d, dv);
        }
    for (int i = 0; i < count; ++i) seg3_copy(&x[i], &buf[i], d, dv);
    for (int i = 0; i < p2; ++i) seg3_free(&buf[i]);
    free(buf);
    seg3_free(&tmp);
    seg3_free(&old_left);
}

typedef struct {
    hla3_args base;
    int chunk;
} hla3_chunk_args;

/*
 * Algorithm 4, per head (zero initial state; the maps make an external
 * initial segment meaningless without its tokens):
 *   token segments T_t; exclusive scan within each chunk -> P_loc_t and the
 *   chunk summary; exclusive scan across chunk summaries -> carry-in;
 *   I_t = carry (x) P_loc_t (x) T_t;  o_t = q_t^T F(I_t)  [/ (q_t^T eta(I_t) + eps)].
 * Unmasked third order has no corrected state; it is not handled here.
 */
static void hla3_chunked_head(void *pargs, int hd)
{
    const hla3_chunk_args *ca = (const hla3_chunk_args *)pargs;
    const hla3_args *a = &ca->base;
    const int n = a->n, d = a->d, dv = a->dv, W = ca->chunk;
    const double *q = a->q + (size_t)hd * n * d;
    tokens3 tk = {a->k + (size_t)hd * n * d, a->v + (size_t)hd * n * dv, d, dv};
    const int nchunks = (n + W - 1) / W;
    double *out = a->out ? a->out + (size_t)hd * n * dv : NULL;
    double *den_out = a->den ? a->den + (size_t)hd * n : NULL;

    seg3 *tok = (seg3 *)calloc((size_t)(n ? n : 1), sizeof(seg3));
    seg3 *tseg = (seg3 *)calloc((size_t)(n ? n : 1), sizeof(seg3));
    seg3 *summ = (seg3 *)calloc((size_t)(nchunks ? nchunks : 1), sizeof(seg3));
    for (int t = 0; t < n; ++t) {
        seg3_alloc(&tok[t], d, dv);
        seg3_alloc(&tseg[t], d, dv);
        seg3_token(&tok[t], q + (size_t)t * d, tk.k + (size_t)t * d, tk.v + (size_t)t * dv, t, d, dv);
        seg3_copy(&tseg[t], &tok[t], d, dv);
    }
    for (int c = 0; c < nchunks; ++c) seg3_alloc(&summ[c], d, dv);
    for (int c = 0; c < nchunks; ++c) {
        int t0 = c * W, t1 = t0 + W < n ? t0 + W : n;
        seg3_blelloch_exclusive(&tk, tok + t0, t1 - t0);
        seg3_combine(&tk, &tok[t1 - 1], &tseg[t1 - 1], &summ[c]);
    }
    seg3_blelloch_exclusive(&tk, summ, nchunks);
    seg3 tmp, incl;
    seg3_alloc(&tmp, d, dv);
    seg3_alloc(&incl, d, dv);
    for (int c = 0; c < nchunks; ++c) {
        int t0 = c * W, t1 = t0 + W < n ? t0 + W : n;
        for (int t = t0; t < t1; ++t) {
            const double *qt = q + (size_t)t * d;
            seg3_combine(&tk, &summ[c], &tok[t], &tmp);
            seg3_combine(&tk, &tmp, &tseg[t], &incl);
            double den = dot(qt, incl.eta, d);
            for (int col = 0; col < dv; ++col) {
                double num = 0.0;
                for (int r = 0; r < d; ++r) num += qt[r] * incl.F[(size_t)r * dv + col];
                if (out) out[(size_t)t * dv + col] = a->normalized ? num / (den + a->eps) : num;
            }
            if (den_out) den_out[t] = den;
        }
    }
    for (int t = 0; t < n; ++t) { seg3_free(&tok[t]); seg3_free(&tseg[t]); }
    for (int c = 0; c < nchunks; ++c) seg3_free(&summ[c]);
    seg3_free(&tmp); seg3_free(&incl);
    free(tok); free(tseg); free(summ);
}

int hla3_chunked_f64(const double *q, const double *k, const double *v, double *out, double *den,
                     int BH, int n, int d, int dv, int normalized, double eps, int chunk, int nthreads)
{
    if (BH < 0 || n < 0 || d < 1 || dv < 1 || chunk < 1) return 1;
    hla3_chunk_args a = {{q, k, v, out, den, n, d, dv, 1, normalized, eps, NULL, NULL}, chunk};
    run_heads(hla3_chunked_head, &a, BH, nthreads);
    return 0;
}

/* ======================================================================== */
/* (S, D, e) form of the masked second-order state                          */
/* ======================================================================== */

size_t hla2_sde_len_f64(int d, int dv)
{
    return (size_t)d * d + (size_t)d * dv + (size_t)d;
}

/*
 * Theorem 1 reads the masked outputs as num_t = q_t^T (S_t C_t - G_t) and
 * den_t = q_t^T (S_t m_t - h_t); this folds each head's tuple (S, C, m, G, h)
 * into [ S | D = S C - G | e = S m - h ] (d*d, d*dv, d).
 */
void hla2_state_to_sde_f64(const double *st, double *out, int BH, int d, int dv)
{
    const size_t len = hla2_state_len_f64(d, dv), olen = hla2_sde_len_f64(d, dv);
    for (int hd = 0; hd < BH; ++hd) {
        const double *S = st + (size_t)hd * len, *C = S + (size_t)d * d, *m = C + (size_t)d * dv;
        const double *G = m + d, *h = G + (size_t)d * dv;
        double *oS = out + (size_t)hd * olen, *oD = oS + (size_t)d * d, *oe = oD + (size_t)d * dv;
        memcpy(oS, S, sizeof(double) * (size_t)d * d);
        mat_mul(S, C, d, d, dv, oD);
        for (size_t i = 0; i < (size_t)d * dv; ++i) oD[i] -= G[i];
        mat_vec(S, m, d, d, oe);
        for (int r = 0; r < d; ++r) oe[r] -= h[r];
    }
}

/* ======================================================================== */
/* Asymmetric second order (AHLA), Sec. "Asymmetric Higher-order Linear      */
/* Attention"                                                               */
/* ======================================================================== */

/* AHLA streaming state per head: [ P (d*dv) | m (d) | E (d*dv) | n (d) ] */
size_t ahla_state_len_f64(int d, int dv)
{
    return 2 * (size_t)d * dv + 2 * (size_t)d;
}

typedef struct {
    const double *q, *k, *v;
    double *out, *den;
    int n, d, dv, normalized;
    double eps;
    const double *state_in;
    double *state_out;
} ahla_args;

/*
 * One head of the AHLA recurrence (masked streaming identity, Theorem AHLA;
 * Algorithm AHLA-stream at gamma = 1).  For t = 1..n:
 *   P_t = P_{t-1} + k_t v_t^T,   m_t = m_{t-1} + k_t
 *   E_t = E_{t-1} + k_t (q_t^T P_t),   n_t = n_{t-1} + k_t (q_t^T m_t)
 *   num = q_t^T E_t,  den = q_t^T n_t,  out = num or num / (den + eps)
 */
static void ahla_serial_head(void *pargs, int hd)
{
    const ahla_args *a = (const ahla_args *)pargs;
    const int n = a->n, d = a->d, dv = a->dv;
    const double *q = a->q + (size_t)hd * n * d;
    const double *k = a->k + (size_t)hd * n * d;
    const double *v = a->v + (size_t)hd * n * dv;
    double *out = a->out ? a->out + (size_t)hd * n * dv : NULL;
    double *den_out = a->den ? a->den + (size_t)hd * n : NULL;
    double *P = zalloc((size_t)d * dv), *m = zalloc(d), *E = zalloc((size_t)d * dv), *nn = zalloc(d);
    double *r = zalloc(dv), *num = zalloc(dv);
    if (a->state_in) {
        const double *st = a->state_in + (size_t)hd * ahla_state_len_f64(d, dv);
        memcpy(P, st, sizeof(double) * (size_t)d * dv);
        memcpy(m, st + (size_t)d * dv, sizeof(double) * d);
        memcpy(E, st + (size_t)d * dv + d, sizeof(double) * (size_t)d * dv);
        memcpy(nn, st + 2 * (size_t)d * dv + d, sizeof(double) * d);
    }
    for (int t = 0; t < n; ++t) {
        const double *qt = q + (size_t)t * d, *kt = k + (size_t)t * d, *vt = v + (size_t)t * dv;
        for (int i = 0; i < d; ++i) {
            for (int c = 0; c < dv; ++c) P[(size_t)i * dv + c] += kt[i] * vt[c];
            m[i] += kt[i];
        }
        rowvec_mat(qt, P, d, dv, r);       /* r = q_t^T P_t  */
        const double s = dot(qt, m, d);    /* s = q_t^T m_t  */
        for (int i = 0; i < d; ++i) {
            for (int c = 0; c < dv; ++c) E[(size_t)i * dv + c] += kt[i] * r[c];
            nn[i] += s * kt[i];
        }
        rowvec_mat(qt, E, d, dv, num);     /* q_t^T E_t      */
        const double den = dot(qt, nn, d); /* q_t^T n_t      */
        if (out)
            for (int c = 0; c < dv; ++c) out[(size_t)t * dv + c] = a->normalized ? num[c] / (den + a->eps) : num[c];
        if (den_out) den_out[t] = den;
    }
    if (a->state_out) {
        double *st = a->state_out + (size_t)hd * ahla_state_len_f64(d, dv);
        memcpy(st, P, sizeof(double) * (size_t)d * dv);
        memcpy(st + (size_t)d * dv, m, sizeof(double) * d);
        memcpy(st + (size_t)d * dv + d, E, sizeof(double) * (size_t)d * dv);
        memcpy(st + 2 * (size_t)d * dv + d, nn, sizeof(double) * d);
    }
    free(P); free(m); free(E); free(nn); free(r); free(num);
}

int ahla_serial_f64(const double *q, const double *k, const double *v, double *out, double *den,
                    int BH, int n, int d, int dv, int normalized, double eps,
                    const double *state_in, double *state_out, int nthreads)
{
    if (BH < 0 || n < 0 || d < 1 || dv < 1) return 1;
    ahla_args a = {q, k, v, out, den, n, d, dv, normalized, eps, state_in, state_out};
    run_heads(ahla_serial_head, &a, BH, nthreads);
    return 0;
}

/* segment summary for the AHLA scan: [ R (d*d) | P (d*dv) | m (d) | E (d*dv) | n (d) ],
 * R = sum over the segment of k_i q_i^T (Sec. "Chunk-parallel scans for AHLA") */
size_t ahla_summary_len_f64(int d, int dv)
{
    return (size_t)d * d + ahla_state_len_f64(d, dv);
}

/*
 * out = A (+)_AHLA B for adjacent segments, A first (Eq. AHLA-semidirect):
 *   R = R_A + R_B,  P = P_A + P_B,  m = m_A + m_B,
 *   E = E_A + E_B + R_B P_A,  n = n_A + n_B + R_B m_A.
 */
void ahla_combine_f64(const double *A, const double *B, double *out, int d, int dv)
{
    const size_t oR = 0, oP = (size_t)d * d, om = oP + (size_t)d * dv, oE = om + d, on = oE + (size_t)d * dv;
    const size_t len = ahla_summary_len_f64(d, dv);
    for (size_t i = 0; i < len; ++i) out[i] = A[i] + B[i];
    double *RP = zalloc((size_t)d * dv), *Rm = zalloc(d);
    mat_mul(B + oR, A + oP, d, d, dv, RP);   /* R_B P_A */
    mat_vec(B + oR, A + om, d, d, Rm);       /* R_B m_A */
    for (size_t i = 0; i < (size_t)d * dv; ++i) out[oE + i] += RP[i];
    for (int i = 0; i < d; ++i) out[on + i] += Rm[i];
    free(RP); free(Rm);
}

/* the summary of the single token (q, k, v): R = k q^T, P = k v^T, m = k, E = k (q . k) v^T, n = k (q . k) */
static void ahla_token_summary(const double *qt, const double *kt, const double *vt, int d, int dv, double *T)
{
    const size_t oP = (size_t)d * d, om = oP + (size_t)d * dv, oE = om + d, on = oE + (size_t)d * dv;
    const double qk = dot(qt, kt, d);
    for (int i = 0; i < d; ++i) {
        for (int j = 0; j < d; ++j) T[(size_t)i * d + j] = kt[i] * qt[j];
        for (int c = 0; c < dv; ++c) {
            T[oP + (size_t)i * dv + c] = kt[i] * vt[c];
            T[oE + (size_t)i * dv + c] = kt[i] * qk * vt[c];
        }
        T[om + i] = kt[i];
        T[on + i] = kt[i] * qk;
    }
}

/* in-place exclusive Blelloch scan (up-sweep, down-sweep) of count summaries under (+)_AHLA */
static void ahla_blelloch_exclusive(double *x, int count, int d, int dv)
{
    const size_t len = ahla_summary_len_f64(d, dv);
    int p2 = 1;
    while (p2 < count) p2 <<= 1;
    double *buf = zalloc(len * (size_t)p2), *tmp = zalloc(len), *old_left = zalloc(len);
    memcpy(buf, x, sizeof(double) * len * (size_t)count);   /* the padding stays the identity (zeros) */
    for (int s = 1; s < p2; s <<= 1)
        for (int i = 2 * s - 1; i < p2; i += 2 * s) {
            ahla_combine_f64(buf + len * (size_t)(i - s), buf + len * (size_t)i, tmp, d, dv);
            memcpy(buf + len * (size_t)i, tmp, sizeof(double) * len);
        }
    memset(buf + len * (size_t)(p2 - 1), 0, sizeof(double) * len);
    for (int s = p2 >> 1; s >= 1; s >>= 1)
        for (int i = 2 * s - 1; i < p2; i += 2 * s) {
            double *l = buf + len * (size_t)(i - s), *r = buf + len * (size_t)i;
            memcpy(old_left, l, sizeof(double) * len);
            memcpy(l, r, sizeof(double) * len);
            ahla_combine_f64(r, old_left, tmp, d, dv);
            memcpy(r, tmp, sizeof(double) * len);
        }
    memcpy(x, buf, sizeof(double) * len * (size_t)count);
    free(buf); free(tmp); free(old_left);
}

typedef struct {
    const double *q, *k, *v;
    double *out, *den;
    int n, d, dv, chunk, normalized;
    double eps;
} ahla_chunk_args;

/*
 * One head by the scan route (Sec. "Chunk-parallel scans for AHLA", scan
 * equivalence): token summaries; within each chunk an exclusive Blelloch scan
 * gives the chunk-local prefix of every token; chunk summaries are scanned
 * the same way across chunks; the state at token t is
 *   carry(chunk) (+) local exclusive prefix (+) token t,
 * and o_t = q_t^T E_t, den_t = q_t^T n_t.
 */
static void ahla_chunked_head(void *pargs, int hd)
{
    const ahla_chunk_args *a = (const ahla_chunk_args *)pargs;
    const int n = a->n, d = a->d, dv = a->dv, C = a->chunk;
    const size_t len = ahla_summary_len_f64(d, dv);
    const size_t oE = (size_t)d * d + (size_t)d * dv + d, on = oE + (size_t)d * dv;
    const double *q = a->q + (size_t)hd * n * d, *k = a->k + (size_t)hd * n * d, *v = a->v + (size_t)hd * n * dv;
    const int nch = (n + C - 1) / C;
    double *tok = zalloc(len * (size_t)(n > 0 ? n : 1)), *pre = zalloc(len * (size_t)(n > 0 ? n : 1));
    double *summ = zalloc(len * (size_t)(nch > 0 ? nch : 1));
    double *tmp = zalloc(len), *st = zalloc(len), *num = zalloc(dv);
    for (int t = 0; t < n; ++t) ahla_token_summary(q + (size_t)t * d, k + (size_t)t * d, v + (size_t)t * dv, d, dv,
                                                   tok + len * (size_t)t);
    memcpy(pre, tok, sizeof(double) * len * (size_t)n);
    for (int c = 0; c < nch; ++c) {
        const int t0 = c * C, cnt = (n - t0 < C) ? n - t0 : C;
        /* chunk summary = fold of its tokens */
        double *sc = summ + len * (size_t)c;
        memcpy(sc, tok + len * (size_t)t0, sizeof(double) * len);
        for (int t = t0 + 1; t < t0 + cnt; ++t) {
            ahla_combine_f64(sc, tok + len * (size_t)t, tmp, d, dv);
            memcpy(sc, tmp, sizeof(double) * len);
        }
        ahla_blelloch_exclusive(pre + len * (size_t)t0, cnt, d, dv);
    }
    ahla_blelloch_exclusive(summ, nch, d, dv);
    for (int t = 0; t < n; ++t) {
        const double *carry = summ + len * (size_t)(t / C);
        ahla_combine_f64(carry, pre + len * (size_t)t, tmp, d, dv);
        ahla_combine_f64(tmp, tok + len * (size_t)t, st, d, dv);
        const double *qt = q + (size_t)t * d;
        rowvec_mat(qt, st + oE, d, dv, num);
        const double den = dot(qt, st + on, d);
        if (a->out)
            for (int c = 0; c < dv; ++c)
                a->out[((size_t)hd * n + t) * dv + c] = a->normalized ? num[c] / (den + a->eps) : num[c];
        if (a->den) a->den[(size_t)hd * n + t] = den;
    }
    free(tok); free(pre); free(summ); free(tmp); free(st); free(num);
}

int ahla_chunked_f64(const double *q, const double *k, const double *v, double *out, double *den,
                     int BH, int n, int d, int dv, int chunk, int normalized, double eps, int nthreads)
{
    if (BH < 0 || n < 0 || d < 1 || dv < 1 || chunk < 1) return 1;
    ahla_chunk_args a = {q, k, v, out, den, n, d, dv, chunk, normalized, eps};
    run_heads(ahla_chunked_head, &a, BH, nthreads);
    return 0;
}

/* ======================================================================== */
/* Gradients of second-order HLA (Sec. "Chunk-parallel training via          */
/* associative scans": the reverse pass, with the forward states             */
/* checkpointed at tile boundaries and recomputed within a tile)             */
/* ======================================================================== */

typedef struct {
    const double *q, *k, *v, *dout;
    double *dq, *dk, *dv;
    int n, d, dvv, masked, normalized, ckpt;
    double eps;
} hla2_bwd_args;

/* one forward token update of the tuple (online updates after Theorem 1) */
static void hla2_token_update(double *st, const double *qt, const double *kt, const double *vt, int d, int dv,
                              int masked, double *kC)
{
    double *S = st, *C = S + (size_t)d * d, *m = C + (size_t)d * dv, *G = m + d, *h = G + (size_t)d * dv;
    if (masked) {
        rowvec_mat(kt, C, d, dv, kC);
        const double km = dot(kt, m, d);
        for (int r = 0; r < d; ++r) {
            for (int c = 0; c < dv; ++c) G[(size_t)r * dv + c] += kt[r] * kC[c];
            h[r] += kt[r] * km;
        }
    }
    for (int r = 0; r < d; ++r) {
        for (int c = 0; c < d; ++c) S[(size_t)r * d + c] += kt[r] * kt[c];
        for (int c = 0; c < dv; ++c) C[(size_t)r * dv + c] += qt[r] * vt[c];
        m[r] += qt[r];
    }
}

/*
 * One head of the reverse sweep: the vector-Jacobian product of the serial
 * recurrence for L = sum_t dout_t . o_t.  The forward states are kept at the
 * start of every ckpt-token tile (checkpoints); each tile is recomputed
 * forward from its checkpoint, then swept backward token by token.  With the
 * adjoint tuple (dS, dC, dm, dG, dh) of the state after token t:
 *   output (num = q^T S C - q^T G, den = q^T S m - q^T h on the state after t):
 *     gnum = dout (unnormalised) or dout / (den + eps), gden = -(dout . o) / (den + eps)
 *     dq += S C gnum - G gnum + gden (S m - h)
 *     dS += q (C gnum)^T + gden q m^T,  dC += (S q) gnum^T,  dm += gden S q
 *     dG -= q gnum^T,  dh -= gden q                     (masked only for G, h)
 *   token update (state before t -> after t), in reverse:
 *     S += k k^T:           dk += (dS + dS^T) k
 *     C += q v^T:           dq += dC v,  dv += dC^T q
 *     m += q:               dq += dm
 *     G += k (k^T C_prev):  dk += dG (C_prev^T k) + C_prev (dG^T k),  dC += k (k^T dG)
 *     h += k (k^T m_prev):  dk += dh (k . m_prev) + m_prev (k . dh),  dm += k (k . dh)
 * (dS, dC, dm, dG, dh then belong to the state before t.)
 */
static void hla2_backward_head(void *pargs, int hd)
{
    const hla2_bwd_args *a = (const hla2_bwd_args *)pargs;
    const int n = a->n, d = a->d, dv = a->dvv, ck = a->ckpt > 0 ? a->ckpt : 1;
    const size_t len = hla2_state_len_f64(d, dv);
    const size_t oC = (size_t)d * d, om = oC + (size_t)d * dv, oG = om + d, oh = oG + (size_t)d * dv;
    const double *q = a->q + (size_t)hd * n * d, *k = a->k + (size_t)hd * n * d, *v = a->v + (size_t)hd * n * dv;
    const double *g = a->dout + (size_t)hd * n * dv;
    double *dq = a->dq + (size_t)hd * n * d, *dk = a->dk + (size_t)hd * n * d, *dvo = a->dv + (size_t)hd * n * dv;
    const int ntile = (n + ck - 1) / ck;
    double *cp = zalloc(len * (size_t)(ntile > 0 ? ntile : 1));   /* state before each tile */
    double *tile = zalloc(len * (size_t)(ck + 1));                 /* states before / after the tile's tokens */
    double *adj = zalloc(len), *kC = zalloc(dv);
    double *u = zalloc(d), *Cg = zalloc(d), *Sm = zalloc(d), *num = zalloc(dv), *gnum = zalloc(dv), *tv = zalloc(d);
    /* forward pass: checkpoints */
    {
        double *st = zalloc(len);
        for (int t = 0; t < n; ++t) {
            if (t % ck == 0) memcpy(cp + len * (size_t)(t / ck), st, sizeof(double) * len);
            hla2_token_update(st, q + (size_t)t * d, k + (size_t)t * d, v + (size_t)t * dv, d, dv, a->masked, kC);
        }
        free(st);
    }
    memset(dq, 0, sizeof(double) * (size_t)n * d);
    memset(dk, 0, sizeof(double) * (size_t)n * d);
    memset(dvo, 0, sizeof(double) * (size_t)n * dv);
    for (int ti = ntile - 1; ti >= 0; --ti) {
        const int t0 = ti * ck, cnt = (n - t0 < ck) ? n - t0 : ck;
        memcpy(tile, cp + len * (size_t)ti, sizeof(double) * len);
        for (int j = 0; j < cnt; ++j) {
            const int t = t0 + j;
            memcpy(tile + len * (size_t)(j + 1), tile + len * (size_t)j, sizeof(double) * len);
            hla2_token_update(tile + len * (size_t)(j + 1), q + (size_t)t * d, k + (size_t)t * d,
                              v + (size_t)t * dv, d, dv, a->masked, kC);
        }
        for (int j = cnt - 1; j >= 0; --j) {
            const int t = t0 + j;
            const double *qt = q + (size_t)t * d, *kt = k + (size_t)t * d, *vt = v + (size_t)t * dv;
            const double *gt = g + (size_t)t * dv;
            const double *post = tile + len * (size_t)(j + 1), *prev = tile + len * (size_t)j;
            const double *S = post, *C = post + oC, *m = post + om, *G = post + oG, *h = post + oh;
            double *dS = adj, *dC = adj + oC, *dm = adj + om, *dG = adj + oG, *dh = adj + oh;
            double *dqt = dq + (size_t)t * d, *dkt = dk + (size_t)t * d, *dvt = dvo + (size_t)t * dv;
            /* forward values of the output at t */
            mat_vec(S, qt, d, d, u);                     /* u = S q (S symmetric) */
            rowvec_mat(u, C, d, dv, num);                /* u^T C     */
            double den = dot(u, m, d);
            if (a->masked) {
                for (int c = 0; c < dv; ++c) {
                    double s = 0.0;
                    for (int r = 0; r < d; ++r) s += qt[r] * G[(size_t)r * dv + c];
                    num[c] -= s;
                }
                den -= dot(qt, h, d);
            }
            double gden = 0.0;
            for (int c = 0; c < dv; ++c) gnum[c] = a->normalized ? gt[c] / (den + a->eps) : gt[c];
            if (a->normalized) {
                double go = 0.0;
                for (int c = 0; c < dv; ++c) go += gt[c] * num[c] / (den + a->eps);
                gden = -go / (den + a->eps);
            }
            /* output adjoints */
            mat_vec(C, gnum, d, dv, Cg);                 /* C gnum    */
            mat_vec(S, Cg, d, d, tv);                    /* S C gnum  */
            for (int r = 0; r < d; ++r) dqt[r] += tv[r];
            mat_vec(S, m, d, d, Sm);                     /* S m       */
            for (int r = 0; r < d; ++r) dqt[r] += gden * Sm[r];
            if (a->masked) {
                mat_vec(G, gnum, d, dv, tv);             /* G gnum    */
                for (int r = 0; r < d; ++r) dqt[r] -= tv[r] + gden * h[r];
            }
            for (int r = 0; r < d; ++r) {
                for (int c = 0; c < d; ++c) dS[(size_t)r * d + c] += qt[r] * Cg[c] + gden * qt[r] * m[c];
                for (int c = 0; c < dv; ++c) dC[(size_t)r * dv + c] += u[r] * gnum[c];
                dm[r] += gden * u[r];
                if (a->masked) {
                    for (int c = 0; c < dv; ++c) dG[(size_t)r * dv + c] -= qt[r] * gnum[c];
                    dh[r] -= gden * qt[r];
                }
            }
            /* reverse of the token update */
            for (int r = 0; r < d; ++r) {
                double s = 0.0;
                for (int c = 0; c < d; ++c) s += (dS[(size_t)r * d + c] + dS[(size_t)c * d + r]) * kt[c];
                dkt[r] += s;
                double sc = 0.0;
                for (int c = 0; c < dv; ++c) sc += dC[(size_t)r * dv + c] * vt[c];
                dqt[r] += sc + dm[r];
            }
            for (int c = 0; c < dv; ++c) {
                double s = 0.0;
                for (int r = 0; r < d; ++r) s += dC[(size_t)r * dv + c] * qt[r];
                dvt[c] += s;
            }
            if (a->masked) {
                const double *Cp = prev + oC, *mp = prev + om;
                double *kdG = zalloc(dv), *Ctk = zalloc(dv);
                rowvec_mat(kt, dG, d, dv, kdG);          /* k^T dG       */
                rowvec_mat(kt, Cp, d, dv, Ctk);          /* k^T C_prev   */
                const double kdh = dot(kt, dh, d), kmp = dot(kt, mp, d);
                for (int r = 0; r < d; ++r) {
                    double s1 = 0.0, s2 = 0.0;
                    for (int c = 0; c < dv; ++c) {
                        s1 += dG[(size_t)r * dv + c] * Ctk[c];
                        s2 += Cp[(size_t)r * dv + c] * kdG[c];
                    }
                    dkt[r] += s1 + s2 + dh[r] * kmp + mp[r] * kdh;
                    for (int c = 0; c < dv; ++c) dC[(size_t)r * dv + c] += kt[r] * kdG[c];
                    dm[r] += kt[r] * kdh;
                }
                free(kdG); free(Ctk);
            }
        }
    }
    free(cp); free(tile); free(adj); free(kC); free(u); free(Cg); free(Sm); free(num); free(gnum); free(tv);
}

int hla2_backward_f64(const double *q, const double *k, const double *v, const double *dout,
                      double *dq, double *dk, double *dv, int BH, int n, int d, int dvv, int masked,
                      int normalized, double eps, int ckpt, int nthreads)
{
    if (BH < 0 || n < 0 || d < 1 || dvv < 1) return 1;
    hla2_bwd_args a = {q, k, v, dout, dq, dk, dv, n, d, dvv, masked, normalized, ckpt, eps};
    run_heads(hla2_backward_head, &a, BH, nthreads);
    return 0;
}
