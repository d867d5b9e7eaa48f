// Chunk-parallel third-order HLA forward (Theorem 4, Algorithm 4 at gamma = 1)
// in fp32 on CUDA cores; calls that ask for state_out take the serial kernel
// (hla3_generic.cu), which also advances G1..G3 and h1..h3 of the state tuple.
//
// Per head, tokens are cut into chunks of W (W = min(chunk, 64), 32 for head
// sizes of 128; the result does not depend on the chunking up to rounding).
// Rows are tokens of one chunk, A = Q K^T (A_ts = q_t . k_s), a = diag(A),
// L / Ls the lower triangle with / without the diagonal.
//
// Masked.  With o_t = q_t^T F_t for the corrected state F (and den_t = q_t^T eta_t),
// the token update of Algorithm 3 is
//   dF_s = k_s a_s q_s^T P_s + k_s (k_s^T S^Q_{s-1} k_s) v_s^T + S^K_{s-1} q_s a_s v_s^T,
// so that, for a chunk with carry-in (S^K, S^Q, P, m, F, eta)_p,
//   Y = Q P_p + (L.A) V,   b_s = k_s^T S^Q_p k_s + sum_{u<s} A_us^2,
//   C_ts = q_t^T S^K_p q_s + sum_{i<s} A_ti A_si,
//   num = Q F_p + (L.A)(diag(a) Y + diag(b) V) + (L.C) diag(a) V,
//   den = Q eta_p + (L.A)(a . (Q m_p + (L.A) 1) + b) + (L.C) a.
// The carries follow the concatenation of Eqs. hla3-base-concat and
// hla3-corrected-concat: S^K, S^Q, P, m add up, and
//   F_{A (x) B} = F_A + F_B + S^K_A R_B + M^KQP_B[S^Q_A] + U_B P_A
// (eta likewise with r, M^KQm, m) with the chunk's R = Q^T diag(a) V,
// r = Q^T a, U = K^T diag(a) Q and the segment map applied by contraction,
// M^KQP_B[Z] = K^T diag(k_t^T Z k_t) V.  Every term is linear in the
// exclusive prefixes of S^K, S^Q, P, m, so the carries are two rounds of
// prefix sums with no sequential matrix chain:
//   F_p(c) = F_0 + sum_{c'<c} [F_{c'} + S^K_p(c') R_{c'} + M_{c'}[S^Q_p(c')] + U_{c'} P_p(c')].
// The chunk-local F of the bracket (zero carry-in) is
//   F_c = K^T (diag(a) Y_loc + diag(b_loc) V + N V),  N_ts = [t < s] A_st a_s.
//
// Unmasked (Sec. 7.1): o_t = q_t^T S^K_t S^Q_t P_t with inclusive prefixes:
//   X = Q S^K_p + (L.A) K,  Z = X S^Q_p + (L.(X Q^T)) Q,  num = Z P_p + (L.(Z K^T)) V,
//   den = Z m_p + (L.(Z K^T)) 1.
//
// Launches: local summaries, prefix sums of (S^K, S^Q, P, m), brackets (masked),
// prefix sums of the brackets (masked), outputs; plus the corrected initial
// carry F_0 = S^K S^Q P - G1 - G2 - G3 (eta_0 likewise) when state_in is given.
#include "hla_internal.h"

namespace hla {
namespace {

constexpr int kT3c = 256;

struct C3Layout {
    int BH, n, d, dv, W, nc;
    int stage_bracket;  // the bracket kernel copies its d x d / d x dv operands to shared memory
    int stage_out;      // the output kernel copies its chunk's prefix record to shared memory
    long long rec_loc, rec_pre, oSK, oSQ, oU, oP, oF, oR, om, oe, orr;  // local record offsets (floats)
    long long pSK, pSQ, pP, pm, pF, pe;                                  // prefix record offsets
    long long loc_base, pre_base, init_base, total;
    __host__ __device__ float *loc(float *ws, int hd, int c) const { return ws + loc_base + ((long long)hd * nc + c) * rec_loc; }
    __host__ __device__ float *pre(float *ws, int hd, int c) const { return ws + pre_base + ((long long)hd * nc + c) * rec_pre; }
    __host__ __device__ float *init(float *ws, int hd) const {
        return ws + init_base + (long long)hd * ((long long)d * dv + d);
    }
};

inline long long up4(long long x) { return (x + 3) / 4 * 4; }

int chunk3_width(int d, int dv, int chunk) {
    const int cap = (d >= 128 || dv >= 128) ? 32 : 64;
    return chunk < cap ? chunk : cap;
}

C3Layout c3_layout(int BH, int n, int d, int dv, int chunk) {
    C3Layout L;
    L.BH = BH; L.n = n; L.d = d; L.dv = dv;
    L.W = chunk3_width(d, dv, chunk);
    L.nc = (n + L.W - 1) / L.W;
    const long long dd = (long long)d * d, ddv = (long long)d * dv;
    long long o = 0;
    L.oSK = o; o += up4(dd); L.oSQ = o; o += up4(dd); L.oU = o; o += up4(dd);
    L.oP = o; o += up4(ddv); L.oF = o; o += up4(ddv); L.oR = o; o += up4(ddv);
    L.om = o; o += up4(d); L.oe = o; o += up4(d); L.orr = o; o += up4(d);
    L.rec_loc = o;
    o = 0;
    L.pSK = o; o += up4(dd); L.pSQ = o; o += up4(dd); L.pP = o; o += up4(ddv);
    L.pm = o; o += up4(d); L.pF = o; o += up4(ddv); L.pe = o; o += up4(d);
    L.rec_pre = o;
    L.loc_base = 0;
    L.pre_base = L.loc_base + (long long)BH * L.nc * L.rec_loc;
    L.init_base = L.pre_base + (long long)BH * L.nc * L.rec_pre;
    L.total = L.init_base + (long long)BH * (ddv + d);
    L.stage_bracket = (3 * dd + 2 * ddv) * 4 <= 96 * 1024;
    L.stage_out = L.rec_pre * 4 <= 32 * 1024;
    return L;
}

template <typename T>
__device__ __forceinline__ float ld_tok(const T *p) { return to_f32(*p); }

// dst (row stride ld) = or += sum_k a(r, k) b(k, c) over rows x cols.  Each thread forms a 2 x 2 block of
// outputs, rows r and r + rows/2, columns c and c + cols/2, so that every operand element it loads is used
// twice (the products are bound by shared-memory loads); with an odd size, one output per thread.  The
// same thread owns the same outputs in every call of the same shape, so accumulating calls need no barrier
// between them.
template <bool kAcc, typename FA, typename FB>
__device__ __forceinline__ void smm2(float *dst, int ld, int rows, int cols, int kdim, FA a, FB b) {
    if ((rows | cols) & 1) {
        for (int i = threadIdx.x; i < rows * cols; i += blockDim.x) {
            const int r = i / cols, c = i % cols;
            float s = 0.f;
            for (int k = 0; k < kdim; ++k) s += a(r, k) * b(k, c);
            dst[r * ld + c] = kAcc ? dst[r * ld + c] + s : s;
        }
        return;
    }
    const int hr = rows >> 1, hc = cols >> 1;
    for (int i = threadIdx.x; i < hr * hc; i += blockDim.x) {
        const int r = i / hc, c = i % hc;
        float s00 = 0.f, s01 = 0.f, s10 = 0.f, s11 = 0.f;
        for (int k = 0; k < kdim; ++k) {
            const float a0 = a(r, k), a1 = a(r + hr, k), b0 = b(k, c), b1 = b(k, c + hc);
            s00 += a0 * b0;
            s01 += a0 * b1;
            s10 += a1 * b0;
            s11 += a1 * b1;
        }
        float *d0 = dst + r * ld + c, *d1 = dst + (r + hr) * ld + c;
        if (kAcc) {
            d0[0] += s00; d0[hc] += s01; d1[0] += s10; d1[hc] += s11;
        } else {
            d0[0] = s00; d0[hc] = s01; d1[0] = s10; d1[hc] = s11;
        }
    }
}

// One of up to four independent products of the same shape computed side by side: the block's threads
// are split into ngrp groups and group grp forms this product with 4 x 4 output blocks per thread (rows
// r + i rows/4, columns c + j cols/4), eight operand loads per sixteen multiply-adds; other threads return
// at once.  Sizes that are not multiples of 4: one output per thread of the group.
template <bool kAcc, typename FA, typename FB>
__device__ __forceinline__ void smm44(int grp, int ngrp, float *dst, int ld, int rows, int cols, int kdim, FA a, FB b) {
    const int per = blockDim.x / ngrp, t = (int)threadIdx.x - grp * per;
    if (t < 0 || t >= per) return;
    if ((rows | cols) & 3) {  // one output per thread of the group
        for (int i = t; i < rows * cols; i += per) {
            const int r = i / cols, c = i % cols;
            float s = 0.f;
            for (int k = 0; k < kdim; ++k) s += a(r, k) * b(k, c);
            dst[r * ld + c] = kAcc ? dst[r * ld + c] + s : s;
        }
        return;
    }
    const int qr = rows >> 2, qc = cols >> 2;
    for (int i = t; i < qr * qc; i += per) {
        const int r = i / qc, c = i % qc;
        float acc[4][4];
#pragma unroll
        for (int x = 0; x < 4; ++x)
#pragma unroll
            for (int y = 0; y < 4; ++y) acc[x][y] = 0.f;
        for (int k = 0; k < kdim; ++k) {
            float av[4], bv[4];
#pragma unroll
            for (int x = 0; x < 4; ++x) av[x] = a(r + x * qr, k);
#pragma unroll
            for (int y = 0; y < 4; ++y) bv[y] = b(k, c + y * qc);
#pragma unroll
            for (int x = 0; x < 4; ++x)
#pragma unroll
                for (int y = 0; y < 4; ++y) acc[x][y] += av[x] * bv[y];
        }
#pragma unroll
        for (int x = 0; x < 4; ++x)
#pragma unroll
            for (int y = 0; y < 4; ++y) {
                float *o = dst + (r + x * qr) * ld + c + y * qc;
                *o = kAcc ? *o + acc[x][y] : acc[x][y];
            }
    }
}

// Triangular products, two outputs per thread that share one operand and their summation range:
// rows:  dst[t][c] (+)= sum_{k in [lo(t), hi(t))} a(t, k) b(k, c), columns c and c + cols/2
// cols:  dst[t][c] (+)= sum_{k in [0, hi(c))} a(t, k) b(k, c), rows t and t + rows/2
// (odd widths: one output per thread)
template <bool kAcc, typename FA, typename FB, typename FL, typename FH>
__device__ __forceinline__ void smm_rows(float *dst, int ld, int rows, int cols, FA a, FB b, FL lo, FH hi) {
    const int hc = (cols & 1) ? cols : cols >> 1, per = (cols & 1) ? 1 : 2;
    for (int i = threadIdx.x; i < rows * hc; i += blockDim.x) {
        const int t = i / hc, c = i % hc;
        float s0 = 0.f, s1 = 0.f;
        const int k1 = hi(t);
        for (int k = lo(t); k < k1; ++k) {
            const float av = a(t, k);
            s0 += av * b(k, c);
            if (per == 2) s1 += av * b(k, c + hc);
        }
        float *d0 = dst + t * ld + c;
        d0[0] = kAcc ? d0[0] + s0 : s0;
        if (per == 2) d0[hc] = kAcc ? d0[hc] + s1 : s1;
    }
}
template <bool kAcc, typename FA, typename FB, typename FH>
__device__ __forceinline__ void smm_cols(float *dst, int ld, int rows, int cols, FA a, FB b, FH hi) {
    const int hr = (rows & 1) ? rows : rows >> 1, per = (rows & 1) ? 1 : 2;
    for (int i = threadIdx.x; i < hr * cols; i += blockDim.x) {
        const int t = i / cols, c = i % cols;
        float s0 = 0.f, s1 = 0.f;
        const int k1 = hi(c);
        for (int k = 0; k < k1; ++k) {
            const float bv = b(k, c);
            s0 += a(t, k) * bv;
            if (per == 2) s1 += a(t + hr, k) * bv;
        }
        float *d0 = dst + t * ld + c;
        d0[0] = kAcc ? d0[0] + s0 : s0;
        if (per == 2) d0[hr * ld] = kAcc ? d0[hr * ld] + s1 : s1;
    }
}

// loads the chunk's Q, K (w x d) and V (w x dv) as fp32 with row strides d + 1 and dv + 1
// (shared-memory rows one float longer than the data, so that column walks hit distinct
// banks); rows past the sequence are zero
template <typename T>
__device__ void load_chunk(const T *q, const T *k, const T *v, float *Qs, float *Ks, float *Vs, int hd, int t0,
                           int w, int W, int n, int d, int dv) {
    const T *Qh = q + ((size_t)hd * n + t0) * d, *Kh = k + ((size_t)hd * n + t0) * d;
    const T *Vh = v + ((size_t)hd * n + t0) * dv;
    for (int i = threadIdx.x; i < W * d; i += blockDim.x) {
        const int r = i / d, c = i % d;
        Qs[r * (d + 1) + c] = r < w ? ld_tok(Qh + i) : 0.f;
        Ks[r * (d + 1) + c] = r < w ? ld_tok(Kh + i) : 0.f;
    }
    for (int i = threadIdx.x; i < W * dv; i += blockDim.x) {
        const int r = i / dv, c = i % dv;
        Vs[r * (dv + 1) + c] = r < w ? ld_tok(Vh + i) : 0.f;
    }
}

// ---------------------------------------------------------------------------
// 1. chunk-local summaries
// ---------------------------------------------------------------------------
// Shared-memory matrices use row strides one longer than their width (ld = d + 1,
// lv = dv + 1, lw = W + 1, lm = max(d, dv) + 1).
template <typename T>
__global__ void __launch_bounds__(kT3c) c3_local_kernel(const T *__restrict__ q, const T *__restrict__ k,
                                                        const T *__restrict__ v, float *ws, C3Layout L, int masked) {
    extern __shared__ float sm[];
    const int c = blockIdx.x, hd = blockIdx.y, W = L.W, d = L.d, dv = L.dv;
    const int ld = d + 1, lv = dv + 1, lw = W + 1;
    const int t0 = c * W, w = min(W, L.n - t0);
    float *Qs = sm, *Ks = Qs + W * ld, *Vs = Ks + W * ld, *A = Vs + W * lv, *Z = A + W * lw, *a = Z + W * lv;
    float *zeta = a + W, *b = zeta + W, *ym = b + W;
    load_chunk(q, k, v, Qs, Ks, Vs, hd, t0, w, W, L.n, d, dv);
    __syncthreads();
    float *rec = L.loc(ws, hd, c);
    // first-order sums (and A below), side by side in four thread groups
    smm44<false>(0, 4, rec + L.oSK, d, d, d, W, [&](int r, int t) { return Ks[t * ld + r]; }, [&](int t, int cc) { return Ks[t * ld + cc]; });
    smm44<false>(1, 4, rec + L.oSQ, d, d, d, W, [&](int r, int t) { return Qs[t * ld + r]; }, [&](int t, int cc) { return Qs[t * ld + cc]; });
    smm44<false>(2, 4, rec + L.oP, dv, d, dv, W, [&](int r, int t) { return Ks[t * ld + r]; }, [&](int t, int cc) { return Vs[t * lv + cc]; });
    for (int r = threadIdx.x; r < d; r += blockDim.x) {
        float s = 0.f;
        for (int t = 0; t < W; ++t) s += Ks[t * ld + r];
        rec[L.om + r] = s;
    }
    if (!masked) return;
    smm44<false>(3, 4, A, lw, W, W, d, [&](int t, int j) { return Qs[t * ld + j]; }, [&](int j, int s) { return Ks[s * ld + j]; });
    __syncthreads();
    for (int t = threadIdx.x; t < W; t += blockDim.x) {
        a[t] = A[t * lw + t];
        float bs = 0.f, ys = 0.f;
        for (int u = 0; u < t; ++u) bs += A[u * lw + t] * A[u * lw + t];
        for (int j = 0; j <= t; ++j) ys += A[t * lw + j];
        b[t] = bs;
        ym[t] = ys;
    }
    // Z = diag(a) Y_loc + diag(b) V + N V with Y_loc = (L.A) V and N_ts = [s > t] A_st a_s
    smm_rows<false>(Z, lv, W, dv, [&](int t, int j) { return A[t * lw + j]; }, [&](int j, int cc) { return Vs[j * lv + cc]; },
                    [](int) { return 0; }, [](int t) { return t + 1; });
    __syncthreads();
    for (int i = threadIdx.x; i < W * dv; i += blockDim.x) {
        const int t = i / dv, cc = i % dv;
        Z[t * lv + cc] = a[t] * Z[t * lv + cc] + b[t] * Vs[t * lv + cc];
    }
    for (int t = threadIdx.x; t < W; t += blockDim.x) {
        float nv = 0.f;
        for (int s = t + 1; s < W; ++s) nv += A[s * lw + t] * a[s];
        zeta[t] = a[t] * ym[t] + b[t] + nv;
    }
    __syncthreads();
    smm_rows<true>(Z, lv, W, dv, [&](int t, int s) { return A[s * lw + t] * a[s]; }, [&](int s, int cc) { return Vs[s * lv + cc]; },
                   [](int t) { return t + 1; }, [&](int) { return W; });
    __syncthreads();
    smm44<false>(0, 4, rec + L.oF, dv, d, dv, W, [&](int r, int t) { return Ks[t * ld + r]; }, [&](int t, int cc) { return Z[t * lv + cc]; });
    smm44<false>(1, 4, rec + L.oR, dv, d, dv, W, [&](int r, int t) { return Qs[t * ld + r] * a[t]; },
                 [&](int t, int cc) { return Vs[t * lv + cc]; });
    smm44<false>(2, 4, rec + L.oU, d, d, d, W, [&](int r, int t) { return Ks[t * ld + r] * a[t]; },
                 [&](int t, int cc) { return Qs[t * ld + cc]; });
    for (int r = threadIdx.x; r < d; r += blockDim.x) {
        float se = 0.f, sr = 0.f;
        for (int t = 0; t < W; ++t) {
            se += Ks[t * ld + r] * zeta[t];
            sr += Qs[t * ld + r] * a[t];
        }
        rec[L.oe + r] = se;
        rec[L.orr + r] = sr;
    }
}

// exclusive scan of one element over the chunks of a head: pre[c][po] = run + sum_{c'<c} loc[c'][lo]
// (eight loads in flight at a time; the additions stay in chunk order)
__device__ __forceinline__ void scan_chunks(float *ws, const C3Layout &L, int hd, long long lo, long long po, float run) {
    const float *src = L.loc(ws, hd, 0) + lo;
    float *dst = L.pre(ws, hd, 0) + po;
    int c = 0;
    for (; c + 8 <= L.nc; c += 8) {
        float x[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) x[u] = __ldcg(src + (long long)(c + u) * L.rec_loc);
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            dst[(long long)(c + u) * L.rec_pre] = run;
            run += x[u];
        }
    }
    for (; c < L.nc; ++c) {
        dst[(long long)c * L.rec_pre] = run;
        run += __ldcg(src + (long long)c * L.rec_loc);
    }
}

// ---------------------------------------------------------------------------
// 2. exclusive prefix sums over chunks of (S^K, S^Q, P, m), starting at state_in
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kT3c) c3_prefix1_kernel(float *ws, C3Layout L, const float *state_in) {
    const int hd = blockIdx.y, d = L.d, dv = L.dv;
    const long long dd = (long long)d * d, ddv = (long long)d * dv;
    const long long nel = 2 * dd + ddv + d;
    const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= nel) return;
    long long lo, po;  // local and prefix offsets; i is also the offset in the state tuple [SK | SQ | P | mK | ...]
    if (i < dd) { lo = L.oSK + i; po = L.pSK + i; }
    else if (i < 2 * dd) { lo = L.oSQ + (i - dd); po = L.pSQ + (i - dd); }
    else if (i < 2 * dd + ddv) { lo = L.oP + (i - 2 * dd); po = L.pP + (i - 2 * dd); }
    else { lo = L.om + (i - 2 * dd - ddv); po = L.pm + (i - 2 * dd - ddv); }
    const long long st_len = 2 * dd + 4 * ddv + 4 * (long long)d;
    float run = state_in ? state_in[(long long)hd * st_len + i] : 0.f;
    scan_chunks(ws, L, hd, lo, po, run);
}

// corrected initial carry F_0 = S^K S^Q P - G1 - G2 - G3, eta_0 = S^K S^Q m - h1 - h2 - h3
__global__ void __launch_bounds__(kT3c) c3_init_kernel(float *ws, C3Layout L, const float *state_in) {
    const int hd = blockIdx.x, d = L.d, dv = L.dv;
    const long long dd = (long long)d * d, ddv = (long long)d * dv;
    const float *st = state_in + (long long)hd * (2 * dd + 4 * ddv + 4 * (long long)d);
    const float *SK = st, *SQ = SK + dd, *P = SQ + dd, *mK = P + ddv, *G1 = mK + d, *G2 = G1 + ddv, *G3 = G2 + ddv;
    const float *h1 = G3 + ddv, *h2 = h1 + d, *h3 = h2 + d;
    float *out = L.init(ws, hd);
    for (long long i = threadIdx.x; i < ddv + d; i += blockDim.x) {
        const bool isF = i < ddv;
        const int r = isF ? (int)(i / dv) : (int)(i - ddv), cc = isF ? (int)(i % dv) : 0;
        float acc = 0.f;
        for (int x = 0; x < d; ++x) {
            float skq = 0.f;
            for (int y = 0; y < d; ++y) skq += SK[(long long)r * d + y] * SQ[(long long)y * d + x];
            acc += skq * (isF ? P[(long long)x * dv + cc] : mK[x]);
        }
        out[i] = acc - (isF ? (G1[i] + G2[i] + G3[i]) : (h1[r] + h2[r] + h3[r]));
    }
}

// ---------------------------------------------------------------------------
// 3. brackets F_c + S^K_p R_c + M_c[S^Q_p] + U_c P_p (and eta), written over F_c / eta_c
// ---------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(kT3c) c3_bracket_kernel(const T *__restrict__ k, const T *__restrict__ v, float *ws,
                                                          C3Layout L) {
    extern __shared__ float sm[];
    const int c = blockIdx.x, hd = blockIdx.y, W = L.W, d = L.d, dv = L.dv;
    const int ld = d + 1, lv = dv + 1;
    const int t0 = c * W, w = min(W, L.n - t0);
    float *Ks = sm, *Vs = Ks + W * ld, *T1 = Vs + W * lv, *bq = T1 + W * ld, *stage = bq + W;
    const T *Kh = k + ((size_t)hd * L.n + t0) * d, *Vh = v + ((size_t)hd * L.n + t0) * dv;
    for (int i = threadIdx.x; i < W * d; i += blockDim.x) Ks[(i / d) * ld + i % d] = (i / d) < w ? ld_tok(Kh + i) : 0.f;
    for (int i = threadIdx.x; i < W * dv; i += blockDim.x)
        Vs[(i / dv) * lv + i % dv] = (i / dv) < w ? ld_tok(Vh + i) : 0.f;
    __syncthreads();
    float *rec = L.loc(ws, hd, c);
    const float *pr = L.pre(ws, hd, c);
    const float *SKp = pr + L.pSK, *SQp = pr + L.pSQ, *Pp = pr + L.pP, *mp = pr + L.pm;
    const float *R = rec + L.oR, *U = rec + L.oU, *rr = rec + L.orr;
    if (L.stage_bracket) {  // copies of the d x d and d x dv operands in shared memory
        const int dd = d * d, ddv = d * dv;
        float *sSK = stage, *sSQ = sSK + dd, *sU = sSQ + dd, *sR = sU + dd, *sP = sR + ddv;
        for (int i = threadIdx.x; i < dd; i += blockDim.x) { sSK[i] = SKp[i]; sSQ[i] = SQp[i]; sU[i] = U[i]; }
        for (int i = threadIdx.x; i < ddv; i += blockDim.x) { sR[i] = R[i]; sP[i] = Pp[i]; }
        SKp = sSK; SQp = sSQ; U = sU; R = sR; Pp = sP;
        __syncthreads();
    }
    // bq_t = k_t^T S^Q_p k_t
    smm2<false>(T1, ld, W, d, d, [&](int t, int j) { return Ks[t * ld + j]; }, [&](int j, int cc) { return SQp[j * d + cc]; });
    __syncthreads();
    for (int t = threadIdx.x; t < W; t += blockDim.x) {
        float s = 0.f;
        for (int j = 0; j < d; ++j) s += T1[t * ld + j] * Ks[t * ld + j];
        bq[t] = s;
    }
    __syncthreads();
    // F_c += S^K_p R + U P_p + K^T diag(bq) V, summed in shared memory (same output owners in all three)
    float *acc = bq + W + (L.stage_bracket ? 3 * d * d + 2 * d * dv : 0);
    smm2<false>(acc, dv, d, dv, d, [&](int r, int x) { return SKp[r * d + x]; }, [&](int x, int cc) { return R[x * dv + cc]; });
    smm2<true>(acc, dv, d, dv, d, [&](int r, int x) { return U[r * d + x]; }, [&](int x, int cc) { return Pp[x * dv + cc]; });
    smm2<true>(acc, dv, d, dv, W, [&](int r, int t) { return Ks[t * ld + r] * bq[t]; },
               [&](int t, int cc) { return Vs[t * lv + cc]; });
    __syncthreads();
    for (int i = threadIdx.x; i < d * dv; i += blockDim.x) rec[L.oF + i] += acc[i];
    for (int r = threadIdx.x; r < d; r += blockDim.x) {
        float a1 = 0.f, a2 = 0.f, a3 = 0.f;
        for (int x = 0; x < d; ++x) {
            a1 += SKp[r * d + x] * rr[x];
            a3 += U[r * d + x] * mp[x];
        }
        for (int t = 0; t < W; ++t) a2 += Ks[t * ld + r] * bq[t];
        rec[L.oe + r] += a1 + a2 + a3;
    }
}

// 4. exclusive prefix sums of the brackets, starting at F_0, eta_0
__global__ void __launch_bounds__(kT3c) c3_prefix2_kernel(float *ws, C3Layout L, int has_init) {
    const int hd = blockIdx.y, d = L.d, dv = L.dv;
    const long long ddv = (long long)d * dv;
    const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= ddv + d) return;
    const bool isF = i < ddv;
    const long long lo = isF ? L.oF + i : L.oe + (i - ddv), po = isF ? L.pF + i : L.pe + (i - ddv);
    float run = has_init ? L.init(ws, hd)[i] : 0.f;
    scan_chunks(ws, L, hd, lo, po, run);
}

// floats of the output kernel's working matrices, rounded up to 4: where the staged prefix record starts
__host__ __device__ inline size_t out_stage_offset(const C3Layout &L) {
    const int lm = (L.d > L.dv ? L.d : L.dv) + 1;
    const size_t f = (size_t)L.W * (2 * (L.d + 1) + (L.dv + 1)) + 2 * (size_t)L.W * (L.W + 1) + 2 * (size_t)L.W * lm +
                     4 * L.W + (size_t)L.W * (L.dv + 1);
    return (f + 3) / 4 * 4;
}

// ---------------------------------------------------------------------------
// 5. outputs of a chunk from its carry-in
// ---------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(kT3c, 4) c3_out_kernel(const T *__restrict__ q, const T *__restrict__ k,
                                                      const T *__restrict__ v, T *__restrict__ out, float *ws,
                                                      C3Layout L, int masked, int normalized, float eps) {
    extern __shared__ float sm[];
    const int c = blockIdx.x, hd = blockIdx.y, W = L.W, d = L.d, dv = L.dv;
    const int ld = d + 1, lv = dv + 1, lw = W + 1, lm = (d > dv ? d : dv) + 1;
    const int t0 = c * W, w = min(W, L.n - t0);
    float *Qs = sm, *Ks = Qs + W * ld, *Vs = Ks + W * ld, *A = Vs + W * lv, *Cm = A + W * lw;
    float *M1 = Cm + W * lw, *M2 = M1 + W * lm, *a = M2 + W * lm, *b = a + W, *x1 = b + W, *den = x1 + W;
    float *Yb = den + W;  // W x dv (row stride dv + 1): Y, then the numerator
    load_chunk(q, k, v, Qs, Ks, Vs, hd, t0, w, W, L.n, d, dv);
    const float *pr = L.pre(ws, hd, c);
    if (L.stage_out) {  // the chunk's prefix record (read many times below) from L2 once, 16-byte aligned
        float *st = sm + out_stage_offset(L);
        for (long long i = threadIdx.x; i < L.rec_pre / 4; i += blockDim.x)
            reinterpret_cast<float4 *>(st)[i] = __ldcg(reinterpret_cast<const float4 *>(pr) + i);
        pr = st;
    }
    __syncthreads();
    const float *SKp = pr + L.pSK, *SQp = pr + L.pSQ, *Pp = pr + L.pP, *mp = pr + L.pm;
    const float *Fp = pr + L.pF, *ep = pr + L.pe;
    T *Oh = out + ((size_t)hd * L.n + t0) * dv;
    if (masked) {
        // A = Q K^T, M1 = K S^Q_p, M2 = Q S^K_p (W x d), Y = Q P_p: side by side in four thread groups
        smm44<false>(0, 4, A, lw, W, W, d, [&](int t, int j) { return Qs[t * ld + j]; }, [&](int j, int s) { return Ks[s * ld + j]; });
        smm44<false>(1, 4, M1, lm, W, d, d, [&](int t, int j) { return Ks[t * ld + j]; }, [&](int j, int cc) { return SQp[j * d + cc]; });
        smm44<false>(2, 4, M2, lm, W, d, d, [&](int t, int j) { return Qs[t * ld + j]; }, [&](int j, int cc) { return SKp[j * d + cc]; });
        smm44<false>(3, 4, Yb, lv, W, dv, d, [&](int s, int j) { return Qs[s * ld + j]; }, [&](int j, int cc) { return Pp[j * dv + cc]; });
        __syncthreads();
        for (int s = threadIdx.x; s < W; s += blockDim.x) {
            a[s] = A[s * lw + s];
            float bs = 0.f, ys = 0.f, qm = 0.f;
            for (int j = 0; j < d; ++j) {
                bs += M1[s * lm + j] * Ks[s * ld + j];
                qm += Qs[s * ld + j] * mp[j];
            }
            for (int u = 0; u < s; ++u) bs += A[u * lw + s] * A[u * lw + s];
            for (int j = 0; j <= s; ++j) ys += A[s * lw + j];
            b[s] = bs;
            x1[s] = qm + ys;  // (Q m_p + (L.A) 1)_s
        }
        // C_ts = q_t^T S^K_p q_s + sum_{i<s} A_ti A_si for s <= t, 0 above the diagonal; Y += (L.A) V
        smm2<false>(Cm, lw, W, W, d, [&](int t, int j) { return M2[t * lm + j]; }, [&](int j, int s) { return Qs[s * ld + j]; });
        __syncthreads();  // the accumulating products below own other elements
        smm_cols<true>(Cm, lw, W, W, [&](int t, int x) { return A[t * lw + x]; }, [&](int x, int s) { return A[s * lw + x]; },
                       [](int s) { return s; });
        smm_rows<true>(Yb, lv, W, dv, [&](int s, int j) { return A[s * lw + j]; }, [&](int j, int cc) { return Vs[j * lv + cc]; },
                       [](int) { return 0; }, [](int s) { return s + 1; });
        __syncthreads();
        for (int i = threadIdx.x; i < W * W; i += blockDim.x) {
            const int t = i / W, s = i % W;
            if (s > t) Cm[t * lw + s] = 0.f;
        }
        // M1 <- G1 = diag(a) Y + diag(b) V;  M2 <- G2 = diag(a) V
        for (int i = threadIdx.x; i < W * dv; i += blockDim.x) {
            const int s = i / dv, cc = i % dv;
            M1[s * lm + cc] = a[s] * Yb[s * lv + cc] + b[s] * Vs[s * lv + cc];
            M2[s * lm + cc] = a[s] * Vs[s * lv + cc];
        }
        __syncthreads();
        for (int t = threadIdx.x; t < W; t += blockDim.x) {
            float dn = 0.f;
            for (int j = 0; j < d; ++j) dn += Qs[t * ld + j] * ep[j];
            for (int s = 0; s <= t; ++s) dn += A[t * lw + s] * (a[s] * x1[s] + b[s]) + Cm[t * lw + s] * a[s];
            den[t] = dn;
        }
        // num = Q F_p + (L.A) G1 + C G2
        smm2<false>(Yb, lv, W, dv, d, [&](int t, int j) { return Qs[t * ld + j]; }, [&](int j, int cc) { return Fp[j * dv + cc]; });
        __syncthreads();
        smm_rows<true>(Yb, lv, W, dv, [&](int t, int s) { return A[t * lw + s]; }, [&](int s, int cc) { return M1[s * lm + cc]; },
                       [](int) { return 0; }, [](int t) { return t + 1; });
        smm_rows<true>(Yb, lv, W, dv, [&](int t, int s) { return Cm[t * lw + s]; }, [&](int s, int cc) { return M2[s * lm + cc]; },
                       [](int) { return 0; }, [](int t) { return t + 1; });
        __syncthreads();
        for (int i = threadIdx.x; i < w * dv; i += blockDim.x) {
            const int t = i / dv, cc = i % dv;
            const float num = Yb[t * lv + cc];
            from_f32(&Oh[i], normalized ? num / (den[t] + eps) : num);
        }
    } else {
        // A = Q K^T; M1 = X = Q S^K_p + (L.A) K
        smm2<false>(A, lw, W, W, d, [&](int t, int j) { return Qs[t * ld + j]; }, [&](int j, int s) { return Ks[s * ld + j]; });
        __syncthreads();
        for (int i = threadIdx.x; i < W * d; i += blockDim.x) {
            const int t = i / d, cc = i % d;
            float x = 0.f;
            for (int j = 0; j < d; ++j) x += Qs[t * ld + j] * SKp[j * d + cc];
            for (int s = 0; s <= t; ++s) x += A[t * lw + s] * Ks[s * ld + cc];
            M1[t * lm + cc] = x;
        }
        __syncthreads();
        // Cm = L.(X Q^T); M2 = Z = X S^Q_p + Cm Q
        for (int i = threadIdx.x; i < W * W; i += blockDim.x) {
            const int t = i / W, u = i % W;
            float s = 0.f;
            if (u <= t)
                for (int j = 0; j < d; ++j) s += M1[t * lm + j] * Qs[u * ld + j];
            Cm[t * lw + u] = s;
        }
        __syncthreads();
        for (int i = threadIdx.x; i < W * d; i += blockDim.x) {
            const int t = i / d, cc = i % d;
            float z = 0.f;
            for (int j = 0; j < d; ++j) z += M1[t * lm + j] * SQp[j * d + cc];
            for (int u = 0; u <= t; ++u) z += Cm[t * lw + u] * Qs[u * ld + cc];
            M2[t * lm + cc] = z;
        }
        __syncthreads();
        // A <- L.(Z K^T); den = Z m_p + A 1
        for (int i = threadIdx.x; i < W * W; i += blockDim.x) {
            const int t = i / W, s = i % W;
            float zk = 0.f;
            if (s <= t)
                for (int j = 0; j < d; ++j) zk += M2[t * lm + j] * Ks[s * ld + j];
            A[t * lw + s] = zk;
        }
        __syncthreads();
        for (int t = threadIdx.x; t < W; t += blockDim.x) {
            float dn = 0.f;
            for (int j = 0; j < d; ++j) dn += M2[t * lm + j] * mp[j];
            for (int s = 0; s <= t; ++s) dn += A[t * lw + s];
            den[t] = dn;
        }
        __syncthreads();
        for (int i = threadIdx.x; i < w * dv; i += blockDim.x) {
            const int t = i / dv, cc = i % dv;
            float num = 0.f;
            for (int j = 0; j < d; ++j) num += M2[t * lm + j] * Pp[j * dv + cc];
            for (int s = 0; s <= t; ++s) num += A[t * lw + s] * Vs[s * lv + cc];
            from_f32(&Oh[i], normalized ? num / (den[t] + eps) : num);
        }
    }
}

size_t smem_local(const C3Layout &L) {
    return sizeof(float) * ((size_t)L.W * (2 * (L.d + 1) + 2 * (L.dv + 1)) + (size_t)L.W * (L.W + 1) + 4 * L.W);
}
size_t smem_bracket(const C3Layout &L) {
    const size_t stage = L.stage_bracket ? 3 * (size_t)L.d * L.d + 2 * (size_t)L.d * L.dv : 0;
    return sizeof(float) * ((size_t)L.W * (2 * (L.d + 1) + (L.dv + 1)) + L.W + stage + (size_t)L.d * L.dv);
}
size_t smem_out(const C3Layout &L) {
    return sizeof(float) * (out_stage_offset(L) + (L.stage_out ? (size_t)L.rec_pre : 0));
}

template <typename T>
cudaError_t launch_all(const Fwd2 &p, const C3Layout &L, float *ws, cudaStream_t s) {
    const T *q = static_cast<const T *>(p.q), *k = static_cast<const T *>(p.k), *v = static_cast<const T *>(p.v);
    T *out = static_cast<T *>(p.out);
    cudaError_t e;
    const dim3 grid(L.nc, L.BH);
    if ((e = cudaFuncSetAttribute(c3_local_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_local(L))))
        return e;
    if ((e = cudaFuncSetAttribute(c3_bracket_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)smem_bracket(L))))
        return e;
    if ((e = cudaFuncSetAttribute(c3_out_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_out(L))))
        return e;
    cudaFuncSetAttribute(c3_out_kernel<T>, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
    cudaFuncSetAttribute(c3_local_kernel<T>, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
    cudaFuncSetAttribute(c3_bracket_kernel<T>, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
    c3_local_kernel<T><<<grid, kT3c, smem_local(L), s>>>(q, k, v, ws, L, p.masked);
    const long long n1 = 2LL * p.d * p.d + (long long)p.d * p.dv + p.d;
    c3_prefix1_kernel<<<dim3((unsigned)((n1 + kT3c - 1) / kT3c), L.BH), kT3c, 0, s>>>(ws, L, p.state_in);
    if (p.masked) {
        if (p.state_in) c3_init_kernel<<<L.BH, kT3c, 0, s>>>(ws, L, p.state_in);
        c3_bracket_kernel<T><<<grid, kT3c, smem_bracket(L), s>>>(k, v, ws, L);
        const long long n2 = (long long)p.d * p.dv + p.d;
        c3_prefix2_kernel<<<dim3((unsigned)((n2 + kT3c - 1) / kT3c), L.BH), kT3c, 0, s>>>(ws, L,
                                                                                       p.state_in ? 1 : 0);
    }
    c3_out_kernel<T><<<grid, kT3c, smem_out(L), s>>>(q, k, v, out, ws, L, p.masked, p.normalized, p.eps);
    return cudaGetLastError();
}

}  // namespace

size_t chunked3_workspace_bytes(int BH, int n, int d, int dv, int chunk) {
    if (n <= 0 || BH <= 0) return kWsHeaderBytes;
    return kWsHeaderBytes + sizeof(float) * (size_t)c3_layout(BH, n, d, dv, chunk).total;
}

// the per-chunk records grow like (n / chunk) * (5 d^2 + 5 d dv); above 1 GiB the
// serial kernel (whose scratch is one state per head) serves the call instead
bool chunked3_eligible(int BH, int n, int d, int dv, int chunk) {
    return BH <= 65535 && chunked3_workspace_bytes(BH, n, d, dv, chunk) <= (size_t(1) << 30);
}

cudaError_t chunked3_forward(const Fwd2 &p, cudaStream_t stream) {
    if (p.n <= 0 || p.BH <= 0) return cudaSuccess;
    const C3Layout L = c3_layout(p.BH, p.n, p.d, p.dv, p.chunk);
    float *ws = reinterpret_cast<float *>(p.ws + kWsHeaderBytes);
    if (p.dt == HLA_BF16) return launch_all<__nv_bfloat16>(p, L, ws, stream);
    return launch_all<float>(p, L, ws, stream);
}

}  // namespace hla
