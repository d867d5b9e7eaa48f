// Gradients of masked second-order HLA: a reverse chunk scan with the forward
// states checkpointed at chunk boundaries (Sec. "Chunk-parallel training via
// associative scans": the adjoint of the semidirect product applied by a
// reverse scan), fp32 SIMT kernels.
//
// With x_j = S_j q_j, T_tj = q_t . x_j and L = sum_t g_t . o_t, the forward is
// o_t = sum_{j<=t} T_tj v_j (proof of Theorem 1), so with P_tj = g_t . v_j:
//   dv_j = sum_{t>=j} T_tj g_t,   y_j = sum_{t>=j} P_tj q_t,
//   dq_t = sum_{j<=t} P_tj x_j + S_t y_t,
//   dk_i = sum_{j>=i} [ (q_j . k_i) y_j + (y_j . k_i) q_j ].
// The ratio-normalised output o = num / (den + eps) is the same computation
// with values [v | 1] (den is the extra column) and upstream gradient
// [g / (den + eps) | -(g . o) / (den + eps)]: every kernel works with the
// augmented width W = dv + 1 (for the plain output the extra gradient column
// is zero).
//
// Per chunk (rows = its tokens; p = prefix before the chunk, s = suffix after):
//   forward:  W_c = L . (Q K^T),  X = W_c K + Q S_p,  T = L . (Q X^T),
//             num' = T V' + Q D_p            (S_p, D_p = sum x v'^T: prefixes)
//   backward: P = L . (G' V'^T),  Y = P^T Q + V' Gam_s,
//             dV' = T^T G' + X Gam_s^T,
//             dQ = P X + G' D_p^T + Y S_p + (L . (Y K^T)) K,
//             dK = K Lam_s + W_c^T Y + (L . (Y K^T))^T Q,
// with the suffix sums Gam_s = sum g' q^T (W x d) and Lam_s = sum (y q^T + q y^T)
// (d x d).  The forward prefixes compose as D_p += X_loc^T V' + S_p (Q^T V')
// (the semidirect product, D-form); the suffixes compose in reverse as
//   Lam += Lam_loc + Gam_s^T M + M^T Gam_s  (M = V'^T Q, Lam_loc from the
//   chunk's own P^T Q),  Gam += G'^T Q,
// the adjoint of that product.  Five launches: forward local summaries, the
// forward prefix scan (the checkpoints), per-chunk gradient inputs and local
// reverse summaries, the reverse scan, per-chunk gradients.
#include <algorithm>

#include "hla_internal.h"
#include "simt_gemm.cuh"

namespace hla {
namespace {

constexpr int kThreads = 256;
constexpr int kCols = 32;

struct BLayout {
    int BH, n, d, dv, W, C, nch;
    long long fl_S, fl_DL, fl_C, fl_len;            // forward local: S_c d*d | DL_c d*W | C_c d*W
    long long fc_S, fc_D, fc_DT, fc_len;            // forward carry: S_p d*d | D_p d*W | D_p^T W*d
    long long bl_G, bl_Gam, bl_M, bl_Lam, bl_len;   // backward local: G' C*W | Gam_c W*d | M_c W*d | Lam_c d*d
    long long bc_Gam, bc_Lam, bc_GamT, bc_len;      // backward carry: Gam_s W*d | Lam_s d*d | Gam_s^T d*W
    long long o_fl, o_fc, o_bl, o_bc, total;        // floats from the scratch start
};

inline long long up16(long long x) { return (x + 15) / 16 * 16; }

BLayout make_layout(int BH, int n, int d, int dv, int chunk) {
    BLayout L;
    L.BH = BH; L.n = n; L.d = d; L.dv = dv; L.W = dv + 1;
    L.C = std::min(chunk, (d == 128 || dv == 128) ? 32 : 64);
    L.nch = (n + L.C - 1) / L.C;
    const long long dd = (long long)d * d, dW = (long long)d * L.W;
    L.fl_S = 0; L.fl_DL = up16(dd); L.fl_C = L.fl_DL + up16(dW); L.fl_len = L.fl_C + up16(dW);
    L.fc_S = 0; L.fc_D = up16(dd); L.fc_DT = L.fc_D + up16(dW); L.fc_len = L.fc_DT + up16(dW);
    L.bl_G = 0; L.bl_Gam = up16((long long)L.C * L.W); L.bl_M = L.bl_Gam + up16(dW); L.bl_Lam = L.bl_M + up16(dW);
    L.bl_len = L.bl_Lam + up16(dd);
    L.bc_Gam = 0; L.bc_Lam = up16(dW); L.bc_GamT = L.bc_Lam + up16(dd); L.bc_len = L.bc_GamT + up16(dW);
    const long long chunks = (long long)BH * L.nch;
    L.o_fl = 0;
    L.o_fc = L.o_fl + chunks * L.fl_len;
    L.o_bl = L.o_fc + chunks * L.fc_len;
    L.o_bc = L.o_bl + chunks * L.bl_len;
    L.total = L.o_bc + chunks * L.bc_len;
    return L;
}

__device__ __forceinline__ float *rec(float *ws, long long base, long long len, const BLayout &L, int hd, int c) {
    return ws + base + ((long long)hd * L.nch + c) * len;
}

// token rows of a chunk into shared memory (zero beyond the sequence); with ones, column
// `width` of each valid row is 1 (the augmented value column)
template <typename T>
__device__ void load_rows(const T *src, float *dst, int rows, int width, int Crows, int stride, bool ones) {
    for (int i = threadIdx.x; i < Crows * stride; i += blockDim.x) {
        const int r = i / stride, c = i % stride;
        float x = 0.f;
        if (r < rows) x = c < width ? to_f32(src[(long long)r * width + c]) : (ones && c == width ? 1.f : 0.f);
        dst[i] = x;
    }
}

// ---------------------------------------------------------------------------
// B1: forward local summaries S_c = K^T K, DL_c = (W_c K)^T V', C_c = Q^T V'
// ---------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(kThreads) bwd_fwd_local(const T *q, const T *k, const T *v, float *ws, BLayout L) {
    extern __shared__ float sm[];
    const int c = blockIdx.x, hd = blockIdx.y, d = L.d, W = L.W, C = L.C, t0 = c * C, len = min(C, L.n - t0);
    const int kd = d + 1;
    float *Qs = sm, *Ks = Qs + C * d, *Vs = Ks + C * kd, *Ws = Vs + C * W, *Xs = Ws + C * C;
    load_rows(q + ((long long)hd * L.n + t0) * d, Qs, len, d, C, d, false);
    load_rows(k + ((long long)hd * L.n + t0) * d, Ks, len, d, C, kd, false);
    load_rows(v + ((long long)hd * L.n + t0) * L.dv, Vs, len, L.dv, C, W, true);
    __syncthreads();
    bgemm(Ws, C, Qs, d, 1, Ks, 1, kd, C, C, d, false, 1);        // W_c = L . Q K^T
    __syncthreads();
    bgemm(Xs, d, Ws, C, 1, Ks, kd, 1, C, d, C, false, 0, 1);     // X_loc = W_c K
    __syncthreads();
    float *fl = rec(ws, L.o_fl, L.fl_len, L, hd, c);
    bgemm(fl + L.fl_S, d, Ks, 1, kd, Ks, kd, 1, d, d, C, false);  // K^T K
    bgemm(fl + L.fl_DL, W, Xs, 1, d, Vs, W, 1, d, W, C, false);   // X_loc^T V'
    bgemm(fl + L.fl_C, W, Qs, 1, d, Vs, W, 1, d, W, C, false);    // Q^T V'
}

// ---------------------------------------------------------------------------
// B2: forward prefix scan (the checkpoints).  Block (column block of D, head) keeps
// the whole S_p and 32 columns of D_p; per chunk it records them, then
// D_p += DL_c + S_p C_c and S_p += S_c.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads) bwd_fwd_scan(float *ws, BLayout L) {
    extern __shared__ float sm[];
    const int hd = blockIdx.y, d = L.d, W = L.W, j0 = blockIdx.x * kCols, ncol = min(kCols, W - j0);
    // S_p (d x d), D_p columns (d x 32), the chunk's C_c and DL_c columns staged per chunk (d x 32 each)
    float *Sp = sm, *Dp = Sp + d * d, *Cc = Dp + d * kCols, *DLc = Cc + d * kCols;
    for (int i = threadIdx.x; i < d * d; i += blockDim.x) Sp[i] = 0.f;
    for (int i = threadIdx.x; i < d * kCols; i += blockDim.x) Dp[i] = 0.f;
    __syncthreads();
    for (int c = 0; c < L.nch; ++c) {
        float *fc = rec(ws, L.o_fc, L.fc_len, L, hd, c);
        const float *fl = rec(ws, L.o_fl, L.fl_len, L, hd, c);
        if (blockIdx.x == 0)
            for (int i = threadIdx.x; i < d * d; i += blockDim.x) fc[L.fc_S + i] = Sp[i];
        for (int i = threadIdx.x; i < d * kCols; i += blockDim.x) {
            const int a = i / kCols, j = i % kCols;
            if (j < ncol) {
                fc[L.fc_D + a * W + j0 + j] = Dp[i];
                Cc[i] = fl[L.fl_C + a * W + j0 + j];
                DLc[i] = fl[L.fl_DL + a * W + j0 + j];
            }
        }
        for (int i = threadIdx.x; i < d * ncol; i += blockDim.x) {  // D_p^T, consecutive threads on consecutive a
            const int j = i / d, a = i % d;
            fc[L.fc_DT + (long long)(j0 + j) * d + a] = Dp[a * kCols + j];
        }
        __syncthreads();
        // D_new = D_p + DL_c + S_p C_c (old S_p); each thread keeps its results in registers
        float dn[128 * kCols / kThreads];
        int cnt = 0;
        for (int i = threadIdx.x; i < d * kCols; i += blockDim.x, ++cnt) {
            const int a = i / kCols, j = i % kCols;
            float x = 0.f;
            if (j < ncol) {
                x = Dp[i] + DLc[i];
                for (int b = 0; b < d; ++b) x += Sp[a * d + b] * Cc[b * kCols + j];
            }
            dn[cnt] = x;
        }
        __syncthreads();
        cnt = 0;
        for (int i = threadIdx.x; i < d * kCols; i += blockDim.x, ++cnt) Dp[i] = dn[cnt];
        for (int i = threadIdx.x; i < d * d; i += blockDim.x) Sp[i] += fl[L.fl_S + i];
        __syncthreads();
    }
}

// Recompute of a chunk's forward quantities shared by B3 and B5: W_c, X, T (rows = tokens).
__device__ void chunk_forward(const float *Qs, const float *Ks, int kd, const float *Sp, float *Ws, float *Xs,
                              float *Ts, int C, int d) {
    bgemm(Ws, C, Qs, d, 1, Ks, 1, kd, C, C, d, false, 1);        // W_c = L . Q K^T
    __syncthreads();
    bgemm(Xs, d, Ws, C, 1, Ks, kd, 1, C, d, C, false, 0, 1);     // X = W_c K
    bgemm(Xs, d, Qs, d, 1, Sp, d, 1, C, d, d, true);             //   + Q S_p
    __syncthreads();
    bgemm(Ts, C, Qs, d, 1, Xs, 1, d, C, C, d, false, 1);         // T = L . Q X^T
    __syncthreads();
}

// ---------------------------------------------------------------------------
// B3: per chunk, the upstream gradient G' (C x W) and the local reverse summaries
// Gam_c = G'^T Q, M_c = V'^T Q, Lam_c = Y_loc^T Q + Q^T Y_loc with Y_loc = P^T Q.
// ---------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(kThreads) bwd_local1(const T *q, const T *k, const T *v, const T *dout, float *ws,
                                                       BLayout L, int normalized, float eps) {
    extern __shared__ float sm[];
    const int c = blockIdx.x, hd = blockIdx.y, d = L.d, W = L.W, dv = L.dv, C = L.C, t0 = c * C;
    const int len = min(C, L.n - t0), kd = d + 1;
    float *Qs = sm, *Ks = Qs + C * d, *Vs = Ks + C * kd, *Gs = Vs + C * W, *Ws = Gs + C * W, *Xs = Ws + C * C;
    float *Ts = Xs + C * d, *Ns = Ts + C * C;  // Ns: num' (C x W), then Y_loc (C x d)
    load_rows(q + ((long long)hd * L.n + t0) * d, Qs, len, d, C, d, false);
    load_rows(k + ((long long)hd * L.n + t0) * d, Ks, len, d, C, kd, false);
    load_rows(v + ((long long)hd * L.n + t0) * dv, Vs, len, dv, C, W, true);
    load_rows(dout + ((long long)hd * L.n + t0) * dv, Gs, len, dv, C, W, false);
    const float *fc = rec(ws, L.o_fc, L.fc_len, L, hd, c);
    __syncthreads();
    chunk_forward(Qs, Ks, kd, fc + L.fc_S, Ws, Xs, Ts, C, d);
    if (normalized) {
        bgemm(Ns, W, Ts, C, 1, Vs, W, 1, C, W, C, false, 0, 1);   // num' = T V'
        bgemm(Ns, W, Qs, d, 1, fc + L.fc_D, W, 1, C, W, d, true);  //   + Q D_p
        __syncthreads();
        // G' = [g / (den + eps) | -(g . o) / (den + eps)], o = num / (den + eps)
        for (int r = threadIdx.x; r < C; r += blockDim.x) {
            if (r >= len) continue;  // rows beyond the sequence keep their zero gradient
            const float inv = 1.f / (Ns[r * W + dv] + eps);
            float go = 0.f;
            for (int j = 0; j < dv; ++j) {
                const float g = Gs[r * W + j];
                go += g * Ns[r * W + j] * inv;
                Gs[r * W + j] = g * inv;
            }
            Gs[r * W + dv] = -go * inv;
        }
        __syncthreads();
    }
    float *bl = rec(ws, L.o_bl, L.bl_len, L, hd, c);
    for (int i = threadIdx.x; i < C * W; i += blockDim.x) bl[L.bl_G + i] = Gs[i];
    float *Ps = Ts;  // T is not needed any more: P = L . (G' V'^T)
    bgemm(Ps, C, Gs, W, 1, Vs, 1, W, C, C, W, false, 1);
    __syncthreads();
    float *Ys = Ns;
    bgemm(Ys, d, Ps, 1, C, Qs, d, 1, C, d, C, false, 0, 3);      // Y_loc = P^T Q (P(t, j) = 0 for t < j)
    bgemm(bl + L.bl_Gam, d, Gs, 1, W, Qs, d, 1, W, d, C, false); // Gam_c = G'^T Q
    bgemm(bl + L.bl_M, d, Vs, 1, W, Qs, d, 1, W, d, C, false);   // M_c = V'^T Q
    __syncthreads();
    // Lam_c = Y_loc^T Q + Q^T Y_loc
    for (int idx = threadIdx.x; idx < d * d; idx += blockDim.x) {
        const int a = idx / d, b = idx % d;
        float s = 0.f;
        for (int t = 0; t < C; ++t) s += Ys[t * d + a] * Qs[t * d + b] + Qs[t * d + a] * Ys[t * d + b];
        bl[L.bl_Lam + idx] = s;
    }
}

// ---------------------------------------------------------------------------
// B4: reverse scan.  Block (column block of Lam, head) keeps the whole Gam_s and 32
// columns of Lam_s; from the last chunk back it records them, then
// Lam_s += Lam_c + Gam_s^T M_c + M_c^T Gam_s (old Gam_s) and Gam_s += Gam_c.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads) bwd_scan(float *ws, BLayout L) {
    extern __shared__ float sm[];
    const int hd = blockIdx.y, d = L.d, W = L.W, j0 = blockIdx.x * kCols, ncol = min(kCols, d - j0);
    // Gam_s (W x d), Lam_s columns (d x 32), the chunk's M_c (W x d) staged per chunk
    float *Gm = sm, *Lm = Gm + W * d, *Mc = Lm + d * kCols;
    for (int i = threadIdx.x; i < W * d; i += blockDim.x) Gm[i] = 0.f;
    for (int i = threadIdx.x; i < d * kCols; i += blockDim.x) Lm[i] = 0.f;
    __syncthreads();
    for (int c = L.nch - 1; c >= 0; --c) {
        float *bc = rec(ws, L.o_bc, L.bc_len, L, hd, c);
        const float *bl = rec(ws, L.o_bl, L.bl_len, L, hd, c);
        if (blockIdx.x == 0) {
            for (int i = threadIdx.x; i < W * d; i += blockDim.x) bc[L.bc_Gam + i] = Gm[i];
            for (int i = threadIdx.x; i < W * d; i += blockDim.x) {  // Gam_s^T, consecutive threads on consecutive w
                const int f = i / W, w = i % W;
                bc[L.bc_GamT + i] = Gm[w * d + f];
            }
        }
        for (int i = threadIdx.x; i < d * ncol; i += blockDim.x) {
            const int a = i / ncol, j = i % ncol;
            bc[L.bc_Lam + a * d + j0 + j] = Lm[a * kCols + j];
        }
        for (int i = threadIdx.x; i < W * d; i += blockDim.x) Mc[i] = bl[L.bl_M + i];
        __syncthreads();
        float ln[128 * kCols / kThreads];
        int cnt = 0;
        for (int i = threadIdx.x; i < d * kCols; i += blockDim.x, ++cnt) {
            const int a = i / kCols, j = i % kCols, b = j0 + j;
            float x = 0.f;
            if (j < ncol) {
                x = Lm[i] + bl[L.bl_Lam + a * d + b];
                for (int w = 0; w < W; ++w) x += Gm[w * d + a] * Mc[w * d + b] + Mc[w * d + a] * Gm[w * d + b];
            }
            ln[cnt] = x;
        }
        __syncthreads();
        cnt = 0;
        for (int i = threadIdx.x; i < d * kCols; i += blockDim.x, ++cnt) Lm[i] = ln[cnt];
        for (int i = threadIdx.x; i < W * d; i += blockDim.x) Gm[i] += bl[L.bl_Gam + i];
        __syncthreads();
    }
}

// ---------------------------------------------------------------------------
// B5: per chunk gradients.
// ---------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(kThreads) bwd_local2(const T *q, const T *k, const T *v, T *dq, T *dk, T *dvo,
                                                       float *ws, BLayout L) {
    extern __shared__ float sm[];
    const int c = blockIdx.x, hd = blockIdx.y, d = L.d, W = L.W, dv = L.dv, C = L.C, t0 = c * C;
    const int len = min(C, L.n - t0), kd = d + 1;
    float *Qs = sm, *Ks = Qs + C * d, *Vs = Ks + C * kd, *Gs = Vs + C * W, *Ws = Gs + C * W, *Xs = Ws + C * C;
    float *Ts = Xs + C * d, *Ps = Ts + C * C, *Ys = Ps + C * C, *Bs = Ys + C * d, *Os = Bs + C * C;  // Os: C x max(d, W)
    load_rows(q + ((long long)hd * L.n + t0) * d, Qs, len, d, C, d, false);
    load_rows(k + ((long long)hd * L.n + t0) * d, Ks, len, d, C, kd, false);
    load_rows(v + ((long long)hd * L.n + t0) * dv, Vs, len, dv, C, W, true);
    const float *fc = rec(ws, L.o_fc, L.fc_len, L, hd, c), *bl = rec(ws, L.o_bl, L.bl_len, L, hd, c);
    const float *bc = rec(ws, L.o_bc, L.bc_len, L, hd, c);
    for (int i = threadIdx.x; i < C * W; i += blockDim.x) Gs[i] = bl[L.bl_G + i];
    __syncthreads();
    chunk_forward(Qs, Ks, kd, fc + L.fc_S, Ws, Xs, Ts, C, d);
    bgemm(Ps, C, Gs, W, 1, Vs, 1, W, C, C, W, false, 1);          // P = L . G' V'^T
    __syncthreads();
    bgemm(Ys, d, Ps, 1, C, Qs, d, 1, C, d, C, false, 0, 3);       // Y = P^T Q
    bgemm(Ys, d, Vs, W, 1, bc + L.bc_Gam, d, 1, C, d, W, true);   //   + V' Gam_s
    __syncthreads();
    bgemm(Bs, C, Ys, d, 1, Ks, 1, kd, C, C, d, false, 1);         // B = L . Y K^T
    // dV' = T^T G' + X Gam_s^T   (columns < dv)
    bgemm(Os, W, Ts, 1, C, Gs, W, 1, C, W, C, false, 0, 3);
    bgemm(Os, W, Xs, d, 1, bc + L.bc_GamT, W, 1, C, W, d, true);
    __syncthreads();
    T *gv = dvo + ((long long)hd * L.n + t0) * dv;
    for (int i = threadIdx.x; i < len * dv; i += blockDim.x) from_f32(&gv[i], Os[(i / dv) * W + i % dv]);
    __syncthreads();
    // dQ = P X + G' D_p^T + Y S_p + B K
    bgemm(Os, d, Ps, C, 1, Xs, d, 1, C, d, C, false, 0, 1);
    bgemm(Os, d, Gs, W, 1, fc + L.fc_DT, d, 1, C, d, W, true);
    bgemm(Os, d, Ys, d, 1, fc + L.fc_S, d, 1, C, d, d, true);
    bgemm(Os, d, Bs, C, 1, Ks, kd, 1, C, d, C, true, 0, 1);
    __syncthreads();
    T *gq = dq + ((long long)hd * L.n + t0) * d;
    for (int i = threadIdx.x; i < len * d; i += blockDim.x) from_f32(&gq[i], Os[i]);
    __syncthreads();
    // dK = K Lam_s + W_c^T Y + B^T Q
    bgemm(Os, d, Ks, kd, 1, bc + L.bc_Lam, d, 1, C, d, d, false);
    bgemm(Os, d, Ws, 1, C, Ys, d, 1, C, d, C, true, 0, 3);
    bgemm(Os, d, Bs, 1, C, Qs, d, 1, C, d, C, true, 0, 3);
    __syncthreads();
    T *gk = dk + ((long long)hd * L.n + t0) * d;
    for (int i = threadIdx.x; i < len * d; i += blockDim.x) from_f32(&gk[i], Os[i]);
}

template <typename T>
cudaError_t backward_t(const Bwd2 &p, cudaStream_t s) {
    const BLayout L = make_layout(p.BH, p.n, p.d, p.dv, p.chunk);
    if (L.nch == 0) return cudaSuccess;
    float *ws = reinterpret_cast<float *>(p.ws + kWsHeaderBytes);
    const int C = L.C, d = L.d, W = L.W, kd = d + 1;
    const T *q = static_cast<const T *>(p.q), *k = static_cast<const T *>(p.k), *v = static_cast<const T *>(p.v);
    const T *g = static_cast<const T *>(p.dout);
    const dim3 grid(L.nch, p.BH);
    cudaError_t e;
    auto smem = [](size_t floats) { return (int)(floats * sizeof(float)); };
    const int sm1 = smem((size_t)C * d + (size_t)C * kd + (size_t)C * W + (size_t)C * C + (size_t)C * d);
    if ((e = cudaFuncSetAttribute(bwd_fwd_local<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm1))) return e;
    bwd_fwd_local<T><<<grid, kThreads, sm1, s>>>(q, k, v, ws, L);
    if ((e = cudaGetLastError())) return e;
    const int sm2 = smem((size_t)d * d + 3 * (size_t)d * kCols);
    if ((e = cudaFuncSetAttribute(bwd_fwd_scan, cudaFuncAttributeMaxDynamicSharedMemorySize, sm2))) return e;
    bwd_fwd_scan<<<dim3((W + kCols - 1) / kCols, p.BH), kThreads, sm2, s>>>(ws, L);
    if ((e = cudaGetLastError())) return e;
    const int sm3 = smem((size_t)C * d + (size_t)C * kd + 2 * (size_t)C * W + 2 * (size_t)C * C + (size_t)C * d +
                         (size_t)C * std::max(W, d));
    if ((e = cudaFuncSetAttribute(bwd_local1<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm3))) return e;
    bwd_local1<T><<<grid, kThreads, sm3, s>>>(q, k, v, g, ws, L, p.normalized, p.eps);
    if ((e = cudaGetLastError())) return e;
    const int sm4 = smem(2 * (size_t)W * d + (size_t)d * kCols);
    if ((e = cudaFuncSetAttribute(bwd_scan, cudaFuncAttributeMaxDynamicSharedMemorySize, sm4))) return e;
    bwd_scan<<<dim3((d + kCols - 1) / kCols, p.BH), kThreads, sm4, s>>>(ws, L);
    if ((e = cudaGetLastError())) return e;
    const int sm5 = smem((size_t)C * d + (size_t)C * kd + 2 * (size_t)C * W + 4 * (size_t)C * C + 2 * (size_t)C * d +
                         (size_t)C * std::max(W, d));
    if ((e = cudaFuncSetAttribute(bwd_local2<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm5))) return e;
    bwd_local2<T><<<grid, kThreads, sm5, s>>>(q, k, v, static_cast<T *>(p.dq), static_cast<T *>(p.dk),
                                               static_cast<T *>(p.dval), ws, L);
    return cudaGetLastError();
}

}  // namespace

size_t backward2_workspace_bytes(int BH, int n, int d, int dv, int chunk) {
    const BLayout L = make_layout(BH, n, d, dv, chunk);
    const size_t simt = kWsHeaderBytes + sizeof(float) * (size_t)L.total, tc = backward2_tc_workspace_bytes(BH, n);
    return simt > tc ? simt : tc;
}

cudaError_t backward2_launch(const Bwd2 &p, cudaStream_t stream) {
    if (backward2_tc_applicable(p)) return backward2_tc_launch(p, stream);
    return p.dt == HLA_BF16 ? backward_t<__nv_bfloat16>(p, stream) : backward_t<float>(p, stream);
}

}  // namespace hla
