// Generic second-order HLA forward: fp32 SIMT kernels for every supported
// shape (d, dv in {16,32,64,128}, any chunk <= 128, ragged last chunk,
// masked/unmasked, normalised or not, fp32 or bf16 tokens, optional states).
//
// Formulation (per head; rows are tokens of one chunk, "p" = carry-in prefix).
// With x_t = S_t q_t (S symmetric), masked second order is a causal linear
// attention with query q and key x (proof of Theorem 1: num_t =
// q_t^T sum_{j<=t} S_j q_j v_j^T), and the unmasked form is o_t = x_t^T C_t:
//   W  = L . (Q K^T)                     (L lower triangular incl. diagonal)
//   XL = W K,   X = XL + Q S_p            (rows x_t = S_t q_t)
//   masked:   T = L . (Q X^T),  num = T V + Q D_p,  den = T 1 + Q e_p
//   unmasked: T = L . (X Q^T),  num = T V + X C_p,  den = T 1 + X m_p
// Carries compose with the semidirect product of Eq. semidirect, written for
// D = S C - G and e = S m - h (D_{AB} = D_A + D_B + S_A C_B):
//   S += K^T K, C += Q^T V, m += Q^T 1,
//   D += XL^T V + S_p (Q^T V),  e += XL^T 1 + S_p (Q^T 1).
// Three launches: chunk-local summaries (all chunks in parallel), the carry
// scan (sequential over chunks, parallel over column tiles), outputs (all
// chunks in parallel).  Intermediates live in the caller's workspace.
#include <algorithm>

#include "hla_internal.h"

namespace hla {
namespace {

constexpr int kThreads = 256;
constexpr int kScanCols = 32;  // D/C columns per scan block

struct GLayout {
    int BH, n, d, dv, C, nch;
    // local record (per head, per chunk), offsets in floats
    int oW, oX, odS, odC, odm, odD, ode;
    long long rec_local;
    // carry record (per head, nch + 1 records)
    int oS, oC, om, oD, oe;
    long long rec_carry;
    long long carry_base;  // floats from scratch start to the carry records

    __host__ __device__ float *local(float *base, int hd, int c) const {
        return base + ((long long)hd * nch + c) * rec_local;
    }
    __host__ __device__ float *carry(float *base, int hd, int c) const {
        return base + carry_base + ((long long)hd * (nch + 1) + c) * rec_carry;
    }
};

inline long long up16(long long x) { return (x + 15) / 16 * 16; }

GLayout make_layout(int BH, int n, int d, int dv, int C) {
    GLayout L;
    L.BH = BH; L.n = n; L.d = d; L.dv = dv; L.C = C;
    L.nch = (n + C - 1) / C;
    long long o = 0;
    L.oW = (int)o; o += up16((long long)C * C);
    L.oX = (int)o; o += up16((long long)C * d);
    L.odS = (int)o; o += up16((long long)d * d);
    L.odC = (int)o; o += up16((long long)d * dv);
    L.odm = (int)o; o += up16(d);
    L.odD = (int)o; o += up16((long long)d * dv);
    L.ode = (int)o; o += up16(d);
    L.rec_local = o;
    o = 0;
    L.oS = (int)o; o += up16((long long)d * d);
    L.oC = (int)o; o += up16((long long)d * dv);
    L.om = (int)o; o += up16(d);
    L.oD = (int)o; o += up16((long long)d * dv);
    L.oe = (int)o; o += up16(d);
    L.rec_carry = o;
    L.carry_base = (long long)BH * L.nch * L.rec_local;
    return L;
}

long long state_floats(const GLayout &L) { return (long long)L.d * L.d + 2LL * L.d * L.dv + 2LL * L.d; }
// carry records, then a staging copy of state_in (used when state_out aliases it)
long long stage_base(const GLayout &L) { return up16(L.carry_base + (long long)L.BH * (L.nch + 1) * L.rec_carry); }
long long scratch_floats(const GLayout &L) { return stage_base(L) + up16((long long)L.BH * state_floats(L)); }

// ---------------------------------------------------------------------------
// kernel 1: chunk-local summaries
// ---------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(kThreads) g2_local_kernel(const T *__restrict__ q, const T *__restrict__ k,
                                                            const T *__restrict__ v, float *ws, GLayout L) {
    extern __shared__ float smem[];
    const int c = blockIdx.x, hd = blockIdx.y;
    const int d = L.d, dv = L.dv, C = L.C;
    const int t0 = c * C, len = min(C, L.n - t0);
    float *Qs = smem, *Ks = Qs + C * d, *Vs = Ks + C * d;
    const T *Qg = q + ((long long)hd * L.n + t0) * d;
    const T *Kg = k + ((long long)hd * L.n + t0) * d;
    const T *Vg = v + ((long long)hd * L.n + t0) * dv;
    for (int i = threadIdx.x; i < len * d; i += blockDim.x) { Qs[i] = to_f32(Qg[i]); Ks[i] = to_f32(Kg[i]); }
    for (int i = threadIdx.x; i < len * dv; i += blockDim.x) Vs[i] = to_f32(Vg[i]);
    __syncthreads();

    float *rec = L.local(ws, hd, c);
    float *W = rec + L.oW, *XL = rec + L.oX;
    // W_ti = q_t . k_i for i <= t (row stride C)
    for (int idx = threadIdx.x; idx < len * len; idx += blockDim.x) {
        const int t = idx / len, i = idx % len;
        float s = 0.f;
        if (i <= t)
            for (int r = 0; r < d; ++r) s += Qs[t * d + r] * Ks[i * d + r];
        W[t * C + i] = s;
    }
    // dS = K^T K, dC = Q^T V, dm = Q^T 1
    for (int idx = threadIdx.x; idx < d * d; idx += blockDim.x) {
        const int a = idx / d, b = idx % d;
        float s = 0.f;
        for (int t = 0; t < len; ++t) s += Ks[t * d + a] * Ks[t * d + b];
        rec[L.odS + idx] = s;
    }
    for (int idx = threadIdx.x; idx < d * dv; idx += blockDim.x) {
        const int a = idx / dv, b = idx % dv;
        float s = 0.f;
        for (int t = 0; t < len; ++t) s += Qs[t * d + a] * Vs[t * dv + b];
        rec[L.odC + idx] = s;
    }
    for (int a = threadIdx.x; a < d; a += blockDim.x) {
        float s = 0.f;
        for (int t = 0; t < len; ++t) s += Qs[t * d + a];
        rec[L.odm + a] = s;
    }
    __syncthreads();
    // XL = W K (row stride d)
    for (int idx = threadIdx.x; idx < len * d; idx += blockDim.x) {
        const int t = idx / d, r = idx % d;
        float s = 0.f;
        for (int i = 0; i <= t; ++i) s += W[t * C + i] * Ks[i * d + r];
        XL[idx] = s;
    }
    __syncthreads();
    // dD = XL^T V, de = XL^T 1
    for (int idx = threadIdx.x; idx < d * dv; idx += blockDim.x) {
        const int a = idx / dv, b = idx % dv;
        float s = 0.f;
        for (int t = 0; t < len; ++t) s += XL[t * d + a] * Vs[t * dv + b];
        rec[L.odD + idx] = s;
    }
    for (int a = threadIdx.x; a < d; a += blockDim.x) {
        float s = 0.f;
        for (int t = 0; t < len; ++t) s += XL[t * d + a];
        rec[L.ode + a] = s;
    }
}

// ---------------------------------------------------------------------------
// kernel 2: carry scan over chunks; block (hd, column tile of C/D)
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads) g2_scan_kernel(float *ws, GLayout L, int masked,
                                                           const float *__restrict__ state_in,
                                                           float *__restrict__ state_out) {
    extern __shared__ float smem[];
    const int hd = blockIdx.x, tile = blockIdx.y;
    const int d = L.d, dv = L.dv;
    const int c0 = tile * kScanCols, c1 = min(dv, c0 + kScanCols), nc = c1 - c0;
    const bool lead = (tile == 0);
    float *S = smem;           // d*d, running carry of S (private copy per block)
    float *m = S + d * d;      // d
    const long long st_len = (long long)d * d + 2LL * d * dv + 2LL * d;
    const long long oC = (long long)d * d, om = oC + (long long)d * dv, oG = om + d, oh = oG + (long long)d * dv;

    float *cur = L.carry(ws, hd, 0);
    const float *st = state_in ? state_in + hd * st_len : nullptr;
    for (int i = threadIdx.x; i < d * d; i += blockDim.x) S[i] = st ? st[i] : 0.f;
    for (int i = threadIdx.x; i < d; i += blockDim.x) m[i] = st ? st[om + i] : 0.f;
    __syncthreads();
    // initial carry: C, and D = S C - G, e = S m - h (masked)
    for (int idx = threadIdx.x; idx < d * nc; idx += blockDim.x) {
        const int a = idx / nc, b = c0 + idx % nc;
        cur[L.oC + a * dv + b] = st ? st[oC + a * dv + b] : 0.f;
        if (masked) {
            float s = 0.f;
            if (st) {
                for (int j = 0; j < d; ++j) s += S[a * d + j] * st[oC + j * dv + b];
                s -= st[oG + a * dv + b];
            }
            cur[L.oD + a * dv + b] = s;
        }
    }
    if (lead) {
        for (int i = threadIdx.x; i < d * d; i += blockDim.x) cur[L.oS + i] = S[i];
        for (int a = threadIdx.x; a < d; a += blockDim.x) {
            cur[L.om + a] = m[a];
            if (masked) {
                float s = 0.f;
                if (st) {
                    for (int j = 0; j < d; ++j) s += S[a * d + j] * st[om + j];
                    s -= st[oh + a];
                }
                cur[L.oe + a] = s;
            }
        }
    }
    __syncthreads();

    for (int c = 0; c < L.nch; ++c) {
        const float *loc = L.local(ws, hd, c);
        const float *prv = L.carry(ws, hd, c);
        float *nxt = L.carry(ws, hd, c + 1);
        for (int idx = threadIdx.x; idx < d * nc; idx += blockDim.x) {
            const int a = idx / nc, b = c0 + idx % nc;
            nxt[L.oC + a * dv + b] = prv[L.oC + a * dv + b] + loc[L.odC + a * dv + b];
            if (masked) {
                float s = prv[L.oD + a * dv + b] + loc[L.odD + a * dv + b];
                for (int j = 0; j < d; ++j) s += S[a * d + j] * loc[L.odC + j * dv + b];
                nxt[L.oD + a * dv + b] = s;
            }
        }
        if (lead && masked) {
            for (int a = threadIdx.x; a < d; a += blockDim.x) {
                float s = prv[L.oe + a] + loc[L.ode + a];
                for (int j = 0; j < d; ++j) s += S[a * d + j] * loc[L.odm + j];
                nxt[L.oe + a] = s;
            }
        }
        __syncthreads();  // the products above use S before this chunk's update
        for (int i = threadIdx.x; i < d * d; i += blockDim.x) S[i] += loc[L.odS + i];
        for (int a = threadIdx.x; a < d; a += blockDim.x) m[a] += loc[L.odm + a];
        __syncthreads();
        if (lead) {
            for (int i = threadIdx.x; i < d * d; i += blockDim.x) nxt[L.oS + i] = S[i];
            for (int a = threadIdx.x; a < d; a += blockDim.x) nxt[L.om + a] = m[a];
        }
    }
    if (!state_out) return;
    // final state in the paper's tuple: S, C, m, G = S C - D, h = S m - e (zeros if unmasked)
    const float *fin = L.carry(ws, hd, L.nch);
    float *so = state_out + hd * st_len;
    __syncthreads();
    for (int idx = threadIdx.x; idx < d * nc; idx += blockDim.x) {
        const int a = idx / nc, b = c0 + idx % nc;
        const float Cab = fin[L.oC + a * dv + b];
        so[oC + a * dv + b] = Cab;
        float g = 0.f;
        if (masked) {
            for (int j = 0; j < d; ++j) g += S[a * d + j] * fin[L.oC + j * dv + b];
            g -= fin[L.oD + a * dv + b];
        }
        so[oG + a * dv + b] = g;
    }
    if (lead) {
        for (int i = threadIdx.x; i < d * d; i += blockDim.x) so[i] = S[i];
        for (int a = threadIdx.x; a < d; a += blockDim.x) {
            so[om + a] = m[a];
            float hh = 0.f;
            if (masked) {
                for (int j = 0; j < d; ++j) hh += S[a * d + j] * m[j];
                hh -= fin[L.oe + a];
            }
            so[oh + a] = hh;
        }
    }
}

// ---------------------------------------------------------------------------
// kernel 3: outputs
// ---------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(kThreads) g2_out_kernel(const T *__restrict__ q, const T *__restrict__ v,
                                                          T *__restrict__ out, float *ws, GLayout L, int masked,
                                                          int normalized, float eps) {
    extern __shared__ float smem[];
    const int c = blockIdx.x, hd = blockIdx.y;
    const int d = L.d, dv = L.dv, C = L.C;
    const int t0 = c * C, len = min(C, L.n - t0);
    float *Qs = smem, *Vs = Qs + C * d, *den = Vs + C * dv;
    const T *Qg = q + ((long long)hd * L.n + t0) * d;
    const T *Vg = v + ((long long)hd * L.n + t0) * dv;
    for (int i = threadIdx.x; i < len * d; i += blockDim.x) Qs[i] = to_f32(Qg[i]);
    for (int i = threadIdx.x; i < len * dv; i += blockDim.x) Vs[i] = to_f32(Vg[i]);
    __syncthreads();
    float *rec = L.local(ws, hd, c);
    const float *cr = L.carry(ws, hd, c);
    float *X = rec + L.oX, *Tm = rec + L.oW;
    // X = XL + Q S_p (in place)
    for (int idx = threadIdx.x; idx < len * d; idx += blockDim.x) {
        const int t = idx / d, i = idx % d;
        float s = X[idx];
        for (int j = 0; j < d; ++j) s += Qs[t * d + j] * cr[L.oS + j * d + i];
        X[idx] = s;
    }
    __syncthreads();
    // T = L . (Q X^T) (masked) or L . (X Q^T) (unmasked)
    for (int idx = threadIdx.x; idx < len * len; idx += blockDim.x) {
        const int t = idx / len, j = idx % len;
        float s = 0.f;
        if (j <= t) {
            if (masked)
                for (int i = 0; i < d; ++i) s += Qs[t * d + i] * X[j * d + i];
            else
                for (int i = 0; i < d; ++i) s += X[t * d + i] * Qs[j * d + i];
        }
        Tm[t * C + j] = s;
    }
    __syncthreads();
    for (int t = threadIdx.x; t < len; t += blockDim.x) {
        float s = 0.f;
        for (int j = 0; j <= t; ++j) s += Tm[t * C + j];
        if (masked)
            for (int i = 0; i < d; ++i) s += Qs[t * d + i] * cr[L.oe + i];
        else
            for (int i = 0; i < d; ++i) s += X[t * d + i] * cr[L.om + i];
        den[t] = s;
    }
    __syncthreads();
    T *Og = out + ((long long)hd * L.n + t0) * dv;
    for (int idx = threadIdx.x; idx < len * dv; idx += blockDim.x) {
        const int t = idx / dv, b = idx % dv;
        float s = 0.f;
        for (int j = 0; j <= t; ++j) s += Tm[t * C + j] * Vs[j * dv + b];
        if (masked)
            for (int i = 0; i < d; ++i) s += Qs[t * d + i] * cr[L.oD + i * dv + b];
        else
            for (int i = 0; i < d; ++i) s += X[t * d + i] * cr[L.oC + i * dv + b];
        if (normalized) s = s / (den[t] + eps);
        from_f32(&Og[idx], s);
    }
}

template <typename T>
cudaError_t launch_all(const Fwd2 &p, const GLayout &L, float *scratch, cudaStream_t stream) {
    const T *q = static_cast<const T *>(p.q), *k = static_cast<const T *>(p.k), *v = static_cast<const T *>(p.v);
    T *out = static_cast<T *>(p.out);
    const size_t sm_local = sizeof(float) * (size_t)L.C * (2 * L.d + L.dv);
    const size_t sm_scan = sizeof(float) * (size_t)(L.d * L.d + L.d);
    const size_t sm_out = sizeof(float) * (size_t)L.C * (L.d + L.dv + 1);
    cudaError_t e;
    if ((e = cudaFuncSetAttribute(g2_local_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm_local)))
        return e;
    if ((e = cudaFuncSetAttribute(g2_scan_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm_scan)))
        return e;
    if ((e = cudaFuncSetAttribute(g2_out_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm_out)))
        return e;
    if (L.nch > 0) {
        g2_local_kernel<T><<<dim3(L.nch, L.BH), kThreads, sm_local, stream>>>(q, k, v, scratch, L);
        if ((e = cudaGetLastError())) return e;
    }
    const int tiles = (L.dv + kScanCols - 1) / kScanCols;
    g2_scan_kernel<<<dim3(L.BH, tiles), kThreads, sm_scan, stream>>>(scratch, L, p.masked, p.state_in, p.state_out);
    if ((e = cudaGetLastError())) return e;
    if (L.nch > 0) {
        g2_out_kernel<T><<<dim3(L.nch, L.BH), kThreads, sm_out, stream>>>(q, v, out, scratch, L, p.masked,
                                                                           p.normalized, p.eps);
        if ((e = cudaGetLastError())) return e;
    }
    return cudaSuccess;
}

}  // namespace

size_t generic2_workspace_bytes(int BH, int n, int d, int dv, int chunk) {
    GLayout L = make_layout(BH, n, d, dv, chunk);
    return kWsHeaderBytes + sizeof(float) * (size_t)scratch_floats(L);
}

cudaError_t generic2_forward(const Fwd2 &p, cudaStream_t stream) {
    GLayout L = make_layout(p.BH, p.n, p.d, p.dv, p.chunk);
    float *scratch = reinterpret_cast<float *>(p.ws + kWsHeaderBytes);
    Fwd2 pp = p;
    if (p.state_in && p.state_out) {
        // several blocks of one head read state_in while others write state_out:
        // read a private copy when the two ranges overlap
        const size_t bytes = sizeof(float) * (size_t)p.BH * (size_t)state_floats(L);
        const char *a = reinterpret_cast<const char *>(p.state_in), *b = reinterpret_cast<const char *>(p.state_out);
        if (a < b + bytes && b < a + bytes) {
            float *copy = scratch + stage_base(L);
            cudaError_t e = cudaMemcpyAsync(copy, p.state_in, bytes, cudaMemcpyDeviceToDevice, stream);
            if (e != cudaSuccess) return e;
            pp.state_in = copy;
        }
    }
    if (p.dt == HLA_BF16) return launch_all<__nv_bfloat16>(pp, L, scratch, stream);
    return launch_all<float>(pp, L, scratch, stream);
}

}  // namespace hla
