// Third-order HLA forward, first correct version: one block per head runs the
// masked third-order streaming recurrence token by token (Algorithm 3 at
// gamma = 1, Theorem 3); the unmasked form outputs q^T S^K S^Q P^KV (Sec. 7.1).
// The state tuple lives in shared memory when it fits and otherwise in the
// caller's workspace.
//
// Masked outputs are read from the corrected state F = S^K S^Q P - G1 - G2 - G3
// and eta = S^K S^Q m^K - h1 - h2 - h3 (Eq. hla3-corrected-state), advanced by
// its own recurrence (Eq. hla3-corrected-recurrence).  Evaluating
// q^T S^K S^Q P - q^T (G1 + G2 + G3) instead would cancel a sum over all t^3
// index triples down to the O(t^2) admissible ones and lose about log10(t)
// digits in fp32.  G1..G3 and h1..h3 are still advanced (for the state tuple).
// Per token, with the previous states:
//   u1 = S^Q k,  a2 = S^K q,  a3 = S^K u1,  r1 = u1^T P,  r2 = q^T P
//   G1 += k r1^T, h1 += k (u1.m);  G2 += a2 r2^T, h2 += a2 (q.m);  G3 += a3 v^T, h3 += a3
//   F   += (a2 (k.q) + k (k.u1) + k (k.q)^2) v^T + k (k.q) r2^T
//   eta +=  a2 (k.q) + k (k.u1) + k (k.q)(q.m) + k (k.q)^2
//   S^K += k k^T, S^Q += q q^T, P += k v^T, m^K += k
//   masked:   num = q^T F,                 den = q^T eta
//   unmasked: num = (q^T S^K) S^Q P,       den = (q^T S^K) S^Q m^K
#include "hla_internal.h"

namespace hla {
namespace {

constexpr int kT3 = 256;

__host__ __device__ size_t state3_floats(int d, int dv) { return 2 * (size_t)d * d + 4 * (size_t)d * dv + 4 * (size_t)d; }
// state tuple followed by the corrected state F (d*dv) and eta (d)
__host__ __device__ size_t work3_floats(int d, int dv) { return state3_floats(d, dv) + (size_t)d * dv + d; }

bool state_in_smem(int d, int dv) {
    return sizeof(float) * (work3_floats(d, dv) + 8 * 128) <= 200 * 1024;
}

template <typename T>
__global__ void __launch_bounds__(kT3) hla3_serial_kernel(const T *__restrict__ q, const T *__restrict__ k,
                                                          const T *__restrict__ v, T *__restrict__ out, int n,
                                                          int d, int dv, int masked, int normalized, float eps,
                                                          const float *state_in,  // may alias state_out
                                                          float *state_out, float *ws_state,
                                                          int smem_state) {
    extern __shared__ float sm[];
    const int hd = blockIdx.x, tid = threadIdx.x;
    const size_t L = state3_floats(d, dv), LW = work3_floats(d, dv);
    float *st = smem_state ? sm : ws_state + (size_t)hd * LW;
    float *vecs = smem_state ? sm + LW : sm;
    float *SK = st, *SQ = SK + d * d, *P = SQ + d * d, *mK = P + d * dv;
    float *G1 = mK + d, *G2 = G1 + d * dv, *G3 = G2 + d * dv;
    float *h1 = G3 + d * dv, *h2 = h1 + d, *h3 = h2 + d;
    float *F = h3 + d, *eta = F + d * dv;
    float *qs = vecs, *ks = qs + 128, *vs = ks + 128, *u1 = vs + 128, *a2 = u1 + 128, *a3 = a2 + 128;
    float *r1 = a3 + 128, *r2 = r1 + 128;
    __shared__ float sc[8];

    const float *si = state_in ? state_in + (size_t)hd * L : nullptr;
    for (size_t i = tid; i < L; i += blockDim.x) {
        const bool gpart = i >= 2 * (size_t)d * d + (size_t)d * dv + d;  // G1..h3
        st[i] = (si && (masked || !gpart)) ? si[i] : 0.f;
    }
    __syncthreads();
    if (masked) {
        // corrected state of the initial tuple: F = S^K S^Q P - G1 - G2 - G3, eta likewise
        for (int i = tid; i < d * dv + d; i += blockDim.x) {
            const bool isF = i < d * dv;
            const int r = isF ? i / dv : i - d * dv, c = isF ? i % dv : 0;
            float acc = 0.f;
            if (si) {
                for (int a = 0; a < d; ++a) {
                    float skq = 0.f;  // (S^K S^Q)[r][a]
                    for (int b = 0; b < d; ++b) skq += SK[(size_t)r * d + b] * SQ[(size_t)b * d + a];
                    acc += skq * (isF ? P[(size_t)a * dv + c] : mK[a]);
                }
                acc -= isF ? (G1[i] + G2[i] + G3[i]) : (h1[r] + h2[r] + h3[r]);
            }
            (isF ? F[i] : eta[r]) = acc;
        }
        __syncthreads();
    }
    const T *Qh = q + (size_t)hd * n * d, *Kh = k + (size_t)hd * n * d, *Vh = v + (size_t)hd * n * dv;
    T *Oh = out + (size_t)hd * n * dv;
    for (int t = 0; t < n; ++t) {
        for (int i = tid; i < d; i += blockDim.x) { qs[i] = to_f32(Qh[(size_t)t * d + i]); ks[i] = to_f32(Kh[(size_t)t * d + i]); }
        for (int i = tid; i < dv; i += blockDim.x) vs[i] = to_f32(Vh[(size_t)t * dv + i]);
        __syncthreads();
        if (masked) {
            // u1 = S^Q k, a2 = S^K q (symmetric matrices: row r dotted with the vector)
            for (int r = tid; r < 2 * d; r += blockDim.x) {
                const float *M = r < d ? SQ + (size_t)r * d : SK + (size_t)(r - d) * d;
                const float *x = r < d ? ks : qs;
                float s = 0.f;
                for (int j = 0; j < d; ++j) s += M[j] * x[j];
                (r < d ? u1 : a2)[r < d ? r : r - d] = s;
            }
            __syncthreads();
            for (int r = tid; r < d; r += blockDim.x) {
                float s = 0.f;
                for (int j = 0; j < d; ++j) s += SK[(size_t)r * d + j] * u1[j];
                a3[r] = s;
            }
            if (tid == 0) {
                float s1 = 0.f, s2 = 0.f, kq = 0.f, ku = 0.f;
                for (int j = 0; j < d; ++j) {
                    s1 += u1[j] * mK[j]; s2 += qs[j] * mK[j]; kq += ks[j] * qs[j]; ku += ks[j] * u1[j];
                }
                sc[0] = s1; sc[1] = s2; sc[3] = kq; sc[4] = ku;
            }
            // row vectors u1^T P and q^T P into r1, r2 (dv long)
            for (int c = tid; c < 2 * dv; c += blockDim.x) {
                const int col = c < dv ? c : c - dv;
                const float *x = c < dv ? u1 : qs;
                float s = 0.f;
                for (int j = 0; j < d; ++j) s += x[j] * P[(size_t)j * dv + col];
                (c < dv ? r1 : r2)[col] = s;
            }
            __syncthreads();
            const float kq = sc[3], ku = sc[4];
            for (int i = tid; i < d * dv; i += blockDim.x) {
                const int r = i / dv, c = i % dv;
                G1[i] += ks[r] * r1[c];
                G2[i] += a2[r] * r2[c];
                G3[i] += a3[r] * vs[c];
                F[i] += (a2[r] * kq + ks[r] * ku + ks[r] * kq * kq) * vs[c] + ks[r] * kq * r2[c];
            }
            for (int r = tid; r < d; r += blockDim.x) {
                h1[r] += ks[r] * sc[0];
                h2[r] += a2[r] * sc[1];
                h3[r] += a3[r];
                eta[r] += a2[r] * kq + ks[r] * ku + ks[r] * kq * sc[1] + ks[r] * kq * kq;
            }
        }
        // inclusive first-order updates
        for (int i = tid; i < d * d; i += blockDim.x) {
            const int r = i / d, c = i % d;
            SK[i] += ks[r] * ks[c];
            SQ[i] += qs[r] * qs[c];
        }
        for (int i = tid; i < d * dv; i += blockDim.x) {
            const int r = i / dv, c = i % dv;
            P[i] += ks[r] * vs[c];
        }
        for (int r = tid; r < d; r += blockDim.x) mK[r] += ks[r];
        __syncthreads();
        // r1 = q^T S^K, then r2 = r1 S^Q
        for (int c = tid; c < d; c += blockDim.x) {
            float s = 0.f;
            for (int j = 0; j < d; ++j) s += qs[j] * SK[(size_t)j * d + c];
            r1[c] = s;
        }
        __syncthreads();
        for (int c = tid; c < d; c += blockDim.x) {
            float s = 0.f;
            for (int j = 0; j < d; ++j) s += r1[j] * SQ[(size_t)j * d + c];
            r2[c] = s;
        }
        __syncthreads();
        if (tid == 0) {
            float den = 0.f;
            if (masked)
                for (int j = 0; j < d; ++j) den += qs[j] * eta[j];
            else
                for (int j = 0; j < d; ++j) den += r2[j] * mK[j];
            sc[2] = den;
        }
        __syncthreads();
        for (int c = tid; c < dv; c += blockDim.x) {
            float num = 0.f;
            if (masked)
                for (int j = 0; j < d; ++j) num += qs[j] * F[(size_t)j * dv + c];
            else
                for (int j = 0; j < d; ++j) num += r2[j] * P[(size_t)j * dv + c];
            from_f32(&Oh[(size_t)t * dv + c], normalized ? num / (sc[2] + eps) : num);
        }
        __syncthreads();
    }
    if (state_out) {
        float *so = state_out + (size_t)hd * L;
        for (size_t i = tid; i < L; i += blockDim.x) so[i] = st[i];
    }
}

}  // namespace

size_t generic3_workspace_bytes(int BH, int n, int d, int dv, int chunk) {
    (void)n; (void)chunk;
    return kWsHeaderBytes + (state_in_smem(d, dv) ? 0 : sizeof(float) * (size_t)BH * work3_floats(d, dv));
}

cudaError_t generic3_forward(const Fwd2 &p, cudaStream_t stream) {
    const int in_smem = state_in_smem(p.d, p.dv) ? 1 : 0;
    const size_t smem = sizeof(float) * ((in_smem ? work3_floats(p.d, p.dv) : 0) + 8 * 128);
    float *ws_state = reinterpret_cast<float *>(p.ws + kWsHeaderBytes);
    cudaError_t e;
    if (p.dt == HLA_BF16) {
        if ((e = cudaFuncSetAttribute(hla3_serial_kernel<__nv_bfloat16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)smem)))
            return e;
        hla3_serial_kernel<__nv_bfloat16><<<p.BH, kT3, smem, stream>>>(
            static_cast<const __nv_bfloat16 *>(p.q), static_cast<const __nv_bfloat16 *>(p.k),
            static_cast<const __nv_bfloat16 *>(p.v), static_cast<__nv_bfloat16 *>(p.out), p.n, p.d, p.dv, p.masked,
            p.normalized, p.eps, p.state_in, p.state_out, ws_state, in_smem);
    } else {
        if ((e = cudaFuncSetAttribute(hla3_serial_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)smem)))
            return e;
        hla3_serial_kernel<float><<<p.BH, kT3, smem, stream>>>(
            static_cast<const float *>(p.q), static_cast<const float *>(p.k), static_cast<const float *>(p.v),
            static_cast<float *>(p.out), p.n, p.d, p.dv, p.masked, p.normalized, p.eps, p.state_in, p.state_out,
            ws_state, in_smem);
    }
    return cudaGetLastError();
}

}  // namespace hla
