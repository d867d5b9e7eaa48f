// Streaming decode step of second-order HLA (online updates after Theorem 1,
// outputs of Theorem 1 / Eq. hla-row), one block per head.
//
// The step is a read-modify-write of the fp32 state tuple (S, C, m, G, h):
//   masked:  G' = G + k (k^T C),  h' = h + k (k^T m)       (previous C, m)
//   S' = S + k k^T,  C' = C + q v^T,  m' = m + q
//   u' = S' q = S q + k (k.q)                               (S symmetric)
//   num = u'^T C' - q^T G' = u'^T C + (u'.q) v^T - q^T G - (q.k)(k^T C)
//   den = u'.m' - q.h'     = u'.(m + q) - q.h - (q.k)(k.m)
// so one pass over S (giving u'), one pass over C (the column sums k^T C and
// u'^T C), then one pass over G that reads q^T G from the old values and writes
// G' = G + k (k^T C) at once.  The unmasked form skips G and h (and leaves them
// untouched).
//
// Memory access: every matrix is read and written once with 16-byte accesses,
// consecutive threads on consecutive columns, all of a thread's loads of a
// matrix issued before any of its arithmetic.
#include "hla_internal.h"

namespace hla {
namespace {

constexpr int kStepThreads = 256;
constexpr int kMaxUnits = 16;  // float4 units per thread for a 128 x 128 matrix

template <int W>
__device__ __forceinline__ float group_sum(float x) {
#pragma unroll
    for (int o = W / 2; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o, W);
    return x;
}

__device__ __forceinline__ float group_sum_rt(float x, int w) {
    switch (w) {
        case 4: return group_sum<4>(x);
        case 8: return group_sum<8>(x);
        case 16: return group_sum<16>(x);
        default: return group_sum<32>(x);
    }
}

// block-wide sum of up to three values; every thread receives the result
__device__ __forceinline__ void block_sum3(float &a, float &b, float &c, float *red) {
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    a = group_sum<32>(a); b = group_sum<32>(b); c = group_sum<32>(c);
    __syncthreads();
    if (lane == 0) { red[wid * 3 + 0] = a; red[wid * 3 + 1] = b; red[wid * 3 + 2] = c; }
    __syncthreads();
    a = b = c = 0.f;
#pragma unroll
    for (int w = 0; w < kStepThreads / 32; ++w) { a += red[w * 3]; b += red[w * 3 + 1]; c += red[w * 3 + 2]; }
}

template <typename T>
__global__ void __launch_bounds__(kStepThreads, 2)
step2_kernel(const T *__restrict__ q, const T *__restrict__ k, const T *__restrict__ v, T *__restrict__ out,
             float *__restrict__ state, int d, int dv, int masked, int normalized, float eps) {
    __shared__ float qs[128], ks[128], vs[128], us[128], ms[128];
    __shared__ float red[3 * (kStepThreads / 32)];
    __shared__ float part[kStepThreads][12];
    __shared__ float kC[128], uC[128], qG[128];

    const int hd = blockIdx.x, tid = threadIdx.x;
    const long long st_len = (long long)d * d + 2LL * d * dv + 2LL * d;
    float *S = state + hd * st_len;
    float *Cm = S + (long long)d * d;
    float *m = Cm + (long long)d * dv;
    float *G = m + d;
    float *h = G + (long long)d * dv;

    float kq = 0.f, km = 0.f, qh = 0.f;
    if (tid < d) {
        const float qi = to_f32(q[(long long)hd * d + tid]), ki = to_f32(k[(long long)hd * d + tid]);
        const float mi = m[tid];
        qs[tid] = qi; ks[tid] = ki; ms[tid] = mi;
        kq = ki * qi; km = ki * mi;
        if (masked) qh = qi * h[tid];
    }
    if (tid < dv) vs[tid] = to_f32(v[(long long)hd * dv + tid]);
    block_sum3(kq, km, qh, red);  // also a barrier: qs, ks, vs visible

    // ---- pass over S: u = S q, S' = S + k k^T --------------------------------
    {
        const int w = d >> 2;  // float4 units per row of S
        const int nunits = (d * d) >> 2;
        const float4 *S4 = reinterpret_cast<const float4 *>(S);
        float4 *S4w = reinterpret_cast<float4 *>(S);
        float4 reg[kMaxUnits];
#pragma unroll
        for (int i = 0; i < kMaxUnits; ++i) {
            const int f = tid + i * kStepThreads;
            if (f < nunits) reg[i] = S4[f];
        }
#pragma unroll
        for (int i = 0; i < kMaxUnits; ++i) {
            const int f = tid + i * kStepThreads;
            if (i * kStepThreads < nunits) {  // uniform per iteration: shuffles stay convergent
                float part_u = 0.f;
                if (f < nunits) {
                    const int row = f / w, c4 = (f % w) * 4;
                    const float4 s = reg[i];
                    part_u = s.x * qs[c4] + s.y * qs[c4 + 1] + s.z * qs[c4 + 2] + s.w * qs[c4 + 3];
                    const float kr = ks[row];
                    S4w[f] = make_float4(s.x + kr * ks[c4], s.y + kr * ks[c4 + 1], s.z + kr * ks[c4 + 2],
                                         s.w + kr * ks[c4 + 3]);
                }
                part_u = group_sum_rt(part_u, w);
                if (f < nunits && (f % w) == 0) {
                    const int row = f / w;
                    us[row] = part_u + ks[row] * kq;  // u' = S q + k (k.q)
                }
            }
        }
    }
    __syncthreads();

    // u'.q and u'.(m + q)
    float uq = 0.f, um = 0.f, dummy = 0.f;
    if (tid < d) { uq = us[tid] * qs[tid]; um = us[tid] * (ms[tid] + qs[tid]); }
    block_sum3(uq, um, dummy, red);

    // ---- pass over C: column sums k^T C, u'^T C; C' = C + q v^T --------------
    const int wv = dv >> 2;
    const int nunits = (d * dv) >> 2;
    const int c4 = (tid % wv) * 4;  // fixed column group of this thread
    {
        float4 acc_kC = make_float4(0.f, 0.f, 0.f, 0.f), acc_uC = acc_kC;
        const float4 *C4 = reinterpret_cast<const float4 *>(Cm);
        float4 *C4w = reinterpret_cast<float4 *>(Cm);
        float4 creg[kMaxUnits];
#pragma unroll
        for (int i = 0; i < kMaxUnits; ++i) {
            const int f = tid + i * kStepThreads;
            if (f < nunits) creg[i] = C4[f];
        }
        const float v0 = vs[c4], v1 = vs[c4 + 1], v2 = vs[c4 + 2], v3 = vs[c4 + 3];
#pragma unroll
        for (int i = 0; i < kMaxUnits; ++i) {
            const int f = tid + i * kStepThreads;
            if (f < nunits) {
                const int row = f / wv;
                const float4 c = creg[i];
                const float kr = ks[row], ur = us[row], qr = qs[row];
                acc_kC.x += kr * c.x; acc_kC.y += kr * c.y; acc_kC.z += kr * c.z; acc_kC.w += kr * c.w;
                acc_uC.x += ur * c.x; acc_uC.y += ur * c.y; acc_uC.z += ur * c.z; acc_uC.w += ur * c.w;
                C4w[f] = make_float4(c.x + qr * v0, c.y + qr * v1, c.z + qr * v2, c.w + qr * v3);
            }
        }
        part[tid][0] = acc_kC.x; part[tid][1] = acc_kC.y; part[tid][2] = acc_kC.z; part[tid][3] = acc_kC.w;
        part[tid][4] = acc_uC.x; part[tid][5] = acc_uC.y; part[tid][6] = acc_uC.z; part[tid][7] = acc_uC.w;
    }
    __syncthreads();
    if (tid < dv) {
        const int grp = tid >> 2, comp = tid & 3;
        float a = 0.f, b = 0.f;
        for (int g = grp; g < kStepThreads; g += wv) { a += part[g][comp]; b += part[g][4 + comp]; }
        kC[tid] = a; uC[tid] = b;
    }
    __syncthreads();

    // ---- pass over G: column sums q^T G (old G); G' = G + k (k^T C) -----------
    if (masked) {
        float4 acc_qG = make_float4(0.f, 0.f, 0.f, 0.f);
        const float4 *G4 = reinterpret_cast<const float4 *>(G);
        float4 *G4w = reinterpret_cast<float4 *>(G);
        float4 greg[kMaxUnits];
#pragma unroll
        for (int i = 0; i < kMaxUnits; ++i) {
            const int f = tid + i * kStepThreads;
            if (f < nunits) greg[i] = G4[f];
        }
        const float a0 = kC[c4], a1 = kC[c4 + 1], a2 = kC[c4 + 2], a3 = kC[c4 + 3];
#pragma unroll
        for (int i = 0; i < kMaxUnits; ++i) {
            const int f = tid + i * kStepThreads;
            if (f < nunits) {
                const int row = f / wv;
                const float kr = ks[row], qr = qs[row];
                const float4 g = greg[i];
                acc_qG.x += qr * g.x; acc_qG.y += qr * g.y; acc_qG.z += qr * g.z; acc_qG.w += qr * g.w;
                G4w[f] = make_float4(g.x + kr * a0, g.y + kr * a1, g.z + kr * a2, g.w + kr * a3);
            }
        }
        part[tid][8] = acc_qG.x; part[tid][9] = acc_qG.y; part[tid][10] = acc_qG.z; part[tid][11] = acc_qG.w;
        if (tid < d) h[tid] += ks[tid] * km;
        __syncthreads();
        if (tid < dv) {
            const int grp = tid >> 2, comp = tid & 3;
            float c = 0.f;
            for (int g = grp; g < kStepThreads; g += wv) c += part[g][8 + comp];
            qG[tid] = c;
        }
        __syncthreads();
    }

    // ---- m' = m + q; output ---------------------------------------------------
    if (tid < d) m[tid] = ms[tid] + qs[tid];
    if (tid < dv) {
        float num = uC[tid] + uq * vs[tid];
        float den = um;
        if (masked) {
            num -= qG[tid] + kq * kC[tid];
            den -= qh + kq * km;
        }
        from_f32(&out[(long long)hd * dv + tid], normalized ? num / (den + eps) : num);
    }
}

}  // namespace

cudaError_t step2_launch(const void *q, const void *k, const void *v, void *out, hla_dtype dt, int BH, int d, int dv,
                         int masked, int normalized, float eps, float *state, cudaStream_t stream) {
    if (BH == 0) return cudaSuccess;
    if (dt == HLA_BF16)
        step2_kernel<__nv_bfloat16><<<BH, kStepThreads, 0, stream>>>(
            static_cast<const __nv_bfloat16 *>(q), static_cast<const __nv_bfloat16 *>(k),
            static_cast<const __nv_bfloat16 *>(v), static_cast<__nv_bfloat16 *>(out), state, d, dv, masked,
            normalized, eps);
    else
        step2_kernel<float><<<BH, kStepThreads, 0, stream>>>(static_cast<const float *>(q),
                                                              static_cast<const float *>(k),
                                                              static_cast<const float *>(v),
                                                              static_cast<float *>(out), state, d, dv, masked,
                                                              normalized, eps);
    return cudaGetLastError();
}

}  // namespace hla
