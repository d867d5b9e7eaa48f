// Streaming decode step of second-order HLA (online updates after Theorem 1,
// outputs of Theorem 1 / Eq. hla-row), one block per SM working through heads.
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
// Memory access: every matrix is read once into shared memory by a 1-D bulk copy
// (one instruction per matrix, completing on an mbarrier), issued a pass or more
// ahead of its use, and written once with 16-byte stores; consecutive threads on
// consecutive columns.
#include "hla_internal.h"
#include "sm103_prims.cuh"

namespace hla {
namespace {

constexpr int kStepThreads = 512;
constexpr int kMaxUnits = 128 * 128 / 4 / kStepThreads;  // float4 units per thread for a 128 x 128 matrix

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

// Sums over the 32 lanes of a warp of eight values v[0..7] at once (9 shuffles instead of 40): on
// return, lane l holds the sum of v[l >> 2] (each step keeps half of the values a lane still holds)
__device__ __forceinline__ float warp_sum8(float (&v)[8]) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const bool up = (lane & 16) != 0;
        const float send = up ? v[i] : v[i + 4], keep = up ? v[i + 4] : v[i];
        v[i] = keep + __shfl_xor_sync(0xffffffffu, send, 16);
    }
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        const bool up = (lane & 8) != 0;
        const float send = up ? v[i] : v[i + 2], keep = up ? v[i + 2] : v[i];
        v[i] = keep + __shfl_xor_sync(0xffffffffu, send, 8);
    }
    {
        const bool up = (lane & 4) != 0;
        const float send = up ? v[0] : v[1], keep = up ? v[1] : v[0];
        v[0] = keep + __shfl_xor_sync(0xffffffffu, send, 4);
    }
    float x = v[0];
    x += __shfl_xor_sync(0xffffffffu, x, 2);
    x += __shfl_xor_sync(0xffffffffu, x, 1);
    return x;
}

// sum_i a[i] b[i] over shared-memory vectors, computed by every warp on its own (no block barrier)
__device__ __forceinline__ float warp_dot(const float *a, const float *b, int n) {
    float s = 0.f;
    for (int i = threadIdx.x & 31; i < n; i += 32) s += a[i] * b[i];
    return group_sum<32>(s);
}

// 1-D bulk copy global -> shared (16-byte aligned, a multiple of 16 bytes), completing on `bar`
__device__ __forceinline__ void bulk_copy(void *dst, const void *src, uint32_t bytes, uint64_t *bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                 ::"r"(sm103::smem_u32(dst)), "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes),
                   "r"(sm103::smem_u32(bar))
                 : "memory");
}
constexpr unsigned long long kCopyWaitNs = 2000000000ull;
__device__ __forceinline__ void store4(float4 *p, float4 v) { *p = v; }

// One block per SM, heads hd = blockIdx.x, + gridDim.x, ...  The state of a head is staged in shared
// memory in three buffers, one per pass (S; C with m; G with h), each refilled with the next head's
// part as soon as its pass has read it, so that while one pass works the copies of the next two
// parts (and of the next head's tokens) are in flight.  Thread 0 issues each refill as one bulk copy
// on the buffer's mbarrier (phase = the block's head count); every thread waits on it, bounded: a
// copy that never lands ends the block.  Updated values go to global memory straight from registers.
//
// kSDE: the state is (S, D, e) with D = S C - G and e = S m - h (masked operator only; rows of the
// per-head record: S d*d | D d*dv | e d).  A token then updates
//   S' = S + k k^T,  u' = S' q,  D' = D + u' v^T,  e' = e + u'
// and num = q^T D' = q^T D + (q.u') v^T, den = q.e' = q.e + q.u': one pass over S and one over D.
template <typename T, bool kSDE>
__global__ void __launch_bounds__(kStepThreads, 1)
step2_kernel(const T *__restrict__ q, const T *__restrict__ k, const T *__restrict__ v, T *__restrict__ out,
             float *__restrict__ state, int BH, int d, int dv, int masked, int normalized, float eps) {
    extern __shared__ float4 dyn[];
    __shared__ float qs[128], ks[128], vs[128], us[128];
    __shared__ float part[kStepThreads][12];
    __shared__ float kC[128], uC[128], qG[128];
    __shared__ uint64_t bar[3];  // S and tokens; (C, m) or (D, e); (G, h)

    const int tid = threadIdx.x;
    if (kSDE) masked = 0;  // staging as for (S, C, m): no third buffer
    const long long st_len = kSDE ? (long long)d * d + (long long)d * dv + d : (long long)d * d + 2LL * d * dv + 2LL * d;
    const int nS = (d * d) >> 2, nCm = (d * dv + d) >> 2;  // float4 units of S and of (C, m) / (G, h)
    const int nt_q = d * (int)sizeof(T) / 16, nt_v = dv * (int)sizeof(T) / 16;  // 16-byte token chunks
    float4 *bS = dyn, *bC = bS + nS, *bG = bC + nCm;
    float4 *bT = bG + (masked ? nCm : 0);  // raw tokens q | k | v
    const T *tq = reinterpret_cast<const T *>(bT), *tk = tq + d, *tv = tk + d;

    // thread 0 issues the copies: after a block barrier that ends the generic reads of the buffer
    auto load_S = [&](int hd) {  // S and the head's tokens
        if (tid == 0) {
            sm103::fence_async_smem();
            sm103::mbar_arrive_expect_tx(&bar[0], (uint32_t)(16 * (nS + 2 * nt_q + nt_v)));
            bulk_copy(bS, state + hd * st_len, 16u * nS, &bar[0]);
            bulk_copy(bT, q + (long long)hd * d, 16u * nt_q, &bar[0]);
            bulk_copy(bT + nt_q, k + (long long)hd * d, 16u * nt_q, &bar[0]);
            bulk_copy(bT + 2 * nt_q, v + (long long)hd * dv, 16u * nt_v, &bar[0]);
        }
    };
    auto load_part = [&](float4 *dst, int hd, long long off, int b) {  // (C, m), (D, e) or (G, h)
        if (tid == 0) {
            sm103::fence_async_smem();
            sm103::mbar_arrive_expect_tx(&bar[b], 16u * nCm);
            bulk_copy(dst, state + hd * st_len + off, 16u * nCm, &bar[b]);
        }
    };
    const long long offC = (long long)d * d, offG = offC + (long long)d * dv + d;

    int hd = blockIdx.x;
    if (hd >= BH) return;
    if (tid == 0) {
        for (int b = 0; b < 3; ++b) sm103::mbar_init(&bar[b], 1);
        sm103::fence_mbar_init();
    }
    __syncthreads();
    load_S(hd);
    load_part(bC, hd, offC, 1);
    if (masked) load_part(bG, hd, offG, 2);
    for (uint32_t par = 0; hd < BH; hd += gridDim.x, par ^= 1u) {
        const int nx = hd + gridDim.x;  // this block's next head (none: empty copy groups)
        float *S = state + hd * st_len;
        float *Cm = S + offC;
        float *m = Cm + (long long)d * dv;
        float *G = S + offG;
        float *h = G + (long long)d * dv;

        // ---- tokens, k.q ----
        if (!sm103::mbar_wait(&bar[0], par, kCopyWaitNs)) return;  // S and tokens of this head
        if (tid < d) {
            qs[tid] = to_f32(tq[tid]);
            ks[tid] = to_f32(tk[tid]);
        }
        if (tid < dv) vs[tid] = to_f32(tv[tid]);
        __syncthreads();
        const float kq = warp_dot(ks, qs, d);

        // ---- pass over S: u = S q, S' = S + k k^T ----
        if (d == 128 && kMaxUnits == 8) {
            // a warp covers one row per unit (rows warp + 16 i): the eight row sums in one reduction
            float4 *Sg = reinterpret_cast<float4 *>(S);
            const int c4 = (tid & 31) * 4;
            const float q0 = qs[c4], q1 = qs[c4 + 1], q2 = qs[c4 + 2], q3 = qs[c4 + 3];
            const float k0 = ks[c4], k1 = ks[c4 + 1], k2 = ks[c4 + 2], k3 = ks[c4 + 3];
            float pu[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const int f = tid + i * kStepThreads;
                const float4 sv = bS[f];
                pu[i] = sv.x * q0 + sv.y * q1 + sv.z * q2 + sv.w * q3;
                const float kr = ks[f >> 5];
                store4(Sg + f, make_float4(sv.x + kr * k0, sv.y + kr * k1, sv.z + kr * k2, sv.w + kr * k3));
            }
            const float su = warp_sum8(pu);
            if ((tid & 3) == 0) {
                const int row = (tid >> 5) + 16 * ((tid & 31) >> 2);
                us[row] = su + ks[row] * kq;  // u' = S q + k (k.q)
            }
        } else {
            const int w = d >> 2;  // float4 units per row of S
            float4 *Sg = reinterpret_cast<float4 *>(S);
#pragma unroll
            for (int i = 0; i < kMaxUnits; ++i) {
                const int f = tid + i * kStepThreads;
                if (i * kStepThreads < nS) {  // uniform per iteration: shuffles stay convergent
                    float part_u = 0.f;
                    if (f < nS) {
                        const int row = f / w, c4 = (f % w) * 4;
                        const float4 sv = bS[f];
                        part_u = sv.x * qs[c4] + sv.y * qs[c4 + 1] + sv.z * qs[c4 + 2] + sv.w * qs[c4 + 3];
                        const float kr = ks[row];
                        store4(Sg + f, make_float4(sv.x + kr * ks[c4], sv.y + kr * ks[c4 + 1],
                                                      sv.z + kr * ks[c4 + 2], sv.w + kr * ks[c4 + 3]));
                    }
                    part_u = group_sum_rt(part_u, w);
                    if (f < nS && (f % w) == 0) {
                        const int row = f / w;
                        us[row] = part_u + ks[row] * kq;  // u' = S q + k (k.q)
                    }
                }
            }
        }
        __syncthreads();  // S buffer read, u' complete
        if (nx < BH) load_S(nx);

        if constexpr (kSDE) {
            // ---- pass over D: column sums q^T D (old D); D' = D + u' v^T; e' = e + u' ----
            if (!sm103::mbar_wait(&bar[1], par, kCopyWaitNs)) return;  // (D, e) of this head
            const float *ev = reinterpret_cast<const float *>(bC + ((d * dv) >> 2));
            float *eg = Cm + (long long)d * dv;
            if (tid < d) eg[tid] = ev[tid] + us[tid];
            const float qe = warp_dot(qs, ev, d), uq = warp_dot(us, qs, d);
            const int wv = dv >> 2, nD = (d * dv) >> 2, c4 = (tid % wv) * 4;
            {
                float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
                float4 *Dg = reinterpret_cast<float4 *>(Cm);
                const float v0 = vs[c4], v1 = vs[c4 + 1], v2 = vs[c4 + 2], v3 = vs[c4 + 3];
#pragma unroll
                for (int i = 0; i < kMaxUnits; ++i) {
                    const int f = tid + i * kStepThreads;
                    if (f < nD) {
                        const int row = f / wv;
                        const float4 c = bC[f];
                        const float qr = qs[row], ur = us[row];
                        acc.x += qr * c.x; acc.y += qr * c.y; acc.z += qr * c.z; acc.w += qr * c.w;
                        store4(Dg + f, make_float4(c.x + ur * v0, c.y + ur * v1, c.z + ur * v2, c.w + ur * v3));
                    }
                }
                part[tid][0] = acc.x; part[tid][1] = acc.y; part[tid][2] = acc.z; part[tid][3] = acc.w;
            }
            __syncthreads();  // (D, e) buffer read
            if (nx < BH) load_part(bC, nx, offC, 1);
            if (tid < dv) {
                const int grp = tid >> 2, comp = tid & 3;
                float a = 0.f;
                for (int g = grp; g < kStepThreads; g += wv) a += part[g][comp];
                const float num = a + uq * vs[tid];
                from_f32(&out[(long long)hd * dv + tid], normalized ? num / (qe + uq + eps) : num);
            }
            __syncthreads();  // qs, ks, vs, us, part read before the next head rewrites them
            continue;
        }

        // ---- pass over C: column sums k^T C, u'^T C; C' = C + q v^T; m' = m + q ----
        if (!sm103::mbar_wait(&bar[1], par, kCopyWaitNs)) return;  // (C, m) of this head
        const float *mv = reinterpret_cast<const float *>(bC + ((d * dv) >> 2));
        if (tid < d) m[tid] = mv[tid] + qs[tid];
        const float uq = warp_dot(us, qs, d), km = warp_dot(ks, mv, d);
        const float um = warp_dot(us, mv, d) + uq;  // u'.(m + q)
        const int wv = dv >> 2;
        const int nC = (d * dv) >> 2;
        const int c4 = (tid % wv) * 4;  // fixed column group of this thread
        {
            float4 acc_kC = make_float4(0.f, 0.f, 0.f, 0.f), acc_uC = acc_kC;
            float4 *Cg = reinterpret_cast<float4 *>(Cm);
            const float v0 = vs[c4], v1 = vs[c4 + 1], v2 = vs[c4 + 2], v3 = vs[c4 + 3];
#pragma unroll
            for (int i = 0; i < kMaxUnits; ++i) {
                const int f = tid + i * kStepThreads;
                if (f < nC) {
                    const int row = f / wv;
                    const float4 c = bC[f];
                    const float kr = ks[row], ur = us[row], qr = qs[row];
                    acc_kC.x += kr * c.x; acc_kC.y += kr * c.y; acc_kC.z += kr * c.z; acc_kC.w += kr * c.w;
                    acc_uC.x += ur * c.x; acc_uC.y += ur * c.y; acc_uC.z += ur * c.z; acc_uC.w += ur * c.w;
                    store4(Cg + f, make_float4(c.x + qr * v0, c.y + qr * v1, c.z + qr * v2, c.w + qr * v3));
                }
            }
            part[tid][0] = acc_kC.x; part[tid][1] = acc_kC.y; part[tid][2] = acc_kC.z; part[tid][3] = acc_kC.w;
            part[tid][4] = acc_uC.x; part[tid][5] = acc_uC.y; part[tid][6] = acc_uC.z; part[tid][7] = acc_uC.w;
        }
        __syncthreads();  // (C, m) buffer read
        if (nx < BH) load_part(bC, nx, offC, 1);
        if (tid < dv) {
            const int grp = tid >> 2, comp = tid & 3;
            float a = 0.f, b = 0.f;
            for (int g = grp; g < kStepThreads; g += wv) { a += part[g][comp]; b += part[g][4 + comp]; }
            kC[tid] = a; uC[tid] = b;
        }
        __syncthreads();

        // ---- pass over G: column sums q^T G (old G); G' = G + k (k^T C); h' = h + k (k.m) ----
        float qh = 0.f;
        if (masked) {
            if (!sm103::mbar_wait(&bar[2], par, kCopyWaitNs)) return;  // (G, h) of this head
            const float *hv = reinterpret_cast<const float *>(bG + nC);
            if (tid < d) h[tid] = hv[tid] + ks[tid] * km;
            qh = warp_dot(qs, hv, d);
            float4 acc_qG = make_float4(0.f, 0.f, 0.f, 0.f);
            float4 *Gg = reinterpret_cast<float4 *>(G);
            const float a0 = kC[c4], a1 = kC[c4 + 1], a2 = kC[c4 + 2], a3 = kC[c4 + 3];
#pragma unroll
            for (int i = 0; i < kMaxUnits; ++i) {
                const int f = tid + i * kStepThreads;
                if (f < nC) {
                    const int row = f / wv;
                    const float kr = ks[row], qr = qs[row];
                    const float4 g = bG[f];
                    acc_qG.x += qr * g.x; acc_qG.y += qr * g.y; acc_qG.z += qr * g.z; acc_qG.w += qr * g.w;
                    store4(Gg + f, make_float4(g.x + kr * a0, g.y + kr * a1, g.z + kr * a2, g.w + kr * a3));
                }
            }
            part[tid][8] = acc_qG.x; part[tid][9] = acc_qG.y; part[tid][10] = acc_qG.z; part[tid][11] = acc_qG.w;
            __syncthreads();  // part written, the (G, h) buffer read
            if (nx < BH) load_part(bG, nx, offG, 2);
            if (tid < dv) {
                const int grp = tid >> 2, comp = tid & 3;
                float c = 0.f;
                for (int g = grp; g < kStepThreads; g += wv) c += part[g][8 + comp];
                qG[tid] = c;
            }
            __syncthreads();
        }

        // ---- output ----
        if (tid < dv) {
            float num = uC[tid] + uq * vs[tid];
            float den = um;
            if (masked) {
                num -= qG[tid] + kq * kC[tid];
                den -= qh + kq * km;
            }
            from_f32(&out[(long long)hd * dv + tid], normalized ? num / (den + eps) : num);
        }
        __syncthreads();  // qs, ks, vs, us, kC, uC, qG read before the next head rewrites them
    }
}

// dynamic shared memory of step2_kernel: S, (C, m), (G, h) if masked, tokens
size_t step2_smem(int d, int dv, int masked, size_t tsize) {
    const size_t nS = (size_t)d * d / 4, nCm = ((size_t)d * dv + d) / 4;
    return 16 * (nS + nCm * (masked ? 2 : 1)) + tsize * (2 * (size_t)d + dv);
}

template <bool kSDE>
cudaError_t step2_launch_t(const void *q, const void *k, const void *v, void *out, hla_dtype dt, int BH, int d,
                           int dv, int masked, int normalized, float eps, float *state, cudaStream_t stream) {
    if (BH == 0) return cudaSuccess;
    int dev = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    const int grid = BH < sms ? BH : sms;
    if (kSDE) masked = 0;  // shared-memory staging of (S, D, e) is that of (S, C, m)
    if (dt == HLA_BF16) {
        auto kern = step2_kernel<__nv_bfloat16, kSDE>;
        const size_t sm = step2_smem(d, dv, masked, sizeof(__nv_bfloat16));
        if ((e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm))) return e;
        kern<<<grid, kStepThreads, sm, stream>>>(static_cast<const __nv_bfloat16 *>(q),
                                                static_cast<const __nv_bfloat16 *>(k),
                                                static_cast<const __nv_bfloat16 *>(v),
                                                static_cast<__nv_bfloat16 *>(out), state, BH, d, dv, masked,
                                                normalized, eps);
    } else {
        auto kern = step2_kernel<float, kSDE>;
        const size_t sm = step2_smem(d, dv, masked, sizeof(float));
        if ((e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm))) return e;
        kern<<<grid, kStepThreads, sm, stream>>>(static_cast<const float *>(q), static_cast<const float *>(k),
                                                static_cast<const float *>(v), static_cast<float *>(out), state,
                                                BH, d, dv, masked, normalized, eps);
    }
    return cudaGetLastError();
}

}  // namespace

cudaError_t step2_launch(const void *q, const void *k, const void *v, void *out, hla_dtype dt, int BH, int d, int dv,
                         int masked, int normalized, float eps, float *state, cudaStream_t stream) {
    return step2_launch_t<false>(q, k, v, out, dt, BH, d, dv, masked, normalized, eps, state, stream);
}

cudaError_t step2_sde_launch(const void *q, const void *k, const void *v, void *out, hla_dtype dt, int BH, int d,
                             int dv, int normalized, float eps, float *state, cudaStream_t stream) {
    return step2_launch_t<true>(q, k, v, out, dt, BH, d, dv, 1, normalized, eps, state, stream);
}

namespace {

// (S, C, m, G, h) -> (S, D = S C - G, e = S m - h) per head, one block per head, the tuple staged in
// shared memory (dst must not overlap src: blocks of other heads may still be reading it).
__global__ void __launch_bounds__(256) state_to_sde_kernel(const float *src, float *dst, int d, int dv) {
    extern __shared__ float st[];
    const int hd = blockIdx.x, tid = threadIdx.x;
    const long long len = (long long)d * d + 2LL * d * dv + 2LL * d;
    const float4 *s4 = reinterpret_cast<const float4 *>(src + hd * len);
    float4 *st4 = reinterpret_cast<float4 *>(st);
    for (int i = tid; i < (int)(len >> 2); i += blockDim.x) st4[i] = s4[i];
    __syncthreads();
    const float *S = st, *C = S + d * d, *m = C + d * dv, *G = m + d, *h = G + d * dv;
    float *o = dst + hd * ((long long)d * d + (long long)d * dv + d);
    for (int i = tid; i < d * d; i += blockDim.x) o[i] = S[i];
    for (int i = tid; i < d * dv + d; i += blockDim.x) {
        const bool is_e = i >= d * dv;
        const int a = is_e ? i - d * dv : i / dv, b = is_e ? 0 : i % dv;
        float acc = 0.f;
        for (int j = 0; j < d; ++j) acc += S[a * d + j] * (is_e ? m[j] : C[j * dv + b]);
        o[d * d + i] = acc - (is_e ? h[a] : G[i]);
    }
}

}  // namespace

cudaError_t state_to_sde_launch(const float *src, float *dst, int BH, int d, int dv, cudaStream_t stream) {
    if (BH == 0) return cudaSuccess;
    const size_t smem = sizeof(float) * ((size_t)d * d + 2 * (size_t)d * dv + 2 * (size_t)d);
    cudaError_t e = cudaFuncSetAttribute(state_to_sde_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e) return e;
    state_to_sde_kernel<<<BH, 256, smem, stream>>>(src, dst, d, dv);
    return cudaGetLastError();
}

}  // namespace hla
