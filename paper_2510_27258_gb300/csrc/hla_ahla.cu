// Asymmetric second-order HLA (AHLA): chunk-parallel forward and decode step,
// fp32 SIMT kernels (Sec. "Asymmetric Higher-order Linear Attention").
//
// AHLA is causal linear attention applied twice: with A = L . (Q K^T) (L lower
// triangular incl. the diagonal), r_t = q_t^T P_t = (A V)_t and
// o_t = q_t^T E_t = (A R)_t (Theorem AHLA: P_t = sum_{j<=t} k_j v_j^T,
// E_t = sum_{i<=t} k_i r_i^T; denominators with v -> 1).  Per chunk, rows are
// its tokens and "p" the carry-in prefix:
//   R = A V + Q P_p,   s = A 1 + Q m_p,   O = A R + Q E_p,   den = A s + Q n_p.
// Chunk summaries compose with Eq. AHLA-semidirect,
//   E_AB = E_A + E_B + R^KQ_B P_A,  n_AB = n_A + n_B + R^KQ_B m_A,
// with R^KQ = sum_i k_i q_i^T over the later chunk, so a chunk's local
// summary (zero carry) is R^KQ = K^T Q, P = K^T V, m = K^T 1, E = K^T (A V),
// n = K^T (A 1).  Three launches: chunk-local summaries (all chunks in
// parallel), the carry scan (sequential over chunks, parallel over column
// blocks of [P | m] and [E | n]), outputs (all chunks in parallel).  The
// chunk argument is the scan granularity; chunks are at most 64 tokens here,
// 32 with a 128-wide head (the result does not depend on it up to rounding).
// Token rows of K are staged with a stride of d + 1 floats, so that the lanes
// of a warp, which take consecutive keys, read distinct banks.
#include <algorithm>

#include "hla_internal.h"
#include "simt_gemm.cuh"
#include "sm103_prims.cuh"

namespace hla {
namespace {

constexpr int kThreads = 256;
constexpr int kCols = 32;  // columns of [P | m] / [E | n] per scan block

struct ALayout {
    int BH, n, d, dv, C, nch;
    // local record per (head, chunk), floats: R^KQ d*d | P d*dv | m d | E d*dv | n d | Rloc C*dv | sloc C
    long long oR, oP, om, oE, on, oRl, osl, rec_local;
    // carry record per (head, chunk): P d*dv | m d | E d*dv | n d  (the state before the chunk)
    long long rec_carry, carry_base;
};

inline long long up16(long long x) { return (x + 15) / 16 * 16; }

ALayout make_layout(int BH, int n, int d, int dv, int chunk) {
    ALayout L;
    L.BH = BH; L.n = n; L.d = d; L.dv = dv;
    L.C = std::min(chunk, (d == 128 || dv == 128) ? 32 : 64);  // shared-memory staging of the output kernel
    L.nch = (n + L.C - 1) / L.C;
    long long o = 0;
    L.oR = o; o += up16((long long)d * d);
    L.oP = o; o += up16((long long)d * dv);
    L.om = o; o += up16(d);
    L.oE = o; o += up16((long long)d * dv);
    L.on = o; o += up16(d);
    L.oRl = o; o += up16((long long)L.C * dv);
    L.osl = o; o += up16(L.C);
    L.rec_local = o;
    L.rec_carry = up16(2LL * d * dv + 2LL * d);
    L.carry_base = (long long)BH * L.nch * L.rec_local;
    return L;
}

long long scratch_floats(const ALayout &L) { return L.carry_base + (long long)L.BH * L.nch * L.rec_carry; }

__device__ __forceinline__ float *local_rec(float *ws, const ALayout &L, int hd, int c) {
    return ws + ((long long)hd * L.nch + c) * L.rec_local;
}
__device__ __forceinline__ float *carry_rec(float *ws, const ALayout &L, int hd, int c) {
    return ws + L.carry_base + ((long long)hd * L.nch + c) * L.rec_carry;
}

template <typename T>
__device__ void load_tokens(const T *src, float *dst, int rows, int width, int Crows, int stride) {
    for (int i = threadIdx.x; i < Crows * width; i += blockDim.x) {
        const int r = i / width, c = i % width;
        dst[r * stride + c] = i < rows * width ? to_f32(src[i]) : 0.f;
    }
}

// ---------------------------------------------------------------------------
// kernel 1: chunk-local summaries (zero carry)
// ---------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(kThreads) ahla_local_kernel(const T *__restrict__ q, const T *__restrict__ k,
                                                              const T *__restrict__ v, float *ws, ALayout L) {
    extern __shared__ float sm[];
    const int c = blockIdx.x, hd = blockIdx.y, d = L.d, dv = L.dv, C = L.C;
    const int t0 = c * C, len = min(C, L.n - t0);
    const int kd = d + 1, w1 = dv + 1;  // row strides of K and of the augmented [V | 1], [R | s]
    float *Qs = sm, *Ks = Qs + C * d, *Vs = Ks + C * kd, *As = Vs + C * w1, *Rs = As + C * C;
    load_tokens(q + ((long long)hd * L.n + t0) * d, Qs, len, d, C, d);
    load_tokens(k + ((long long)hd * L.n + t0) * d, Ks, len, d, C, kd);
    load_tokens(v + ((long long)hd * L.n + t0) * dv, Vs, len, dv, C, w1);
    for (int t = threadIdx.x; t < C; t += blockDim.x) Vs[t * w1 + dv] = t < len ? 1.f : 0.f;
    __syncthreads();
    bgemm(As, C, Qs, d, 1, Ks, 1, kd, C, C, d, false, 1);          // A = L . Q K^T
    __syncthreads();
    bgemm(Rs, w1, As, C, 1, Vs, w1, 1, C, w1, C, false, 0, 1);     // [R_loc | s_loc] = A [V | 1]
    __syncthreads();
    float *rec = local_rec(ws, L, hd, c);
    for (int idx = threadIdx.x; idx < C * w1; idx += blockDim.x) {
        const int t = idx / w1, col = idx % w1;
        if (col < dv) rec[L.oRl + t * dv + col] = Rs[idx];
        else rec[L.osl + t] = Rs[idx];
    }
    bgemm(rec + L.oR, d, Ks, 1, kd, Qs, d, 1, d, d, C, false);      // R^KQ = K^T Q
    bgemm(rec + L.oP, dv, Ks, 1, kd, Vs, w1, 1, d, dv, C, false);   // P = K^T V
    bgemm(rec + L.om, 1, Ks, 1, kd, Vs + dv, w1, 1, d, 1, C, false); // m = K^T 1
    bgemm(rec + L.oE, dv, Ks, 1, kd, Rs, w1, 1, d, dv, C, false);   // E = K^T R_loc
    bgemm(rec + L.on, 1, Ks, 1, kd, Rs + dv, w1, 1, d, 1, C, false); // n = K^T s_loc
}

// ---------------------------------------------------------------------------
// kernel 2: carry scan.  Block (column block, head) keeps columns [j0, j0 + 32) of
// the augmented P' = [P | m] and E' = [E | n] (d x (dv + 1)); for every chunk it
// records the carry-in, then E' += E'_c + R^KQ_c P'  (old P') and P' += P'_c.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads) ahla_scan_kernel(float *ws, ALayout L, const float *state_in,
                                                             float *state_out) {
    extern __shared__ float sm[];
    const int hd = blockIdx.y, d = L.d, dv = L.dv, j0 = blockIdx.x * kCols;
    float *Pp = sm, *Ep = Pp + d * kCols, *Rq = Ep + d * kCols;  // d x 32, d x 32, d x d
    const int ncol = min(kCols, dv + 1 - j0);
    const long long st_len = 2LL * d * dv + 2LL * d;
    auto P_at = [&](const float *base, int a, int j) { return j < dv ? base[a * dv + j] : base[(long long)d * dv + a]; };
    // base layout of a state / carry record: P d*dv | m d | E d*dv | n d
    const float *sin = state_in ? state_in + hd * st_len : nullptr;
    for (int idx = threadIdx.x; idx < d * kCols; idx += blockDim.x) {
        const int a = idx / kCols, j = idx % kCols;
        const bool ok = j < ncol;
        Pp[idx] = (ok && sin) ? P_at(sin, a, j0 + j) : 0.f;
        Ep[idx] = (ok && sin) ? P_at(sin + (long long)d * dv + d, a, j0 + j) : 0.f;
    }
    __syncthreads();
    for (int c = 0; c < L.nch; ++c) {
        float *cr = carry_rec(ws, L, hd, c);
        const float *lr = local_rec(ws, L, hd, c);
        for (int idx = threadIdx.x; idx < d * ncol; idx += blockDim.x) {
            const int a = idx / ncol, j = idx % ncol, col = j0 + j;
            if (col < dv) {
                cr[a * dv + col] = Pp[a * kCols + j];
                cr[(long long)d * dv + d + a * dv + col] = Ep[a * kCols + j];
            } else {
                cr[(long long)d * dv + a] = Pp[a * kCols + j];
                cr[2LL * d * dv + d + a] = Ep[a * kCols + j];
            }
        }
        for (int idx = threadIdx.x; idx < d * d; idx += blockDim.x) Rq[idx] = lr[L.oR + idx];
        __syncthreads();
        // E' += E'_c + R^KQ_c P' (each thread owns elements (a, j); P' is read before it changes)
        float newE[128 * kCols / kThreads], newP[128 * kCols / kThreads];
        int cnt = 0;
        for (int idx = threadIdx.x; idx < d * kCols; idx += blockDim.x, ++cnt) {
            const int a = idx / kCols, j = idx % kCols;
            float e = Ep[idx], p = Pp[idx];
            if (j < ncol) {
                float s = 0.f;
                for (int b = 0; b < d; ++b) s += Rq[a * d + b] * Pp[b * kCols + j];
                const int col = j0 + j;
                e += s + (col < dv ? lr[L.oE + a * dv + col] : lr[L.on + a]);
                p += col < dv ? lr[L.oP + a * dv + col] : lr[L.om + a];
            }
            newE[cnt] = e;
            newP[cnt] = p;
        }
        __syncthreads();  // every P' read before it is updated
        cnt = 0;
        for (int idx = threadIdx.x; idx < d * kCols; idx += blockDim.x, ++cnt) {
            Ep[idx] = newE[cnt];
            Pp[idx] = newP[cnt];
        }
        __syncthreads();
    }
    if (state_out) {
        float *so = state_out + hd * st_len;
        for (int idx = threadIdx.x; idx < d * ncol; idx += blockDim.x) {
            const int a = idx / ncol, j = idx % ncol, col = j0 + j;
            if (col < dv) {
                so[a * dv + col] = Pp[a * kCols + j];
                so[(long long)d * dv + d + a * dv + col] = Ep[a * kCols + j];
            } else {
                so[(long long)d * dv + a] = Pp[a * kCols + j];
                so[2LL * d * dv + d + a] = Ep[a * kCols + j];
            }
        }
    }
}

// ---------------------------------------------------------------------------
// kernel 3: outputs.  R = R_loc + Q P_p, s = s_loc + Q m_p, O = A R + Q E_p,
// den = A s + Q n_p.
// ---------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(kThreads) ahla_out_kernel(const T *__restrict__ q, const T *__restrict__ k,
                                                            T *__restrict__ out, float *ws, ALayout L, int normalized,
                                                            float eps) {
    extern __shared__ float sm[];
    const int c = blockIdx.x, hd = blockIdx.y, d = L.d, dv = L.dv, C = L.C;
    const int t0 = c * C, len = min(C, L.n - t0);
    const int kd = d + 1, w1 = dv + 1;
    // Rs = [R | s] and Os = [O | den] (C x (dv + 1)); Ps = [P_p | m_p], Es = [E_p | n_p] (d x (dv + 1));
    // Os takes the place of K, which is dead once A is formed
    const int kw = kd > w1 ? kd : w1;
    float *Qs = sm, *Ks = Qs + C * d, *Rs = Ks + C * kw, *As = Rs + C * w1, *Ps = As + C * C, *Es = Ps + d * w1;
    float *Os = Ks;
    load_tokens(q + ((long long)hd * L.n + t0) * d, Qs, len, d, C, d);
    load_tokens(k + ((long long)hd * L.n + t0) * d, Ks, len, d, C, kd);
    const float *lr = local_rec(ws, L, hd, c), *cr = carry_rec(ws, L, hd, c);
    for (int idx = threadIdx.x; idx < d * w1; idx += blockDim.x) {
        const int f = idx / w1, col = idx % w1;
        Ps[idx] = col < dv ? cr[f * dv + col] : cr[(long long)d * dv + f];
        Es[idx] = col < dv ? cr[(long long)d * dv + d + f * dv + col] : cr[2LL * d * dv + d + f];
    }
    for (int idx = threadIdx.x; idx < C * w1; idx += blockDim.x) {
        const int t = idx / w1, col = idx % w1;
        Rs[idx] = col < dv ? lr[L.oRl + t * dv + col] : lr[L.osl + t];
    }
    __syncthreads();
    bgemm(Rs, w1, Qs, d, 1, Ps, w1, 1, C, w1, d, true);             // [R | s] += Q [P_p | m_p]
    bgemm(As, C, Qs, d, 1, Ks, 1, kd, C, C, d, false, 1);           // A = L . Q K^T
    __syncthreads();
    bgemm(Os, w1, As, C, 1, Rs, w1, 1, C, w1, C, false, 0, 1);      // [O | den] = A [R | s]
    bgemm(Os, w1, Qs, d, 1, Es, w1, 1, C, w1, d, true);             //   + Q [E_p | n_p]
    __syncthreads();
    T *o = out + ((long long)hd * L.n + t0) * dv;
    for (int idx = threadIdx.x; idx < len * dv; idx += blockDim.x) {
        const int t = idx / dv, col = idx % dv;
        const float x = Os[t * w1 + col];
        from_f32(&o[idx], normalized ? x / (Os[t * w1 + dv] + eps) : x);
    }
}

// ---------------------------------------------------------------------------
// decode step: P' = P + k v^T, m' = m + k, r = q^T P', s = q . m',
// E' = E + k r^T, n' = n + s k, o = q^T E', den = q . n'.  P and E are read and
// written once with 16-byte accesses, consecutive threads on consecutive column
// groups; every thread keeps one column group of the column sums q^T P' (then
// q^T E'), combined across row groups in shared memory.
// ---------------------------------------------------------------------------
// One 512-thread block per SM works through heads (hd = blockIdx.x, + gridDim.x,
// ...), each head's [P | m] and [E | n] staged in shared memory by one 1-D bulk copy each, issued
// a pass or more before use: while the P pass of a head runs, its [E | n] is in flight, and each
// buffer takes the next head's part as soon as its pass has read it.  Updated values go to global
// memory straight from registers.  Every thread waits on the buffer's mbarrier (phase = the block's
// head count), bounded: a copy that never lands ends the block.
constexpr int kStepPThreads = 512;
constexpr unsigned long long kCopyWaitNs = 2000000000ull;

__device__ __forceinline__ void bulk_copy(void *dst, const void *src, uint32_t bytes, uint64_t *bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                 ::"r"(sm103::smem_u32(dst)), "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes),
                   "r"(sm103::smem_u32(bar))
                 : "memory");
}

template <typename T>
__global__ void __launch_bounds__(kStepPThreads, 1)
ahla_step_staged_kernel(const T *__restrict__ q, const T *__restrict__ k, const T *__restrict__ v, T *__restrict__ out,
                        float *__restrict__ state, int BH, int d, int dv, int normalized, float eps) {
    extern __shared__ float4 dyn[];
    __shared__ float qs[128], ks[128], vs[128], rs[128], part[kStepPThreads][4], red[kStepPThreads / 32];
    __shared__ float s_sc;
    __shared__ uint64_t bar[2];  // [P | m] and tokens; [E | n]
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const long long st = 2LL * d * dv + 2 * d;
    const int nP = (d * dv + d) >> 2;  // float4 units of [P | m], of [E | n]
    const int nt_q = d * (int)sizeof(T) / 16, nt_v = dv * (int)sizeof(T) / 16;
    float4 *bP = dyn, *bE = bP + nP, *bT = bE + nP;
    const T *tq = reinterpret_cast<const T *>(bT), *tk = tq + d, *tv = tk + d;
    // thread 0 issues the copies, after a block barrier that ends the generic reads of the buffer
    auto load_P = [&](int hd) {
        if (tid == 0) {
            sm103::fence_async_smem();
            sm103::mbar_arrive_expect_tx(&bar[0], (uint32_t)(16 * (nP + 2 * nt_q + nt_v)));
            bulk_copy(bP, state + hd * st, 16u * nP, &bar[0]);
            bulk_copy(bT, q + (long long)hd * d, 16u * nt_q, &bar[0]);
            bulk_copy(bT + nt_q, k + (long long)hd * d, 16u * nt_q, &bar[0]);
            bulk_copy(bT + 2 * nt_q, v + (long long)hd * dv, 16u * nt_v, &bar[0]);
        }
    };
    auto load_E = [&](int hd) {
        if (tid == 0) {
            sm103::fence_async_smem();
            sm103::mbar_arrive_expect_tx(&bar[1], 16u * nP);
            bulk_copy(bE, state + hd * st + (long long)d * dv + d, 16u * nP, &bar[1]);
        }
    };
    // block sum of one value per thread (all threads call it; ends with a block barrier)
    auto block_sum = [&](float x) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
        if (lane == 0) red[wid] = x;
        __syncthreads();
        float t = 0.f;
        for (int w = 0; w < kStepPThreads / 32; ++w) t += red[w];
        __syncthreads();
        return t;
    };
    int hd = blockIdx.x;
    if (hd >= BH) return;
    if (tid == 0) {
        sm103::mbar_init(&bar[0], 1);
        sm103::mbar_init(&bar[1], 1);
        sm103::fence_mbar_init();
    }
    __syncthreads();
    load_P(hd);
    load_E(hd);
    const int wv = dv >> 2, n4 = (d * dv) >> 2, c4 = (tid % wv) * 4;  // kStepPThreads is a multiple of wv
    for (uint32_t par = 0; hd < BH; hd += gridDim.x, par ^= 1u) {
        const int nx = hd + gridDim.x;  // this block's next head
        float *P = state + hd * st, *m = P + (long long)d * dv, *E = m + d, *nn = E + (long long)d * dv;
        if (!sm103::mbar_wait(&bar[0], par, kCopyWaitNs)) return;  // [P | m] and tokens of this head
        if (tid < d) {
            qs[tid] = to_f32(tq[tid]);
            ks[tid] = to_f32(tk[tid]);
        }
        if (tid < dv) vs[tid] = to_f32(tv[tid]);
        __syncthreads();
        // ---- [P | m]: P' = P + k v^T, m' = m + k, r = q^T P', s = q . m' ----
        {
            float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
            float4 *P4 = reinterpret_cast<float4 *>(P);
            const float v0 = vs[c4], v1 = vs[c4 + 1], v2 = vs[c4 + 2], v3 = vs[c4 + 3];
            for (int f = tid; f < n4; f += kStepPThreads) {
                const int row = f / wv;
                float4 pv = bP[f];
                const float kr = ks[row], qr = qs[row];
                pv.x += kr * v0; pv.y += kr * v1; pv.z += kr * v2; pv.w += kr * v3;
                P4[f] = pv;
                acc.x += qr * pv.x; acc.y += qr * pv.y; acc.z += qr * pv.z; acc.w += qr * pv.w;
            }
            part[tid][0] = acc.x; part[tid][1] = acc.y; part[tid][2] = acc.z; part[tid][3] = acc.w;
            float sm = 0.f;
            if (tid < d) {
                const float mv = reinterpret_cast<const float *>(bP + n4)[tid] + ks[tid];
                m[tid] = mv;
                sm = qs[tid] * mv;
            }
            const float s_tot = block_sum(sm);  // s = q . m' (also: part written, the [P | m] buffer read)
            if (nx < BH) load_P(nx);
            if (tid < dv) {
                const int grp = tid >> 2, comp = tid & 3;
                float a = 0.f;
                for (int g = grp; g < kStepPThreads; g += wv) a += part[g][comp];
                rs[tid] = a;  // r = q^T P'
            }
            if (tid == 0) s_sc = s_tot;
            __syncthreads();
        }
        // ---- [E | n]: E' = E + k r^T, n' = n + s k, o = q^T E', den = q . n' ----
        if (!sm103::mbar_wait(&bar[1], par, kCopyWaitNs)) return;  // [E | n] of this head
        {
            float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
            float4 *E4 = reinterpret_cast<float4 *>(E);
            const float r0 = rs[c4], r1 = rs[c4 + 1], r2 = rs[c4 + 2], r3 = rs[c4 + 3];
            for (int f = tid; f < n4; f += kStepPThreads) {
                const int row = f / wv;
                float4 e = bE[f];
                const float kr = ks[row], qr = qs[row];
                e.x += kr * r0; e.y += kr * r1; e.z += kr * r2; e.w += kr * r3;
                E4[f] = e;
                acc.x += qr * e.x; acc.y += qr * e.y; acc.z += qr * e.z; acc.w += qr * e.w;
            }
            part[tid][0] = acc.x; part[tid][1] = acc.y; part[tid][2] = acc.z; part[tid][3] = acc.w;
            float sn = 0.f;
            if (tid < d) {
                const float nv = reinterpret_cast<const float *>(bE + n4)[tid] + s_sc * ks[tid];
                nn[tid] = nv;
                sn = qs[tid] * nv;
            }
            const float den = block_sum(sn);  // den = q . n' (also: part written, the [E | n] buffer read)
            if (nx < BH) load_E(nx);
            if (tid < dv) {
                const int grp = tid >> 2, comp = tid & 3;
                float a = 0.f;
                for (int g = grp; g < kStepPThreads; g += wv) a += part[g][comp];
                from_f32(&out[(long long)hd * dv + tid], normalized ? a / (den + eps) : a);
            }
            __syncthreads();  // qs, ks, vs, rs, part, s_sc read before the next head rewrites them
        }
    }
}

template <typename T>
cudaError_t forward_t(const Fwd2 &p, cudaStream_t stream) {
    const ALayout L = make_layout(p.BH, p.n, p.d, p.dv, p.chunk);
    float *ws = reinterpret_cast<float *>(p.ws + kWsHeaderBytes);
    const T *q = static_cast<const T *>(p.q), *k = static_cast<const T *>(p.k), *v = static_cast<const T *>(p.v);
    cudaError_t e;
    if (L.nch > 0) {
        const size_t sm1 = sizeof(float) * ((size_t)L.C * (2 * L.d + 1 + 2 * (L.dv + 1)) + (size_t)L.C * L.C);
        if ((e = cudaFuncSetAttribute(ahla_local_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm1)))
            return e;
        ahla_local_kernel<T><<<dim3(L.nch, p.BH), kThreads, sm1, stream>>>(q, k, v, ws, L);
        if ((e = cudaGetLastError())) return e;
    }
    const size_t sm2 = sizeof(float) * ((size_t)2 * p.d * kCols + (size_t)p.d * p.d);
    if ((e = cudaFuncSetAttribute(ahla_scan_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm2))) return e;
    ahla_scan_kernel<<<dim3((p.dv + 1 + kCols - 1) / kCols, p.BH), kThreads, sm2, stream>>>(ws, L, p.state_in,
                                                                                            p.state_out);
    if ((e = cudaGetLastError())) return e;
    if (L.nch > 0) {
        const size_t sm3 = sizeof(float) * ((size_t)L.C * (L.d + std::max(L.d + 1, L.dv + 1) + L.dv + 1) +
                                            (size_t)L.C * L.C + 2 * (size_t)L.d * (L.dv + 1));
        if ((e = cudaFuncSetAttribute(ahla_out_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm3)))
            return e;
        ahla_out_kernel<T><<<dim3(L.nch, p.BH), kThreads, sm3, stream>>>(q, k, static_cast<T *>(p.out), ws, L,
                                                                         p.normalized, p.eps);
        if ((e = cudaGetLastError())) return e;
    }
    return cudaSuccess;
}

}  // namespace

size_t ahla_workspace_bytes_internal(int BH, int n, int d, int dv, int chunk) {
    const ALayout L = make_layout(BH, n, d, dv, chunk);
    return kWsHeaderBytes + sizeof(float) * (size_t)scratch_floats(L);
}

cudaError_t ahla_forward_launch(const Fwd2 &p, cudaStream_t stream) {
    if (ahla_tc_applicable(p)) return ahla_tc_forward(p, stream);
    return p.dt == HLA_BF16 ? forward_t<__nv_bfloat16>(p, stream) : forward_t<float>(p, stream);
}

cudaError_t ahla_step_launch(const void *q, const void *k, const void *v, void *out, hla_dtype dt, int BH, int d,
                             int dv, int normalized, float eps, float *state, cudaStream_t stream) {
    if (BH == 0) return cudaSuccess;
    // the staged kernel copies whole 16-byte units (token rows, [P | m], [E | n], the head stride):
    // the entry point checks the 16-byte alignment of q, k, v and the state, and d, dv in
    // {16, 32, 64, 128} make every row a multiple of 16 bytes
    const size_t tsz = dt == HLA_BF16 ? 2 : 4;
    if ((d * tsz) % 16 != 0 || (dv * tsz) % 16 != 0 || d % 4 != 0 || dv % 4 != 0 || d > 128 || dv > 128)
        return cudaErrorInvalidValue;
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int grid = BH < sms ? BH : sms;
    const size_t smem = 2 * 16 * (size_t)((d * dv + d) / 4) + tsz * (2 * (size_t)d + dv);
    cudaError_t e;
    if (dt == HLA_BF16) {
        if ((e = cudaFuncSetAttribute(ahla_step_staged_kernel<__nv_bfloat16>,
                                      cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)))
            return e;
        ahla_step_staged_kernel<__nv_bfloat16><<<grid, kStepPThreads, smem, stream>>>(
            static_cast<const __nv_bfloat16 *>(q), static_cast<const __nv_bfloat16 *>(k),
            static_cast<const __nv_bfloat16 *>(v), static_cast<__nv_bfloat16 *>(out), state, BH, d, dv, normalized, eps);
    } else {
        if ((e = cudaFuncSetAttribute(ahla_step_staged_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)smem)))
            return e;
        ahla_step_staged_kernel<float><<<grid, kStepPThreads, smem, stream>>>(
            static_cast<const float *>(q), static_cast<const float *>(k), static_cast<const float *>(v),
            static_cast<float *>(out), state, BH, d, dv, normalized, eps);
    }
    return cudaGetLastError();
}

}  // namespace hla
