// Block-level fp32 matrix products on the CUDA cores (shared or global operands with
// arbitrary strides), used by the SIMT kernels of the AHLA forward and the backward.
#pragma once

namespace hla {
namespace {

// C[r][c] (+)= sum_k A(r, k) B(k, c) for r < M, c < N over the block's threads, with
// A(r, k) = A[r * ar + k * ak], B(k, c) = B[k * bk + c * bc], C[r * ldc + c].
// mask 1: only c <= r (others set to 0 unless accumulating).  kmode cuts the k range
// where A or B holds stored zeros: 1 k <= r (A lower triangular by rows), 2 k >= c
// (B(k, c) = 0 for k < c), 3 k >= r (A(r, k) = 0 for k < r); a thread's range is the
// union over its outputs, which only adds products with those stored zeros.
// Each thread computes 4 x 4 outputs: rows r0 .. r0 + 3 and columns cb + j tn
// (j = 0..3, tn = ceil(N / 4)), so that consecutive threads read consecutive columns of B.
__device__ void bgemm(float *Cm, int ldc, const float *A, int ar, int ak, const float *B, int bk, int bc, int M, int N,
                      int K, bool accumulate, int mask = 0, int kmode = 0) {
    const int tn = (N + 3) >> 2, tiles = ((M + 3) >> 2) * tn;
    for (int tile = threadIdx.x; tile < tiles; tile += blockDim.x) {
        const int r0 = (tile / tn) * 4, cb = tile % tn;
        int k0 = 0, k1 = K;
        if (kmode == 1) k1 = min(K, r0 + 4);
        else if (kmode == 2) k0 = cb;
        else if (kmode == 3) k0 = r0;
        float acc[4][4];
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
        if (!(mask == 1 && cb > r0 + 3)) {
            int ra[4], cc[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) ra[i] = min(r0 + i, M - 1) * ar;  // rows / columns beyond the
#pragma unroll
            for (int j = 0; j < 4; ++j) cc[j] = min(cb + j * tn, N - 1) * bc;  // output are not stored
            for (int kk = k0; kk < k1; ++kk) {
                float x[4], y[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) x[i] = A[ra[i] + kk * ak];
#pragma unroll
                for (int j = 0; j < 4; ++j) y[j] = B[kk * bk + cc[j]];
#pragma unroll
                for (int i = 0; i < 4; ++i)
#pragma unroll
                    for (int j = 0; j < 4; ++j) acc[i][j] += x[i] * y[j];
            }
        }
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int r = r0 + i, c = cb + j * tn;
                if (r >= M || c >= N) continue;
                float *o = &Cm[r * ldc + c];
                if (mask == 1 && c > r) {
                    if (!accumulate) *o = 0.f;
                } else {
                    *o = (accumulate ? *o : 0.f) + acc[i][j];
                }
            }
    }
}

}  // namespace
}  // namespace hla
