// Masked third-order HLA forward on the tensor cores (sm_103a): tcgen05 MMAs
// with TMEM accumulators, every chunk contraction split into bf16 hi + lo parts
// so that the fp32 result keeps about 16 bits of every operand.
//
// Per 128-token tile of a head (rows = tokens; p = carry before the tile;
// A = Q K^T, a = diag(A), LA = L . A with L the lower triangle including the
// diagonal), from the token update of Algorithm 3 (Theorem 4's chunk form):
//   Y   = Q P_p + LA V                         (y_s = q_s^T P_s)
//   b_s = k_s^T S^Q_p k_s + sum_{u<s} A_us^2   (k_s^T S^Q_{s-1} k_s)
//   Z'  = diag(a) Y + diag(b - a^2) V
//   C'  = LA LA^T + (Q S^K_p) Q^T              (on the lower triangle:
//                                               q_t^T S^K_{s-1} q_s + A_ts a_s)
//   num = Q F_p + LA Z' + (L . C') diag(a) V
//   carries: S^K += K^T K,  S^Q += Q^T Q,  P += K^T V,
//            F += K^T G' + (Q S^K_p)^T diag(a) V,  G' = Z' + LA^T diag(a) V.
// (The diagonal terms a_s^2 fold the strict triangles of the token update into
// the inclusive LA: C'_ts - A_ts a_s is the strict sum sum_{i<s} A_ti A_si, and
// LA^T aV - a^2 V is the strict sum over s > i.)
//
// F enters the outputs only linearly (q_t^T F_t) and its update does not read F,
// so a head is cut into segments of L tiles that run on different SMs: a
// pre-pass kernel sums S^K, S^Q, P over each segment; the sweep of segment g
// starts from the sums of the segments before it (exact fp32) and from F = 0,
// writes q_t^T F_t(local) and its own total of F; a fix-up kernel adds
// q_t^T F_start(g) with F_start(g) the sum of the earlier segments' totals.
//
// Operands live in shared memory as 128-row x 64-column bf16 blocks in the
// 128-byte-swizzled layout.  A 32-wide operand keeps its hi part in columns
// 0..31 and its lo part in columns 32..63 of the same rows:
//   * products over the 32 features issue six K = 16 steps pairing
//     (hi, hi), (hi, lo), (lo, hi) slices of the two operands;
//   * products over the 128 tokens read such a block MN-major with N = 64 (or
//     M = 64 of an M = 128 product), so the result holds the hi and lo halves
//     side by side (or the four hi/lo quadrants), summed by the epilogue.
// LA (128 x 128) has separate hi and lo tiles.  L . C' is packed as bf16 into TMEM over
// C' itself (each thread's 32 columns: hi in the first 16, lo in the last 16) and read
// from there as the A operand of its product.
//
// TMEM (512 columns): A -> C' -> L . C' packed (128), Y -> num (64), Q S^K_p and
// K S^Q_p (32 + 32, then G'' = LA^T aV over them), and 64-column carry regions
// holding the hi/lo quadrants of [K V]^T K (rows 0..63: S^K, rows 64..127: P^T, V's
// block following K's), Q^T Q (= S^Q) and G'^T K + aV^T (Q S^K_p) (= F^T).  Rows
// 64..127 of the other carry products read the block after the operand's own and
// are never used.
//
// Roles: warp 16 issues the MMAs (one thread); warps 0..15 are the epilogue
// (warp w: TMEM lanes 32 (w % 4) .. +31, one token row each; column block w / 4),
// which also loads the fp32 tokens (the next tile's during this one) and splits
// them into hi + lo.  A tile's outputs are read out while the next tile's first
// product (A = Q K^T) runs, and that product starts on the split tokens while the
// epilogue folds the carries.
//
// Scope: fp32 tokens, d = dv = 32, masked, plain (unnormalised) output, no
// initial or final state.
#include <cstdlib>

#include "hla_internal.h"
#include "sm103_prims.cuh"

namespace hla {
namespace {

using namespace sm103;

constexpr int kTile = 128, kD = 32;
constexpr int kEpiWarps = 16, kEpiThreads = kEpiWarps * 32, kIssuerWarp = kEpiWarps;
constexpr int kThreads = kEpiThreads + 32;
constexpr int kMaxSegments = 160;

// shared-memory blocks of 16 KiB
enum Block { bQ = 0, bK = 1, bV = 2, bQS = 3, bAV = 4, bZ = 5, bG = 6, bLh = 7, bLl = 9, bCar = 11, kBlocks = 12 };
// bLh / bLl: 128 x 128 tiles (two blocks each): LA, hi and lo parts.
// bCar: four 32-row K-major operands (hi | lo): S^K_p, S^Q_p, P_p^T, F_p^T.
// The pre-pass alternates two sets of Q, K, V blocks (0..2 and 3..5: a tile's split runs
// while the products of the tile before read the other set) and holds two stages of fp32
// tokens in blocks 6..11 (Q, K, V of one tile: 128 rows of 128 bytes each, copied as one
// contiguous piece per operand).
constexpr int kStages = 2;
__device__ __forceinline__ int stage_block(int s, int t) { return 6 + 3 * s + t; }
constexpr uint32_t kSmemBlocks = kBlocks * kBlockBytes;

// TMEM columns
constexpr uint32_t kTA = 0, kTY = 128, kTQS = 192, kTKS = 224, kTG = 192, kTCar = 256;  // + 64 per carry

enum Bar {
    bEvA = 0, bEvQ = 1, bEvY = 2, bEvC = 3, bEvO = 4,  // MMA commits
    bEp0 = 5, bEp1 = 6, bEp2 = 7, bEp3 = 8,            // epilogue hand-offs (16 warp arrivals)
    bTear = 9,
    bSt0 = 10,                                         // + stage: pre-pass token copies
    bEvO1 = 12,                                        // pre-pass: products of the second block set
    bEpQK = 13,                                        // sweep: Q, K, V (hi | lo) stored (16 warp arrivals)
    kNumBars = 14
};

struct Misc {
    uint64_t bar[kNumBars];
    uint32_t tmem_base;
    int abort_flag;
    float sa[kTile];          // a_t = A_tt
    float sdp[4][kTile];      // per column block: partial q_t . k_t in fp32
    float sbp[4][kTile];      // per lane quadrant: column sums of A_us^2 over u < s
    float sbp2[4][kTile];     // per column block: partial k_s^T S^Q_p k_s
    float fold[4][32][33];    // carry read-out: each carry folded to 32 x 32 (hi/lo rows, columns added)
};
constexpr uint32_t kMiscBytes = 24 * 1024;
static_assert(sizeof(Misc) <= kMiscBytes, "misc smem");
constexpr uint32_t kSmemBytes = kSmemBlocks + kMiscBytes;

struct Params {
    const float *q, *k, *v;
    float *out;
    float *rec;  // [BH][G][3][32][32]: S^K, S^Q, P^T summed over each segment (pre-pass)
    float *dF;   // [BH][G][32][32]: F^T summed over each segment (sweep)
    int BH, n, M, G, L;
    WsHeader *err;
};

constexpr unsigned long long kBarWaitNs = 2000000000ull;

__device__ __forceinline__ void set_error(WsHeader *err, unsigned where, unsigned detail) {
    if (atomicCAS(&err->error, 0u, (unsigned)kDevTimeout) == 0u) {
        err->where = where;
        err->detail = detail;
    }
}

__device__ __forceinline__ bool bar_wait(Misc *ms, int b, uint32_t parity, const Params &p) {
    if (ms->abort_flag) return false;
    if (mbar_wait(&ms->bar[b], parity, kBarWaitNs)) return true;
    set_error(p.err, 400 + b, parity);
    ms->abort_flag = 1;
    return false;
}

__device__ __forceinline__ void epi_sync() { asm volatile("bar.sync 1, %0;" ::"n"(kEpiThreads) : "memory"); }

__device__ __forceinline__ void epi_arrive(Misc *ms, int b) {
    tc_fence_before();
    __syncwarp();
    if ((threadIdx.x & 31) == 0) mbar_arrive(&ms->bar[b]);
}

// 32 lanes x 8 consecutive TMEM columns
__device__ __forceinline__ void tmem_ld8(uint32_t taddr, uint32_t (&v)[8]) {
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
                 : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7])
                 : "r"(taddr));
}

// 1-D bulk copy global -> shared (both addresses 16-byte aligned, size a multiple of 16),
// completing as transaction bytes on `bar`
__device__ __forceinline__ void bulk_load(void *dst, const void *src, uint32_t bytes, uint64_t *bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                 ::"r"(smem_u32(dst)), "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(smem_u32(bar))
                 : "memory");
}

// ------------------------------- MMA issue -------------------------------
// Shared-memory descriptors: the high word is fixed (1 KiB between 8-row groups, tcgen05
// version, 128-byte swizzle); the low word is the start address / 16 plus the leading-byte
// offset (unused for K-major operands; 16 KiB between the 64-element blocks of an MN-major
// operand), so every K step adds a constant to a per-block low word.
constexpr uint32_t kDescHi = (1024u >> 4) | (1u << 14) | (2u << 29);
constexpr uint32_t kLboK = 1u << 16, kLboMN = (kBlockBytes >> 4) << 16;
constexpr uint32_t kBlk16 = kBlockBytes >> 4;  // one block in 16-byte units

__device__ __forceinline__ uint64_t dsc(uint32_t lo) { return (static_cast<uint64_t>(kDescHi) << 32) | lo; }

// D (+)= A B over the 32 features, both operands K-major blocks with hi in columns
// 0..31 and lo in columns 32..63: hi.hi + hi.lo + lo.hi (six K = 16 steps; a step of 16
// columns is 32 bytes).  a, b: low descriptor words of K-major blocks.
template <int N>
__device__ __forceinline__ void mma_feat3(uint32_t d, uint32_t a, uint32_t b, uint32_t acc) {
    constexpr uint32_t id = idesc_bf16(128, N, 0, 0);
    umma_bf16(d, dsc(a), dsc(b), id, acc);
    umma_bf16(d, dsc(a + 2), dsc(b + 2), id, 1u);
    umma_bf16(d, dsc(a), dsc(b + 4), id, 1u);
    umma_bf16(d, dsc(a + 2), dsc(b + 6), id, 1u);
    umma_bf16(d, dsc(a + 4), dsc(b), id, 1u);
    umma_bf16(d, dsc(a + 6), dsc(b + 2), id, 1u);
}

// D (+)= A B over the 128 tokens of a tile (eight K = 16 steps).  K-major operands
// span a 128 x 128 tile (two blocks); MN-major ones hold the tokens in their rows
// (16 rows = 2 KiB per step; M = 128 reads the block after as columns 64..127).
template <bool A_MN, bool B_MN, int N>
__device__ __forceinline__ void mma_tok(uint32_t d, uint32_t a, uint32_t b, uint32_t acc) {
    constexpr uint32_t id = idesc_bf16(128, N, A_MN, B_MN);
#pragma unroll
    for (int kk = 0; kk < 8; ++kk) {
        const uint32_t ka = A_MN ? kk * 128u : (kk >> 2) * kBlk16 + (kk & 3) * 2u;
        const uint32_t kb = B_MN ? kk * 128u : (kk >> 2) * kBlk16 + (kk & 3) * 2u;
        umma_bf16(d, dsc(a + ka), dsc(b + kb), id, kk > 0 ? 1u : acc);
    }
}

// D (+)= A B over the 128 tokens with A in TMEM (bf16 pairs packed in the first 16 of each 32
// columns: K elements 32g .. 32g + 31 of a row in columns a + 32g .. +15, so K step kk starts at
// column 32 (kk / 2) + 8 (kk % 2)); B MN-major
template <int N>
__device__ __forceinline__ void mma_ts_tok(uint32_t d, uint32_t a_tmem, uint32_t b, uint32_t acc) {
    constexpr uint32_t id = idesc_bf16(128, N, 0, 1);
#pragma unroll
    for (int kk = 0; kk < 8; ++kk)
        umma_bf16_ts(d, a_tmem + 32u * (kk >> 1) + 8u * (kk & 1), dsc(b + kk * 128u), id, kk > 0 ? 1u : acc);
}

// ------------------------------- epilogue helpers -------------------------------
// x -> bf16 hi, bf16 lo = x - hi (8 values, packed in pairs)
__device__ __forceinline__ void split8(const float (&x)[8], uint4 &hi, uint4 &lo) {
    uint32_t h[4], l[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        h[i] = pack_bf16x2(x[2 * i], x[2 * i + 1]);
        const float h0 = __uint_as_float(h[i] << 16), h1 = __uint_as_float(h[i] & 0xFFFF0000u);
        l[i] = pack_bf16x2(x[2 * i] - h0, x[2 * i + 1] - h1);
    }
    hi = make_uint4(h[0], h[1], h[2], h[3]);
    lo = make_uint4(l[0], l[1], l[2], l[3]);
}

__device__ __forceinline__ void st16(uint8_t *tile, int r, int c, const uint4 &v) {
    *reinterpret_cast<uint4 *>(tile + tile_off(r, c)) = v;
}

// 8 values of a 32-wide operand row: hi at column c, lo at column 32 + c of the block
__device__ __forceinline__ void store_hl8(uint8_t *blk, int r, int c, const float (&x)[8]) {
    uint4 h, l;
    split8(x, h, l);
    st16(blk, r, c, h);
    st16(blk, r, 32 + c, l);
}

// the 8 values written by store_hl8, as hi + lo
__device__ __forceinline__ void load_hl8(const uint8_t *blk, int r, int c, float (&x)[8]) {
    const uint4 h = *reinterpret_cast<const uint4 *>(blk + tile_off(r, c));
    const uint4 l = *reinterpret_cast<const uint4 *>(blk + tile_off(r, 32 + c));
    const uint32_t hh[4] = {h.x, h.y, h.z, h.w}, ll[4] = {l.x, l.y, l.z, l.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        x[2 * i] = __uint_as_float(hh[i] << 16) + __uint_as_float(ll[i] << 16);
        x[2 * i + 1] = __uint_as_float(hh[i] & 0xFFFF0000u) + __uint_as_float(ll[i] & 0xFFFF0000u);
    }
}

__device__ __forceinline__ void load_row8(const float *base, int n, int head, int tok, int c, float (&x)[8]) {
    if (tok < n) {
        const float4 *s = reinterpret_cast<const float4 *>(base + ((size_t)head * n + tok) * kD + c);
        const float4 u = __ldg(s), w = __ldg(s + 1);
        x[0] = u.x; x[1] = u.y; x[2] = u.z; x[3] = u.w; x[4] = w.x; x[5] = w.y; x[6] = w.z; x[7] = w.w;
    } else {
#pragma unroll
        for (int i = 0; i < 8; ++i) x[i] = 0.f;
    }
}

// 8 staged fp32 values, or zeros for a row beyond the sequence
__device__ __forceinline__ void ld_stage8(const float *src, bool ok, float (&x)[8]) {
    const float4 u = *reinterpret_cast<const float4 *>(src), w = *reinterpret_cast<const float4 *>(src + 4);
    x[0] = ok ? u.x : 0.f; x[1] = ok ? u.y : 0.f; x[2] = ok ? u.z : 0.f; x[3] = ok ? u.w : 0.f;
    x[4] = ok ? w.x : 0.f; x[5] = ok ? w.y : 0.f; x[6] = ok ? w.z : 0.f; x[7] = ok ? w.w : 0.f;
}

// the 32 column sums of a warp's 32 x 32 values: lane i returns the sum of column i
__device__ __forceinline__ float reduce_scatter32(float (&x)[32], int lane) {
#pragma unroll
    for (int w = 16; w >= 1; w >>= 1) {
        const bool up = (lane & w) != 0;
#pragma unroll
        for (int i = 0; i < w; ++i) {
            const float keep = up ? x[i + w] : x[i], send = up ? x[i] : x[i + w];
            x[i] = keep + __shfl_xor_sync(0xFFFFFFFFu, send, w);
        }
    }
    return x[0];
}

template <bool kPre>
__global__ void __launch_bounds__(kThreads, 1) hla3_tc_kernel(Params p) {
    extern __shared__ __align__(1024) uint8_t smem[];
    Misc *ms = reinterpret_cast<Misc *>(smem + kSmemBlocks);
    auto blk = [&](int b) { return smem + b * kBlockBytes; };
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const bool issuer = warp == kIssuerWarp;

    if (smem_u32(smem) & 1023u) {  // the swizzled layout needs 1 KiB alignment
        if (tid == 0) set_error(p.err, 399, smem_u32(smem));
        return;
    }
    if (tid == 0) {
        for (int b = 0; b < kNumBars; ++b)
            mbar_init(&ms->bar[b], ((b >= bEp0 && b <= bEp3) || b == bEpQK) ? kEpiWarps : 1);
        ms->abort_flag = 0;
        fence_mbar_init();
    }
    if (issuer) {
        tmem_alloc(&ms->tmem_base, 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tb = ms->tmem_base;
    const int items = p.BH * p.G;

    if (issuer) {
        if (lane == 0) {
            const uint32_t sb4 = smem_u32(smem) >> 4;
            auto lk = [&](int b) { return sb4 + (uint32_t)b * kBlk16 + kLboK; };   // K-major block
            auto lm = [&](int b) { return sb4 + (uint32_t)b * kBlk16 + kLboMN; };  // MN-major block
            const uint32_t car = lk(bCar);  // + 256 per 32-row carry operand
            uint32_t n_tiles = 0, st_pend = 0, st_iss = 0;  // st_iss bit s: copies into stage s, mod 2
            auto stage_copy = [&](int s, int head, int j) {  // pre-pass: tile j's Q, K, V into stage s
                const int tok0 = j * kTile, rows = min(kTile, p.n - tok0);
                const uint32_t bytes = (uint32_t)rows * kD * sizeof(float);
                const size_t off = ((size_t)head * p.n + tok0) * kD;
                st_pend |= 1u << s;
                st_iss ^= 1u << s;
                mbar_arrive_expect_tx(&ms->bar[bSt0 + s], 3 * bytes);
                bulk_load(blk(stage_block(s, 0)), p.q + off, bytes, &ms->bar[bSt0 + s]);
                bulk_load(blk(stage_block(s, 1)), p.k + off, bytes, &ms->bar[bSt0 + s]);
                bulk_load(blk(stage_block(s, 2)), p.v + off, bytes, &ms->bar[bSt0 + s]);
            };
            for (int item = blockIdx.x; item < items && !ms->abort_flag; item += gridDim.x) {
                const int head = item / p.G, g = item % p.G;
                if (kPre && g == p.G - 1) continue;  // nobody reads the last segment's sums
                const int j0 = g * p.L, j1 = min(p.M, j0 + p.L);
                if (kPre)  // the first tiles' copies (every stage is free between items)
                    for (int t = 0; t < kStages && j0 + t < j1; ++t) stage_copy((n_tiles + t) % kStages, head, j0 + t);
                for (int j = j0; j < j1; ++j, ++n_tiles) {
                    const uint32_t tp = n_tiles & 1;
                    if (!bar_wait(ms, kPre ? bEp0 : bEpQK, tp, p)) break;  // Q, K, V in shared memory
                    tc_fence_after();
                    if (kPre) {
                        st_pend &= ~(1u << (n_tiles % kStages));  // read by the epilogue
                        if (j + kStages < j1) stage_copy(n_tiles % kStages, head, j + kStages);
                        const int o = 3 * (int)(n_tiles & 1);  // block set of this tile
                        mma_tok<true, true, 64>(tb + kTCar + 0, lm(o + 1), lm(o + 1), 1u);   // [S^K; P^T] += [K V]^T K
                        mma_tok<true, true, 64>(tb + kTCar + 64, lm(o), lm(o), 1u);          // S^Q += Q^T Q
                        umma_commit(&ms->bar[(n_tiles & 1) ? bEvO1 : bEvO]);
                        continue;
                    }
                    mma_feat3<128>(tb + kTA, lk(bQ), lk(bK), 0u);        // A = Q K^T (under the carry fold)
                    umma_commit(&ms->bar[bEvA]);
                    if (!bar_wait(ms, bEp0, tp, p)) break;              // the carries (bf16) in shared memory
                    tc_fence_after();
                    mma_feat3<32>(tb + kTQS, lk(bQ), car, 0u);           // Q S^K_p
                    mma_feat3<32>(tb + kTKS, lk(bK), car + 256, 0u);     // K S^Q_p
                    umma_commit(&ms->bar[bEvQ]);
                    // carries that need only this tile's tokens, while the epilogue forms LA
                    mma_tok<true, true, 64>(tb + kTCar + 0, lm(bK), lm(bK), 1u);   // [S^K; P^T] += [K V]^T K
                    mma_tok<true, true, 64>(tb + kTCar + 64, lm(bQ), lm(bQ), 1u);  // S^Q += Q^T Q
                    if (!bar_wait(ms, bEp1, tp, p)) break;              // LA (hi, lo)
                    tc_fence_after();
                    mma_tok<false, true, 64>(tb + kTY, lk(bLh), lm(bV), 0u);   // Y = LA V (hi | lo halves)
                    mma_tok<false, true, 64>(tb + kTY, lk(bLl), lm(bV), 1u);
                    mma_feat3<32>(tb + kTY, lk(bQ), car + 512, 1u);           //   + Q P_p
                    umma_commit(&ms->bar[bEvY]);
                    // C' = LA LA^T while the epilogue forms Z', aV and Q S^K_p
                    mma_tok<false, false, 128>(tb + kTA, lk(bLh), lk(bLh), 0u);
                    mma_tok<false, false, 128>(tb + kTA, lk(bLh), lk(bLl), 1u);
                    mma_tok<false, false, 128>(tb + kTA, lk(bLl), lk(bLh), 1u);
                    if (!bar_wait(ms, bEp2, tp, p)) break;              // Q S^K_p, aV, Z' (hi | lo)
                    tc_fence_after();
                    mma_feat3<128>(tb + kTA, lk(bQS), lk(bQ), 1u);             // C' += (Q S^K_p) Q^T
                    mma_tok<true, true, 64>(tb + kTG, lm(bLh), lm(bAV), 0u);   // G'' = LA^T aV
                    mma_tok<true, true, 64>(tb + kTG, lm(bLl), lm(bAV), 1u);
                    umma_commit(&ms->bar[bEvC]);
                    // while the epilogue forms L . C' and G': num = LA Z' + Q F_p, F^T += aV^T (Q S^K_p)
                    mma_tok<false, true, 64>(tb + kTY, lk(bLh), lm(bZ), 0u);
                    mma_tok<false, true, 64>(tb + kTY, lk(bLl), lm(bZ), 1u);
                    mma_feat3<32>(tb + kTY, lk(bQ), car + 768, 1u);
                    mma_tok<true, true, 64>(tb + kTCar + 192, lm(bAV), lm(bQS), 1u);
                    if (!bar_wait(ms, bEp3, tp, p)) break;              // L . C' (packed over C'), G'
                    tc_fence_after();
                    mma_ts_tok<64>(tb + kTY, tb + kTA, lm(bAV), 1u);        // num += (L . C') aV: hi
                    mma_ts_tok<64>(tb + kTY, tb + kTA + 16, lm(bAV), 1u);   //   and lo (packed in TMEM)
                    mma_tok<true, true, 64>(tb + kTCar + 192, lm(bG), lm(bK), 1u);    // F^T += G'^T K
                    umma_commit(&ms->bar[bEvO]);
                }
            }
            if (ms->abort_flag) {  // copies and MMAs in flight finish (bounded) before release
                for (int st = 0; st < kStages; ++st)
                    if ((st_pend >> st) & 1u) mbar_wait(&ms->bar[bSt0 + st], ((st_iss >> st) & 1u) ^ 1u, kBarWaitNs);
                umma_commit(&ms->bar[bTear]);
                mbar_wait(&ms->bar[bTear], 0, kBarWaitNs);
            }
        }
        __syncwarp();
    } else {
        // ================================ epilogue ================================
        const int qd = warp & 3, cq = warp >> 2;
        const int r = 32 * qd + lane;
        const uint32_t lb = (uint32_t)(32 * qd) << 16;
        // carry cq (S^K, S^Q, P^T, F^T) lives in TMEM region 0, 1, 0, 3 (P^T in lanes 64..127 of the
        // [K; V]^T K product); the two warps on its lanes fold it (c_half: rows 0..31 or 32..63)
        const int c_reg = cq == 2 ? 0 : cq;
        const bool c_act = cq == 2 ? qd >= 2 : qd < 2;
        const int c_half = qd & 1;
        const uint32_t treg = tb + lb + kTCar + 64u * (uint32_t)c_reg;  // this warp's lanes of it
        uint32_t n_tiles = 0, st_par = 0;
        // tokens are read 4 threads to a row (a warp covers 8 consecutive rows, 1 KiB)
        const int e_row = tid >> 2, e_c = (tid & 3) * 8;
        float pq[8], pk[8], pv[8];  // sweep: fp32 (8 columns) of the tile to come

        // rows 0..63 of carry region cq (lanes of the quadrant-0 and -1 warps) folded into
        // ms->fold[cq] as the fp32 32 x 32 carry: hi and lo columns added, rows 32..63 onto 0..31
        auto carry_fold = [&]() {
#pragma unroll
            for (int pass = 1; pass >= 0; --pass) {
                if (c_act && c_half == pass) {
#pragma unroll
                    for (int h = 0; h < 32; h += 16) {
                        uint32_t d0[16], d1[16];
                        tmem_ld16(treg + h, d0);
                        tmem_ld16(treg + 32 + h, d1);
                        tmem_ld_wait();
#pragma unroll
                        for (int f = 0; f < 16; ++f) {
                            const float x = __uint_as_float(d0[f]) + __uint_as_float(d1[f]);
                            float &dst = ms->fold[cq][lane][h + f];
                            dst = pass ? x : dst + x;
                        }
                    }
                }
                epi_sync();
            }
        };
        // after carry_fold: thread et owns 8 values of the folded carries (region, row, columns)
        const int f_rg = tid >> 7, f_row = (tid >> 2) & 31, f_c = (tid & 3) * 8;

        for (int item = blockIdx.x; item < items; item += gridDim.x) {
            const int head = item / p.G, g = item % p.G;
            if (kPre && g == p.G - 1) continue;
            const int j0 = g * p.L, j1 = min(p.M, j0 + p.L);
            // carries at the segment start: S^K, S^Q, P^T summed over the earlier segments, F = 0
            if (c_act) {
                uint32_t z[32];
#pragma unroll
                for (int f = 0; f < 32; ++f) z[f] = 0u;
                if (!kPre && c_half == 0 && cq < 3) {
                    float s[32];
#pragma unroll
                    for (int f = 0; f < 32; ++f) s[f] = 0.f;
                    for (int h = 0; h < g; ++h) {
                        const float4 *src = reinterpret_cast<const float4 *>(
                            p.rec + (((size_t)head * p.G + h) * 3 + cq) * 1024 + lane * 32);
#pragma unroll
                        for (int f = 0; f < 8; ++f) {
                            const float4 u = __ldcg(src + f);
                            s[4 * f] += u.x; s[4 * f + 1] += u.y; s[4 * f + 2] += u.z; s[4 * f + 3] += u.w;
                        }
                    }
#pragma unroll
                    for (int f = 0; f < 32; ++f) z[f] = __float_as_uint(s[f]);
                }
                tmem_st32(treg, z);
#pragma unroll
                for (int f = 0; f < 32; ++f) z[f] = 0u;
                tmem_st32(treg + 32, z);
                tmem_st_wait();
            }
            if (!kPre) {
                load_row8(p.q, p.n, head, j0 * kTile + e_row, e_c, pq);
                load_row8(p.k, p.n, head, j0 * kTile + e_row, e_c, pk);
                load_row8(p.v, p.n, head, j0 * kTile + e_row, e_c, pv);
            }

            // tiles j0 .. j1 - 1, then (j = j1) the segment totals once the last tile's MMAs are done
            for (int j = j0; j <= j1; ++j) {
                const uint32_t tp = n_tiles & 1;
                const int tok0 = j * kTile;
                const bool totals = j == j1;
                if (!kPre && j > j0) {  // the previous tile's products are done (its outputs are read below)
                    bar_wait(ms, bEvO, tp ^ 1u, p);
                    tc_fence_after();
                }
                // ---- E0: Q, K, V -> hi | lo blocks (A = Q K^T starts on them); the previous tile's
                // outputs; carries -> bf16 operands ----
                if (!totals) {
                    if (kPre) {  // this tile's copies in stage n_tiles % 2 (rows beyond n are stale: zero)
                        const int st = n_tiles % kStages;
                        if (n_tiles >= 2) {  // the products of tile n_tiles - 2 have read this block set
                            bar_wait(ms, (n_tiles & 1) ? bEvO1 : bEvO, ((n_tiles >> 1) + 1) & 1, p);
                            tc_fence_after();
                        }
                        bar_wait(ms, bSt0 + st, (st_par >> st) & 1u, p);
                        st_par ^= 1u << st;
                        const int so = e_row * kD + e_c;
                        const bool ok = tok0 + e_row < p.n;
                        ld_stage8(reinterpret_cast<const float *>(blk(stage_block(st, 0))) + so, ok, pq);
                        ld_stage8(reinterpret_cast<const float *>(blk(stage_block(st, 1))) + so, ok, pk);
                        ld_stage8(reinterpret_cast<const float *>(blk(stage_block(st, 2))) + so, ok, pv);
                    }
                    const int o = kPre ? 3 * (int)(n_tiles & 1) : 0;  // block set (Q, K, V at o, o + 1, o + 2)
                    store_hl8(blk(o + bQ), e_row, e_c, pq);
                    store_hl8(blk(o + bK), e_row, e_c, pk);
                    store_hl8(blk(o + bV), e_row, e_c, pv);
                    if (!kPre) {
                        float dp = 0.f;
#pragma unroll
                        for (int u = 0; u < 8; ++u) dp = fmaf(pq[u], pk[u], dp);
                        ms->sdp[e_c / 8][e_row] = dp;
                        fence_async_smem();
                        epi_arrive(ms, bEpQK);
                    }
                }
                if (!kPre && j > j0) {  // ---- E4 of the previous tile: its outputs ----
                    uint32_t o0[8], o1[8];
                    tmem_ld8(tb + lb + kTY + 8 * cq, o0);
                    tmem_ld8(tb + lb + kTY + 32 + 8 * cq, o1);
                    tmem_ld_wait();
                    const int t = tok0 - kTile + r;
                    if (t < p.n) {
                        float4 *dst = reinterpret_cast<float4 *>(p.out + ((size_t)head * p.n + t) * kD + 8 * cq);
                        float o[8];
#pragma unroll
                        for (int u = 0; u < 8; ++u) o[u] = __uint_as_float(o0[u]) + __uint_as_float(o1[u]);
                        dst[0] = make_float4(o[0], o[1], o[2], o[3]);
                        dst[1] = make_float4(o[4], o[5], o[6], o[7]);
                    }
                }
                if (kPre && totals && n_tiles > 0) {  // the last tile's products (and so all) are done
                    const uint32_t c = n_tiles - 1;
                    bar_wait(ms, (c & 1) ? bEvO1 : bEvO, (c >> 1) & 1, p);
                    tc_fence_after();
                }
                if (!kPre || totals) {
                    carry_fold();
                    float x[8];
#pragma unroll
                    for (int u = 0; u < 8; ++u) x[u] = ms->fold[f_rg][f_row][f_c + u];
                    if (!totals) {
                        store_hl8(blk(bCar), 32 * f_rg + f_row, f_c, x);
                    } else if (kPre ? f_rg < 3 : f_rg == 3) {
                        float *dst = kPre ? p.rec + (((size_t)head * p.G + g) * 3 + f_rg) * 1024
                                          : p.dF + ((size_t)head * p.G + g) * 1024;
                        float4 *d4 = reinterpret_cast<float4 *>(dst + f_row * 32 + f_c);
                        __stcg(d4, make_float4(x[0], x[1], x[2], x[3]));
                        __stcg(d4 + 1, make_float4(x[4], x[5], x[6], x[7]));
                    }
                }
                if (totals) {
                    epi_sync();  // every fold read before the next item's stores
                    break;
                }
                fence_async_smem();
                epi_arrive(ms, bEp0);
                auto prefetch = [&]() {  // the next tile's rows load while this one is worked on
                    if (j + 1 < j1) {
                        load_row8(p.q, p.n, head, tok0 + kTile + e_row, e_c, pq);
                        load_row8(p.k, p.n, head, tok0 + kTile + e_row, e_c, pk);
                        load_row8(p.v, p.n, head, tok0 + kTile + e_row, e_c, pv);
                    }
                };
                if (kPre) {
                    ++n_tiles;
                    continue;
                }
                // ---- E1: A -> a, column sums of squares above the diagonal, LA (hi, lo) ----
                // The diagonal a_t = q_t . k_t is taken from the fp32 tokens, not from the split
                // product: the first output of a head is a_0^3 v_0, so a_0 needs a small error
                // relative to itself, not to |q_0| |k_0|.
                bar_wait(ms, bEvA, tp, p);
                tc_fence_after();
                epi_sync();  // every partial q_t . k_t written
                {
                    uint32_t a[32];
                    tmem_ld32(tb + lb + kTA + 32 * cq, a);
                    tmem_ld_wait();
                    const bool diag = cq == qd;  // this block holds the diagonal element of row r
                    const float dg = ((ms->sdp[0][r] + ms->sdp[1][r]) + (ms->sdp[2][r] + ms->sdp[3][r]));
                    if (diag) {
#pragma unroll
                        for (int i = 0; i < 32; ++i) a[i] = (i == lane) ? __float_as_uint(dg) : a[i];
                        ms->sa[r] = dg;
                    }
                    // this warp's 32 x 32 block lies above the diagonal (blk_zero), below it (blk_full) or on it
                    const bool blk_zero = cq > qd, blk_full = cq < qd;
#pragma unroll
                    for (int jj = 0; jj < 32; jj += 8) {
                        uint4 h = make_uint4(0u, 0u, 0u, 0u), l = h;
                        if (!blk_zero) {
                            float x[8];
#pragma unroll
                            for (int u = 0; u < 8; ++u)
                                x[u] = (blk_full || 32 * cq + jj + u <= r) ? __uint_as_float(a[jj + u]) : 0.f;
                            split8(x, h, l);
                        }
                        st16(blk(bLh), r, 32 * cq + jj, h);
                        st16(blk(bLl), r, 32 * cq + jj, l);
                    }
                    if (blk_full) {  // no entry above the diagonal
                        ms->sbp[qd][32 * cq + lane] = 0.f;
                    } else {
                        float x[32];
#pragma unroll
                        for (int i = 0; i < 32; ++i) {
                            const float av = __uint_as_float(a[i]);
                            x[i] = (blk_zero || r < 32 * cq + i) ? av * av : 0.f;
                        }
                        ms->sbp[qd][32 * cq + lane] = reduce_scatter32(x, lane);
                    }
                }
                fence_async_smem();
                epi_arrive(ms, bEp1);
                // ---- E2: b, Z' = a Y + (b - a^2) V, aV, Q S^K_p -> hi | lo ----
                bar_wait(ms, bEvQ, tp, p);
                bar_wait(ms, bEvY, tp, p);
                tc_fence_after();
                float zf[8];
                {
                    float kf[8], vf[8];  // K and V rows as the products see them (hi + lo)
                    load_hl8(blk(bK), r, 8 * cq, kf);
                    load_hl8(blk(bV), r, 8 * cq, vf);
                    uint32_t ks[8], y0[8], y1[8], qs[8];
                    tmem_ld8(tb + lb + kTKS + 8 * cq, ks);
                    tmem_ld8(tb + lb + kTY + 8 * cq, y0);
                    tmem_ld8(tb + lb + kTY + 32 + 8 * cq, y1);
                    tmem_ld8(tb + lb + kTQS + 8 * cq, qs);
                    tmem_ld_wait();
                    float part = 0.f;
#pragma unroll
                    for (int u = 0; u < 8; ++u) part += __uint_as_float(ks[u]) * kf[u];
                    ms->sbp2[cq][r] = part;
                    epi_sync();
                    const float a = ms->sa[r];
                    const float b = ((ms->sbp[0][r] + ms->sbp[1][r]) + (ms->sbp[2][r] + ms->sbp[3][r])) +
                                    ((ms->sbp2[0][r] + ms->sbp2[1][r]) + (ms->sbp2[2][r] + ms->sbp2[3][r]));
                    const float bz = b - a * a;
                    float av[8], qsf[8];
#pragma unroll
                    for (int u = 0; u < 8; ++u) {
                        zf[u] = a * (__uint_as_float(y0[u]) + __uint_as_float(y1[u])) + bz * vf[u];
                        av[u] = a * vf[u];
                        qsf[u] = __uint_as_float(qs[u]);
                    }
                    store_hl8(blk(bZ), r, 8 * cq, zf);
                    store_hl8(blk(bAV), r, 8 * cq, av);
                    store_hl8(blk(bQS), r, 8 * cq, qsf);
                }
                fence_async_smem();
                epi_arrive(ms, bEp2);
                // ---- E3: G' = Z' + LA^T aV -> hi | lo; L . C' -> hi, lo packed over C' in TMEM ----
                // (each thread packs its own 32 columns into their first 16 (hi) and last 16 (lo),
                // so no thread overwrites columns another still reads; LA stays in shared memory
                // for the products issued meanwhile)
                bar_wait(ms, bEvC, tp, p);
                tc_fence_after();
                {
                    uint32_t g0[8], g1[8];
                    tmem_ld8(tb + lb + kTG + 8 * cq, g0);
                    tmem_ld8(tb + lb + kTG + 32 + 8 * cq, g1);
                    tmem_ld_wait();
                    float gf[8];
#pragma unroll
                    for (int u = 0; u < 8; ++u) gf[u] = zf[u] + (__uint_as_float(g0[u]) + __uint_as_float(g1[u]));
                    store_hl8(blk(bG), r, 8 * cq, gf);
                }
                {
                    const bool blk_zero = cq > qd, blk_full = cq < qd;  // above, below or on the diagonal
                    uint32_t hp[16], lp[16];
                    if (blk_zero) {
#pragma unroll
                        for (int i = 0; i < 16; ++i) hp[i] = lp[i] = 0u;
                    } else {
                        uint32_t c[32];
                        tmem_ld32(tb + lb + kTA + 32 * cq, c);
                        tmem_ld_wait();
#pragma unroll
                        for (int i = 0; i < 16; ++i) {
                            const int c0 = 32 * cq + 2 * i;
                            const float x0 = (blk_full || c0 <= r) ? __uint_as_float(c[2 * i]) : 0.f;
                            const float x1 = (blk_full || c0 + 1 <= r) ? __uint_as_float(c[2 * i + 1]) : 0.f;
                            hp[i] = pack_bf16x2(x0, x1);
                            lp[i] = pack_bf16x2(x0 - __uint_as_float(hp[i] << 16), x1 - __uint_as_float(hp[i] & 0xFFFF0000u));
                        }
                    }
                    tmem_st16(tb + lb + kTA + 32 * cq, hp);
                    tmem_st16(tb + lb + kTA + 32 * cq + 16, lp);
                    tmem_st_wait();
                }
                fence_async_smem();
                epi_arrive(ms, bEp3);
                prefetch();
                ++n_tiles;
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (issuer) {
        tc_fence_after();
        tmem_dealloc(tb, 512);
    }
}

// out[t] += q_t^T F_start(g) for the tiles of segments g >= 1 (F_start: the F^T totals of the
// segments before g); one block per tile of a head: the tile's Q rows and F_start staged in
// shared memory, each thread forms 4 tokens x 4 outputs.  Every global load (Q rows, the
// thread's outputs, the totals) is issued before the first shared-memory store.
__global__ void __launch_bounds__(256) hla3_tc_fixup_kernel(const float *__restrict__ q, float *__restrict__ out,
                                                             const float *__restrict__ dF, int n, int G, int L) {
    __shared__ __align__(16) float Qs[kTile][kD + 4];
    __shared__ __align__(16) float Fs[kD][kD + 4];  // Fs[f][j] = F_start[f][j]
    const int head = blockIdx.y, j = blockIdx.x + L, g = j / L, tok0 = j * kTile;
    const int tid = threadIdx.x;
    const int tg = tid >> 3, c0 = (tid & 7) * 4;  // tokens 4 tg .. +3, outputs c0 .. +3
    float4 qv[4], ov[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {  // Q rows: element e = tid + 256 i of the tile's 128 x 8 float4
        const int e = tid + 256 * i, row = e >> 3, c4 = (e & 7) * 4;
        qv[i] = tok0 + row < n ? __ldg(reinterpret_cast<const float4 *>(q + ((size_t)head * n + tok0 + row) * kD + c4))
                               : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int t = tok0 + 4 * tg + i;
        ov[i] = t < n ? *reinterpret_cast<const float4 *>(out + ((size_t)head * n + t) * kD + c0)
                      : make_float4(0.f, 0.f, 0.f, 0.f);
    }
    float fs[4] = {0.f, 0.f, 0.f, 0.f};  // F^T elements tid + 256 i summed over the earlier segments
    for (int h = 0; h < g; ++h)
#pragma unroll
        for (int i = 0; i < 4; ++i) fs[i] += __ldcg(dF + ((size_t)head * G + h) * 1024 + tid + 256 * i);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int e = tid + 256 * i;
        *reinterpret_cast<float4 *>(&Qs[e >> 3][(e & 7) * 4]) = qv[i];
        Fs[e % kD][e / kD] = fs[i];
    }
    __syncthreads();
    float acc[4][4] = {};
#pragma unroll 8
    for (int f = 0; f < kD; f += 4) {
        float4 a4[4], f4[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) a4[i] = *reinterpret_cast<const float4 *>(&Qs[4 * tg + i][f]);
#pragma unroll
        for (int u = 0; u < 4; ++u) f4[u] = *reinterpret_cast<const float4 *>(&Fs[f + u][c0]);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float qq[4] = {a4[i].x, a4[i].y, a4[i].z, a4[i].w};
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                acc[i][0] += qq[u] * f4[u].x;
                acc[i][1] += qq[u] * f4[u].y;
                acc[i][2] += qq[u] * f4[u].z;
                acc[i][3] += qq[u] * f4[u].w;
            }
        }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int t = tok0 + 4 * tg + i;
        if (t >= n) break;
        float4 x = ov[i];
        x.x += acc[i][0]; x.y += acc[i][1]; x.z += acc[i][2]; x.w += acc[i][3];
        *reinterpret_cast<float4 *>(out + ((size_t)head * n + t) * kD + c0) = x;
    }
}

struct Plan {
    int M, G, L;
};

Plan plan(int BH, int n, int sms) {
    Plan pl;
    pl.M = (n + kTile - 1) / kTile;
    int G = sms / (BH > 0 ? BH : 1);
    if (const char *e = getenv("HLA3_SEGMENT_TILES")) {  // tests: force the segment length
        const int L = atoi(e);
        if (L > 0) G = (pl.M + L - 1) / L;
    }
    G = G < 1 ? 1 : (G > pl.M ? pl.M : G);
    G = G > kMaxSegments ? kMaxSegments : G;
    pl.L = (pl.M + G - 1) / G;
    pl.G = (pl.M + pl.L - 1) / pl.L;
    return pl;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

size_t hla3_tc_workspace_bytes(int BH, int n) {
    if (BH <= 0 || n <= 0) return kWsHeaderBytes;
    const long long M = (n + kTile - 1) / kTile;
    const long long G = M < kMaxSegments ? M : kMaxSegments;
    return kWsHeaderBytes + sizeof(float) * (size_t)BH * G * 4 * 1024;
}

bool hla3_tc_applicable(const Fwd2 &p) {
    if (getenv("HLA_DISABLE_FUSED")) return false;
    if (p.dt != HLA_F32 || p.d != kD || p.dv != kD || !p.masked || p.normalized) return false;
    if (p.state_in || p.state_out || p.n <= 0 || p.BH <= 0) return false;
    if (!aligned16(p.q) || !aligned16(p.k) || !aligned16(p.v) || !aligned16(p.out)) return false;
    if (p.ws_bytes < hla3_tc_workspace_bytes(p.BH, p.n)) return false;
    int dev = 0, major = 0, minor = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return false;
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    return major == 10 && minor == 3;
}

int hla3_tc_launches(int BH, int n) {
    int dev = 0, sms = 152;
    if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    return plan(BH, n, sms).G > 1 ? 3 : 1;
}

cudaError_t hla3_tc_forward(const Fwd2 &p, cudaStream_t stream) {
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const Plan pl = plan(p.BH, p.n, sms);
    Params kp{};
    kp.q = static_cast<const float *>(p.q);
    kp.k = static_cast<const float *>(p.k);
    kp.v = static_cast<const float *>(p.v);
    kp.out = static_cast<float *>(p.out);
    float *ws = reinterpret_cast<float *>(p.ws + kWsHeaderBytes);
    kp.dF = ws;
    kp.rec = ws + (size_t)p.BH * pl.G * 1024;
    kp.BH = p.BH;
    kp.n = p.n;
    kp.M = pl.M;
    kp.G = pl.G;
    kp.L = pl.L;
    kp.err = reinterpret_cast<WsHeader *>(p.ws);
    cudaError_t e;
    if ((e = cudaFuncSetAttribute(hla3_tc_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes)))
        return e;
    if ((e = cudaFuncSetAttribute(hla3_tc_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)kSmemBytes)))
        return e;
    const int items = p.BH * pl.G;
    if (pl.G > 1) hla3_tc_kernel<true><<<items < sms ? items : sms, kThreads, kSmemBytes, stream>>>(kp);
    hla3_tc_kernel<false><<<items < sms ? items : sms, kThreads, kSmemBytes, stream>>>(kp);
    if (pl.G > 1)
        hla3_tc_fixup_kernel<<<dim3(pl.M - pl.L, p.BH), 256, 0, stream>>>(kp.q, kp.out, kp.dF, p.n, pl.G, pl.L);
    return cudaGetLastError();
}

}  // namespace hla
