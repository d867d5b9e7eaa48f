// Backward of masked second-order HLA on the tensor cores (sm_103a): tcgen05 MMAs
// with TMEM accumulators, TMA tile loads, one persistent CTA per head.
//
// The gradients are the adjoint of the chunked forward (Sec. "Chunk-parallel
// training via associative scans": the reverse scan with the adjoint of the
// semidirect product, checkpoints at tile boundaries).  With x_j = S_j q_j,
// T_tj = q_t . x_j and P_tj = g_t . v_j (both for j <= t), per 128-token tile
// (rows = tokens; p = prefix before the tile, s = suffix after it):
//   forward:  W = L . (Q K^T),  X = W K + Q S_p,  T = L . (Q X^T)
//   backward: P = L . (G V^T),  Y = P^T Q + V Gam_s     (y_j = sum_{t>=j} P_tj q_t)
//             dV = T^T G + X Gam_s^T
//             B = L . (Y K^T)
//             dQ = P X + G D_p^T + Y S_p + B K
//             dK = K Lam_s + W^T Y + B^T Q
// with the forward prefixes S_p = sum k k^T, D_p = sum x v^T and the suffix sums
// Gam_s^T = sum q g^T and Lam_s = sum (y q^T + q y^T), which the reverse sweep
// carries as Gam^T += Q^T G and Lam'' += Q^T Y with Lam_s = Lam'' + Lam''^T (K Lam_s
// reads Lam'' once K-major and once MN-major; one N = 128 product serves both carries).
//
// One kernel, per head: a forward sweep over the tiles carries S and D in TMEM
// and stores per tile a record of X (hi, lo) and the bf16 checkpoints S_p, D_p
// (the swizzled shared-memory image of three blocks, one 1-D bulk copy); a
// reverse sweep reloads the records, so it never forms W or X again, and
// carries Gam^T and Lam in TMEM.  No CTA waits on another.
//
// Precision.  A gradient row can be a small difference of large terms (dq_0 is
// k_0 times k_0 . y_0 plus a P X term, for one), so an intermediate rounded once
// to bf16 can miss the row by far more than its own 2^-9.  Every intermediate
// that feeds such a sum is therefore an exact pair hi + lo of bf16 values
// (lo = bf16(x - hi), 2^-17 together) and its products take the terms hi.hi,
// hi.lo and lo.hi: W, P, X, Y, B and the carries Gam_s, Lam_s.  T (it only
// scales rows of G) and the checkpoints S_p, D_p stay single.
//
// Layout.  Token operands are bf16 in the 128-byte-swizzled layout TMA writes
// (128 rows x 64 columns per 16 KiB block; 64 x 64 matrices in the first 64
// rows of an 8 KiB half); X and Y go to shared memory as hi and lo blocks.  The
// 128 x 128 masked tiles never touch shared memory: each is formed in TMEM, the
// epilogue masks it and writes it back over its own columns as packed bf16
// hi/lo, and the next product reads it there as its A operand.  A transposed
// use (P^T, T^T, W^T, B^T) is its own product (V G^T, X Q^T, K Q^T, K Y^T) with
// the mask turned over.  Products on the carries read K^T, X^T, Q^T MN-major
// as the M side of an M = 128 product; rows 64..127 come from the next block
// and land in TMEM lanes nobody reads.
//
// TMEM (512 columns): DQ (64) dQ; DK (64) X (forward), Y -> dV -> dK (reverse);
// GAM, LAM (64 each) the carries (forward S, D; reverse Gam^T, Lam''), rows
// 0..63; T0, T1 (128 each) the masked tiles: forward W in T0; reverse P^T, T^T,
// B^T in T0 and P, B, W^T in T1.
//
// Roles: warp 16 issues TMA copies and MMAs (one thread); in the reverse sweep
// warp 17 issues the second half of the MMAs (P, B, W^T in T1, dQ, the carries),
// since one thread issues a 128 x 64 x 16 MMA with A in TMEM no faster than
// about one per 55 cycles and two threads overlap them; warps 0..15 are the
// epilogue (warp w: TMEM lanes 32 (w % 4) .. +31, one token row each; column
// quarter w / 4).
//
// Scope: bf16 tokens, d = dv = 64, masked, plain (unnormalised) output.
#include <cstdlib>

#include "hla_internal.h"
#include "sm103_prims.cuh"

namespace hla {
namespace {

using namespace sm103;

constexpr int kTile = 128, kD = 64;
constexpr int kEpiWarps = 16, kEpiThreads = kEpiWarps * 32, kIssuerWarp = kEpiWarps, kIssuer2Warp = kEpiWarps + 1;
constexpr int kThreads = kEpiThreads + 64;

// shared-memory blocks of 16 KiB (128 rows x 64 bf16)
enum Block {
    bQ = 0, bK = 1, bV = 2, bG = 3,
    bYh = 4, bYl = 5,  // Y = hi + lo (Y_hi right after G: Q^T [G | Y_hi] is one N = 128 product)
    bXh = 6, bXl = 7,  // X = hi + lo
    bCk = 8,           // S_p (rows 0..63 of the first 8 KiB), D_p (the second 8 KiB): the checkpoint image
    bGam = 9,          // Gam_s^T: hi (first 8 KiB), lo (second 8 KiB)
    bLam = 10,         // Lam''_s (Lam_s = Lam'' + Lam''^T): hi, lo
    bQ2 = 11,          // the second Q, K, V set at 11, 12, 13 (tiles alternate between the sets)
    kBlocks = 14
};
static_assert(bXl == bXh + 1 && bCk == bXh + 2, "a tile's record is three consecutive blocks");
constexpr uint32_t kHalf = kBlockBytes / 2;
constexpr uint32_t kSmemBlocks = kBlocks * kBlockBytes;
// one record per tile, the image of blocks bXh, bXl, bCk: X (hi, lo), then S_p and D_p
constexpr uint32_t kCkBytes = 3 * kBlockBytes;

constexpr uint32_t kDQ = 0, kDK = 64, kGAM = 128, kLAM = 192, kT0 = 256, kT1 = 384;  // TMEM columns

enum Bar {
    bLd0 = 0, bLd1 = 1,  // tile copies: the two Q, K, V sets
    bLdG = 2,            // reverse sweep: G and the tile's record
    // MMA commits (forward: A, X, the carries; reverse: P^T, P, Y, T^T, B, dV, B^T, W^T, all)
    bEvA = 3, bEvA2 = 4, bEvX = 5, bEvC = 6, bEvT = 7, bEvB = 8, bEvV = 9, bEvB2 = 10, bEvW = 11, bEvO = 12,
    // epilogue hand-offs (16 warp arrivals each)
    bEp0 = 13, bEp1 = 14, bEp2 = 15,                             // both sweeps
    bEp1b = 16, bEp3 = 17, bEp4a = 18, bEp4b = 19, bEp5 = 20,  // reverse sweep
    bTear = 21,
    bCkDone = 22,  // a head's records are in global memory
    bEvCar = 23,   // reverse sweep, second issuer: the carries (its last reads of G, X and the checkpoint)
    bTear2 = 24,
    bEp5b = 25,   // reverse sweep: dQ read out of TMEM (DQ free for K Lam_s)
    bEvKL = 26,   // reverse sweep, second issuer: K Lam_s in DQ
    kNumBars = 27
};
__host__ __device__ constexpr bool epi_bar(int b) { return (b >= bEp0 && b <= bEp5) || b == bEp5b; }

struct Misc {
    uint64_t bar[kNumBars];
    uint32_t tmem_base;
    int abort_flag;
};
constexpr uint32_t kMiscBytes = 1024;
static_assert(sizeof(Misc) <= kMiscBytes, "misc smem");
constexpr uint32_t kSmemBytes = kSmemBlocks + kMiscBytes;

struct Params {
    uint8_t *ck;  // [BH][M] checkpoints of kCkBytes
    int BH, n, M;
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
    set_error(p.err, 500 + b, parity);
    ms->abort_flag = 1;
    return false;
}

__device__ __forceinline__ void epi_sync() { asm volatile("bar.sync 1, %0;" ::"n"(kEpiThreads) : "memory"); }

__device__ __forceinline__ void epi_arrive(Misc *ms, int b) {
    tc_fence_before();
    __syncwarp();
    if ((threadIdx.x & 31) == 0) mbar_arrive(&ms->bar[b]);
}

// 1-D bulk copies between global and shared memory (16-byte aligned, sizes a multiple of 16)
__device__ __forceinline__ void bulk_load(void *dst, const void *src, uint32_t bytes, uint64_t *bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                 ::"r"(smem_u32(dst)), "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(smem_u32(bar))
                 : "memory");
}
__device__ __forceinline__ void bulk_store(void *dst, const void *src, uint32_t bytes) {
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;"
                 ::"l"(reinterpret_cast<uint64_t>(dst)), "r"(smem_u32(src)), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void bulk_prefetch_l2(const void *src, uint32_t bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(reinterpret_cast<uint64_t>(src)), "r"(bytes)
                 : "memory");
}

// ------------------------------- MMA issue -------------------------------
constexpr uint32_t kDescHi = (1024u >> 4) | (1u << 14) | (2u << 29);
constexpr uint32_t kLboK = 1u << 16, kLboMN = (kBlockBytes >> 4) << 16;
constexpr uint32_t kBlk16 = kBlockBytes >> 4;
constexpr uint32_t kH16 = kHalf >> 4;  // the second 8 KiB of a block, in descriptor units

__device__ __forceinline__ uint64_t dsc(uint32_t lo) { return (static_cast<uint64_t>(kDescHi) << 32) | lo; }

// D (+)= A B over KS steps of K = 16, both operands in shared memory.  K-major operands:
// 64 K elements per 128-byte row, the next 64 in the next block; MN-major operands: 16 K
// rows (2 KiB) per step.
template <bool A_MN, bool B_MN, int N, int KS>
__device__ __forceinline__ void mma(uint32_t d, uint32_t a, uint32_t b, uint32_t acc) {
    constexpr uint32_t id = idesc_bf16(128, N, A_MN, B_MN);
#pragma unroll
    for (int kk = 0; kk < KS; ++kk) {
        const uint32_t ka = A_MN ? kk * 128u : (kk >> 2) * kBlk16 + (kk & 3) * 2u;
        const uint32_t kb = B_MN ? kk * 128u : (kk >> 2) * kBlk16 + (kk & 3) * 2u;
        umma_bf16(d, dsc(a + ka), dsc(b + kb), id, kk > 0 ? 1u : acc);
    }
}

// D (+)= A B over the 128 tokens of a tile, A a masked tile in TMEM (bf16 pairs packed in
// the first 16 of each 32 columns: K elements 32g .. 32g + 31 of a row in columns
// a + 32g .. +15, so K step kk starts at column 32 (kk / 2) + 8 (kk % 2); the lo parts sit
// 16 columns further), B a token block read MN-major, N = 64
__device__ __forceinline__ void mma_ts(uint32_t d, uint32_t a_tmem, uint32_t b, uint32_t acc) {
    constexpr uint32_t id = idesc_bf16(128, 64, 0, 1);
#pragma unroll
    for (int kk = 0; kk < 8; ++kk)
        umma_bf16_ts(d, a_tmem + 32u * (kk >> 1) + 8u * (kk & 1), dsc(b + kk * 128u), id, kk > 0 ? 1u : acc);
}

// ------------------------------- epilogue helpers -------------------------------
__device__ __forceinline__ uint4 pack8(const float *x) {
    return make_uint4(pack_bf16x2(x[0], x[1]), pack_bf16x2(x[2], x[3]), pack_bf16x2(x[4], x[5]),
                      pack_bf16x2(x[6], x[7]));
}

__device__ __forceinline__ void st16(uint8_t *tile, int r, int c, const uint4 &v) {
    *reinterpret_cast<uint4 *>(tile + tile_off(r, c)) = v;
}

// bf16 hi of a pair and lo = bf16(x - hi), packed
__device__ __forceinline__ void split2(float x0, float x1, uint32_t &h, uint32_t &l) {
    h = pack_bf16x2(x0, x1);
    l = pack_bf16x2(x0 - __uint_as_float(h << 16), x1 - __uint_as_float(h & 0xFFFF0000u));
}

// One warp's 32 columns (c0 .. c0 + 31) of row r of a 128 x 128 product in TMEM at `t`:
// masked (kUpper: column >= r, else column <= r) and written back over the same columns
// as packed bf16, hi at c0 and (kLo) lo at c0 + 16.
template <bool kUpper, bool kLo>
__device__ __forceinline__ void mask_pack(uint32_t t, int r, int c0) {
    // the warp's 32 x 32 block (rows 32 qd .., columns c0 ..) lies wholly outside the mask, wholly
    // inside it, or on the diagonal (warp-uniform)
    const int qd = r >> 5, cq = c0 >> 5;
    const bool zero = kUpper ? cq < qd : cq > qd, full = kUpper ? cq > qd : cq < qd;
    uint32_t hp[16], lp[16];
    if (zero) {
#pragma unroll
        for (int i = 0; i < 16; ++i) hp[i] = lp[i] = 0u;
    } else {
        uint32_t a[32];
        tmem_ld32(t + c0, a);
        tmem_ld_wait();
        if (full) {
#pragma unroll
            for (int i = 0; i < 16; ++i) split2(__uint_as_float(a[2 * i]), __uint_as_float(a[2 * i + 1]), hp[i], lp[i]);
        } else {
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                const int c = c0 + 2 * i;
                const bool k0 = kUpper ? c >= r : c <= r, k1 = kUpper ? c + 1 >= r : c + 1 <= r;
                split2(k0 ? __uint_as_float(a[2 * i]) : 0.f, k1 ? __uint_as_float(a[2 * i + 1]) : 0.f, hp[i], lp[i]);
            }
        }
    }
    tmem_st16(t + c0, hp);
    if (kLo) tmem_st16(t + c0 + 16, lp);
    tmem_st_wait();
}

// 16 fp32 TMEM values (columns c0 .. c0 + 15 of a 64-wide result) of row r as bf16 hi and
// lo into the same row of two blocks
__device__ __forceinline__ void store16_hl(uint8_t *hi, uint8_t *lo, int r, int c0, const uint32_t (&a)[16]) {
    uint32_t h[8], l[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) split2(__uint_as_float(a[2 * i]), __uint_as_float(a[2 * i + 1]), h[i], l[i]);
    st16(hi, r, c0, make_uint4(h[0], h[1], h[2], h[3]));
    st16(hi, r, c0 + 8, make_uint4(h[4], h[5], h[6], h[7]));
    st16(lo, r, c0, make_uint4(l[0], l[1], l[2], l[3]));
    st16(lo, r, c0 + 8, make_uint4(l[4], l[5], l[6], l[7]));
}

// the same, bf16 only
__device__ __forceinline__ void store16(uint8_t *blk, int r, int c0, const uint32_t (&a)[16]) {
    float x[16];
#pragma unroll
    for (int u = 0; u < 16; ++u) x[u] = __uint_as_float(a[u]);
    st16(blk, r, c0, pack8(x));
    st16(blk, r, c0 + 8, pack8(x + 8));
}

struct Tok {  // raw token pointers, for the L2 prefetch of the next reverse tile
    const __nv_bfloat16 *q, *k, *v, *g;
};

__global__ void __launch_bounds__(kThreads, 1)
bwd_tc_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
              const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_g,
              const __grid_constant__ CUtensorMap tm_dq, const __grid_constant__ CUtensorMap tm_dk,
              const __grid_constant__ CUtensorMap tm_dv, Params p, Tok tok) {
    extern __shared__ __align__(1024) uint8_t smem[];
    Misc *ms = reinterpret_cast<Misc *>(smem + kSmemBlocks);
    auto blk = [&](int b) { return smem + b * kBlockBytes; };
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const bool issuer = warp == kIssuerWarp, issuer2 = warp == kIssuer2Warp;

    if (smem_u32(smem) & 1023u) {  // the swizzled layout needs 1 KiB alignment
        if (tid == 0) set_error(p.err, 499, smem_u32(smem));
        return;
    }
    if (tid == 0) {
        for (int b = 0; b < kNumBars; ++b) mbar_init(&ms->bar[b], epi_bar(b) ? kEpiWarps : 1);
        ms->abort_flag = 0;
        fence_mbar_init();
    }
    if (issuer) {
        tmem_alloc(&ms->tmem_base, 512);
        tmem_relinquish();
        if (lane == 0) {
            prefetch_tmap(&tm_q); prefetch_tmap(&tm_k); prefetch_tmap(&tm_v); prefetch_tmap(&tm_g);
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tb = ms->tmem_base;
    const int M = p.M;

    if (issuer) {
        if (lane == 0) {
            const uint32_t sb4 = smem_u32(smem) >> 4;
            auto lk = [&](int b) { return sb4 + (uint32_t)b * kBlk16 + kLboK; };   // K-major block
            auto lm = [&](int b) { return sb4 + (uint32_t)b * kBlk16 + kLboMN; };  // MN-major block
            const uint32_t DK = tb + kDK, GAM = tb + kGAM, LAM = tb + kLAM;
            const uint32_t T0 = tb + kT0, T1 = tb + kT1;
            // tile counters: n_s every tile of both sweeps (the barriers both use), n_f forward
            // tiles, n_b reverse tiles
            uint32_t ld_par = 0, ld_pend = 0, n_s = 0, n_f = 0, n_b = 0, n_head = 0;
            auto load_fwd = [&](int set, int head, int j) {  // Q, K, V of tile j into blocks 0..2 or 11..13
                const int b0 = set ? bQ2 : bQ;
                ld_pend |= 1u << set;
                mbar_arrive_expect_tx(&ms->bar[bLd0 + set], 3 * kBlockBytes);
                tma_load_3d(blk(b0), &tm_q, &ms->bar[bLd0 + set], 0, j * kTile, head);
                tma_load_3d(blk(b0 + 1), &tm_k, &ms->bar[bLd0 + set], 0, j * kTile, head);
                tma_load_3d(blk(b0 + 2), &tm_v, &ms->bar[bLd0 + set], 0, j * kTile, head);
            };
            auto wait_ld = [&](int set) {  // set 0, 1: a Q, K, V set; 2: G and the record
                if (!bar_wait(ms, bLd0 + set, (ld_par >> set) & 1u, p)) return false;
                ld_par ^= 1u << set;
                ld_pend &= ~(1u << set);
                return true;
            };
            for (int head = blockIdx.x; head < p.BH && !ms->abort_flag; head += gridDim.x, ++n_head) {
                // ---------------- forward sweep: checkpoints of S and D ----------------
                load_fwd(0, head, 0);
                if (M > 1) load_fwd(1, head, 1);
                bool ok = true;
                for (int j = 0; j < M && ok; ++j, ++n_f, ++n_s) {
                    const uint32_t tp = n_s & 1, tf = n_f & 1;
                    const int set = j & 1, qb = set ? bQ2 : bQ, kb = qb + 1, vb = qb + 2;
                    ok = false;
                    if (!bar_wait(ms, bEp0, tp, p) || !wait_ld(set)) break;  // S_p (bf16) in bCk; tokens
                    tc_fence_after();
                    mma<false, false, 128, 4>(T0, lk(qb), lk(kb), 0u);  // A = Q K^T
                    umma_commit(&ms->bar[bEvA]);
                    mma<true, true, 64, 8>(GAM, lm(kb), lm(kb), 1u);  // S += K^T K (under E1)
                    if (!bar_wait(ms, bEp1, tp, p)) break;           // W (hi, lo) packed in T0
                    tc_fence_after();
                    mma_ts(DK, T0, lm(kb), 0u);                       // X = W K
                    mma_ts(DK, T0 + 16, lm(kb), 1u);
                    mma<false, false, 64, 4>(DK, lk(qb), lk(bCk), 1u);  //   + Q S_p
                    umma_commit(&ms->bar[bEvX]);
                    if (!bar_wait(ms, bEp2, tp, p)) break;  // X (hi, lo) in bXh, bXl
                    tc_fence_after();
                    mma<true, true, 64, 8>(LAM, lm(bXh), lm(vb), 1u);  // D += X^T V
                    mma<true, true, 64, 8>(LAM, lm(bXl), lm(vb), 1u);
                    umma_commit(&ms->bar[bEvC]);
                    if (!bar_wait(ms, bEvC, tf, p)) break;  // this set is free again
                    if (j + 2 < M) load_fwd(set, head, j + 2);
                    ok = true;
                }
                if (!ok) break;
                // the checkpoints are in global memory (the epilogue waited for its copies)
                if (!bar_wait(ms, bCkDone, n_head & 1, p)) break;
                // ---------------- reverse sweep: gradients (the second issuer makes the copies) ----
                for (int j = M - 1; j >= 0 && ok; --j, ++n_b, ++n_s) {
                    const uint32_t ts = n_s & 1, tp = n_b & 1;
                    const int set = (M - 1 - j) & 1, qb = set ? bQ2 : bQ, kb = qb + 1, vb = qb + 2;
                    ok = false;
                    // Q, K, V; G and the record.  P^T starts at once (T0 was last read by this
                    // thread's B^T Q); the epilogue packs it after the carry hand-off E0, so the
                    // arrival of E1 also says Gam_s, Lam_s (hi, lo) are in shared memory.
                    if (!wait_ld(set) || !wait_ld(2)) break;
                    tc_fence_after();
                    mma<false, false, 128, 4>(T0, lk(vb), lk(bG), 0u);  // P^T = V G^T
                    umma_commit(&ms->bar[bEvA]);
                    if (!bar_wait(ms, bEp1, ts, p)) break;  // P^T in T0; E0 done
                    tc_fence_after();
                    mma_ts(DK, T0, lm(qb), 0u);  // Y = P^T Q
                    mma_ts(DK, T0 + 16, lm(qb), 1u);
                    mma<false, false, 64, 4>(DK, lk(vb), lk(bGam), 1u);  //   + V Gam_s
                    mma<false, false, 64, 4>(DK, lk(vb), lk(bGam) + kH16, 1u);
                    umma_commit(&ms->bar[bEvX]);
                    mma<false, false, 128, 4>(T0, lk(bXh), lk(qb), 0u);  // T^T = X Q^T
                    mma<false, false, 128, 4>(T0, lk(bXl), lk(qb), 1u);
                    umma_commit(&ms->bar[bEvT]);
                    if (!bar_wait(ms, bEp3, tp, p)) break;  // T^T in T0
                    tc_fence_after();
                    mma_ts(DK, T0, lm(bG), 0u);                                 // dV = T^T G
                    mma<false, true, 64, 4>(DK, lk(bXh), lm(bGam), 1u);         //   + X Gam_s^T
                    mma<false, true, 64, 4>(DK, lk(bXh), lm(bGam) + kH16, 1u);
                    mma<false, true, 64, 4>(DK, lk(bXl), lm(bGam), 1u);
                    umma_commit(&ms->bar[bEvV]);
                    mma<false, false, 128, 4>(T0, lk(kb), lk(bYh), 0u);  // B^T = K Y^T
                    mma<false, false, 128, 4>(T0, lk(kb), lk(bYl), 1u);
                    umma_commit(&ms->bar[bEvB2]);
                    if (!bar_wait(ms, bEp4b, tp, p)) break;  // B^T in T0 and dV out of DK
                    tc_fence_after();
                    mma_ts(DK, T0, lm(qb), 0u);  // dK = B^T Q (+ W^T Y below; K Lam_s goes to DQ)
                    mma_ts(DK, T0 + 16, lm(qb), 1u);
                    if (!bar_wait(ms, bEp5, tp, p)) break;  // W^T in T1
                    tc_fence_after();
                    mma_ts(DK, T1, lm(bYh), 1u);  //   + W^T Y
                    mma_ts(DK, T1, lm(bYl), 1u);
                    mma_ts(DK, T1 + 16, lm(bYh), 1u);
                    umma_commit(&ms->bar[bEvO]);
                    if (!bar_wait(ms, bEvO, tp, p)) break;  // every operand of this set read
                    ok = true;
                }
                // the second issuer's last K Lam_s has read its set before the next head's copies
                if (!ok || !bar_wait(ms, bEvKL, (n_b - 1) & 1u, p)) break;
            }
            if (ms->abort_flag) {  // copies and MMAs in flight finish (bounded) before release
                for (int s = 0; s < 2; ++s)
                    if ((ld_pend >> s) & 1u) mbar_wait(&ms->bar[bLd0 + s], (ld_par >> s) & 1u, kBarWaitNs);
                if ((ld_pend >> 2) & 1u) mbar_wait(&ms->bar[bLdG], (ld_par >> 2) & 1u, kBarWaitNs);
                umma_commit(&ms->bar[bTear]);
                mbar_wait(&ms->bar[bTear], 0, kBarWaitNs);
            }
        }
        __syncwarp();
    } else if (issuer2) {
        // ====== second issuer: the reverse sweep's P, B, W^T tiles (T1), dQ (DQ) and the carries ======
        if (lane == 0) {
            const uint32_t sb4 = smem_u32(smem) >> 4;
            auto lk = [&](int b) { return sb4 + (uint32_t)b * kBlk16 + kLboK; };
            auto lm = [&](int b) { return sb4 + (uint32_t)b * kBlk16 + kLboMN; };
            const uint32_t DQ = tb + kDQ, GAM = tb + kGAM, LAM = tb + kLAM, T1 = tb + kT1;
            // the same tile counters as the first issuer; ld_par follows every completed copy phase,
            // the forward sweep's included (set j % 2 for forward tile j)
            uint32_t ld_par = 0, ld_pend = 0, n_s = 0, n_b = 0, n_head = 0;
            auto wait_ld = [&](int set) {
                if (!bar_wait(ms, bLd0 + set, (ld_par >> set) & 1u, p)) return false;
                ld_par ^= 1u << set;
                ld_pend &= ~(1u << set);
                return true;
            };
            auto load_qkv = [&](int set, int head, int j) {  // Q, K, V of tile j into blocks 0..2 or 11..13
                const int b0 = set ? bQ2 : bQ;
                ld_pend |= 1u << set;
                mbar_arrive_expect_tx(&ms->bar[bLd0 + set], 3 * kBlockBytes);
                tma_load_3d(blk(b0), &tm_q, &ms->bar[bLd0 + set], 0, j * kTile, head);
                tma_load_3d(blk(b0 + 1), &tm_k, &ms->bar[bLd0 + set], 0, j * kTile, head);
                tma_load_3d(blk(b0 + 2), &tm_v, &ms->bar[bLd0 + set], 0, j * kTile, head);
            };
            auto load_gck = [&](int head, int j) {  // G of tile j and its record (X hi, lo; S_p, D_p)
                ld_pend |= 4u;
                mbar_arrive_expect_tx(&ms->bar[bLdG], kBlockBytes + kCkBytes);
                tma_load_3d(blk(bG), &tm_g, &ms->bar[bLdG], 0, j * kTile, head);
                bulk_load(blk(bXh), p.ck + ((size_t)head * M + j) * kCkBytes, kCkBytes, &ms->bar[bLdG]);
            };
            for (int head = blockIdx.x; head < p.BH && !ms->abort_flag; head += gridDim.x, ++n_head) {
                n_s += (uint32_t)M;
                ld_par ^= (uint32_t)(((M + 1) / 2) & 1) | ((uint32_t)((M / 2) & 1) << 1);
                if (!bar_wait(ms, bCkDone, n_head & 1, p)) break;  // every record written, every forward product done
                load_qkv(0, head, M - 1);
                load_gck(head, M - 1);
                bool ok = true;
                for (int j = M - 1; j >= 0 && ok; --j, ++n_b, ++n_s) {
                    const uint32_t ts = n_s & 1, tp = n_b & 1;
                    const int set = (M - 1 - j) & 1, qb = set ? bQ2 : bQ, kb = qb + 1, vb = qb + 2;
                    ok = false;
                    // the previous tile's products are done (the first issuer's, the last of which
                    // read T1, and this thread's K Lam_s): its set takes the next tile's Q, K, V
                    if (j < M - 1 && (!bar_wait(ms, bEvO, tp ^ 1u, p) || !bar_wait(ms, bEvKL, tp ^ 1u, p))) break;
                    if (j > 0) {
                        load_qkv(set ^ 1, head, j - 1);
                        const size_t t0 = (size_t)head * p.n + (size_t)(j - 1) * kTile;
                        const uint32_t bytes = (uint32_t)min(kTile, p.n - (j - 1) * kTile) * kD * 2;
                        bulk_prefetch_l2(tok.g + t0 * kD, bytes);  // G and the record towards L2
                        bulk_prefetch_l2(p.ck + ((size_t)head * M + j - 1) * kCkBytes, kCkBytes);
                    }
                    if (!wait_ld(set) || !wait_ld(2)) break;
                    tc_fence_after();
                    mma<false, false, 128, 4>(T1, lk(bG), lk(vb), 0u);  // P = G V^T
                    umma_commit(&ms->bar[bEvA2]);
                    if (!bar_wait(ms, bEp1b, tp, p)) break;  // P in T1
                    tc_fence_after();
                    mma_ts(DQ, T1, lm(bXh), 0u);  // dQ = P X
                    mma_ts(DQ, T1, lm(bXl), 1u);
                    mma_ts(DQ, T1 + 16, lm(bXh), 1u);
                    mma<false, false, 64, 4>(DQ, lk(bG), lk(bCk) + kH16, 1u);  //   + G D_p^T
                    if (!bar_wait(ms, bEp2, ts, p)) break;  // Y (hi, lo) in shared memory
                    tc_fence_after();
                    mma<false, false, 64, 4>(DQ, lk(bYh), lk(bCk), 1u);  //   + Y S_p
                    mma<false, false, 64, 4>(DQ, lk(bYl), lk(bCk), 1u);
                    mma<false, false, 128, 4>(T1, lk(bYh), lk(kb), 0u);  // B = Y K^T
                    mma<false, false, 128, 4>(T1, lk(bYl), lk(kb), 1u);
                    umma_commit(&ms->bar[bEvB]);
                    // the carries, under the B epilogue: [Gam^T | Lam''] += Q^T [G | Y_hi], Lam'' += Q^T Y_lo
                    mma<true, true, 128, 8>(GAM, lm(qb), lm(bG), 1u);
                    mma<true, true, 64, 8>(LAM, lm(qb), lm(bYl), 1u);
                    umma_commit(&ms->bar[bEvCar]);
                    if (!bar_wait(ms, bEp4a, tp, p)) break;  // B in T1
                    tc_fence_after();
                    mma_ts(DQ, T1, lm(kb), 1u);  // dQ += B K
                    mma_ts(DQ, T1 + 16, lm(kb), 1u);
                    mma<false, false, 128, 4>(T1, lk(kb), lk(qb), 0u);  // W^T = K Q^T
                    umma_commit(&ms->bar[bEvW]);
                    // every product that reads G or the record is done (the first issuer's by the
                    // B^T hand-off, this thread's by its carry commit): the next tile's G and record
                    if (!bar_wait(ms, bEp4b, tp, p) || !bar_wait(ms, bEvCar, tp, p)) break;
                    if (j > 0) load_gck(head, j - 1);
                    if (!bar_wait(ms, bEp5b, tp, p)) break;  // dQ read out of DQ
                    tc_fence_after();
                    mma<false, false, 64, 4>(DQ, lk(kb), lk(bLam), 0u);  // K Lam_s = K Lam''^T
                    mma<false, false, 64, 4>(DQ, lk(kb), lk(bLam) + kH16, 1u);
                    mma<false, true, 64, 4>(DQ, lk(kb), lm(bLam), 1u);  //   + K Lam''
                    mma<false, true, 64, 4>(DQ, lk(kb), lm(bLam) + kH16, 1u);
                    umma_commit(&ms->bar[bEvKL]);
                    ok = true;
                }
                if (!ok) break;
            }
            if (ms->abort_flag) {  // this thread's copies and MMAs in flight finish (bounded) before release
                for (int s = 0; s < 3; ++s)
                    if ((ld_pend >> s) & 1u) mbar_wait(&ms->bar[bLd0 + s], (ld_par >> s) & 1u, kBarWaitNs);
                umma_commit(&ms->bar[bTear2]);
                mbar_wait(&ms->bar[bTear2], 0, kBarWaitNs);
            }
        }
        __syncwarp();
    } else {
        // ================================ epilogue ================================
        const int qd = warp & 3, cq = warp >> 2;
        const int r = 32 * qd + lane;
        const uint32_t lb = (uint32_t)(32 * qd) << 16;
        const uint32_t t0 = tb + lb + kT0, t1 = tb + lb + kT1, c32 = 32u * cq, c16 = 16u * cq;
        uint32_t n_s = 0, n_f = 0, n_b = 0, n_head = 0;
        auto zero_carries = [&]() {  // rows 0..63 of GAM and LAM
            if (qd < 2) {
                uint32_t z[16];
#pragma unroll
                for (int u = 0; u < 16; ++u) z[u] = 0u;
                tmem_st16(tb + lb + kGAM + c16, z);
                tmem_st16(tb + lb + kLAM + c16, z);
                tmem_st_wait();
            }
        };
        // a 64-wide result in TMEM at column `col` -> row r of a block as bf16 hi and lo
        auto to_smem_hl = [&](uint32_t col, int bh, int bl) {
            uint32_t a[16];
            tmem_ld16(tb + lb + col + c16, a);
            tmem_ld_wait();
            store16_hl(blk(bh), blk(bl), r, c16, a);
        };
        // a 64-wide result -> bf16 in a free block -> one TMA store of the tile (rows past n are
        // not written); row-wise stores from the threads would cost a 16-byte piece per row
        auto drain2 = [&](uint32_t col, uint32_t col2, int stage, const CUtensorMap *map, int tok0, int head) {
            uint32_t a[16], b[16];
            tmem_ld16(tb + lb + col + c16, a);
            tmem_ld16(tb + lb + col2 + c16, b);
            tmem_ld_wait();
#pragma unroll
            for (int u = 0; u < 16; ++u) a[u] = __float_as_uint(__uint_as_float(a[u]) + __uint_as_float(b[u]));
            if (tid == 0) tma_store_wait_read();
            epi_sync();
            store16(blk(stage), r, c16, a);
            fence_async_smem();
            epi_sync();
            if (tid == 0) {
                tma_store_3d(map, blk(stage), 0, tok0, head);
                tma_store_commit();
            }
        };
        auto drain = [&](uint32_t col, int stage, const CUtensorMap *map, int tok0, int head) {
            uint32_t a[16];
            tmem_ld16(tb + lb + col + c16, a);
            tmem_ld_wait();
            if (tid == 0) tma_store_wait_read();  // the block's previous copy has read it
            epi_sync();
            store16(blk(stage), r, c16, a);
            fence_async_smem();
            epi_sync();
            if (tid == 0) {
                tma_store_3d(map, blk(stage), 0, tok0, head);
                tma_store_commit();
            }
        };
        for (int head = blockIdx.x; head < p.BH; head += gridDim.x, ++n_head) {
            // ---------------- forward sweep ----------------
            zero_carries();
            for (int j = 0; j < M; ++j, ++n_f, ++n_s) {
                const uint32_t tp = n_s & 1, tf = n_f & 1;
                // E0: S_p, D_p -> bf16 checkpoint image in bCk (also the B operand of Q S_p)
                if (j > 0) {
                    bar_wait(ms, bEvC, tf ^ 1u, p);  // the previous tile's carry products
                    tc_fence_after();
                    if (tid == 0) tma_store_wait_read();  // its record has left bXh, bXl, bCk
                    epi_sync();
                }
                if (qd < 2) {
                    uint32_t a[16], b[16];
                    tmem_ld16(tb + lb + kGAM + c16, a);
                    tmem_ld16(tb + lb + kLAM + c16, b);
                    tmem_ld_wait();
                    store16(blk(bCk), r, c16, a);
                    store16(blk(bCk) + kHalf, r, c16, b);
                }
                fence_async_smem();
                epi_arrive(ms, bEp0);
                // E1: W = L . A, packed hi/lo over A
                bar_wait(ms, bEvA, tp, p);
                tc_fence_after();
                mask_pack<false, true>(t0, r, c32);
                epi_arrive(ms, bEp1);
                // E2: X -> hi, lo; the tile's record (X hi, lo; S_p, D_p) -> global
                bar_wait(ms, bEvX, tp, p);
                tc_fence_after();
                to_smem_hl(kDK, bXh, bXl);
                fence_async_smem();
                epi_sync();
                if (tid == 0) {
                    bulk_store(p.ck + ((size_t)head * M + j) * kCkBytes, blk(bXh), kCkBytes);
                    tma_store_commit();
                }
                epi_arrive(ms, bEp2);
            }
            bar_wait(ms, bEvC, (n_f - 1) & 1u, p);  // the last carry products (before GAM, LAM are reset)
            tc_fence_after();
            if (tid == 0) {
                tma_store_wait_all();  // every record is in global memory
                mbar_arrive(&ms->bar[bCkDone]);
            }
            // ---------------- reverse sweep ----------------
            zero_carries();
            for (int j = M - 1; j >= 0; --j, ++n_b, ++n_s) {
                const uint32_t ts = n_s & 1, tp = n_b & 1;
                const int tok0 = j * kTile;
                // E0: Gam_s^T, Lam''_s -> hi, lo (the previous tile's products are done: waited in E6;
                // the copies of its dV and dQ have read bGam, the one of dK may still read bYh)
                if (tid == 0) tma_store_wait_read1();
                epi_sync();
                if (qd < 2) {
                    uint32_t a[16], b[16];
                    tmem_ld16(tb + lb + kGAM + c16, a);
                    tmem_ld16(tb + lb + kLAM + c16, b);
                    tmem_ld_wait();
                    store16_hl(blk(bGam), blk(bGam) + kHalf, r, c16, a);
                    store16_hl(blk(bLam), blk(bLam) + kHalf, r, c16, b);
                }
                fence_async_smem();
                epi_arrive(ms, bEp0);
                // E1: P^T = L^T . (V G^T) over T0, P = L . (G V^T) over T1
                bar_wait(ms, bEvA, ts, p);
                tc_fence_after();
                mask_pack<true, true>(t0, r, c32);
                epi_arrive(ms, bEp1);
                bar_wait(ms, bEvA2, tp, p);
                tc_fence_after();
                mask_pack<false, true>(t1, r, c32);
                epi_arrive(ms, bEp1b);
                // E2: Y -> hi, lo (the previous dK copy has read bYh)
                bar_wait(ms, bEvX, ts, p);
                tc_fence_after();
                if (tid == 0) tma_store_wait_read();
                epi_sync();
                to_smem_hl(kDK, bYh, bYl);
                fence_async_smem();
                epi_arrive(ms, bEp2);
                // E3: T^T = L^T . (X Q^T) over T0 (bf16 only)
                bar_wait(ms, bEvT, tp, p);
                tc_fence_after();
                mask_pack<true, false>(t0, r, c32);
                epi_arrive(ms, bEp3);
                // E4: B = L . (Y K^T) over T1; dV out; B^T over T0
                bar_wait(ms, bEvB, tp, p);
                tc_fence_after();
                mask_pack<false, true>(t1, r, c32);
                epi_arrive(ms, bEp4a);
                bar_wait(ms, bEvV, tp, p);
                tc_fence_after();
                drain(kDK, bGam, &tm_dv, tok0, head);  // Gam_s read by its last product (dV)
                bar_wait(ms, bEvB2, tp, p);
                tc_fence_after();
                mask_pack<true, true>(t0, r, c32);
                epi_arrive(ms, bEp4b);
                // E5: W^T = L^T . (K Q^T) over T1, then dQ out
                bar_wait(ms, bEvW, tp, p);
                tc_fence_after();
                mask_pack<true, true>(t1, r, c32);
                epi_arrive(ms, bEp5);
                drain(kDQ, bGam, &tm_dq, tok0, head);
                epi_arrive(ms, bEp5b);
                // E6: dK = (B^T Q + W^T Y from DK) + (K Lam_s from DQ) out
                bar_wait(ms, bEvO, tp, p);
                bar_wait(ms, bEvKL, tp, p);
                tc_fence_after();
                drain2(kDK, kDQ, bYh, &tm_dk, tok0, head);  // Y read by its last product (W^T Y)
            }
        }
        if (tid == 0) tma_store_wait_all();
    }
    tc_fence_before();
    __syncthreads();
    if (issuer) {
        tc_fence_after();
        tmem_dealloc(tb, 512);
    }
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        cudaDriverEntryPointQueryResult qr;
        void *f = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &qr) ==
                cudaSuccess &&
            qr == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(f);
    }
    return fn;
}

// [BH][n][64] bf16, boxes of 64 columns x 128 tokens, 128-byte swizzle, zero fill beyond n
bool make_map(CUtensorMap *m, const void *base, int BH, int n) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[3] = {(cuuint64_t)kD, (cuuint64_t)n, (cuuint64_t)BH};
    cuuint64_t strides[2] = {(cuuint64_t)kD * 2, (cuuint64_t)n * kD * 2};
    cuuint32_t box[3] = {(cuuint32_t)kD, (cuuint32_t)kTile, 1};
    cuuint32_t es[3] = {1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims, strides, box, es,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool aligned16(const void *q) { return (reinterpret_cast<uintptr_t>(q) & 15u) == 0; }

}  // namespace

size_t backward2_tc_workspace_bytes(int BH, int n) {
    if (BH <= 0 || n <= 0) return kWsHeaderBytes;
    return kWsHeaderBytes + (size_t)BH * ((n + kTile - 1) / kTile) * kCkBytes;
}

bool backward2_tc_applicable(const Bwd2 &p) {
    if (getenv("HLA_DISABLE_FUSED")) return false;
    if (p.dt != HLA_BF16 || p.d != kD || p.dv != kD || p.normalized || p.n <= 0 || p.BH <= 0) return false;
    if (!aligned16(p.q) || !aligned16(p.k) || !aligned16(p.v) || !aligned16(p.dout)) return false;
    if (!aligned16(p.dq) || !aligned16(p.dk) || !aligned16(p.dval)) return false;
    if (p.ws_bytes < backward2_tc_workspace_bytes(p.BH, p.n)) return false;
    int dev = 0, major = 0, minor = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return false;
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    return major == 10 && minor == 3 && encode_fn() != nullptr;
}

cudaError_t backward2_tc_launch(const Bwd2 &p, cudaStream_t stream) {
    CUtensorMap mq, mk, mv, mg, mdq, mdk, mdv;
    if (!make_map(&mq, p.q, p.BH, p.n) || !make_map(&mk, p.k, p.BH, p.n) || !make_map(&mv, p.v, p.BH, p.n) ||
        !make_map(&mg, p.dout, p.BH, p.n) || !make_map(&mdq, p.dq, p.BH, p.n) || !make_map(&mdk, p.dk, p.BH, p.n) ||
        !make_map(&mdv, p.dval, p.BH, p.n))
        return cudaErrorInvalidValue;
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    Params kp{};
    kp.ck = reinterpret_cast<uint8_t *>(p.ws + kWsHeaderBytes);
    kp.BH = p.BH;
    kp.n = p.n;
    kp.M = (p.n + kTile - 1) / kTile;
    kp.err = reinterpret_cast<WsHeader *>(p.ws);
    Tok tok{static_cast<const __nv_bfloat16 *>(p.q), static_cast<const __nv_bfloat16 *>(p.k),
            static_cast<const __nv_bfloat16 *>(p.v), static_cast<const __nv_bfloat16 *>(p.dout)};
    cudaError_t e = cudaMemsetAsync(p.ws, 0, kWsHeaderBytes, stream);
    if (e) return e;
    if ((e = cudaFuncSetAttribute(bwd_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes)))
        return e;
    const int grid = p.BH < sms ? p.BH : sms;
    bwd_tc_kernel<<<grid, kThreads, kSmemBytes, stream>>>(mq, mk, mv, mg, mdq, mdk, mdv, kp, tok);
    return cudaGetLastError();
}

}  // namespace hla
