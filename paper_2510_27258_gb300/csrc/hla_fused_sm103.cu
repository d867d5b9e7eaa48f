// Fused forward of masked second-order HLA for sm_103a (GB300): tcgen05 MMAs
// with TMEM accumulators, TMA tile loads/stores, one persistent CTA per SM.
//
// Per head the sequence is cut into 128-token tiles; with x_t = S_t q_t the
// masked operator is  o_t = sum_{j<=t} (q_t . x_j) v_j  (proof of Theorem 1),
// and per tile (rows = tokens, p = carry before the tile):
//   A = Q K^T,  W = L . A                        (L: lower triangle incl. diagonal)
//   X = W K + Q S_p                              (rows x_t = S_t q_t)
//   T = L . (Q X^T),  O = T V + Q D_p            (D = sum_j x_j v_j^T = S C - G)
//   den_t = sum_{j<=t} T_tj + q_t . e_p          (e = sum_j x_j = S m - h)
//   S_p += K^T K,  D_p += X^T V,  e_p += X^T 1
// The carries compose across tiles as the semidirect product of Eq. semidirect
// does (D_AB = D_A + D_B + S_A C_B is the D-form of G_AB = G_A + G_B + S_B C_A).
//
// The unmasked operator o_t = q_t^T S_t C_t (the online updates after Theorem 1
// without G, h) is  o_t = sum_{j<=t} (x_t . q_j) v_j + x_t^T C_p: the same X, then
//   T = L . (X Q^T),  O = T V + X C_p,  C_p += Q^T V
// in the same slots and TMEM regions (C where D sits): the kUnmasked
// instantiation.  It runs the plain output only, one segment per head (the fix-up
// of later segments would need X, which is not kept) and no state.
//
// Parallel structure: a work item is (head, segment of L consecutive tiles);
// items are handed out by an atomic ticket in segment-major order, so the
// segments of one head run on different SMs at staggered times.  Each item
//   1. sums K^T K over its tiles (its S aggregate), waits for the inclusive S
//      prefix of the previous segment (a two-slot ring in global memory read
//      through L2, guarded by release/acquire flags) and publishes its own;
//   2. sweeps its tiles with the S carry and a segment-local D carry in TMEM,
//      writing provisional outputs (exact for the first segment of a head);
//   3. waits for the inclusive D prefix of the previous segment, publishes its
//      own, and (segments > 0) adds the missing carry term Q D_prefix (and
//      q . e_prefix to the denominator) to its provisional outputs.
// The exclusive scan across segments is a chained scan; Theorem 2 guarantees
// the result equals the serial recurrence.
//
// Roles: warp 16 issues TMA loads and MMAs (one thread); warp 17 releases the
// cross-SM prefix flags once the epilogue has written a prefix (the GPU-scope
// fence this takes stays off the epilogue's path); warps 0-15 are the epilogue
// (TMEM -> registers -> shared memory): warp w reads TMEM lanes 32 (w % 4) ..
// +31 (one row each) and columns 32 (w / 4) .. +31.
//
// Head sizes: d = dv = 64 has its own instantiation whose products run over 64
// features (the tiles and TMEM regions keep their 128-column layout).  A mix of
// 64 and 128 runs as 128 with zero features 64..127: the TMA box of those
// columns lies wholly outside the tensor and is zero-filled, so S, x_t, D and e
// have zero rows / columns there (the S shift cancels exactly: q_f = 0) and the
// padded output columns, which are zero, are not stored.  The tile is 128
// tokens whatever the requested chunk (Theorem 2: the result does not depend on
// the chunking up to rounding).
//
// Precision: tokens are bf16, every product accumulates in fp32 (TMEM).  The S
// operand is split as S = c I + R (c = bf16(trace / d), the trace of the S carry
// at most one tile old) with c q_t added in
// fp32, so x_t is accurate although |S| grows like t/d.  X enters T = Q X^T as
// bf16 hi + lo (with X rounded once, q_t . x_t = (q_t . k_t)^2 at t = 0 would
// lose |q||k| / |q.k| times the bf16 rounding when q and k are nearly
// orthogonal).  For the normalised output, whose denominator cancels heavily,
// R and W are also split into hi + lo, so X and T are accurate to ~2^-16 of
// each term; the denominator is the fp32 row sum of T plus q_t . e_p, with the
// e carry summed in fp32 on CUDA cores.  T and D enter T V and Q D as bf16.
#include <algorithm>
#include <functional>
#include <queue>
#include <vector>

#include "hla_internal.h"
#include "sm103_prims.cuh"

namespace hla {
namespace {

using namespace sm103;

constexpr int kD = 128;           // layout width of tiles, carries and TMEM regions (head sizes 64, 128)
constexpr int kTile = 128;        // tokens per tile (MMA M)
constexpr int kEpiWarps = 16;     // 4 per TMEM lane quadrant
constexpr int kEpiThreads = kEpiWarps * 32;
constexpr int kIssuerWarp = kEpiWarps;
constexpr int kPubWarp = kEpiWarps + 1;  // releases the cross-SM prefix flags
constexpr int kThreads = kEpiThreads + 64;
constexpr int kSlots = 7;
constexpr uint32_t kSmemTiles = kSlots * kTileBytes;
constexpr uint32_t kMiscBytes = 3072;
constexpr uint32_t kSmemBytes = kSmemTiles + kMiscBytes;  // = 227 KiB; base must be 1 KiB aligned

// shared-memory slots (32 KiB each)
enum Slot { kQ0 = 0, kQ1 = 1, kK = 2, kV = 3, kW = 4, kSX = 5, kSD = 6 };

// TMEM columns: S carry, D carry, A -> T, X -> O
constexpr uint32_t kTS = 0, kTD = 128, kTA = 256, kTX = 384;

// fix-up buffers (three tiles in flight): Q slot, provisional output slot, TMEM columns of F
__device__ __forceinline__ int fix_q(int i) { return i == 0 ? kQ0 : i == 1 ? kQ1 : kW; }
__device__ __forceinline__ int fix_o(int i) { return i == 0 ? kK : i == 1 ? kV : kSX; }
__device__ __forceinline__ uint32_t fix_t(int i) { return i == 0 ? kTA : i == 1 ? kTX : kTD; }

// barrier indices
enum Bar {
    bLd0 = 0,  // + slot index for the TMA-loaded slots (Q0, Q1, K, V, W, SX)
    bPre = 6,  // pre-pass MMA done (per K tile)
    bEvP = 7, bEvA = 8, bEvX = 9, bEvS = 10, bEvT = 11, bEvO = 12, bEvD = 13,
    bEvF = 14,  // + fix-up buffer (0..2)
    bEpW = 17, bEpX = 18, bEpT = 19,
    bEpR = 20,  // next tile's S split written
    bEpF = 21,  // + fix-up buffer: its slots and TMEM region are free again
    bEpDF = 24,
    bEpO = 25,  // O read out of TMEM
    bEpOut = 26,  // provisional outputs of the segment written (segments > 0)
    bTear = 27,   // (count 1) all MMAs done, after a wait gave up
    kNumBars = 28
};
constexpr int kFirstEpiBar = bEpW;

struct Misc {
    uint64_t bar[kNumBars];
    uint32_t tmem_base;
    int item;        // current ticket
    int abort_flag;  // an mbarrier wait gave up
    int pad;
    float red[kEpiWarps];
    float eloc[kD];      // segment-local e carry
    float den[kTile];    // denominators of the current tile
    float part[3][kD];   // partial sums of the other three column quarters / lane quadrants
    float dtr[2][4];     // diagonal sums of the S carry per lane quadrant, by tile parity
};
static_assert(sizeof(Misc) <= kMiscBytes, "misc smem");

struct Params {
    int BH, n, M, L, G, n_items;
    int normalized;
    float eps;
    const float *state_in;  // S_0 of each head (paper tuple), or null
    const float *init_De;   // D_0 (d*dv) and e_0 (d) of each head, or null
    float *ring;            // [BH][2][d*d + d*dv + d]; S and D parts thread-major (see ring4)
    unsigned *flags;        // [2][BH][2]: S flags then D flags
    unsigned *ticket;
    float *den_loc;         // [BH][n] provisional denominators (normalised, segments > 0)
    WsHeader *err;
    unsigned long long wait_ns;  // budget of a cross-SM chain wait
    int inject_skip_item;        // testing: this item does not publish its S prefix
    int out_blocks;              // 64-column blocks of an output row (dv / 64)
};

constexpr int kRingFloats = kD * kD + kD * kD + kD;

// The S and D prefixes in the ring are stored in the order the epilogue holds
// them: float4 c (columns c0 + 4c .. +3 of row r) of epilogue thread et at
// float4 index c * kEpiThreads + et, so that every warp access is 512
// contiguous bytes.
// Writer and reader (the next segment of the head) use the same thread mapping.
__device__ __forceinline__ int ring4(int c, int et) { return c * kEpiThreads + et; }
// floats of one head's state tuple [S | C | m | G | h] with d = dv = kD
constexpr int kStateFloats = kD * kD + 2 * kD * kD + 2 * kD;
// budget of an intra-CTA mbarrier wait (TMA or MMA completion, epilogue hand-off)
constexpr unsigned long long kBarWaitNs = 2000000000ull;

// ---------------------------------------------------------------------------
__device__ __forceinline__ void st_release(unsigned *p, unsigned v) {
    asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ unsigned ld_acquire(const unsigned *p) {
    unsigned v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
// named barrier of the epilogue warps
__device__ __forceinline__ void epi_sync() { asm volatile("bar.sync 1, %0;" ::"n"(kEpiThreads) : "memory"); }
// Hand-offs epilogue -> publisher warp (named barriers 2 and 3, 288 threads): the
// epilogue arrives after writing a prefix to the ring and goes on; the publisher
// waits, then makes the ring writes visible GPU-wide and releases the flag.
constexpr int kBarPubS = 2, kBarPubD = 3;
__device__ __forceinline__ void pub_arrive(int id) {
    asm volatile("bar.arrive %0, %1;" ::"r"(id), "r"(kEpiThreads + 32) : "memory");
}
__device__ __forceinline__ void pub_wait(int id) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(kEpiThreads + 32) : "memory");
}

__device__ __forceinline__ void set_error(WsHeader *err, unsigned where, unsigned detail) {
    if (atomicCAS(&err->error, 0u, (unsigned)kDevTimeout) == 0u) {
        err->where = where;
        err->detail = detail;
    }
}

// Spin (one thread) until *flag == want; bounded by wall time and by the error word.
__device__ bool chain_wait(const unsigned *flag, unsigned want, const Params &p, unsigned where, unsigned detail) {
    const uint64_t t0 = globaltimer_ns();
    while (true) {
        if (ld_acquire(flag) == want) return true;
        if (*(volatile unsigned *)&p.err->error != 0u) return false;
        if (globaltimer_ns() - t0 > p.wait_ns) {
            set_error(p.err, where, detail);
            return false;
        }
        __nanosleep(64);
    }
}

// Bounded mbarrier wait.  On timeout the error word is set and the CTA is marked
// aborted: later waits return at once, the epilogue keeps its (uniform) control
// flow so that its named barriers still match, and the issuer stops issuing.
__device__ __forceinline__ bool bar_wait(Misc *ms, int b, uint32_t parity, const Params &p) {
    if (ms->abort_flag) return false;
    if (mbar_wait(&ms->bar[b], parity, kBarWaitNs)) return true;
    set_error(p.err, 100 + b, parity);
    ms->abort_flag = 1;
    return false;
}

// epilogue warps arrive (count kEpiWarps): lane 0 after the warp's own fences
__device__ __forceinline__ void epi_arrive(Misc *ms, int b) {
    tc_fence_before();
    __syncwarp();
    if ((threadIdx.x & 31) == 0) mbar_arrive(&ms->bar[b]);
}

// 8 consecutive bf16 of row r (columns c..c+7) of a tile, as floats
__device__ __forceinline__ void tile_row8(const uint8_t *tile, int r, int c, float (&f)[8]) {
    const uint4 u = *reinterpret_cast<const uint4 *>(tile + tile_off(r, c));
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        f[2 * i] = __uint_as_float(w[i] << 16);
        f[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
    }
}

__device__ __forceinline__ void store_row8(uint8_t *tile, int r, int c, const float *f) {
    uint4 u;
    u.x = pack_bf16x2(f[0], f[1]);
    u.y = pack_bf16x2(f[2], f[3]);
    u.z = pack_bf16x2(f[4], f[5]);
    u.w = pack_bf16x2(f[6], f[7]);
    *reinterpret_cast<uint4 *>(tile + tile_off(r, c)) = u;
}

__device__ __forceinline__ float bf16_round(float x) { return __bfloat162float(__float2bfloat16_rn(x)); }

// a, b -> bf16 pair hi (a in the low half) and the bf16 pair of the remainders a - hi_a, b - hi_b
__device__ __forceinline__ void split2(float a, float b, uint32_t &hi, uint32_t &lo) {
    hi = pack_bf16x2(a, b);
    lo = pack_bf16x2(a - __uint_as_float(hi << 16), b - __uint_as_float(hi & 0xffff0000u));
}

// row r, columns c0..c0+31: v -> bf16 hi in tile th and, if lo, the bf16 remainder in tile tl
__device__ __forceinline__ void store_split32(uint8_t *th, uint8_t *tl, int r, int c0, const float (&v)[32], bool lo) {
#pragma unroll
    for (int jj = 0; jj < 32; jj += 8) {
        uint32_t h[4], l[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) split2(v[jj + 2 * i], v[jj + 2 * i + 1], h[i], l[i]);
        *reinterpret_cast<uint4 *>(th + tile_off(r, c0 + jj)) = make_uint4(h[0], h[1], h[2], h[3]);
        if (lo) *reinterpret_cast<uint4 *>(tl + tile_off(r, c0 + jj)) = make_uint4(l[0], l[1], l[2], l[3]);
    }
}

// zero the entries of columns c0..c0+31 above the diagonal of row r (c > r); for the
// 32 x 32 diagonal block of the tile, r - c0 = lane
// kSel: by selects (no branch that diverges the warp); else by a branch per element, which for the
// 128-feature instantiation measured faster overall (it staggers the diagonal warps)
template <bool kSel>
__device__ __forceinline__ void mask_upper32(float (&f)[32], int r, int c0) {
#pragma unroll
    for (int jj = 0; jj < 32; ++jj) {
        if constexpr (kSel) {
            f[jj] = (c0 + jj > r) ? 0.f : f[jj];
        } else {
            if (c0 + jj > r) f[jj] = 0.f;
        }
    }
}

// subtract c from the entry of column r (the diagonal), which this thread holds when
// its block is the diagonal block
template <bool kSel>
__device__ __forceinline__ void shift_diag32(float (&f)[32], int lane, float c) {
#pragma unroll
    for (int jj = 0; jj < 32; ++jj) {
        if constexpr (kSel) {
            f[jj] -= (jj == lane) ? c : 0.f;
        } else {
            if (jj == lane) f[jj] -= c;
        }
    }
}

// f[lane] (the diagonal entry of row r when this thread's block is the diagonal block)
template <bool kSel>
__device__ __forceinline__ float pick_lane32(const float (&f)[32], int lane) {
    float x = 0.f;
#pragma unroll
    for (int jj = 0; jj < 32; ++jj) {
        if constexpr (kSel) {
            x = (jj == lane) ? f[jj] : x;
        } else {
            if (jj == lane) x = f[jj];
        }
    }
    return x;
}

// 32 values -> 16 packed bf16 pairs (the tensor-memory A-operand layout)
__device__ __forceinline__ void pack32(const float (&v)[32], uint32_t (&h)[16]) {
#pragma unroll
    for (int i = 0; i < 16; ++i) h[i] = pack_bf16x2(v[2 * i], v[2 * i + 1]);
}

// 32 values -> packed bf16 pairs hi and packed bf16 remainders lo
__device__ __forceinline__ void split_pack32(const float (&v)[32], uint32_t (&h)[16], uint32_t (&l)[16]) {
#pragma unroll
    for (int i = 0; i < 16; ++i) split2(v[2 * i], v[2 * i + 1], h[i], l[i]);
}

__device__ __forceinline__ void ld32(uint32_t addr, float (&f)[32]) {
    uint32_t a[32];
    tmem_ld32(addr, a);
    tmem_ld_wait();
#pragma unroll
    for (int j = 0; j < 32; ++j) f[j] = __uint_as_float(a[j]);
}

// Column sums of v over the 32 lanes of a warp: returns, in lane l, the sum of
// column l (31 shuffles: each step halves the columns a lane keeps).
__device__ __forceinline__ float warp_colsum32(float (&v)[32]) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) {
        const bool upper = (lane & o) != 0;
#pragma unroll
        for (int i = 0; i < o; ++i) {
            const float send = upper ? v[i] : v[i + o];
            const float keep = upper ? v[i + o] : v[i];
            v[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
        }
    }
    return v[0];
}

__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

// High word of every shared-memory descriptor used here: stride between 8-row
// groups 1024 B, tcgen05 descriptor version, 128-byte swizzle.
constexpr uint32_t kDescHi = (1024u >> 4) | (1u << 14) | (2u << 29);
// low-word leading-byte-offset fields of K-major (unused, 16 B) and MN-major
// (stride between 64-element blocks) operands
constexpr uint32_t kLboK = 1u << 16, kLboMN = (kBlockBytes >> 4) << 16;

// One 128 x N x 16 KS product D (+)= A B as KS steps of K = 16 (N = 128, KS = 8 unless given), from the
// low descriptor words of the two operand tiles (address >> 4 | LBO field).  The step offsets are
// compile-time constants, so each MMA costs one add per operand.
template <bool A_MN, bool B_MN, int N = 128, int KS = 8>
__device__ __forceinline__ void mma128(uint32_t d_tmem, uint32_t a_lo, uint32_t b_lo, uint32_t accumulate) {
    constexpr uint32_t id = idesc_bf16(128, N, A_MN, B_MN);
#pragma unroll
    for (int kk = 0; kk < KS; ++kk) {
        // K-major: the second 64-element column block is 16 KiB on, 32 B per K step within a block;
        // MN-major: 8 K rows of 128 B (2 KiB with the swizzle atom) per K step
        const uint32_t ka = A_MN ? kk * 128u : (kk >> 2) * (kBlockBytes >> 4) + (kk & 3) * 2u;
        const uint32_t kb = B_MN ? kk * 128u : (kk >> 2) * (kBlockBytes >> 4) + (kk & 3) * 2u;
        umma_bf16(d_tmem, (static_cast<uint64_t>(kDescHi) << 32) | (a_lo + ka),
                  (static_cast<uint64_t>(kDescHi) << 32) | (b_lo + kb), id, kk > 0 ? 1u : accumulate);
    }
}

// The same product with A (128 x 128 bf16) in tensor memory, in the layout the epilogue
// writes: K elements 32g .. 32g+31 of every row packed as bf16 pairs in columns
// a_tmem + 32g .. +15 (g = 0..3), so that K step kk starts at column 32 (kk / 2) + 8 (kk % 2).
template <bool B_MN, int N = 128>
__device__ __forceinline__ void mma128_ts(uint32_t d_tmem, uint32_t a_tmem, uint32_t b_lo, uint32_t accumulate) {
    constexpr uint32_t id = idesc_bf16(128, N, 0, B_MN);
#pragma unroll
    for (int kk = 0; kk < 8; ++kk) {
        const uint32_t kb = B_MN ? kk * 128u : (kk >> 2) * (kBlockBytes >> 4) + (kk & 3) * 2u;
        umma_bf16_ts(d_tmem, a_tmem + 32u * (kk >> 1) + 8u * (kk & 1), (static_cast<uint64_t>(kDescHi) << 32) | (b_lo + kb),
                     id, kk > 0 ? 1u : accumulate);
    }
}

// ---------------------------------------------------------------------------
// the kernel
// ---------------------------------------------------------------------------
// kState: the final state is wanted.  Then W and R are split hi + lo and the e carry kept
// whatever the output (as for the normalised output), and D += X_hi^T V + X_lo^T V is issued
// before O (X_lo is still in slot W), so that the prefixes in the ring are accurate to fp32 level.
template <bool kState, bool kNarrow, bool kUnmasked = false>
__global__ void __launch_bounds__(kThreads, 1)
hla2_fused_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                  const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_o, Params p) {
    extern __shared__ __align__(1024) uint8_t smem[];
    Misc *ms = reinterpret_cast<Misc *>(smem + kSmemTiles);
    auto slot = [&](int s) { return smem + s * kTileBytes; };

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const bool issuer = (warp == kIssuerWarp), publisher = (warp == kPubWarp);
    const bool precise = kState || p.normalized;  // hi + lo splits of W and R
    // head size of the products: 128, or 64 for d = dv = 64 (then the feature columns 64..127 of the tiles,
    // carries and TMEM regions are neither computed nor read; see the narrow notes in the epilogue)
    constexpr int kF = kNarrow ? 64 : 128;
    constexpr int kFS = kF / 16;  // K steps of a contraction over the head size
    const bool need_e = !kUnmasked && (kState || p.normalized);  // the e carry (never unmasked)
    constexpr bool d_lo = kState;                 // D with X_lo, issued before O

    // the tile layout needs 1 KiB alignment of the dynamic shared memory
    if (smem_u32(smem) & 1023u) {
        if (tid == 0) set_error(p.err, 99, smem_u32(smem));
        return;
    }
    if (tid == 0) {
        for (int b = 0; b < kNumBars; ++b) mbar_init(&ms->bar[b], (b >= kFirstEpiBar && b != bTear) ? kEpiWarps : 1);
        ms->abort_flag = 0;
        fence_mbar_init();
    }
    if (issuer) {
        tmem_alloc(&ms->tmem_base, 512);
        tmem_relinquish();
        if (lane == 0) {
            prefetch_tmap(&tm_q); prefetch_tmap(&tm_k); prefetch_tmap(&tm_v); prefetch_tmap(&tm_o);
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tb = ms->tmem_base;

    // per-CTA event counters (identical sequences on both sides)
    uint32_t n_tiles = 0, n_items = 0, n_pre = 0, n_dfix = 0;
    uint32_t ld_par = 0;  // bit s: parity of the next load completion of slot s
    uint32_t ld_pend = 0; // bit s: a load of slot s issued and not waited for yet
    uint32_t fx_par = 0;  // bit i: parity of the next fix-up hand-off of buffer i
    uint32_t n_r = 0;     // S-split hand-offs (one per tile that has a successor in its segment)

    // descriptor low words of the slots, as K-major (lk) and MN-major (lm) operands
    const uint32_t sb4 = smem_u32(smem) >> 4;
    auto lk = [&](int s) { return sb4 + (uint32_t)s * (kTileBytes >> 4) + kLboK; };
    auto lm = [&](int s) { return sb4 + (uint32_t)s * (kTileBytes >> 4) + kLboMN; };

    // L2 priorities: tiles read again later (Q and the provisional outputs of segments > 0, until the
    // fix-up; K from the pre-pass to the sweep) are kept, tiles at their last use go first
    const uint64_t pol_first = l2_policy_evict_first(), pol_last = l2_policy_evict_last();
    const uint64_t pol_normal = l2_policy_evict_normal();
    auto load_tile = [&](int s, const CUtensorMap *map, int head, int tok0, uint64_t pol) {
        ld_pend |= 1u << s;
        mbar_arrive_expect_tx(&ms->bar[bLd0 + s], kTileBytes);
        tma_load_3d_hint(slot(s), map, &ms->bar[bLd0 + s], 0, tok0, head, pol);
        tma_load_3d_hint(slot(s) + kBlockBytes, map, &ms->bar[bLd0 + s], 64, tok0, head, pol);
    };
    auto wait_ld = [&](int s) {
        if (!bar_wait(ms, bLd0 + s, (ld_par >> s) & 1u, p)) return false;  // still pending
        ld_par ^= 1u << s;
        ld_pend &= ~(1u << s);
        return true;
    };

    // Pre-pass of an item: S aggregate of its tiles (sum of K^T K) into TMEM columns S, from K tiles
    // in four slots (K, V, W, Q1); none for the last segment of a head unless the final state is
    // wanted.  It runs at the start of a CTA's first item and, for later items,
    // while the previous item's epilogue waits for its D prefix (the S carry is dead by then and the
    // fix-up has not started).  Returns false if a wait gave up.
    bool pre_done = false;  // issuer: the current item's pre-pass ran in the previous item's tail
    auto prepass = [&](int pitem) {
        const int psig = pitem / p.BH, phead = pitem % p.BH;
        const int pt0 = psig * p.L, pnt = min(p.L, p.M - pt0);
        if (!kState && psig + 1 >= p.G) {  // the last segment of a head: nothing reads its S prefix
            mbar_arrive(&ms->bar[bEvP]);
            return true;
        }
        auto ps = [](int j) { return (j & 3) == 0 ? kK : (j & 3) == 1 ? kV : (j & 3) == 2 ? kW : kQ1; };
        for (int j = 0; j < pnt && j < 4; ++j) load_tile(ps(j), &tm_k, phead, (pt0 + j) * kTile, pol_normal);
        for (int j = 0; j < pnt; ++j) {
            const int sl = ps(j);
            if (!wait_ld(sl)) return false;
            tc_fence_after();
            mma128<true, true, kF>(tb + kTS, lm(sl), lm(sl), j > 0 ? 1u : 0u);  // S_agg += K^T K
            if (j + 4 < pnt) {  // long segment: reuse this slot once its MMA is done
                umma_commit(&ms->bar[bPre]);
                if (!bar_wait(ms, bPre, (n_pre++) & 1, p)) return false;
                load_tile(sl, &tm_k, phead, (pt0 + j + 4) * kTile, pol_normal);
            }
        }
        umma_commit(&ms->bar[bEvP]);
        return true;
    };

    if (tid == 0) ms->item = (int)atomicAdd(p.ticket, 1u);  // later tickets are taken by the issuer
    while (true) {
        tc_fence_before();
        __syncthreads();
        tc_fence_after();
        const int item = ms->item;
        if (item >= p.n_items || ms->abort_flag) break;
        const int sigma = item / p.BH, head = item % p.BH;
        const int t0 = sigma * p.L;           // first tile of the segment
        const int nt = min(p.L, p.M - t0);    // tiles in this segment
        const int ip = n_items & 1;

        if (issuer) {
            // one thread issues; a wait that gives up leaves this item's issuing (break) with the CTA
            // marked aborted, so that every role runs on to the end of the item and the loop stops
            if (lane == 0) do {
                // ---- 1. pre-pass (unless it ran in the previous item's tail), first tile's A ----
                const bool early = pre_done;
                pre_done = false;
                if (!early && !prepass(item)) break;
                if (!bar_wait(ms, bEvP, ip, p)) break;  // the pre-pass slots are free again
                // first tile's inputs (K tile 0 is still in slot K after a pre-pass of <= 4 tiles that
                // ran just now, if there was one)
                const uint64_t pol_q = sigma > 0 ? pol_last : pol_first;  // Q is read again by the fix-up
                load_tile(kQ0, &tm_q, head, t0 * kTile, pol_q);
                const bool reload_k = early || nt > 4 || (!kState && sigma + 1 >= p.G);
                if (reload_k) load_tile(kK, &tm_k, head, t0 * kTile, pol_first);
                load_tile(kV, &tm_v, head, t0 * kTile, pol_first);
                if (wait_ld(kQ0) && (!reload_k || wait_ld(kK))) {
                    tc_fence_after();
                    mma128<false, false, 128, kFS>(tb + kTA, lk(kQ0), lk(kK), 0u);  // A = Q K^T
                    umma_commit(&ms->bar[bEvA]);
                }

                // ---- 2. sweep ----
                // Slots per tile: SX holds R_hi, then X_hi; W holds R_lo, then X_lo; SD holds D_p, then
                // the output staging.  The split of the next tile's S_p is written once T and D have
                // read X (while T V + Q D_p run), so that only the output read-out separates O from
                // the next tile's Q R.
                for (int j = 0; j < nt && !ms->abort_flag; ++j) {
                    const uint32_t tp = n_tiles & 1;
                    const int qs = (j & 1) ? kQ1 : kQ0, qo = (j & 1) ? kQ0 : kQ1;
                    // slot qo (Q of the previous tile, last read by its O MMA) takes the next Q
                    if (j + 1 < nt) load_tile(qo, &tm_q, head, (t0 + j + 1) * kTile, pol_q);
                    // X = Q R_hi + Q R_lo + W_hi K + W_lo K; the Q R part runs while W is built.  For the
                    // first tile of a segment the split of S_p comes with W; later ones wait for the
                    // split and for the previous output to have left TMEM columns X.
                    if (j > 0 && !bar_wait(ms, bEpR, (n_r++) & 1, p)) break;
                    if (j > 0 && !bar_wait(ms, bEpO, tp ^ 1u, p)) break;
                    if (j == 0 && !bar_wait(ms, bEpW, tp, p)) break;
                    tc_fence_after();
                    mma128<false, false, kF, kFS>(tb + kTX, lk(qs), lk(kSX), 0u);      // X = Q R_hi
                    if (precise) mma128<false, false, kF, kFS>(tb + kTX, lk(qs), lk(kW), 1u);  // += Q R_lo
                    // S += K^T K while the W epilogue runs (the S carry was read by the previous split,
                    // before Q R could start)
                    if (kState || j + 1 < nt) mma128<true, true, kF>(tb + kTS, lm(kK), lm(kK), 1u);
                    if (j > 0 && !bar_wait(ms, bEpW, tp, p)) break;  // W (hi, lo) ready
                    tc_fence_after();
                    mma128_ts<true, kF>(tb + kTX, tb + kTA, lm(kK), 1u);          // += W_hi K (W in TMEM)
                    if (precise) mma128_ts<true, kF>(tb + kTX, tb + kTA + 16, lm(kK), 1u);  // += W_lo K
                    umma_commit(&ms->bar[bEvX]);
                    if (!bar_wait(ms, bEvX, tp, p)) break;  // X and S MMAs done: slot K free
                    if (j + 1 < nt) load_tile(kK, &tm_k, head, (t0 + j + 1) * kTile, pol_first);
                    if (!bar_wait(ms, bEpX, tp, p)) break;  // X_hi, X_lo in SX, W; D_p read out of TMEM
                    tc_fence_after();
                    if constexpr (!kUnmasked) {
                        mma128<false, false, 128, kFS>(tb + kTA, lk(qs), lk(kSX), 0u);  // T = Q X_hi^T
                        mma128<false, false, 128, kFS>(tb + kTA, lk(qs), lk(kW), 1u);   // += Q X_lo^T
                    } else {
                        mma128<false, false, 128, kFS>(tb + kTA, lk(kSX), lk(qs), 0u);  // T = X_hi Q^T
                        mma128<false, false, 128, kFS>(tb + kTA, lk(kW), lk(qs), 1u);   // += X_lo Q^T
                    }
                    umma_commit(&ms->bar[bEvT]);
                    if (!wait_ld(kV)) break;
                    tc_fence_after();
                    if constexpr (!kUnmasked) {
                        mma128<true, true, kF>(tb + kTD, lm(kSX), lm(kV), 1u);        // D += X_hi^T V
                        if (d_lo) mma128<true, true, kF>(tb + kTD, lm(kW), lm(kV), 1u);  // D += X_lo^T V
                        umma_commit(&ms->bar[bEvD]);
                        // O = Q D_p (D_p in SD since the X hand-off; TMEM X was read out then) runs
                        // while the epilogue forms T
                        mma128<false, true, kF, kFS>(tb + kTX, lk(qs), lm(kSD), 0u);
                    } else {
                        mma128<true, true, kF>(tb + kTD, lm(qs), lm(kV), 1u);  // C += Q^T V
                        mma128<false, true, kF, kFS>(tb + kTX, lk(kSX), lm(kSD), 0u);  // O = X_hi C_p
                        umma_commit(&ms->bar[bEvD]);  // X (slot SX) read: the S split may overwrite it
                    }
                    if (!bar_wait(ms, bEpT, tp, p)) break;  // T (bf16) in TMEM A
                    tc_fence_after();
                    mma128_ts<true, kF>(tb + kTX, tb + kTA, lm(kV), 1u);          // O += T V (T in TMEM)
                    umma_commit(&ms->bar[bEvO]);
                    if (!bar_wait(ms, bEvO, tp, p)) break;  // T, V and D_p read
                    if (j + 1 < nt) {  // next tile's A = Q K^T overlaps this tile's output epilogue
                        if (!wait_ld(qo) || !wait_ld(kK)) break;
                        tc_fence_after();
                        mma128<false, false, 128, kFS>(tb + kTA, lk(qo), lk(kK), 0u);
                        umma_commit(&ms->bar[bEvA]);
                        load_tile(kV, &tm_v, head, (t0 + j + 1) * kTile, pol_first);
                    }
                    ++n_tiles;
                }

                // ---- next ticket; its pre-pass while the epilogue publishes this item's D prefix ----
                if (!ms->abort_flag) {
                    const int next = (int)atomicAdd(p.ticket, 1u);
                    ms->item = next;  // every thread read this item's ticket at the top of the loop
                    if (next < p.n_items) {
                        if (!prepass(next)) break;
                        pre_done = true;
                        if (!bar_wait(ms, bEvP, ip ^ 1, p)) break;  // its slots are free for the fix-up
                    }
                }

                // ---- 3. fix-up of segments > 0 ----
                if (sigma > 0 && !ms->abort_flag) {
                    // three tiles in flight: tile j uses buffer j % 3 (Q slot, provisional output slot,
                    // which also stages the result, and TMEM region for F)
                    auto load_fix = [&](int j) {
                        const int i = j % 3;
                        load_tile(fix_q(i), &tm_q, head, (t0 + j) * kTile, pol_first);
                        load_tile(fix_o(i), &tm_o, head, (t0 + j) * kTile, pol_first);
                    };
                    // the first loads as soon as the provisional outputs are written, while the D
                    // prefix may still be on its way
                    if (bar_wait(ms, bEpOut, n_dfix & 1, p))
                        for (int j = 0; j < nt && j < 3; ++j) load_fix(j);
                    if (bar_wait(ms, bEpDF, n_dfix & 1, p)) {  // D prefix (bf16) in SD
                        for (int j = 0; j < nt; ++j) {
                            const int i = j % 3;
                            if (!wait_ld(fix_q(i)) || !wait_ld(fix_o(i))) break;
                            tc_fence_after();
                            mma128<false, true, kF, kFS>(tb + fix_t(i), lk(fix_q(i)), lm(kSD), 0u);  // F = Q D_prefix
                            umma_commit(&ms->bar[bEvF + i]);
                            if (j >= 1) {  // tile j-1 done: its buffer takes tile j+2
                                const int g = (j - 1) % 3;
                                const bool ok = bar_wait(ms, bEpF + g, (fx_par >> g) & 1u, p);
                                fx_par ^= 1u << g;
                                if (!ok) break;
                                if (j + 2 < nt) load_fix(j + 2);
                            }
                        }
                        {  // the last tile
                            const int g = (nt - 1) % 3;
                            bar_wait(ms, bEpF + g, (fx_par >> g) & 1u, p);
                            fx_par ^= 1u << g;
                        }
                    }
                }
            } while (0);
            __syncwarp();
        } else if (publisher) {
            // one S prefix and one D prefix per item (the epilogue arrives once at each, on every path)
            unsigned *flagS = p.flags, *flagD = p.flags + 2 * p.BH;
            pub_wait(kBarPubS);
            if (lane == 0 && item != p.inject_skip_item) {
                __threadfence();
                st_release(&flagS[head * 2 + (sigma & 1)], (unsigned)(sigma + 1));
            }
            pub_wait(kBarPubD);
            if (lane == 0) {
                __threadfence();
                st_release(&flagD[head * 2 + (sigma & 1)], (unsigned)(sigma + 1));
            }
            __syncwarp();
        } else {
            // ===================== epilogue warps =====================
            const int et = tid;
            const int qd = warp & 3, cq = warp >> 2;
            const int r = 32 * qd + lane;        // TMEM lane = row handled by this thread
            const int c0 = 32 * cq;              // first of the 32 columns handled by this thread
            const uint32_t lane_base = (uint32_t)(32 * qd) << 16;
            // this thread's 32-column block of L . A and L . T lies above the diagonal (zero), on it, or below
            const bool blk_zero = cq > qd;
            // Head size 64 (kNarrow): the products write feature columns 0..63 only, so the threads of
            // column blocks 2, 3 (fcol false) hold zeros in the S carry and the e carry, skip their share
            // of X, R, D_p, O and F, and never read the TMEM columns no product wrote.  Rows 64..127 of
            // D (from the unwritten columns of X_hi / X_lo) are never read by a product over the head size.
            const bool fcol = !kNarrow || cq < 2;
            const float *ring_prev = p.ring + ((size_t)head * 2 + ((sigma + 1) & 1)) * kRingFloats;
            float *ring_cur = p.ring + ((size_t)head * 2 + (sigma & 1)) * kRingFloats;
            const unsigned *flagS = p.flags, *flagD = p.flags + 2 * p.BH;

            // Shift of the S split: cs = bf16(trace / d) with the trace of the carry-in for the first
            // tile and, for later ones, of the S carry one tile back (read at the previous split; a
            // shift one tile stale keeps R small just the same); every epilogue thread holds the same
            // value.  Any shift is exact (x = R q + cs q in fp32).
            float tr_s = 0.f, cs = 0.f;

            // ---- 1. S chain: carry-in S of the segment, publish the inclusive prefix ----
            // (the last segment of a head publishes none unless the final state is wanted)
            const bool s_agg = kState || sigma + 1 < p.G;
            bar_wait(ms, bEvP, ip, p);
            tc_fence_after();
            if (sigma > 0 && et == 0) chain_wait(&flagS[head * 2 + ((sigma - 1) & 1)], (unsigned)sigma, p, 1, item);
            epi_sync();
            {
                // carry-in S: the previous segment's prefix (ring) or the initial state (row-major)
                const float4 *ringS = sigma > 0 ? reinterpret_cast<const float4 *>(ring_prev) : nullptr;
                const float4 *st_row = (sigma == 0 && p.state_in)
                    ? reinterpret_cast<const float4 *>(p.state_in + (size_t)head * kStateFloats + r * kD + c0)
                    : nullptr;
                float sp[32];
#pragma unroll
                for (int c = 0; c < 8; ++c) {
                    const float4 v4 = (ringS && fcol) ? __ldcg(ringS + ring4(c, et))
                                      : st_row ? __ldcg(st_row + c) : make_float4(0.f, 0.f, 0.f, 0.f);
                    sp[4 * c] = v4.x; sp[4 * c + 1] = v4.y; sp[4 * c + 2] = v4.z; sp[4 * c + 3] = v4.w;
                }
                if (s_agg) {
                    // inclusive S prefix of this segment -> ring, published before this segment's set-up
                    float agg[32];
                    if (fcol) {
                        ld32(tb + lane_base + kTS + c0, agg);
                    } else {
#pragma unroll
                        for (int j = 0; j < 32; ++j) agg[j] = 0.f;
                    }
                    float4 *rc = reinterpret_cast<float4 *>(ring_cur);
#pragma unroll
                    for (int j = 0; j < 32; j += 4)
                        __stcg(rc + ring4(j / 4, et), make_float4(sp[j] + agg[j], sp[j + 1] + agg[j + 1],
                                                                 sp[j + 2] + agg[j + 2], sp[j + 3] + agg[j + 3]));
                }
                pub_arrive(kBarPubS);  // S prefix in the ring
                // trace -> shift (the diagonal element of row r lies in column block qd)
                float s = 0.f;
                if (cq == qd) s = pick_lane32<kNarrow>(sp, lane);
                s = warp_sum(s);
                if (lane == 0) ms->red[warp] = s;
                epi_sync();
#pragma unroll
                for (int w = 0; w < kEpiWarps; ++w) tr_s += ms->red[w];
                cs = bf16_round(tr_s / kD);
                // S carry in TMEM
                uint32_t u[32];
#pragma unroll
                for (int j = 0; j < 32; ++j) u[j] = __float_as_uint(sp[j]);
                tmem_st32(tb + lane_base + kTS + c0, u);
                // split S_p = cs I + R into R_hi (slot SX) and R_lo (slot W)
                if (cq == qd) shift_diag32<kNarrow>(sp, lane, cs);
                if (fcol) store_split32(slot(kSX), slot(kW), r, c0, sp, precise);
                // segment-local D carry: the initial state's D for the first segment
                const float *d0 = (sigma == 0 && p.init_De) ? p.init_De + (size_t)head * (kD * kD + kD) : nullptr;
#pragma unroll
                for (int j = 0; j < 32; j += 4) {
                    const float4 v4 = d0 ? __ldcg(reinterpret_cast<const float4 *>(d0 + r * kD + c0 + j))
                                         : make_float4(0.f, 0.f, 0.f, 0.f);
                    u[j] = __float_as_uint(v4.x); u[j + 1] = __float_as_uint(v4.y);
                    u[j + 2] = __float_as_uint(v4.z); u[j + 3] = __float_as_uint(v4.w);
                }
                tmem_st32(tb + lane_base + kTD + c0, u);
                if (cq == 0) ms->eloc[r] = d0 ? d0[kD * kD + r] : 0.f;
                tmem_st_wait();
            }
            fence_async_smem();

            // ---- 2. sweep ----
            // e carry += column sums of X (sum over the four lane quadrants, in a fixed order)
            auto add_ecol = [&](float ec) {
                if (qd > 0) ms->part[qd - 1][c0 + lane] = ec;
                epi_sync();
                if (qd == 0)
                    ms->eloc[c0 + lane] += (ec + ms->part[0][c0 + lane]) + (ms->part[1][c0 + lane] + ms->part[2][c0 + lane]);
                epi_sync();
            };
            float ecol = 0.f;  // this thread's column sum of the last tile's X, added in the next tile's X wait
            for (int j = 0; j < nt; ++j) {
                const uint32_t tp = n_tiles & 1;
                const uint8_t *qt = slot((j & 1) ? kQ1 : kQ0);
                const int tok0 = (t0 + j) * kTile;

                // W = L . A -> bf16 hi and lo, written over this thread's own A columns in TMEM
                // (the A operand of X += W K): hi in columns c0 .. +15, lo in c0 + 16 .. +31
                bar_wait(ms, bEvA, tp, p);
                tc_fence_after();
                {
                    uint32_t h[16], l[16];
                    if (blk_zero) {
#pragma unroll
                        for (int i = 0; i < 16; ++i) h[i] = l[i] = 0u;
                    } else {
                        float f[32];
                        ld32(tb + lane_base + kTA + c0, f);
                        if (cq == qd) mask_upper32<kNarrow>(f, r, c0);
                        split_pack32(f, h, l);
                    }
                    tmem_st16(tb + lane_base + kTA + c0, h);
                    if (precise) tmem_st16(tb + lane_base + kTA + c0 + 16, l);
                    tmem_st_wait();
                }
                epi_arrive(ms, bEpW);

                if (et == 0) tma_store_wait_read();  // the previous output tile has left slot SD
                epi_sync();
                if (need_e && j > 0) add_ecol(ecol);  // the previous tile's X, before q_t . e_p below

                // while X = W K + Q S_p runs: D_p (bf16, final since the previous O) -> slot SD, read
                // out of TMEM before this tile's D MMA (issued after the X hand-off), and q_t . e_p,
                // the carried part of the denominator
                if (fcol) {
                    float f[32];
                    ld32(tb + lane_base + kTD + c0, f);
#pragma unroll
                    for (int jj = 0; jj < 32; jj += 8) store_row8(slot(kSD), r, c0 + jj, f + jj);
                }
                float den_part = 0.f;
                if (!kUnmasked && p.normalized && fcol) {
#pragma unroll
                    for (int jj = 0; jj < 32; jj += 8) {
                        float q8[8];
                        tile_row8(qt, r, c0 + jj, q8);
#pragma unroll
                        for (int u = 0; u < 8; ++u) den_part += q8[u] * ms->eloc[c0 + jj + u];
                    }
                }

                // X -> X_hi (slot SX), X_lo (slot W)
                bar_wait(ms, bEvX, tp, p);
                tc_fence_after();
                float x[32];
                if (fcol) {
                    ld32(tb + lane_base + kTX + c0, x);
#pragma unroll
                    for (int jj = 0; jj < 32; jj += 8) {
                        float q8[8];
                        tile_row8(qt, r, c0 + jj, q8);
#pragma unroll
                        for (int u = 0; u < 8; ++u) x[jj + u] += cs * q8[u];
                    }
                    store_split32(slot(kSX), slot(kW), r, c0, x, true);
                } else {
#pragma unroll
                    for (int jj = 0; jj < 32; ++jj) x[jj] = 0.f;
                }
                fence_async_smem();  // X_hi, X_lo and D_p (above) visible to the MMAs
                epi_arrive(ms, bEpX);

                // while T = Q X^T runs: column sums of X (e carry)
                if (need_e) ecol = warp_colsum32(x);  // column c0 + lane over this warp's rows

                // T = L . (Q X^T) -> bf16 in TMEM; row sums
                bar_wait(ms, bEvT, tp, p);
                tc_fence_after();
                {
                    // bf16 T over this thread's own T columns in TMEM (the A operand of O += T V)
                    uint32_t h[16];
                    if (blk_zero) {
#pragma unroll
                        for (int i = 0; i < 16; ++i) h[i] = 0u;
                    } else {
                        float f[32];
                        ld32(tb + lane_base + kTA + c0, f);
                        if (cq == qd) mask_upper32<kNarrow>(f, r, c0);
#pragma unroll
                        for (int jj = 0; jj < 32; ++jj) den_part += f[jj];
                        pack32(f, h);
                    }
                    tmem_st16(tb + lane_base + kTA + c0, h);
                    tmem_st_wait();
                }
                epi_arrive(ms, bEpT);

                // denominators: partial sums of the four column quarters, added in a fixed order
                if (p.normalized) {
                    if (cq == 0) ms->den[r] = den_part;
                    else ms->part[cq - 1][r] = den_part;
                }
                epi_sync();
                const float den = p.normalized ? ((ms->den[r] + ms->part[0][r]) + ms->part[1][r]) + ms->part[2][r] : 1.f;

                // D += X^T V done (T too): slots SX and W are free, the S carry is current.  Split of
                // S_p for the next tile while T V + Q D_p run.
                bar_wait(ms, bEvD, tp, p);
                tc_fence_after();
                if (j + 1 < nt) {
                    float f[32];
                    if (fcol) {
                        ld32(tb + lane_base + kTS + c0, f);
                    } else {
#pragma unroll
                        for (int jj = 0; jj < 32; ++jj) f[jj] = 0.f;
                    }
                    const float *dt = ms->dtr[(j + 1) & 1];
                    cs = bf16_round((j == 0 ? tr_s : (dt[0] + dt[1]) + (dt[2] + dt[3])) / kD);
                    {
                        float dg = 0.f;
                        if (cq == qd) dg = pick_lane32<kNarrow>(f, lane);
                        dg = warp_sum(dg);
                        if (cq == qd && lane == 0) ms->dtr[j & 1][qd] = dg;
                    }
                    if (cq == qd) shift_diag32<kNarrow>(f, lane, cs);
                    if (fcol) store_split32(slot(kSX), slot(kW), r, c0, f, precise);
                    fence_async_smem();
                    epi_arrive(ms, bEpR);  // R of the next tile ready: Q R may start once O is read
                }

                // O (provisional for segments > 0, final for the first) -> slot SD, TMA store
                bar_wait(ms, bEvO, tp, p);
                tc_fence_after();
                {
                    const bool final_out = (sigma == 0);
                    float f[32];
                    if (fcol) {
                        ld32(tb + lane_base + kTX + c0, f);
                    } else {
#pragma unroll
                        for (int jj = 0; jj < 32; ++jj) f[jj] = 0.f;
                    }
                    epi_arrive(ms, bEpO);  // TMEM columns X are free for the next tile's X
                    if (final_out && p.normalized) {
                        const float inv = 1.f / (den + p.eps);
#pragma unroll
                        for (int jj = 0; jj < 32; ++jj) f[jj] *= inv;
                    }
                    if (fcol) {
#pragma unroll
                        for (int jj = 0; jj < 32; jj += 8) store_row8(slot(kSD), r, c0 + jj, f + jj);
                    }
                    if (!final_out && p.normalized && cq == 0 && tok0 + r < p.n)
                        p.den_loc[(size_t)head * p.n + tok0 + r] = den;
                }
                fence_async_smem();
                epi_sync();  // also: every denominator read before part is reused
                if (et == 0) {  // provisional outputs stay in L2 for the fix-up
                    const uint64_t pol = sigma > 0 ? l2_policy_evict_last() : l2_policy_evict_first();
                    tma_store_3d_hint(&tm_o, slot(kSD), 0, tok0, head, pol);
                    if (p.out_blocks > 1) tma_store_3d_hint(&tm_o, slot(kSD) + kBlockBytes, 64, tok0, head, pol);
                    tma_store_commit();
                }
                ++n_tiles;
            }
            if (need_e && nt > 0) add_ecol(ecol);  // the last tile's X
            if (sigma > 0) {  // the fix-up may load the provisional outputs once they are written
                if (et == 0) tma_store_wait_all();
                epi_arrive(ms, bEpOut);
            }

            // ---- 3. D chain and fix-up ----
            {
                if (et == 0) {
                    tma_store_wait_read();  // the last output tile has left slot SD (D prefix below)
                    if (sigma > 0) chain_wait(&flagD[head * 2 + ((sigma - 1) & 1)], (unsigned)sigma, p, 2, item);
                }
                epi_sync();
                const float4 *dprev = sigma > 0 ? reinterpret_cast<const float4 *>(ring_prev + kD * kD) : nullptr;
                float4 *dcur = reinterpret_cast<float4 *>(ring_cur + kD * kD);
                {
                    float f[32], dp[32];
                    ld32(tb + lane_base + kTD + c0, f);
#pragma unroll
                    for (int jj = 0; jj < 32; jj += 4) {
                        const float4 v4 = dprev ? __ldcg(dprev + ring4(jj / 4, et)) : make_float4(0.f, 0.f, 0.f, 0.f);
                        dp[jj] = v4.x; dp[jj + 1] = v4.y; dp[jj + 2] = v4.z; dp[jj + 3] = v4.w;
                    }
#pragma unroll
                    for (int jj = 0; jj < 32; jj += 4)
                        __stcg(dcur + ring4(jj / 4, et), make_float4(dp[jj] + f[jj], dp[jj + 1] + f[jj + 1],
                                                                    dp[jj + 2] + f[jj + 2], dp[jj + 3] + f[jj + 3]));
                    if (sigma > 0) {  // D prefix (bf16) for the fix-up
#pragma unroll
                        for (int jj = 0; jj < 32; jj += 8) store_row8(slot(kSD), r, c0 + jj, dp + jj);
                    }
                }
                float eprev = 0.f;
                if (cq == 0) {
                    eprev = sigma > 0 ? __ldcg(ring_prev + 2 * kD * kD + r) : 0.f;
                    __stcg(ring_cur + 2 * kD * kD + r, eprev + ms->eloc[r]);
                }
                pub_arrive(kBarPubD);  // D and e prefixes in the ring
                if (sigma > 0) {
                    if (cq == 0) ms->eloc[r] = eprev;  // now e of the prefix, for the fix-up denominators
                    fence_async_smem();
                    epi_sync();
                    epi_arrive(ms, bEpDF);
                    for (int j = 0; j < nt; ++j) {
                        const int i = j % 3;
                        const uint8_t *qt = slot(fix_q(i));
                        uint8_t *ot = slot(fix_o(i));  // provisional output, overwritten by the result
                        const int tok0 = (t0 + j) * kTile;
                        const float dl = (p.normalized && cq == 0 && tok0 + r < p.n)
                                             ? __ldcg(p.den_loc + (size_t)head * p.n + tok0 + r) : 0.f;
                        bar_wait(ms, bEvF + i, (fx_par >> i) & 1u, p);
                        tc_fence_after();
                        if (p.normalized) {
                            // den_t = provisional denominator + q_t . e_prefix (four column quarters)
                            // (q is zero beyond the head size)
                            float qe = 0.f;
#pragma unroll
                            for (int jj = 0; jj < 32; jj += 8) {
                                float q8[8];
                                tile_row8(qt, r, c0 + jj, q8);
#pragma unroll
                                for (int u = 0; u < 8; ++u) qe += q8[u] * ms->eloc[c0 + jj + u];
                            }
                            if (cq == 0) ms->den[r] = dl + qe;
                            else ms->part[cq - 1][r] = qe;
                        }
                        if (j >= 1 && et == 0) tma_store_wait_read();  // tile j-1's result has left its slot
                        epi_sync();
                        if (j >= 1) epi_arrive(ms, bEpF + (j - 1) % 3);  // tile j-1's buffer is free
                        const float inv = p.normalized
                            ? 1.f / ((((ms->den[r] + ms->part[0][r]) + ms->part[1][r]) + ms->part[2][r]) + p.eps)
                            : 1.f;
                        if (fcol) {
                            float f[32];
                            ld32(tb + lane_base + fix_t(i) + c0, f);
#pragma unroll
                            for (int jj = 0; jj < 32; jj += 8) {
                                float o8[8], w8[8];
                                tile_row8(ot, r, c0 + jj, o8);
#pragma unroll
                                for (int u = 0; u < 8; ++u) w8[u] = (o8[u] + f[jj + u]) * inv;
                                store_row8(ot, r, c0 + jj, w8);
                            }
                        }
                        fence_async_smem();
                        epi_sync();  // also: every denominator read before the next tile's partials
                        if (et == 0) {
                            const uint64_t pol = l2_policy_evict_first();
                            tma_store_3d_hint(&tm_o, ot, 0, tok0, head, pol);
                            if (p.out_blocks > 1) tma_store_3d_hint(&tm_o, ot + kBlockBytes, 64, tok0, head, pol);
                            tma_store_commit();
                        }
                        fx_par ^= 1u << i;
                    }
                    if (et == 0) tma_store_wait_read();  // the last result has left its slot
                    epi_sync();
                    epi_arrive(ms, bEpF + (nt - 1) % 3);
                }
            }
        }
        ++n_items;
        if (sigma > 0) ++n_dfix;
        // every role has finished this item (output stores may still be in flight)
        if (!issuer && tid == 0) tma_store_wait_all();
    }

    if (issuer && lane == 0 && ms->abort_flag) {
        // a wait gave up: the copies and MMAs this CTA still has in flight finish (each wait bounded)
        // before its shared memory and TMEM are released
        for (int s = 0; s <= kSX; ++s)
            if ((ld_pend >> s) & 1u) mbar_wait(&ms->bar[bLd0 + s], (ld_par >> s) & 1u, kBarWaitNs);
        umma_commit(&ms->bar[bTear]);
        mbar_wait(&ms->bar[bTear], 0, kBarWaitNs);
    }
    tc_fence_before();
    __syncthreads();
    if (issuer) {
        tc_fence_after();
        tmem_dealloc(tb, 512);
    }
}

// initial-state carries D_0 = S_0 C_0 - G_0 and e_0 = S_0 m_0 - h_0 of each head (fp32)
__global__ void __launch_bounds__(256) init_carry_kernel(const float *__restrict__ st, float *__restrict__ out) {
    const int hd = blockIdx.x;
    const size_t L = kStateFloats;
    const float *S = st + hd * L, *C = S + kD * kD, *m = C + kD * kD, *G = m + kD, *h = G + kD * kD;
    float *D = out + (size_t)hd * (kD * kD + kD), *e = D + kD * kD;
    for (int idx = threadIdx.x; idx < kD * kD + kD; idx += blockDim.x) {
        if (idx < kD * kD) {
            const int a = idx / kD, b = idx % kD;
            float s = 0.f;
            for (int j = 0; j < kD; ++j) s += S[a * kD + j] * C[j * kD + b];
            D[idx] = s - G[idx];
        } else {
            const int a = idx - kD * kD;
            float s = 0.f;
            for (int j = 0; j < kD; ++j) s += S[a * kD + j] * m[j];
            e[a] = s - h[a];
        }
    }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        cudaDriverEntryPointQueryResult q;
        void *f = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(f);
    }
    return fn;
}

// [BH][n][inner] bf16 tensor (inner = 64 or 128), boxes of 64 columns x 128 tokens,
// 128-byte swizzle, zero fill out of range (the box at column 64 of a 64-wide tensor
// is all fill)
bool make_map(CUtensorMap *m, const void *base, int BH, int n, int inner) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[3] = {(cuuint64_t)inner, (cuuint64_t)n, (cuuint64_t)BH};
    cuuint64_t strides[2] = {(cuuint64_t)inner * 2, (cuuint64_t)n * inner * 2};
    cuuint32_t box[3] = {64, (cuuint32_t)kTile, 1};
    cuuint32_t es[3] = {1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims, strides, box, es,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

struct FusedLayout {
    size_t off_ticket, off_flags, off_ring, off_den, off_init, off_part, total, total_state;
};

int state_groups(int BH, int M);

FusedLayout fused_layout(int BH, int n) {
    FusedLayout L;
    size_t o = kWsHeaderBytes;
    L.off_ticket = o; o += 256;
    L.off_flags = o; o = align_up(o + sizeof(unsigned) * 4 * (size_t)BH, 256);
    L.off_ring = o; o = align_up(o + sizeof(float) * 2 * (size_t)BH * kRingFloats, 256);
    L.off_den = o; o = align_up(o + sizeof(float) * (size_t)BH * n, 256);
    L.off_init = o; o = align_up(o + sizeof(float) * (size_t)BH * (kD * kD + kD), 256);
    L.total = o;
    // C / m partials of the final state (only when state_out is asked for)
    const int M = (n + kTile - 1) / kTile;
    L.off_part = o; o = align_up(o + sizeof(float) * (size_t)BH * state_groups(BH, M) * (kD * kD + kD), 256);
    L.total_state = o;
    return L;
}

// Predicted duration (us) of the ticket schedule with segments of L tiles: items in ticket order go
// to the SM that frees first; an item costs 5.5 us per tile of sweep and, for segments > 0, 2.1 us
// per fix-up tile and 7 us of chain set-up (2 us for a first segment); in the first wave the S
// prefix ripples through the concurrent segments of a head (about 5.6 us per segment, after a cold
// pre-pass of 4.7 us).  Constants measured on B2 H16 n16384 d128.
double predicted_span(int BH, int M, int L, int sms) {
    std::priority_queue<double, std::vector<double>, std::greater<double>> free_at;
    for (int i = 0; i < sms; ++i) free_at.push(0.0);
    double span = 0.0;
    const int G = (M + L - 1) / L;
    for (int sg = 0; sg < G; ++sg) {
        const int li = std::min(L, M - sg * L);
        for (int h = 0; h < BH; ++h) {
            const double t = free_at.top();
            free_at.pop();
            double c = 5.5 * li + (sg > 0 ? 2.1 * li + 7.0 : 2.0);
            if (t == 0.0) c += 4.7 + 5.6 * sg;
            free_at.push(t + c);
            span = std::max(span, t + c);
        }
    }
    return span;
}

int segment_tiles(int BH, int M, int sms) {
    if (const char *e = getenv("HLA_FUSED_SEGMENT_TILES")) {
        int v = atoi(e);
        if (v > 0) return v < M ? v : M;
    }
    if (2 * BH >= sms) return M;  // heads enough to occupy the SMs: one segment per head, no chains
    // Segments of 2..8 tiles (the range measured): the length whose schedule is predicted to end
    // first (on B2 H16 n16384 the prediction picks 7, measured best among 4..13; 6 is 3.5 % slower
    // there because 704 items leave the last wave of the 152 SMs partly idle).
    int best = 2;
    double best_t = 1e300;
    for (int L = 2; L <= 8 && L <= M; ++L) {
        const double t = predicted_span(BH, M, L, sms);
        if (t < best_t) {
            best_t = t;
            best = L;
        }
    }
    return best < M ? best : M;
}

// ---------------------------------------------------------------------------
// final state (state_out): C = C_0 + Q^T V and m = m_0 + Q^T 1 on the tensor
// cores, then the paper tuple from the prefixes the forward left in its ring:
// S, D = S C - G and e = S m - h of the whole sequence, so G = S C - D and
// h = S m - e (the D-form of Eq. semidirect read backwards)
// ---------------------------------------------------------------------------
constexpr int kCThreads = 160;            // 4 warps read TMEM (one lane quadrant each), warp 4 issues
constexpr uint32_t kCOnesBytes = 4096;    // 16 x 128 bf16 ones operand (row 0 ones), K-major
constexpr uint32_t kCSmemBytes = 4 * kTileBytes + kCOnesBytes + 1024;
constexpr int kCPartFloats = kD * kD + kD;  // C (d x dv) then m (d) of one group of tiles

// C and m of tiles [g * tiles_per, ...) of a head, from tiles of 128 tokens (Q^T V: A = Q^T and
// B = V both MN-major; m: B = a 16-row K-major operand whose row 0 is ones)
__global__ void __launch_bounds__(kCThreads, 1)
state_c_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_v, float *part,
               int M, int groups, int tiles_per, WsHeader *err) {
    extern __shared__ __align__(1024) uint8_t csm[];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int head = blockIdx.x / groups, g = blockIdx.x % groups;
    const int j0 = g * tiles_per, j1 = min(M, j0 + tiles_per);
    uint8_t *ones = csm + 4 * kTileBytes;
    // after the tiles and the ones operand: loads of slot pair 0 / 1, MMAs of pair 0 / 1, all done
    uint64_t *bars = reinterpret_cast<uint64_t *>(ones + kCOnesBytes);
    uint32_t &tmem_base_s = *reinterpret_cast<uint32_t *>(bars + 5);
    int &abort_c = *reinterpret_cast<int *>(bars + 6);
    if (smem_u32(csm) & 1023u) {
        if (tid == 0) set_error(err, 98, smem_u32(csm));
        return;
    }
    // ones operand: element (row, token k) of the 128-byte swizzled K-major layout
    for (int i = tid; i < 16 * 128; i += blockDim.x) {
        const int row = i / 128, kk = i % 128;
        const uint32_t off = (kk >> 6) * 2048 + row * 128 + ((((kk & 63) >> 3) ^ (row & 7)) << 4) + (kk & 7) * 2;
        *reinterpret_cast<uint16_t *>(ones + off) = row == 0 ? (uint16_t)0x3F80 : (uint16_t)0;
    }
    if (tid == 0) {
        for (int b = 0; b < 5; ++b) mbar_init(&bars[b], 1);
        abort_c = 0;
        fence_mbar_init();
    }
    if (warp == 4) {
        tmem_alloc(&tmem_base_s, 256);
        tmem_relinquish();
    }
    fence_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tb = tmem_base_s;
    auto cwait = [&](int b, uint32_t par) {
        if (abort_c) return false;
        if (mbar_wait(&bars[b], par, kBarWaitNs)) return true;
        set_error(err, 150 + b, par);
        abort_c = 1;
        return false;
    };
    if (warp == 4) {
        if (lane == 0) {
            const uint32_t sb4 = smem_u32(csm) >> 4;
            auto lmn = [&](int s) { return sb4 + (uint32_t)s * (kTileBytes >> 4) + kLboMN; };
            const uint32_t ones_lo = (smem_u32(ones) >> 4) + kLboK;
            auto load_pair = [&](int j) {
                const int sl = (j - j0) & 1;
                mbar_arrive_expect_tx(&bars[sl], 2 * kTileBytes);
                uint8_t *qs = csm + (2 * sl) * kTileBytes, *vs = csm + (2 * sl + 1) * kTileBytes;
                tma_load_3d(qs, &tm_q, &bars[sl], 0, j * kTile, head);
                tma_load_3d(qs + kBlockBytes, &tm_q, &bars[sl], 64, j * kTile, head);
                tma_load_3d(vs, &tm_v, &bars[sl], 0, j * kTile, head);
                tma_load_3d(vs + kBlockBytes, &tm_v, &bars[sl], 64, j * kTile, head);
            };
            if (j0 < j1) load_pair(j0);
            if (j0 + 1 < j1) load_pair(j0 + 1);
            constexpr uint32_t id_m = idesc_bf16(128, 16, 1, 0);
            for (int j = j0; j < j1; ++j) {
                const int i = j - j0, sl = i & 1;
                if (!cwait(sl, (i >> 1) & 1)) break;
                tc_fence_after();
                mma128<true, true>(tb, lmn(2 * sl), lmn(2 * sl + 1), i > 0 ? 1u : 0u);  // C += Q^T V
#pragma unroll
                for (int kk = 0; kk < 8; ++kk)  // m += Q^T 1 (column 128)
                    umma_bf16(tb + 128, (static_cast<uint64_t>(kDescHi) << 32) | (lmn(2 * sl) + kk * 128u),
                              (static_cast<uint64_t>(kDescHi) << 32) | (ones_lo + (kk >> 2) * 128u + (kk & 3) * 2u),
                              id_m, (i > 0 || kk > 0) ? 1u : 0u);
                umma_commit(&bars[2 + sl]);
                if (j + 2 < j1) {
                    if (!cwait(2 + sl, (i >> 1) & 1)) break;
                    load_pair(j + 2);
                }
            }
            umma_commit(&bars[4]);
        }
        __syncwarp();
    } else {
        // C rows (features f = 32 warp + lane), 128 columns, then m
        float *out = part + (size_t)blockIdx.x * kCPartFloats;
        const uint32_t lb = (uint32_t)(32 * warp) << 16;
        const int f = 32 * warp + lane;
        const bool ok = (j0 < j1) && cwait(4, 0);
        tc_fence_after();
        for (int c0 = 0; c0 < kD; c0 += 32) {
            float v[32];
            if (ok) ld32(tb + lb + c0, v);
            for (int jj = 0; jj < 32; ++jj) out[(size_t)f * kD + c0 + jj] = ok ? v[jj] : 0.f;
        }
        float mv[32];
        if (ok) ld32(tb + lb + 128, mv);
        out[kD * kD + f] = ok ? mv[0] : 0.f;
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 4) {
        tc_fence_after();
        tmem_dealloc(tb, 256);
    }
}

// per head: the paper tuple [S | C | m | G | h] (d x d, d x dv, d, d x dv, d) from the ring slot of
// the head's last segment and the C / m partials; state_in (may alias state_out) supplies C_0, m_0
__global__ void __launch_bounds__(256) state_finalize_kernel(const float *ring, int last_slot, const float *part,
                                                             int groups, const float *state_in, float *state_out,
                                                             int d, int dv) {
    extern __shared__ float fs[];
    float *S = fs, *C = S + kD * kD, *m = C + kD * kD;  // 128 x 128, 128 x 128, 128 (zero outside d, dv)
    const int hd = blockIdx.x, tid = threadIdx.x;
    const float *rg = ring + ((size_t)hd * 2 + last_slot) * kRingFloats;
    const size_t st_len = (size_t)d * d + 2 * (size_t)d * dv + 2 * (size_t)d;
    const float *sin = state_in ? state_in + (size_t)hd * st_len : nullptr;
    // the ring stores float4 c (columns c0 + 4c..) of epilogue thread et = 32 (qd + 4 cq) + lane at c * 512 + et
    auto ring_at = [&](const float *base, int r, int col) {
        const int et = 32 * ((r >> 5) + 4 * (col >> 5)) + (r & 31);
        return base[(size_t)(((col & 31) >> 2) * kEpiThreads + et) * 4 + (col & 3)];
    };
    for (int i = tid; i < kD * kD; i += blockDim.x) {
        const int r = i / kD, c = i % kD;
        S[i] = ring_at(rg, r, c);
        float cv = 0.f;
        if (r < d && c < dv) {
            for (int g = 0; g < groups; ++g) cv += part[((size_t)hd * groups + g) * kCPartFloats + (size_t)r * kD + c];
            if (sin) cv += sin[(size_t)d * d + (size_t)r * dv + c];
        }
        C[i] = cv;
    }
    for (int r = tid; r < kD; r += blockDim.x) {
        float mv = 0.f;
        if (r < d) {
            for (int g = 0; g < groups; ++g) mv += part[((size_t)hd * groups + g) * kCPartFloats + kD * kD + r];
            if (sin) mv += sin[(size_t)d * d + (size_t)d * dv + r];
        }
        m[r] = mv;
    }
    __syncthreads();  // everything read from state_in before state_out (possibly the same memory) is written
    float *so = state_out + (size_t)hd * st_len;
    float *oS = so, *oC = oS + (size_t)d * d, *om = oC + (size_t)d * dv, *oG = om + d, *oh = oG + (size_t)d * dv;
    for (int i = tid; i < d * d; i += blockDim.x) oS[i] = S[(i / d) * kD + i % d];
    for (int i = tid; i < d * dv; i += blockDim.x) {
        const int r = i / dv, c = i % dv;
        float sc = 0.f;
        for (int x = 0; x < d; ++x) sc += S[r * kD + x] * C[x * kD + c];
        oC[i] = C[r * kD + c];
        oG[i] = sc - ring_at(rg + kD * kD, r, c);  // G = S C - D
    }
    for (int r = tid; r < d; r += blockDim.x) {
        float sm_ = 0.f;
        for (int x = 0; x < d; ++x) sm_ += S[r * kD + x] * m[x];
        om[r] = m[r];
        oh[r] = sm_ - rg[2 * kD * kD + r];  // h = S m - e
    }
}

int state_groups(int BH, int M) {
    int g = 256 / (BH > 0 ? BH : 1);
    if (g < 1) g = 1;
    if (g > 8) g = 8;
    return g < M ? g : M;
}

}  // namespace

// head sizes the fused kernel serves (64 as zero-padded 128)
bool fused_dim(int x) { return x == 64 || x == kD; }

size_t fused2_workspace_bytes(int BH, int n, int d, int dv, int chunk, hla_dtype dt, bool with_state) {
    if (dt != HLA_BF16 || !fused_dim(d) || !fused_dim(dv)) return 0;
    (void)chunk;
    const FusedLayout L = fused_layout(BH, n);
    return with_state ? L.total_state : L.total;
}

bool fused2_applicable(const Fwd2 &p) {
    if (getenv("HLA_DISABLE_FUSED")) return false;
    if (p.dt != HLA_BF16 || !fused_dim(p.d) || !fused_dim(p.dv)) return false;
    // unmasked: plain output, no state.  Its denominator x_t . m_t would carry the 2^-17 relative
    // error of the hi/lo products that form x_t times |m_t| ~ sqrt(t), beyond what the fp32 bar of
    // the parity criterion allows; the ratio-normalised unmasked output stays on the fp32 path.
    if (!p.masked && (p.state_in || p.state_out || p.normalized)) return false;
    if (p.n <= 0 || p.BH <= 0) return false;
    if (p.state_in && (p.d != kD || p.dv != kD)) return false;  // initial states in the 128 x 128 layout only
    const FusedLayout FL = fused_layout(p.BH, p.n);
    if (p.ws_bytes < (p.state_out ? FL.total_state : FL.total)) return false;
    int dev = 0, major = 0, minor = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return false;
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    return major == 10 && minor == 3 && encode_fn() != nullptr;
}

cudaError_t fused2_forward(const Fwd2 &p, cudaStream_t stream) {
    FusedLayout FL = fused_layout(p.BH, p.n);
    CUtensorMap mq, mk, mv, mo;
    if (!make_map(&mq, p.q, p.BH, p.n, p.d) || !make_map(&mk, p.k, p.BH, p.n, p.d) ||
        !make_map(&mv, p.v, p.BH, p.n, p.dv) || !make_map(&mo, p.out, p.BH, p.n, p.dv))
        return cudaErrorInvalidValue;
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    Params kp{};
    kp.BH = p.BH;
    kp.n = p.n;
    kp.M = (p.n + kTile - 1) / kTile;
    kp.L = p.masked ? segment_tiles(p.BH, kp.M, sms) : kp.M;  // unmasked: one segment per head
    kp.G = (kp.M + kp.L - 1) / kp.L;
    kp.n_items = kp.G * p.BH;
    kp.normalized = p.normalized;
    kp.eps = p.eps;
    kp.state_in = p.state_in;
    kp.init_De = nullptr;
    kp.ring = reinterpret_cast<float *>(p.ws + FL.off_ring);
    kp.flags = reinterpret_cast<unsigned *>(p.ws + FL.off_flags);
    kp.ticket = reinterpret_cast<unsigned *>(p.ws + FL.off_ticket);
    kp.den_loc = reinterpret_cast<float *>(p.ws + FL.off_den);
    kp.err = reinterpret_cast<WsHeader *>(p.ws);
    kp.wait_ns = 2000000000ull;
    kp.inject_skip_item = -1;
    kp.out_blocks = p.dv / 64;
    if (const char *e = getenv("HLA_TEST_WAIT_NS")) kp.wait_ns = strtoull(e, nullptr, 10);
    if (const char *e = getenv("HLA_TEST_SKIP_PUBLISH_ITEM")) kp.inject_skip_item = atoi(e);
    cudaError_t e;
    // ticket and chain flags start at zero every launch
    if ((e = cudaMemsetAsync(p.ws + FL.off_ticket, 0, FL.off_ring - FL.off_ticket, stream))) return e;
    if (p.state_in) {
        float *init = reinterpret_cast<float *>(p.ws + FL.off_init);
        init_carry_kernel<<<p.BH, 256, 0, stream>>>(p.state_in, init);
        if ((e = cudaGetLastError())) return e;
        kp.init_De = init;
    }
    const int grid = kp.n_items < sms ? kp.n_items : sms;
    // instantiation: final state or not, head size 64 (d = dv = 64) or 128 (also 64 x 128 mixes, padded)
    auto launch = [&](auto kern) -> cudaError_t {
        cudaError_t err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
        if (err) return err;
        kern<<<grid, kThreads, kSmemBytes, stream>>>(mq, mk, mv, mo, kp);
        return cudaGetLastError();
    };
    const bool narrow = p.d == 64 && p.dv == 64;
    if (!p.masked)  // no state (fused2_applicable)
        e = narrow ? launch(hla2_fused_kernel<false, true, true>) : launch(hla2_fused_kernel<false, false, true>);
    else if (p.state_out)
        e = narrow ? launch(hla2_fused_kernel<true, true>) : launch(hla2_fused_kernel<true, false>);
    else
        e = narrow ? launch(hla2_fused_kernel<false, true>) : launch(hla2_fused_kernel<false, false>);
    if (e) return e;
    if ((e = cudaGetLastError()) || !p.state_out) return e;
    // final state: C and m partials, then the tuple (state_in, read by the kernel above, may alias)
    const int groups = state_groups(p.BH, kp.M);
    const int tiles_per = (kp.M + groups - 1) / groups;
    float *part = reinterpret_cast<float *>(p.ws + FL.off_part);
    if ((e = cudaFuncSetAttribute(state_c_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kCSmemBytes)))
        return e;
    state_c_kernel<<<p.BH * groups, kCThreads, kCSmemBytes, stream>>>(mq, mv, part, kp.M, groups, tiles_per, kp.err);
    if ((e = cudaGetLastError())) return e;
    const int fin_smem = (int)(sizeof(float) * (2 * kD * kD + kD));
    if ((e = cudaFuncSetAttribute(state_finalize_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, fin_smem)))
        return e;
    state_finalize_kernel<<<p.BH, 256, fin_smem, stream>>>(kp.ring, (kp.G - 1) & 1, part, groups, p.state_in,
                                                            p.state_out, p.d, p.dv);
    return cudaGetLastError();
}

}  // namespace hla
