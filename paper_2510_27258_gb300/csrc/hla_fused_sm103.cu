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
// Roles: warp 8 issues TMA loads and MMAs (one thread); warps 0-7 are the
// epilogue (TMEM -> registers -> shared memory): warp w reads TMEM lanes
// 32 (w % 4) .. +31 (one row each) and columns 64 (w / 4) .. +63.
//
// Precision: tokens are bf16, every product accumulates in fp32 (TMEM).  The S
// operand is split as S = c I + R (c = bf16(trace S / d)) with c q_t added in
// fp32, so x_t is accurate although |S| grows like t/d.  X enters T = Q X^T as
// bf16 hi + lo (with X rounded once, q_t . x_t = (q_t . k_t)^2 at t = 0 would
// lose |q||k| / |q.k| times the bf16 rounding when q and k are nearly
// orthogonal).  For the normalised output, whose denominator cancels heavily,
// R and W are also split into hi + lo, so X and T are accurate to ~2^-16 of
// each term; the denominator is the fp32 row sum of T plus q_t . e_p, with the
// e carry summed in fp32 on CUDA cores.  T and D enter T V and Q D as bf16.
#include "hla_internal.h"
#include "sm103_prims.cuh"

namespace hla {
namespace {

using namespace sm103;

constexpr int kD = 128;           // d = dv handled by this kernel
constexpr int kTile = 128;        // tokens per tile (MMA M)
constexpr int kEpiWarps = 8;      // 2 per TMEM lane quadrant
constexpr int kEpiThreads = kEpiWarps * 32;
constexpr int kIssuerWarp = kEpiWarps;
constexpr int kThreads = kEpiThreads + 32;
constexpr int kSlots = 7;
constexpr uint32_t kSmemTiles = kSlots * kTileBytes;
constexpr uint32_t kMiscBytes = 3072;
constexpr uint32_t kSmemBytes = kSmemTiles + kMiscBytes;  // = 227 KiB; base must be 1 KiB aligned

// shared-memory slots (32 KiB each)
enum Slot { kQ0 = 0, kQ1 = 1, kK = 2, kV = 3, kW = 4, kSX = 5, kSD = 6 };

// TMEM columns: S carry, D carry, A -> T, X -> O
constexpr uint32_t kTS = 0, kTD = 128, kTA = 256, kTX = 384;

// barrier indices
enum Bar {
    bLd0 = 0,  // + slot index for the four input slots (Q0, Q1, K, V)
    bPre = 4,  // pre-pass MMA done (per K tile)
    bEvP = 5, bEvA = 6, bEvX = 7, bEvT = 8, bEvO = 9, bEvF = 10,
    bEpW = 11, bEpX = 12, bEpT = 13, bEpF = 14, bEpDF = 15,
    kNumBars = 16
};
constexpr int kFirstEpiBar = bEpW;

struct Misc {
    uint64_t bar[kNumBars];
    uint32_t tmem_base;
    int item;        // current ticket
    int abort_flag;  // an mbarrier wait gave up
    int pad;
    float cshift[2]; // S shift of the current / next tile
    float red[kEpiWarps];
    float eloc[kD];      // segment-local e carry
    float den[kTile];    // denominators of the current tile
    float ebuf[2][kD];   // cross-quadrant partial column sums of X
};
static_assert(sizeof(Misc) <= kMiscBytes, "misc smem");

struct Params {
    int BH, n, M, L, G, n_items;
    int normalized;
    float eps;
    const float *state_in;  // S_0 of each head (paper tuple), or null
    const float *init_De;   // D_0 (d*dv) and e_0 (d) of each head, or null
    float *ring;            // [BH][2][d*d + d*dv + d]
    unsigned *flags;        // [2][BH][2]: S flags then D flags
    unsigned *ticket;
    float *den_loc;         // [BH][n] provisional denominators (normalised, segments > 0)
    WsHeader *err;
    unsigned long long wait_ns;  // budget of a cross-SM chain wait
    int inject_skip_item;        // testing: this item does not publish its S prefix
};

constexpr int kRingFloats = kD * kD + kD * kD + kD;
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
__device__ __forceinline__ void epi_sync() { asm volatile("bar.sync 1, 256;" ::: "memory"); }

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

__device__ __forceinline__ void store_zero32(uint8_t *tile, int r, int c0) {
#pragma unroll
    for (int j = 0; j < 32; j += 8) *reinterpret_cast<uint4 *>(tile + tile_off(r, c0 + j)) = make_uint4(0, 0, 0, 0);
}

__device__ __forceinline__ float bf16_round(float x) { return __bfloat162float(__float2bfloat16_rn(x)); }

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

// ---------------------------------------------------------------------------
// the kernel
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads, 1)
hla2_fused_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                  const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_o, Params p) {
    extern __shared__ __align__(1024) uint8_t smem[];
    Misc *ms = reinterpret_cast<Misc *>(smem + kSmemTiles);
    auto slot = [&](int s) { return smem + s * kTileBytes; };

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const bool issuer = (warp == kIssuerWarp);

    // the tile layout needs 1 KiB alignment of the dynamic shared memory
    if (smem_u32(smem) & 1023u) {
        if (tid == 0) set_error(p.err, 99, smem_u32(smem));
        return;
    }
    if (tid == 0) {
        for (int b = 0; b < kNumBars; ++b) mbar_init(&ms->bar[b], b >= kFirstEpiBar ? kEpiWarps : 1);
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
    uint32_t n_tiles = 0, n_items = 0, n_fix = 0, n_pre = 0, n_dfix = 0;
    uint32_t ld_cnt[4] = {0, 0, 0, 0};

    constexpr uint32_t idA = idesc_bf16(128, 128, 0, 0);   // Q K^T, Q R, Q X^T: both K-major
    constexpr uint32_t idKmn = idesc_bf16(128, 128, 0, 1); // W K, T V, Q D: B MN-major
    constexpr uint32_t idMM = idesc_bf16(128, 128, 1, 1);  // K^T K, X^T V: both MN-major
    const uint32_t tileQ[2] = {smem_u32(slot(kQ0)), smem_u32(slot(kQ1))};
    const uint32_t sK = smem_u32(slot(kK)), sV = smem_u32(slot(kV)), sW = smem_u32(slot(kW));
    const uint32_t sSX = smem_u32(slot(kSX)), sSD = smem_u32(slot(kSD));

    auto load_tile = [&](int s, const CUtensorMap *map, int head, int tok0) {
        mbar_arrive_expect_tx(&ms->bar[bLd0 + s], kTileBytes);
        tma_load_3d(slot(s), map, &ms->bar[bLd0 + s], 0, tok0, head);
        tma_load_3d(slot(s) + kBlockBytes, map, &ms->bar[bLd0 + s], 64, tok0, head);
    };
    auto wait_ld = [&](int s) { return bar_wait(ms, bLd0 + s, (ld_cnt[s]++) & 1, p); };

    while (true) {
        if (tid == 0) ms->item = (int)atomicAdd(p.ticket, 1u);
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
            if (lane == 0) {
                // ---- 1. pre-pass: S aggregate of the segment into TMEM cols kTX ----
                const int ps[2] = {kK, kV};
                load_tile(ps[0], &tm_k, head, (t0 + 0) * kTile);
                if (nt > 1) load_tile(ps[1], &tm_k, head, (t0 + 1) * kTile);
                for (int j = 0; j < nt; ++j) {
                    const int s = ps[j & 1];
                    if (!wait_ld(s)) break;
                    tc_fence_after();
                    for (int kk = 0; kk < 8; ++kk)
                        umma_bf16(tb + kTX, desc_mnmajor(smem_u32(slot(s)), kk), desc_mnmajor(smem_u32(slot(s)), kk),
                                  idMM, (j > 0 || kk > 0) ? 1u : 0u);
                    umma_commit(&ms->bar[bPre]);
                    if (!bar_wait(ms, bPre, (n_pre++) & 1, p)) break;
                    if (j + 2 < nt) load_tile(s, &tm_k, head, (t0 + j + 2) * kTile);
                }
                umma_commit(&ms->bar[bEvP]);
                // first tile's inputs and its A = Q K^T
                load_tile(kQ0, &tm_q, head, t0 * kTile);
                load_tile(kK, &tm_k, head, t0 * kTile);
                load_tile(kV, &tm_v, head, t0 * kTile);
                if (wait_ld(kQ0) && wait_ld(kK)) {
                    tc_fence_after();
                    for (int kk = 0; kk < 8; ++kk)
                        umma_bf16(tb + kTA, desc_kmajor(tileQ[0], kk), desc_kmajor(sK, kk), idA, kk > 0);
                    umma_commit(&ms->bar[bEvA]);
                }

                // ---- 2. sweep ----
                for (int j = 0; j < nt && !ms->abort_flag; ++j) {
                    const uint32_t tp = n_tiles & 1;
                    const uint32_t sQ = tileQ[j & 1], sQo = tileQ[(j + 1) & 1];
                    if (!bar_wait(ms, bEpW, tp, p)) break;  // W (hi, lo), S split ready; TMEM X free
                    tc_fence_after();
                    for (int kk = 0; kk < 8; ++kk)  // X = W_hi K
                        umma_bf16(tb + kTX, desc_kmajor(sW, kk), desc_mnmajor(sK, kk), idKmn, kk > 0);
                    if (p.normalized)
                        for (int kk = 0; kk < 8; ++kk)  // X += W_lo K  (W_lo staged in the other Q slot)
                            umma_bf16(tb + kTX, desc_kmajor(sQo, kk), desc_mnmajor(sK, kk), idKmn, 1u);
                    for (int kk = 0; kk < 8; ++kk)  // X += Q R_hi
                        umma_bf16(tb + kTX, desc_kmajor(sQ, kk), desc_kmajor(sSX, kk), idA, 1u);
                    if (p.normalized)
                        for (int kk = 0; kk < 8; ++kk)  // X += Q R_lo
                            umma_bf16(tb + kTX, desc_kmajor(sQ, kk), desc_kmajor(sSD, kk), idA, 1u);
                    for (int kk = 0; kk < 8; ++kk)  // S += K^T K
                        umma_bf16(tb + kTS, desc_mnmajor(sK, kk), desc_mnmajor(sK, kk), idMM, 1u);
                    umma_commit(&ms->bar[bEvX]);
                    if (!bar_wait(ms, bEvX, tp, p)) break;
                    if (j + 1 < nt) {
                        load_tile(kK, &tm_k, head, (t0 + j + 1) * kTile);
                        load_tile((j & 1) ? kQ0 : kQ1, &tm_q, head, (t0 + j + 1) * kTile);
                    }
                    if (!bar_wait(ms, bEpX, tp, p)) break;  // X_hi, X_lo and D_hi ready
                    if (!wait_ld(kV)) break;
                    tc_fence_after();
                    for (int kk = 0; kk < 8; ++kk)  // T = Q X_hi^T
                        umma_bf16(tb + kTA, desc_kmajor(sQ, kk), desc_kmajor(sSX, kk), idA, kk > 0);
                    for (int kk = 0; kk < 8; ++kk)  // T += Q X_lo^T  (X_lo staged in slot W)
                        umma_bf16(tb + kTA, desc_kmajor(sQ, kk), desc_kmajor(sW, kk), idA, 1u);
                    for (int kk = 0; kk < 8; ++kk)  // D += X^T V
                        umma_bf16(tb + kTD, desc_mnmajor(sSX, kk), desc_mnmajor(sV, kk), idMM, 1u);
                    umma_commit(&ms->bar[bEvT]);
                    if (!bar_wait(ms, bEpT, tp, p)) break;  // T ready; TMEM A free
                    tc_fence_after();
                    for (int kk = 0; kk < 8; ++kk)  // O = Q D_p
                        umma_bf16(tb + kTX, desc_kmajor(sQ, kk), desc_mnmajor(sSD, kk), idKmn, kk > 0);
                    for (int kk = 0; kk < 8; ++kk)  // O += T V
                        umma_bf16(tb + kTX, desc_kmajor(sW, kk), desc_mnmajor(sV, kk), idKmn, 1u);
                    umma_commit(&ms->bar[bEvO]);
                    if (j + 1 < nt) {  // next tile's A = Q K^T overlaps this tile's output epilogue
                        if (!wait_ld((j & 1) ? kQ0 : kQ1) || !wait_ld(kK)) break;
                        tc_fence_after();
                        for (int kk = 0; kk < 8; ++kk)
                            umma_bf16(tb + kTA, desc_kmajor(sQo, kk), desc_kmajor(sK, kk), idA, kk > 0);
                        umma_commit(&ms->bar[bEvA]);
                    }
                    if (!bar_wait(ms, bEvO, tp, p)) break;
                    if (j + 1 < nt) load_tile(kV, &tm_v, head, (t0 + j + 1) * kTile);
                    ++n_tiles;
                }

                // ---- 3. fix-up of segments > 0 ----
                if (sigma > 0 && !ms->abort_flag) {
                    if (bar_wait(ms, bEpDF, n_dfix & 1, p)) {  // D prefix (bf16) in SD; outputs written
                        load_tile(kQ0, &tm_q, head, t0 * kTile);
                        load_tile(kK, &tm_o, head, t0 * kTile);
                        for (int j = 0; j < nt; ++j) {
                            const int qs = (j & 1) ? kQ1 : kQ0, os = (j & 1) ? kV : kK;
                            if (!wait_ld(qs) || !wait_ld(os)) break;
                            tc_fence_after();
                            for (int kk = 0; kk < 8; ++kk)  // F = Q D_prefix
                                umma_bf16(tb + kTA, desc_kmajor(tileQ[j & 1], kk), desc_mnmajor(sSD, kk), idKmn,
                                          kk > 0);
                            umma_commit(&ms->bar[bEvF]);
                            if (j + 1 < nt) {
                                // the other pair of slots was released by the previous fix-up epilogue
                                load_tile((j & 1) ? kQ0 : kQ1, &tm_q, head, (t0 + j + 1) * kTile);
                                load_tile((j & 1) ? kK : kV, &tm_o, head, (t0 + j + 1) * kTile);
                            }
                            if (!bar_wait(ms, bEpF, (n_fix++) & 1, p)) break;
                        }
                    }
                }
            }
            __syncwarp();
        } else {
            // ===================== epilogue warps =====================
            const int et = tid;
            const int qd = warp & 3, hf = warp >> 2;
            const int r = 32 * qd + lane;        // TMEM lane = row handled by this thread
            const int cb0 = 64 * hf;             // first of the 64 columns handled by this thread
            const uint32_t lane_base = (uint32_t)(32 * qd) << 16;
            const float *ring_prev = p.ring + ((size_t)head * 2 + ((sigma + 1) & 1)) * kRingFloats;
            float *ring_cur = p.ring + ((size_t)head * 2 + (sigma & 1)) * kRingFloats;
            unsigned *flagS = p.flags, *flagD = p.flags + 2 * p.BH;

            // ---- 1. S chain: carry-in S of the segment, publish the inclusive prefix ----
            bar_wait(ms, bEvP, ip, p);
            tc_fence_after();
            if (sigma > 0 && et == 0) chain_wait(&flagS[head * 2 + ((sigma - 1) & 1)], (unsigned)sigma, p, 1, item);
            epi_sync();
            {
                const float *sprev = nullptr;
                if (sigma > 0) sprev = ring_prev + r * kD;
                else if (p.state_in) sprev = p.state_in + (size_t)head * kStateFloats + r * kD;
                float s = (sprev && (r >> 6) == hf) ? __ldcg(sprev + r) : 0.f;  // diagonal -> trace
                s = warp_sum(s);
                if (lane == 0) ms->red[warp] = s;
                epi_sync();
                float tr = 0.f;
#pragma unroll
                for (int w = 0; w < kEpiWarps; ++w) tr += ms->red[w];
                const float c = bf16_round(tr / kD);
                if (et == 0) ms->cshift[0] = c;
                const float *d0 = (sigma == 0 && p.init_De) ? p.init_De + (size_t)head * (kD * kD + kD) : nullptr;
#pragma unroll 1
                for (int c0 = cb0; c0 < cb0 + 64; c0 += 32) {
                    float agg[32], sp[32];
                    ld32(tb + lane_base + kTX + c0, agg);
#pragma unroll
                    for (int j = 0; j < 32; j += 4) {
                        const float4 v4 = sprev ? __ldcg(reinterpret_cast<const float4 *>(sprev + c0 + j))
                                                : make_float4(0.f, 0.f, 0.f, 0.f);
                        sp[j] = v4.x; sp[j + 1] = v4.y; sp[j + 2] = v4.z; sp[j + 3] = v4.w;
                    }
#pragma unroll
                    for (int j = 0; j < 32; j += 4)
                        __stcg(reinterpret_cast<float4 *>(ring_cur + r * kD + c0 + j),
                               make_float4(sp[j] + agg[j], sp[j + 1] + agg[j + 1], sp[j + 2] + agg[j + 2],
                                           sp[j + 3] + agg[j + 3]));
                    uint32_t u[32];
#pragma unroll
                    for (int j = 0; j < 32; ++j) u[j] = __float_as_uint(sp[j]);
                    tmem_st32(tb + lane_base + kTS + c0, u);
                    // split S_p = c I + R into R_hi (slot SX) and R_lo (slot SD)
                    float hi[32], lo[32];
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        const float rr = sp[j] - ((c0 + j) == r ? c : 0.f);
                        hi[j] = bf16_round(rr);
                        lo[j] = rr - hi[j];
                    }
#pragma unroll
                    for (int j = 0; j < 32; j += 8) {
                        store_row8(slot(kSX), r, c0 + j, hi + j);
                        if (p.normalized) store_row8(slot(kSD), r, c0 + j, lo + j);
                    }
                    // segment-local D carry: the initial state's D for the first segment
#pragma unroll
                    for (int j = 0; j < 32; ++j) u[j] = __float_as_uint(d0 ? d0[r * kD + c0 + j] : 0.f);
                    tmem_st32(tb + lane_base + kTD + c0, u);
                }
                if (hf == 0) ms->eloc[r] = d0 ? d0[kD * kD + r] : 0.f;
                tmem_st_wait();
            }
            fence_async_smem();
            epi_sync();
            if (et == 0 && item != p.inject_skip_item) {
                __threadfence();
                st_release(&flagS[head * 2 + (sigma & 1)], (unsigned)(sigma + 1));
            }

            // ---- 2. sweep ----
            for (int j = 0; j < nt; ++j) {
                const uint32_t tp = n_tiles & 1;
                const uint8_t *qt = slot((j & 1) ? kQ1 : kQ0);
                uint8_t *wlo = slot((j & 1) ? kQ0 : kQ1);  // W_lo staging (the other Q slot)
                const int tok0 = (t0 + j) * kTile;

                // W = L . A (hi, lo)
                bar_wait(ms, bEvA, tp, p);
                tc_fence_after();
                if (et == 0) tma_store_wait_read();  // the previous output tile has left slot W
                epi_sync();
#pragma unroll 1
                for (int c0 = cb0; c0 < cb0 + 64; c0 += 32) {
                    if ((c0 >> 5) > qd) {  // block entirely above the diagonal
                        store_zero32(slot(kW), r, c0);
                        if (p.normalized) store_zero32(wlo, r, c0);
                        continue;
                    }
                    float f[32], g[32];
                    ld32(tb + lane_base + kTA + c0, f);
#pragma unroll
                    for (int jj = 0; jj < 32; ++jj) {
                        if (c0 + jj > r) f[jj] = 0.f;
                        g[jj] = f[jj] - bf16_round(f[jj]);
                    }
#pragma unroll
                    for (int jj = 0; jj < 32; jj += 8) {
                        store_row8(slot(kW), r, c0 + jj, f + jj);
                        if (p.normalized) store_row8(wlo, r, c0 + jj, g + jj);
                    }
                }
                fence_async_smem();
                epi_arrive(ms, bEpW);

                // X -> X_hi (slot SX), X_lo (slot W); D_p -> bf16 (slot SD); e carry
                bar_wait(ms, bEvX, tp, p);
                tc_fence_after();
                const float cs = ms->cshift[j & 1];
                float den_part = 0.f, ecol[2] = {0.f, 0.f};
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int c0 = cb0 + 32 * h;
                    float x[32];
                    ld32(tb + lane_base + kTX + c0, x);
#pragma unroll
                    for (int jj = 0; jj < 32; jj += 8) {
                        float q8[8], lo8[8];
                        tile_row8(qt, r, c0 + jj, q8);
#pragma unroll
                        for (int u = 0; u < 8; ++u) {
                            x[jj + u] += cs * q8[u];
                            lo8[u] = x[jj + u] - bf16_round(x[jj + u]);
                            if (p.normalized) den_part += q8[u] * ms->eloc[c0 + jj + u];
                        }
                        store_row8(slot(kSX), r, c0 + jj, x + jj);
                        store_row8(slot(kW), r, c0 + jj, lo8);
                    }
                    if (p.normalized) ecol[h] = warp_colsum32(x);  // column c0 + lane over this warp's rows
                }
#pragma unroll 1
                for (int c0 = cb0; c0 < cb0 + 64; c0 += 32) {
                    float f[32];
                    ld32(tb + lane_base + kTD + c0, f);
#pragma unroll
                    for (int jj = 0; jj < 32; jj += 8) store_row8(slot(kSD), r, c0 + jj, f + jj);
                }
                fence_async_smem();
                epi_arrive(ms, bEpX);

                // T = L . (Q X^T) -> bf16 (slot W); denominators; next S split (hi)
                bar_wait(ms, bEvT, tp, p);
                tc_fence_after();
#pragma unroll 1
                for (int c0 = cb0; c0 < cb0 + 64; c0 += 32) {
                    if ((c0 >> 5) > qd) {
                        store_zero32(slot(kW), r, c0);
                        continue;
                    }
                    float f[32];
                    ld32(tb + lane_base + kTA + c0, f);
#pragma unroll
                    for (int jj = 0; jj < 32; ++jj) {
                        if (c0 + jj > r) f[jj] = 0.f;
                        den_part += f[jj];
                    }
#pragma unroll
                    for (int jj = 0; jj < 32; jj += 8) store_row8(slot(kW), r, c0 + jj, f + jj);
                }
                if (p.normalized) {  // den_t = both halves' partial sums
                    if (hf == 1) ms->den[r] = den_part;
                    epi_sync();
                    if (hf == 0) ms->den[r] += den_part;
                }
                if (j + 1 < nt) {
                    // shift of the next tile from the trace of the updated S
                    float dg = 0.f;
                    if ((qd >> 1) == hf) {
                        float f[32];
                        ld32(tb + lane_base + kTS + 32 * qd, f);  // block holding the diagonal of these rows
#pragma unroll
                        for (int jj = 0; jj < 32; ++jj)
                            if (jj == lane) dg = f[jj];
                    }
                    dg = warp_sum(dg);
                    if (lane == 0) ms->red[warp] = dg;
                    epi_sync();
                    float tr = 0.f;
#pragma unroll
                    for (int w = 0; w < kEpiWarps; ++w) tr += ms->red[w];
                    const float c = bf16_round(tr / kD);
                    if (et == 0) ms->cshift[(j + 1) & 1] = c;
#pragma unroll 1
                    for (int c0 = cb0; c0 < cb0 + 64; c0 += 32) {
                        float f[32];
                        ld32(tb + lane_base + kTS + c0, f);
#pragma unroll
                        for (int jj = 0; jj < 32; ++jj) f[jj] -= ((c0 + jj) == r ? c : 0.f);
#pragma unroll
                        for (int jj = 0; jj < 32; jj += 8) store_row8(slot(kSX), r, c0 + jj, f + jj);
                    }
                }
                fence_async_smem();
                epi_sync();
                epi_arrive(ms, bEpT);

                // e carry += column sums of X (fixed order ((q0 + q1) + (q2 + q3)))
                if (p.normalized) {
                    const int ca = cb0 + lane, cbx = cb0 + 32 + lane;
                    if (qd & 1) { ms->ebuf[qd >> 1][ca] = ecol[0]; ms->ebuf[qd >> 1][cbx] = ecol[1]; }
                    epi_sync();
                    if (!(qd & 1)) { ecol[0] += ms->ebuf[qd >> 1][ca]; ecol[1] += ms->ebuf[qd >> 1][cbx]; }
                    epi_sync();
                    if (qd == 2) { ms->ebuf[0][ca] = ecol[0]; ms->ebuf[0][cbx] = ecol[1]; }
                    epi_sync();
                    if (qd == 0) {
                        ms->eloc[ca] += ecol[0] + ms->ebuf[0][ca];
                        ms->eloc[cbx] += ecol[1] + ms->ebuf[0][cbx];
                    }
                }

                // O (provisional for segments > 0, final for the first) -> slot W, TMA store
                bar_wait(ms, bEvO, tp, p);
                tc_fence_after();
                {
                    const bool final_out = (sigma == 0);
                    const float den = p.normalized ? ms->den[r] : 1.f;
                    const bool divide = final_out && p.normalized;
#pragma unroll 1
                    for (int c0 = cb0; c0 < cb0 + 64; c0 += 32) {
                        float f[32];
                        ld32(tb + lane_base + kTX + c0, f);
                        if (divide) {
#pragma unroll
                            for (int jj = 0; jj < 32; ++jj) f[jj] = f[jj] / (den + p.eps);
                        }
#pragma unroll
                        for (int jj = 0; jj < 32; jj += 8) store_row8(slot(kW), r, c0 + jj, f + jj);
                    }
                    if (!final_out && p.normalized && hf == 0 && tok0 + r < p.n)
                        p.den_loc[(size_t)head * p.n + tok0 + r] = den;
                }
                if (j + 1 < nt && p.normalized) {  // next S split (lo): D_p (bf16) in SD is dead now
                    const float c = ms->cshift[(j + 1) & 1];
#pragma unroll 1
                    for (int c0 = cb0; c0 < cb0 + 64; c0 += 32) {
                        float f[32];
                        ld32(tb + lane_base + kTS + c0, f);
#pragma unroll
                        for (int jj = 0; jj < 32; ++jj) {
                            const float rr = f[jj] - ((c0 + jj) == r ? c : 0.f);
                            f[jj] = rr - bf16_round(rr);
                        }
#pragma unroll
                        for (int jj = 0; jj < 32; jj += 8) store_row8(slot(kSD), r, c0 + jj, f + jj);
                    }
                }
                fence_async_smem();
                epi_sync();
                if (et == 0) {
                    tma_store_3d(&tm_o, slot(kW), 0, tok0, head);
                    tma_store_3d(&tm_o, slot(kW) + kBlockBytes, 64, tok0, head);
                    tma_store_commit();
                }
                ++n_tiles;
            }

            // ---- 3. D chain and fix-up ----
            {
                if (sigma > 0 && et == 0) chain_wait(&flagD[head * 2 + ((sigma - 1) & 1)], (unsigned)sigma, p, 2, item);
                epi_sync();
                const float *dprev = sigma > 0 ? ring_prev + kD * kD + r * kD : nullptr;
#pragma unroll 1
                for (int c0 = cb0; c0 < cb0 + 64; c0 += 32) {
                    float f[32], dp[32];
                    ld32(tb + lane_base + kTD + c0, f);
#pragma unroll
                    for (int jj = 0; jj < 32; jj += 4) {
                        const float4 v4 = dprev ? __ldcg(reinterpret_cast<const float4 *>(dprev + c0 + jj))
                                                : make_float4(0.f, 0.f, 0.f, 0.f);
                        dp[jj] = v4.x; dp[jj + 1] = v4.y; dp[jj + 2] = v4.z; dp[jj + 3] = v4.w;
                    }
#pragma unroll
                    for (int jj = 0; jj < 32; jj += 4)
                        __stcg(reinterpret_cast<float4 *>(ring_cur + kD * kD + r * kD + c0 + jj),
                               make_float4(dp[jj] + f[jj], dp[jj + 1] + f[jj + 1], dp[jj + 2] + f[jj + 2],
                                           dp[jj + 3] + f[jj + 3]));
                    if (sigma > 0) {
#pragma unroll
                        for (int jj = 0; jj < 32; jj += 8) store_row8(slot(kSD), r, c0 + jj, dp + jj);
                    }
                }
                float eprev = 0.f;
                if (hf == 0) {
                    eprev = sigma > 0 ? __ldcg(ring_prev + 2 * kD * kD + r) : 0.f;
                    __stcg(ring_cur + 2 * kD * kD + r, eprev + ms->eloc[r]);
                }
                tc_fence_before();
                epi_sync();
                if (et == 0) {
                    __threadfence();
                    st_release(&flagD[head * 2 + (sigma & 1)], (unsigned)(sigma + 1));
                }
                if (sigma > 0) {
                    if (hf == 0) ms->eloc[r] = eprev;  // now e of the prefix, for the fix-up denominators
                    if (et == 0) tma_store_wait_all();  // provisional outputs written before they are re-read
                    fence_async_smem();
                    epi_sync();
                    epi_arrive(ms, bEpDF);
                    for (int j = 0; j < nt; ++j) {
                        const uint8_t *qt = slot((j & 1) ? kQ1 : kQ0), *ot = slot((j & 1) ? kV : kK);
                        const int tok0 = (t0 + j) * kTile;
                        bar_wait(ms, bEvF, n_fix & 1, p);
                        tc_fence_after();
                        float den = 1.f;
                        if (p.normalized) {
                            // den_t = provisional denominator + q_t . e_prefix (two column halves)
                            float qe = 0.f;
#pragma unroll
                            for (int c0 = cb0; c0 < cb0 + 64; c0 += 8) {
                                float q8[8];
                                tile_row8(qt, r, c0, q8);
#pragma unroll
                                for (int u = 0; u < 8; ++u) qe += q8[u] * ms->eloc[c0 + u];
                            }
                            if (hf == 1) ms->den[r] = qe;
                            epi_sync();
                            if (hf == 0)
                                ms->den[r] += qe + (tok0 + r < p.n ? p.den_loc[(size_t)head * p.n + tok0 + r] : 0.f);
                            epi_sync();
                            den = ms->den[r];
                        }
                        if (et == 0) tma_store_wait_read();
                        epi_sync();
#pragma unroll 1
                        for (int c0 = cb0; c0 < cb0 + 64; c0 += 32) {
                            float f[32];
                            ld32(tb + lane_base + kTA + c0, f);
#pragma unroll
                            for (int jj = 0; jj < 32; jj += 8) {
                                float o8[8];
                                tile_row8(ot, r, c0 + jj, o8);
#pragma unroll
                                for (int u = 0; u < 8; ++u) {
                                    const float num = o8[u] + f[jj + u];
                                    f[jj + u] = p.normalized ? num / (den + p.eps) : num;
                                }
                            }
#pragma unroll
                            for (int jj = 0; jj < 32; jj += 8) store_row8(slot(kW), r, c0 + jj, f + jj);
                        }
                        fence_async_smem();
                        epi_sync();
                        if (et == 0) {
                            tma_store_3d(&tm_o, slot(kW), 0, tok0, head);
                            tma_store_3d(&tm_o, slot(kW) + kBlockBytes, 64, tok0, head);
                            tma_store_commit();
                        }
                        epi_arrive(ms, bEpF);
                        ++n_fix;
                    }
                }
            }
        }
        ++n_items;
        if (sigma > 0) ++n_dfix;
        // every role has finished this item (output stores may still be in flight)
        if (!issuer && tid == 0) tma_store_wait_all();
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

// [BH][n][128] bf16 tensor, boxes of 64 x 128 tokens, 128-byte swizzle, zero fill out of range
bool make_map(CUtensorMap *m, const void *base, int BH, int n) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[3] = {(cuuint64_t)kD, (cuuint64_t)n, (cuuint64_t)BH};
    cuuint64_t strides[2] = {(cuuint64_t)kD * 2, (cuuint64_t)n * kD * 2};
    cuuint32_t box[3] = {64, (cuuint32_t)kTile, 1};
    cuuint32_t es[3] = {1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims, strides, box, es,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

struct FusedLayout {
    size_t off_ticket, off_flags, off_ring, off_den, off_init, total;
};

FusedLayout fused_layout(int BH, int n) {
    FusedLayout L;
    size_t o = kWsHeaderBytes;
    L.off_ticket = o; o += 256;
    L.off_flags = o; o = align_up(o + sizeof(unsigned) * 4 * (size_t)BH, 256);
    L.off_ring = o; o = align_up(o + sizeof(float) * 2 * (size_t)BH * kRingFloats, 256);
    L.off_den = o; o = align_up(o + sizeof(float) * (size_t)BH * n, 256);
    L.off_init = o; o = align_up(o + sizeof(float) * (size_t)BH * (kD * kD + kD), 256);
    L.total = o;
    return L;
}

int segment_tiles(int BH, int M, int sms) {
    if (const char *e = getenv("HLA_FUSED_SEGMENT_TILES")) {
        int v = atoi(e);
        if (v > 0) return v < M ? v : M;
    }
    // enough segments that the heads fill the SMs several times over, but long
    // enough that the chained scans stay short; tuned on the long workload
    int L = 4;
    if ((long long)BH * ((M + L - 1) / L) < 2LL * sms) L = 2;
    if (BH >= 2 * sms) L = M;  // plenty of heads: one segment per head, no chains
    return L < M ? L : M;
}

}  // namespace

size_t fused2_workspace_bytes(int BH, int n, int d, int dv, int chunk, hla_dtype dt) {
    if (dt != HLA_BF16 || d != kD || dv != kD) return 0;
    (void)chunk;
    return fused_layout(BH, n).total;
}

bool fused2_applicable(const Fwd2 &p) {
    if (getenv("HLA_DISABLE_FUSED")) return false;
    if (p.dt != HLA_BF16 || p.d != kD || p.dv != kD || !p.masked || p.chunk != kTile) return false;
    if (p.state_out || p.n <= 0 || p.BH <= 0) return false;
    if (p.ws_bytes < fused_layout(p.BH, p.n).total) return false;
    int dev = 0, major = 0, minor = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return false;
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    return major == 10 && minor == 3 && encode_fn() != nullptr;
}

cudaError_t fused2_forward(const Fwd2 &p, cudaStream_t stream) {
    FusedLayout FL = fused_layout(p.BH, p.n);
    CUtensorMap mq, mk, mv, mo;
    if (!make_map(&mq, p.q, p.BH, p.n) || !make_map(&mk, p.k, p.BH, p.n) || !make_map(&mv, p.v, p.BH, p.n) ||
        !make_map(&mo, p.out, p.BH, p.n))
        return cudaErrorInvalidValue;
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    Params kp{};
    kp.BH = p.BH;
    kp.n = p.n;
    kp.M = (p.n + kTile - 1) / kTile;
    kp.L = segment_tiles(p.BH, kp.M, sms);
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
    if ((e = cudaFuncSetAttribute(hla2_fused_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes)))
        return e;
    const int grid = kp.n_items < sms ? kp.n_items : sms;
    hla2_fused_kernel<<<grid, kThreads, kSmemBytes, stream>>>(mq, mk, mv, mo, kp);
    return cudaGetLastError();
}

}  // namespace hla
