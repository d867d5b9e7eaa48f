// AHLA forward on the tensor cores (sm_103a): tcgen05 MMAs with TMEM accumulators,
// TMA tile loads and stores, one persistent CTA per SM working through heads.
//
// The asymmetric operator (Sec. "Asymmetric Higher-order Linear Attention",
// Theorem AHLA) is causal linear attention applied twice.  Per 128-token tile of
// a head (rows = tokens, p = carry before the tile):
//   A = Q K^T,  W = L . A                    (L: lower triangle incl. the diagonal)
//   R = W V + Q P_p                          (rows r_t = q_t^T P_t)
//   O = W R + Q E_p                          (rows o_t = q_t^T E_t)
//   P_p += K^T V,  E_p += K^T R
// Each head is swept by one CTA from its first tile to its last, with the P and
// E carries in TMEM (the scan of Eq. AHLA-semidirect done serially over tiles,
// which the scan equivalence makes equal to the serial recurrence).
//
// TMEM (512 columns): P carry, E carry, region A (A, then W as packed bf16, the
// A operand of W V and W R straight from tensor memory), region R (R, then O).
// Shared memory, seven 32 KB tiles: Q and K double-buffered (the next tile's
// copies are in flight during this one), V, R (bf16, the B operand of W R and of
// K^T R), and one slot that holds P_p (bf16), then E_p (bf16), then the output
// staging of the TMA store.
//
// Roles: warp 16 issues TMA copies and MMAs (one thread); warps 0-15 are the
// epilogue: warp w reads TMEM lanes 32 (w % 4) .. +31 (one row each) and columns
// 32 (w / 4) .. +31.
//
// Scope: bf16 tokens, d and dv in {64, 128}, the plain (unnormalised) output, no
// initial or final state.  d = dv = 64 has its own instantiation (kNarrow): the
// products over the head size take 4 K steps and N = 64, and the epilogue reads
// and writes 64 columns.  A mix of 64 and 128 runs as 128 with zero features
// 64..127 (the TMA box of those columns lies outside the tensor and is
// zero-filled).  Precision: W, R and
// the bf16 copies of the carries are rounded to bf16 once; every product
// accumulates in fp32.
#include <vector>

#include "hla_internal.h"
#include "sm103_prims.cuh"

namespace hla {
namespace {

using namespace sm103;

constexpr int kTile = 128;
constexpr int kEpiWarps = 16;
constexpr int kEpiThreads = kEpiWarps * 32;
constexpr int kIssuerWarp = kEpiWarps;
constexpr int kThreads = kEpiThreads + 32;
constexpr int kSlots = 7;
constexpr uint32_t kSmemTiles = kSlots * kTileBytes;
constexpr uint32_t kMiscBytes = 1024;
constexpr uint32_t kSmemBytes = kSmemTiles + kMiscBytes;

enum Slot { kQ0 = 0, kQ1 = 1, kK0 = 2, kK1 = 3, kV = 4, kC = 5, kR = 6 };
constexpr uint32_t kTP = 0, kTE = 128, kTA = 256, kTR = 384;  // TMEM columns

enum Bar {
    bLd0 = 0,  // + slot, for the TMA-loaded slots Q0, Q1, K0, K1, V
    bEvA = 5, bEvR = 6, bEvO = 7,  // MMA commits
    bEpW = 8, bEpR = 9,            // epilogue hand-offs (16 warp arrivals)
    bTear = 10,
    bEvV = 11, bEvE = 12,          // commits: V read (after P += K^T V); E += K^T R done
    kNumBars = 13
};

struct Misc {
    uint64_t bar[kNumBars];
    uint32_t tmem_base;
    int abort_flag;
};
static_assert(sizeof(Misc) <= kMiscBytes, "misc smem");

struct Params {
    int BH, n, M;
    int out_blocks;  // 64-column blocks of an output row (dv / 64)
    WsHeader *err;
};

constexpr unsigned long long kBarWaitNs = 2000000000ull;

__device__ __forceinline__ void set_error(WsHeader *err, unsigned where, unsigned detail) {
    if (atomicCAS(&err->error, 0u, (unsigned)kDevTimeout) == 0u) {
        err->where = where;
        err->detail = detail;
    }
}

// bounded mbarrier wait; on timeout the error word is set and the CTA is marked aborted
__device__ __forceinline__ bool bar_wait(Misc *ms, int b, uint32_t parity, const Params &p) {
    if (ms->abort_flag) return false;
    if (mbar_wait(&ms->bar[b], parity, kBarWaitNs)) return true;
    set_error(p.err, 300 + b, parity);
    ms->abort_flag = 1;
    return false;
}

__device__ __forceinline__ void epi_sync() { asm volatile("bar.sync 1, %0;" ::"n"(kEpiThreads) : "memory"); }

__device__ __forceinline__ void epi_arrive(Misc *ms, int b) {
    tc_fence_before();
    __syncwarp();
    if ((threadIdx.x & 31) == 0) mbar_arrive(&ms->bar[b]);
}

// 32 fp32 values of row r (columns c0 .. c0 + 31) -> bf16 in a tile (the swizzled layout TMA uses)
__device__ __forceinline__ void store_row32(uint8_t *tile, int r, int c0, const uint32_t (&a)[32]) {
#pragma unroll
    for (int jj = 0; jj < 32; jj += 8) {
        uint4 u;
        u.x = pack_bf16x2(__uint_as_float(a[jj]), __uint_as_float(a[jj + 1]));
        u.y = pack_bf16x2(__uint_as_float(a[jj + 2]), __uint_as_float(a[jj + 3]));
        u.z = pack_bf16x2(__uint_as_float(a[jj + 4]), __uint_as_float(a[jj + 5]));
        u.w = pack_bf16x2(__uint_as_float(a[jj + 6]), __uint_as_float(a[jj + 7]));
        *reinterpret_cast<uint4 *>(tile + tile_off(r, c0 + jj)) = u;
    }
}

// Descriptor high word (1 KiB between 8-row groups, tcgen05 version, 128-byte swizzle) and the
// leading-byte-offset fields of K-major (unused) and MN-major (64-element blocks) operands.
constexpr uint32_t kDescHi = (1024u >> 4) | (1u << 14) | (2u << 29);
constexpr uint32_t kLboK = 1u << 16, kLboMN = (kBlockBytes >> 4) << 16;

// D (+)= A B over K = 16 KS (KS steps of 16), N columns, A and B from shared memory (low
// descriptor words)
template <bool A_MN, bool B_MN, int N = 128, int KS = 8>
__device__ __forceinline__ void mma_ss(uint32_t d_tmem, uint32_t a_lo, uint32_t b_lo, uint32_t accumulate) {
    constexpr uint32_t id = idesc_bf16(128, N, A_MN, B_MN);
#pragma unroll
    for (int kk = 0; kk < KS; ++kk) {
        const uint32_t ka = A_MN ? kk * 128u : (kk >> 2) * (kBlockBytes >> 4) + (kk & 3) * 2u;
        const uint32_t kb = B_MN ? kk * 128u : (kk >> 2) * (kBlockBytes >> 4) + (kk & 3) * 2u;
        umma_bf16(d_tmem, (static_cast<uint64_t>(kDescHi) << 32) | (a_lo + ka),
                  (static_cast<uint64_t>(kDescHi) << 32) | (b_lo + kb), id, kk > 0 ? 1u : accumulate);
    }
}

// D (+)= A B with A (128 x 128 bf16) in TMEM: K elements 32g .. 32g + 31 of a row packed in
// columns a_tmem + 32g .. +15, so K step kk starts at column 32 (kk / 2) + 8 (kk % 2); B MN-major,
// N columns
template <int N = 128>
__device__ __forceinline__ void mma_ts(uint32_t d_tmem, uint32_t a_tmem, uint32_t b_lo, uint32_t accumulate) {
    constexpr uint32_t id = idesc_bf16(128, N, 0, 1);
#pragma unroll
    for (int kk = 0; kk < 8; ++kk)
        umma_bf16_ts(d_tmem, a_tmem + 32u * (kk >> 1) + 8u * (kk & 1),
                     (static_cast<uint64_t>(kDescHi) << 32) | (b_lo + kk * 128u), id, kk > 0 ? 1u : accumulate);
}

template <bool kNarrow>
__global__ void __launch_bounds__(kThreads, 1)
ahla_tc_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
               const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_o, Params p) {
    extern __shared__ __align__(1024) uint8_t smem[];
    Misc *ms = reinterpret_cast<Misc *>(smem + kSmemTiles);
    auto slot = [&](int s) { return smem + s * kTileBytes; };
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const bool issuer = warp == kIssuerWarp;

    if (smem_u32(smem) & 1023u) {  // the tile layout needs 1 KiB alignment
        if (tid == 0) set_error(p.err, 299, smem_u32(smem));
        return;
    }
    if (tid == 0) {
        for (int b = 0; b < kNumBars; ++b) mbar_init(&ms->bar[b], (b == bEpW || b == bEpR) ? kEpiWarps : 1);
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
    uint32_t n_tiles = 0;  // tiles swept by this CTA (barrier parities)
    constexpr int kF = kNarrow ? 64 : 128, kFS = kF / 16;  // head size: N of the products, K steps over it

    if (issuer) {
        if (lane == 0) {
            uint32_t ld_par = 0, ld_pend = 0;
            const uint32_t sb4 = smem_u32(smem) >> 4;
            auto lk = [&](int s) { return sb4 + (uint32_t)s * (kTileBytes >> 4) + kLboK; };
            auto lm = [&](int s) { return sb4 + (uint32_t)s * (kTileBytes >> 4) + kLboMN; };
            auto load_tile = [&](int s, const CUtensorMap *map, int head, int tok0) {
                ld_pend |= 1u << s;
                mbar_arrive_expect_tx(&ms->bar[bLd0 + s], kTileBytes);
                tma_load_3d(slot(s), map, &ms->bar[bLd0 + s], 0, tok0, head);
                tma_load_3d(slot(s) + kBlockBytes, map, &ms->bar[bLd0 + s], 64, tok0, head);
            };
            auto wait_ld = [&](int s) {
                if (!bar_wait(ms, bLd0 + s, (ld_par >> s) & 1u, p)) return false;
                ld_par ^= 1u << s;
                ld_pend &= ~(1u << s);
                return true;
            };
            for (int head = blockIdx.x; head < p.BH && !ms->abort_flag; head += gridDim.x) {
                load_tile(kQ0, &tm_q, head, 0);
                load_tile(kK0, &tm_k, head, 0);
                load_tile(kV, &tm_v, head, 0);
                if (!wait_ld(kQ0) || !wait_ld(kK0)) break;
                tc_fence_after();
                mma_ss<false, false, 128, kFS>(tb + kTA, lk(kQ0), lk(kK0), 0u);  // A = Q K^T
                umma_commit(&ms->bar[bEvA]);
                for (int j = 0; j < p.M; ++j) {
                    const uint32_t tp = n_tiles & 1;
                    const int qs = (j & 1) ? kQ1 : kQ0, ks = (j & 1) ? kK1 : kK0;
                    const int qo = (j & 1) ? kQ0 : kQ1, ko = (j & 1) ? kK0 : kK1;
                    const bool more = j + 1 < p.M;
                    if (more) {
                        // slots qo, ko were last read by the previous tile's products, the last of
                        // them E += K^T R (bEvE)
                        if (j > 0 && !bar_wait(ms, bEvE, tp ^ 1u, p)) break;
                        load_tile(qo, &tm_q, head, (j + 1) * kTile);
                        load_tile(ko, &tm_k, head, (j + 1) * kTile);
                    }
                    if (!bar_wait(ms, bEpW, tp, p) || !wait_ld(kV)) break;  // W and P_p (bf16) ready
                    tc_fence_after();
                    mma_ts<kF>(tb + kTR, tb + kTA, lm(kV), 0u);                // R = W V
                    mma_ss<false, true, kF, kFS>(tb + kTR, lk(qs), lm(kC), 1u);  //   + Q P_p
                    umma_commit(&ms->bar[bEvR]);
                    mma_ss<true, true, kF>(tb + kTP, lm(ks), lm(kV), 1u);  // P += K^T V (under the R epilogue)
                    umma_commit(&ms->bar[bEvV]);
                    if (!bar_wait(ms, bEvV, tp, p)) break;                // V read
                    if (more) load_tile(kV, &tm_v, head, (j + 1) * kTile);
                    if (!bar_wait(ms, bEpR, tp, p)) break;                // R and E_p (bf16) ready
                    tc_fence_after();
                    mma_ts<kF>(tb + kTR, tb + kTA, lm(kR), 0u);                // O = W R
                    mma_ss<false, true, kF, kFS>(tb + kTR, lk(qs), lm(kC), 1u);  //   + Q E_p
                    umma_commit(&ms->bar[bEvO]);
                    mma_ss<true, true, kF>(tb + kTE, lm(ks), lm(kR), 1u);  // E += K^T R (under the O epilogue)
                    umma_commit(&ms->bar[bEvE]);
                    if (more) {  // the next A runs behind them (the products execute in issue order)
                        if (!wait_ld(qo) || !wait_ld(ko)) break;
                        tc_fence_after();
                        mma_ss<false, false, 128, kFS>(tb + kTA, lk(qo), lk(ko), 0u);  // next A = Q K^T
                        umma_commit(&ms->bar[bEvA]);
                    } else if (!bar_wait(ms, bEvE, tp, p)) {  // every product of the head is done
                        break;
                    }
                    ++n_tiles;
                }
            }
            if (ms->abort_flag) {
                // a wait gave up: copies and MMAs in flight finish (bounded) before shared memory
                // and TMEM are released
                for (int s = 0; s <= kV; ++s)
                    if ((ld_pend >> s) & 1u) mbar_wait(&ms->bar[bLd0 + s], (ld_par >> s) & 1u, kBarWaitNs);
                umma_commit(&ms->bar[bTear]);
                mbar_wait(&ms->bar[bTear], 0, kBarWaitNs);
            }
        }
        __syncwarp();
    } else {
        // ============================ epilogue ============================
        const int et = tid, qd = warp & 3, cq = warp >> 2;
        const int r = 32 * qd + lane, c0 = 32 * cq;
        const uint32_t lane_base = (uint32_t)(32 * qd) << 16;
        const bool blk_zero = cq > qd;  // this 32-column block of W lies above the diagonal
        // head size 64: the 64-column results (R, O) live in column quarters 0, 1 and the 64 x 64
        // carries P, E also in lane quadrants 0, 1; the other warps skip them
        const bool fcol = !kNarrow || cq < 2, frow = !kNarrow || qd < 2;
        for (int head = blockIdx.x; head < p.BH; head += gridDim.x) {
            if (n_tiles > 0) {  // the previous head's last E += K^T R is done before E is reset
                bar_wait(ms, bEvE, (n_tiles - 1) & 1u, p);
                tc_fence_after();
            }
            {  // carries start at zero
                uint32_t z[32];
#pragma unroll
                for (int i = 0; i < 32; ++i) z[i] = 0u;
                tmem_st32(tb + lane_base + kTP + c0, z);
                tmem_st32(tb + lane_base + kTE + c0, z);
                tmem_st_wait();
            }
            for (int j = 0; j < p.M; ++j) {
                const uint32_t tp = n_tiles & 1;
                // (a) W = L . A -> packed bf16 over this thread's own A columns; P_p -> bf16 (slot C)
                bar_wait(ms, bEvA, tp, p);
                tc_fence_after();
                {
                    uint32_t h[16];
                    if (blk_zero) {
#pragma unroll
                        for (int i = 0; i < 16; ++i) h[i] = 0u;
                    } else {
                        uint32_t a[32];
                        tmem_ld32(tb + lane_base + kTA + c0, a);
                        tmem_ld_wait();
                        if (cq < qd) {  // wholly below the diagonal: no compares
#pragma unroll
                            for (int i = 0; i < 16; ++i) h[i] = pack_bf16x2(__uint_as_float(a[2 * i]), __uint_as_float(a[2 * i + 1]));
                        } else {
#pragma unroll
                            for (int i = 0; i < 16; ++i) {
                                const float x0 = (c0 + 2 * i <= r) ? __uint_as_float(a[2 * i]) : 0.f;
                                const float x1 = (c0 + 2 * i + 1 <= r) ? __uint_as_float(a[2 * i + 1]) : 0.f;
                                h[i] = pack_bf16x2(x0, x1);
                            }
                        }
                    }
                    tmem_st16(tb + lane_base + kTA + c0, h);
                }
                if (et == 0) tma_store_wait_read();  // the previous output has left slot C
                epi_sync();
                if (fcol && frow) {
                    uint32_t a[32];
                    tmem_ld32(tb + lane_base + kTP + c0, a);
                    tmem_ld_wait();
                    store_row32(slot(kC), r, c0, a);  // row = feature, columns = dv
                }
                tmem_st_wait();
                fence_async_smem();
                epi_arrive(ms, bEpW);
                // (b) R -> bf16 (slot R); E_p -> bf16 (slot C, P_p read by now)
                bar_wait(ms, bEvR, tp, p);
                tc_fence_after();
                if (fcol) {
                    uint32_t a[32];
                    tmem_ld32(tb + lane_base + kTR + c0, a);
                    tmem_ld_wait();
                    store_row32(slot(kR), r, c0, a);  // row = token
                    if (frow) {
                        tmem_ld32(tb + lane_base + kTE + c0, a);
                        tmem_ld_wait();
                        store_row32(slot(kC), r, c0, a);  // row = feature
                    }
                }
                fence_async_smem();
                epi_arrive(ms, bEpR);
                // (c) O -> bf16 (slot C, E_p read by now) -> TMA store
                bar_wait(ms, bEvO, tp, p);
                tc_fence_after();
                if (fcol) {
                    uint32_t a[32];
                    tmem_ld32(tb + lane_base + kTR + c0, a);
                    tmem_ld_wait();
                    store_row32(slot(kC), r, c0, a);
                }
                fence_async_smem();
                epi_sync();
                if (et == 0) {
                    tma_store_3d(&tm_o, slot(kC), 0, j * kTile, head);
                    if (p.out_blocks > 1) tma_store_3d(&tm_o, slot(kC) + kBlockBytes, 64, j * kTile, head);
                    tma_store_commit();
                }
                ++n_tiles;
            }
        }
        if (et == 0) tma_store_wait_all();
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

// [BH][n][inner] bf16 (inner = 64 or 128), boxes of 64 columns x 128 tokens, 128-byte swizzle, zero
// fill out of range (the box at column 64 of a 64-wide tensor is all fill)
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

}  // namespace

bool ahla_tc_applicable(const Fwd2 &p) {
    if (getenv("HLA_DISABLE_FUSED")) return false;
    if (p.dt != HLA_BF16 || (p.d != 64 && p.d != 128) || (p.dv != 64 && p.dv != 128)) return false;
    if (p.normalized || p.state_in || p.state_out || p.n <= 0 || p.BH <= 0) return false;
    if (p.ws_bytes < kWsHeaderBytes) return false;
    int dev = 0, major = 0, minor = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return false;
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    return major == 10 && minor == 3 && encode_fn() != nullptr;
}

cudaError_t ahla_tc_forward(const Fwd2 &p, cudaStream_t stream) {
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
    kp.out_blocks = p.dv / 64;
    kp.err = reinterpret_cast<WsHeader *>(p.ws);
    const int grid = p.BH < sms ? p.BH : sms;
    auto launch = [&](auto kern) -> cudaError_t {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
        if (e) return e;
        kern<<<grid, kThreads, kSmemBytes, stream>>>(mq, mk, mv, mo, kp);
        return cudaGetLastError();
    };
    return (p.d == 64 && p.dv == 64) ? launch(ahla_tc_kernel<true>) : launch(ahla_tc_kernel<false>);
}

}  // namespace hla
