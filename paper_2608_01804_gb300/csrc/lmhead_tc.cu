// Vocabulary-tiled lm-head on the 5th-generation tensor cores (tcgen05):
// logits = hidden . W^T are produced 128 x 256 tiles at a time into tensor
// memory and consumed there, so the [N x V] logits never exist in HBM.
//
// One persistent, warp-specialised GEMM kernel (bf16 operands, each either
// K-major or MN-major in global memory, fp32 accumulation) with four
// epilogues:
//   EPI_LSE      online (max, sum of 2^((z - max) c1)) per row over a range
//                of vocabulary tiles, plus the target logit: the log-sum-exp
//                partials of the token log-probs;
//   EPI_DLOGITS  recomputed logits tile -> dlogits = coef (1[v = y] -
//                softmax) in bf16, into a transient token-chunk buffer;
//   EPI_STORE    the accumulator as bf16 (dhidden = dlogits . W, W read
//                MN-major in place);
//   EPI_ACC_F32  the accumulator added into (or stored to) an fp32 matrix:
//                the weight gradient dW = dlogits^T . hidden, summed over
//                token chunks, with both operands read MN-major.
// Warp 0 issues TMA tile loads (128-byte swizzle) into a 4-stage shared-memory
// ring; one thread of warp 1 issues tcgen05.mma (M = 128, N = 256, K = 16)
// into one of two 256-column fp32 accumulators in tensor memory; warps 2-5
// read the other accumulator with tcgen05.ld (one row per thread).
#include "../../include/leap.h"
#include "leap_common.cuh"
#include "leap_internal.h"
#include "loss_math.cuh"

#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <math.h>
#include <mutex>

namespace leap {
namespace {

constexpr int BM = 128;   // tokens per tile (tensor-memory lanes)
constexpr int BN = 256;   // columns per tile (accumulator columns)
constexpr int BK = 64;      // K per stage: one 128-byte swizzle row of bf16
constexpr int STAGES = 4;   // 4 x 48 KB; 3 stages measured 9 % slower, K = 32 stages (64-byte swizzle) slower still
// K-major tiles: rows of BK bf16 (128 bytes, the swizzle span), 8-row swizzle
// atoms KROW_ATOM bytes apart; descriptor swizzle code 2 = 128-byte.
constexpr uint32_t KROW_ATOM = 8 * BK * 2;
constexpr uint64_t KSWZ_CODE = 2;
constexpr uint32_t A_TILE = BM * BK * 2;
constexpr uint32_t B_TILE = BN * BK * 2;
constexpr uint32_t STAGE_BYTES = A_TILE + B_TILE;
constexpr uint32_t TMEM_COLS = 2 * BN;  // two accumulators
constexpr int GEMM_THREADS = 192;       // warp 0 TMA, warp 1 MMA, warps 2-5 epilogue
constexpr size_t GEMM_DYN_SMEM = (size_t)STAGES * STAGE_BYTES + 1024;
constexpr int LSE_TILES_PER_UNIT = 8;   // 2,048 vocabulary columns per LSE work unit
// Token tiles per group of the grouped tile order (measured; see the tile
// order note at unit_coords):
constexpr int kLseGroupM = 16;  // forward: the 152 CTAs in flight cover 16 hidden tiles x ~10 vocabulary units
constexpr int kDlGroupM = 32;   // dlogits chunk: 32 token tiles x ~5 vocabulary tiles in flight
constexpr int kStGroupM = 8;    // dhidden: 8 token tiles x 20 hidden tiles (the whole N) in flight
constexpr int64_t DLOGITS_CHUNK_ROWS = 16384;

// Instruction descriptor of tcgen05.mma kind::f16: D fp32 (bits 4-5 = 1),
// A and B bf16 (bits 7-9 = 1, 10-12 = 1), A / B major-ness at bits 15 / 16
// (0 = K-major, 1 = MN-major), N >> 3 at bits 17-22, M >> 4 at bits 24-28.
template <bool AMN, bool BMN>
__host__ __device__ constexpr uint32_t idesc() {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((AMN ? 1u : 0u) << 15) | ((BMN ? 1u : 0u) << 16) |
           ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);
}
// An MN-major operand tile is loaded as 64-element (128-byte) wide column
// blocks of BK rows each; the blocks sit MN_BLOCK bytes apart in the stage.
constexpr uint32_t MN_BLOCK = BK * 128;

enum { EPI_STORE = 0, EPI_LSE = 1, EPI_DLOGITS = 2, EPI_ACC_F32 = 3 };

struct GemmArgs {
    int32_t M, N, K;
    int32_t tiles_m, tiles_n, tiles_per_unit, units_n;
    int64_t num_units;
    uint16_t* out;            // STORE / DLOGITS: bf16 [M x ldo]
    float* outf;              // ACC_F32: fp32 [M x ldo]
    int64_t ldo;
    int32_t accumulate;       // ACC_F32: add into outf (else overwrite)
    int32_t n_fastest;        // unit order: 0 = consecutive units walk M, 1 = walk N
    int32_t group_m;          // with n_fastest == 0 and > 0: M tiles walked in groups of group_m
    float2* part;             // LSE: (max, sum) per (unit column, row) at [nu * M + row]
    float* zy;                // LSE: target logit per row
    const int32_t* ids;       // LSE / DLOGITS: target id per row
    const float* rowK;        // DLOGITS: log2 of the softmax denominator per row
    const float* rowcoef;     // DLOGITS: dlogits scale per row (0 = zeros)
    float c1;                 // inv_temp * log2(e)
    unsigned int* status;
};

struct TcSmem {
    uint64_t full[STAGES];
    uint64_t empty[STAGES];
    uint64_t acc_full[2];
    uint64_t acc_empty[2];
    uint32_t tmem_base;
    int abort_flag;
};

// ---- tcgen05 / TMA primitives (inline PTX) ----
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

__device__ __forceinline__ void tmem_alloc(uint32_t* dst_smem, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(dst_smem)),
                 "r"(ncols)
                 : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

// D[tmem] (+)= A[smem] . B[smem]^T, issued by one thread.
__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                          uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
        : "memory");
}
// Arrive on `bar` once every tcgen05.mma issued so far by this thread is done.
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_addr(bar))
                 : "memory");
}

__device__ __forceinline__ void tma_load_2d(uint32_t smem_dst, const CUtensorMap* tm, int32_t x, int32_t y,
                                            uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
            smem_dst),
        "l"(tm), "r"(x), "r"(y), "r"(smem_addr(bar))
        : "memory");
}

// Shared-memory matrix descriptor of a K-major tile written by TMA with the
// 128-byte swizzle: rows of BK * 2 = 128 bytes, 8-row groups KROW_ATOM = 1024
// bytes apart.  Fields: start address >> 4 (bits 0-13), leading byte offset
// >> 4 (16-29, unused for this layout), stride byte offset >> 4 (32-45),
// descriptor version 1 (bit 46), swizzle mode (bits 61-63).
__device__ __forceinline__ uint64_t kmajor_desc(uint32_t saddr) {
    return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)1 << 16) | ((uint64_t)(KROW_ATOM >> 4) << 32) |
           ((uint64_t)1 << 46) | (KSWZ_CODE << 61);
}
// The same for an MN-major tile: each 128-byte row holds 64 consecutive M (or
// N) elements of one k, 8-row (8 k) groups are 1024 bytes apart (stride byte
// offset) and the 64-element column blocks MN_BLOCK bytes apart (leading
// byte offset).
__device__ __forceinline__ uint64_t sw128_mn_desc(uint32_t saddr) {
    return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)(MN_BLOCK >> 4) << 16) |
           ((uint64_t)(1024 >> 4) << 32) | ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

// Work unit u -> (vocabulary-unit / N-tile group nu, M tile mb).  Grouped
// order: group_m consecutive M tiles are walked M-fastest across all N units
// before the next group, so the CTAs in flight hold few distinct A tiles
// (reused from L2 across their N tiles) and few distinct B tiles.
__device__ __forceinline__ void unit_coords(const GemmArgs& g, int64_t u, int& nu, int& mb) {
    if (g.n_fastest) {
        nu = (int)(u % g.units_n);
        mb = (int)(u / g.units_n);
    } else if (g.group_m > 0) {
        const int64_t per_group = (int64_t)g.group_m * g.units_n;
        const int64_t grp = u / per_group;
        const int m0 = (int)(grp * g.group_m);
        const int gm = min(g.group_m, g.tiles_m - m0);   // the last group may be short
        const int64_t local = u - grp * per_group;
        nu = (int)(local / gm);
        mb = m0 + (int)(local % gm);
    } else {
        nu = (int)(u / g.tiles_m);
        mb = (int)(u % g.tiles_m);
    }
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
    uint32_t r[32];
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
                 : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
}

__device__ __forceinline__ void store_bf16_8(uint16_t* dst, const float* v, int nvalid) {
    uint32_t w[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) w[q] = pack_bf16x2(v[2 * q], v[2 * q + 1]);
    if (nvalid >= 8) {
        st_stream(reinterpret_cast<uint4*>(dst), make_uint4(w[0], w[1], w[2], w[3]));
    } else {
        for (int j = 0; j < nvalid; ++j) dst[j] = (uint16_t)((j & 1) ? (w[j >> 1] >> 16) : (w[j >> 1] & 0xffffu));
    }
}

template <int EPI, bool AMN, bool BMN>
__global__ void __launch_bounds__(GEMM_THREADS, 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, GemmArgs g) {
    extern __shared__ uint8_t dsmem[];
    __shared__ __align__(8) TcSmem sm;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t stage0 = (smem_addr(dsmem) + 1023u) & ~1023u;  // 1024-byte aligned for the swizzle
    const int nk = (g.K + BK - 1) / BK;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&sm.full[s], 1);
            mbar_init(&sm.empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&sm.acc_full[b], 1);
            mbar_init(&sm.acc_empty[b], 4 * 32);
        }
        sm.abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(&sm.tmem_base, TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sm.tmem_base;

    if (warp == 0) {
        // ---------------- TMA producer ----------------
        if (lane == 0) {
            uint32_t it = 0;
            for (int64_t u = blockIdx.x; u < g.num_units; u += gridDim.x) {
                int nu, mb;
                unit_coords(g, u, nu, mb);
                const int t1 = min(g.tiles_n, (nu + 1) * g.tiles_per_unit);
                for (int nt = nu * g.tiles_per_unit; nt < t1; ++nt) {
                    for (int kb = 0; kb < nk; ++kb, ++it) {
                        const uint32_t s = it % STAGES;
                        if (it >= STAGES) mbar_wait(&sm.empty[s], ((it / STAGES) - 1) & 1u, g.status, &sm.abort_flag);
                        mbar_arrive_expect_tx(&sm.full[s], STAGE_BYTES);
                        const uint32_t a_dst = stage0 + s * STAGE_BYTES, b_dst = a_dst + A_TILE;
                        if (AMN) {
#pragma unroll
                            for (int j = 0; j < BM / 64; ++j)
                                tma_load_2d(a_dst + j * MN_BLOCK, &tmA, mb * BM + 64 * j, kb * BK, &sm.full[s]);
                        } else {
                            tma_load_2d(a_dst, &tmA, kb * BK, mb * BM, &sm.full[s]);
                        }
                        if (BMN) {
#pragma unroll
                            for (int j = 0; j < BN / 64; ++j)
                                tma_load_2d(b_dst + j * MN_BLOCK, &tmB, nt * BN + 64 * j, kb * BK, &sm.full[s]);
                        } else {
                            tma_load_2d(b_dst, &tmB, kb * BK, nt * BN, &sm.full[s]);
                        }
                    }
                }
            }
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        if (lane == 0) {
            uint32_t it = 0, tc = 0;
            for (int64_t u = blockIdx.x; u < g.num_units; u += gridDim.x) {
                int nu, mb;
                unit_coords(g, u, nu, mb);
                const int t1 = min(g.tiles_n, (nu + 1) * g.tiles_per_unit);
                for (int nt = nu * g.tiles_per_unit; nt < t1; ++nt, ++tc) {
                    const uint32_t ab = tc & 1u;
                    if (tc >= 2) mbar_wait(&sm.acc_empty[ab], ((tc >> 1) - 1) & 1u, g.status, &sm.abort_flag);
                    tc_fence_after();
                    const uint32_t d = tmem + ab * BN;
                    for (int kb = 0; kb < nk; ++kb, ++it) {
                        const uint32_t s = it % STAGES;
                        mbar_wait(&sm.full[s], (it / STAGES) & 1u, g.status, &sm.abort_flag);
                        tc_fence_after();
                        const uint32_t a0 = stage0 + s * STAGE_BYTES, b0 = a0 + A_TILE;
#pragma unroll
                        for (int k = 0; k < BK / 16; ++k) {
                            // K = 16 per MMA: 32 bytes along a K-major row, or
                            // 16 rows (two 1024-byte groups) of an MN-major tile.
                            const uint64_t da = AMN ? sw128_mn_desc(a0 + k * 2048) : kmajor_desc(a0 + k * 32);
                            const uint64_t db = BMN ? sw128_mn_desc(b0 + k * 2048) : kmajor_desc(b0 + k * 32);
                            umma_bf16(d, da, db, idesc<AMN, BMN>(), (kb | k) != 0);
                        }
                        umma_commit(&sm.empty[s]);  // the stage is free once these MMAs are done
                    }
                    umma_commit(&sm.acc_full[ab]);
                }
            }
        }
    } else {
        // ---------------- epilogue: one accumulator row per thread ----------------
        const int ew = warp & 3;  // tensor-memory lane quarter this warp may access
        const int rl = ew * 32 + lane;
        uint32_t tc = 0;
        for (int64_t u = blockIdx.x; u < g.num_units; u += gridDim.x) {
            int nu, mb;
            unit_coords(g, u, nu, mb);
            const int t1 = min(g.tiles_n, (nu + 1) * g.tiles_per_unit);
            const int64_t row = (int64_t)mb * BM + rl;
            const bool valid = row < g.M;
            int y = -1;
            float rk = 0.f, coef = 0.f;
            if (valid && (EPI == EPI_LSE || EPI == EPI_DLOGITS)) y = g.ids[row];
            if (valid && EPI == EPI_DLOGITS) {
                rk = g.rowK[row];
                coef = g.rowcoef[row];
            }
            float m = -INFINITY, ssum = 0.f, zyv = 0.f;
            bool hasy = false;
            for (int nt = nu * g.tiles_per_unit; nt < t1; ++nt, ++tc) {
                const uint32_t ab = tc & 1u;
                mbar_wait(&sm.acc_full[ab], (tc >> 1) & 1u, g.status, &sm.abort_flag);
                tc_fence_after();
                const uint32_t taddr = tmem + ((uint32_t)(ew * 32) << 16) + ab * BN;
#pragma unroll 1
                for (int c0 = 0; c0 < BN; c0 += 32) {
                    float v[32];
                    tmem_ld32(taddr + c0, v);
                    const int col0 = nt * BN + c0;
                    if (EPI == EPI_LSE) {
                        float cmax = -INFINITY;
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            if (col0 + j < g.N) cmax = fmaxf(cmax, v[j]);
                        if (cmax > m) {
                            if (ssum != 0.f) ssum *= ex2((m - cmax) * g.c1);
                            m = cmax;
                        }
                        if (cmax != -INFINITY) {
                            const float mc = m * g.c1;
                            float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                            for (int j = 0; j < 32; ++j)
                                if (col0 + j < g.N) acc[j & 3] += ex2(fmaf(v[j], g.c1, -mc));
                            ssum += (acc[0] + acc[1]) + (acc[2] + acc[3]);
                        }
                        if (y >= col0 && y < col0 + 32) {
#pragma unroll
                            for (int j = 0; j < 32; ++j)
                                if (y == col0 + j) zyv = v[j];
                            hasy = true;
                        }
                    } else if (EPI == EPI_ACC_F32) {
                        if (valid) {
                            float* dst = g.outf + row * g.ldo + col0;
                            if (col0 + 32 <= g.N) {
#pragma unroll
                                for (int q = 0; q < 8; ++q) {
                                    float4 o = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
                                    float4* p4 = reinterpret_cast<float4*>(dst + 4 * q);
                                    if (g.accumulate) {
                                        const float4 c = *p4;
                                        o.x += c.x;
                                        o.y += c.y;
                                        o.z += c.z;
                                        o.w += c.w;
                                    }
                                    *p4 = o;
                                }
                            } else {
#pragma unroll
                                for (int j = 0; j < 32; ++j)
                                    if (col0 + j < g.N) dst[j] = g.accumulate ? dst[j] + v[j] : v[j];
                            }
                        }
                    } else if (valid) {
                        float o[32];
                        if (EPI == EPI_DLOGITS) {
#pragma unroll
                            for (int j = 0; j < 32; ++j) {
                                o[j] = (coef == 0.f) ? 0.f : -coef * ex2(fmaf(v[j], g.c1, -rk));
                                if (col0 + j == y) o[j] += coef;
                            }
                        } else {
#pragma unroll
                            for (int j = 0; j < 32; ++j) o[j] = v[j];
                        }
                        uint16_t* dst = g.out + row * g.ldo + col0;
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            const int nv = g.N - (col0 + 8 * q);
                            if (nv > 0) store_bf16_8(dst + 8 * q, o + 8 * q, nv);
                        }
                    }
                }
                tc_fence_before();
                mbar_arrive(&sm.acc_empty[ab]);
            }
            if (EPI == EPI_LSE && valid) {
                g.part[(int64_t)nu * g.M + row] = make_float2(m, ssum);
                if (hasy) g.zy[row] = zyv;
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, TMEM_COLS);
    }
}

// Per row: merge the (max, sum) partials, then the clipped surrogate (Eq. 3)
// and the per-row coefficients of the backward.
__global__ void __launch_bounds__(256) lmhead_combine_kernel(RowArgs a, const float2* part, const float* zy,
                                                             int32_t units_n, float* rowK, float* rowcoef) {
    const int64_t row = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (row >= a.N) return;
    const float wk = a.w[row];
    const int id = a.ids[row];
    const bool bad = (wk != 0.f) && (id < 0 || id >= a.V);
    const float c1 = a.inv_temp * kLog2e;
    if (wk == 0.f || bad) {
        write_masked_outputs(a, row);
        if (bad) flag_status(a.status, LEAP_DEV_BAD_ID);
        rowK[row] = 0.f;
        rowcoef[row] = 0.f;
        return;
    }
    float m = -INFINITY, s = 0.f;
    for (int nu = 0; nu < units_n; ++nu) {
        const float2 p = part[(int64_t)nu * a.N + row];
        lse_merge(m, s, p.x, p.y, c1);
    }
    const TokenLoss r = token_loss(a, m, s, zy[row], a.old_logp[row], a.adv[row], wk);
    write_row_outputs(a, row, r, wk);
    rowK[row] = fmaf(m, c1, log2f(s));
    rowcoef[row] = a.grad_scale * r.g * a.inv_temp;
}

// ---- host side ----
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static std::once_flag once;
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

// 2-D bf16 tensor map: `inner` contiguous elements per row, `outer` rows of
// `row_bytes`, box inner 64 (128 bytes, the swizzle span) x box_outer rows.
bool make_tmap_box(CUtensorMap* tm, const void* base, uint64_t inner, uint64_t outer, uint64_t row_bytes,
                   uint32_t box_inner, uint32_t box_outer, CUtensorMapSwizzle swz) {
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {inner, outer};
    cuuint64_t strides[1] = {row_bytes};
    cuuint32_t box[2] = {box_inner, box_outer};
    cuuint32_t es[2] = {1, 1};
    return fn(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
              CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}
// A K-major operand: `inner` = K contiguous, boxes of BK x box_outer rows.
bool make_tmap(CUtensorMap* tm, const void* base, uint64_t inner, uint64_t outer, uint64_t row_bytes,
               uint32_t box_outer) {
    return make_tmap_box(tm, base, inner, outer, row_bytes, BK, box_outer, CU_TENSOR_MAP_SWIZZLE_128B);
}
// An MN-major operand: `inner` = M (or N) contiguous, boxes of 64 x BK rows (128-byte swizzle).
bool make_tmap_mn(CUtensorMap* tm, const void* base, uint64_t inner, uint64_t outer, uint64_t row_bytes) {
    return make_tmap_box(tm, base, inner, outer, row_bytes, 64, BK, CU_TENSOR_MAP_SWIZZLE_128B);
}

// Tensor maps: a K-major operand [rows x K] is read in boxes of BK x BM (or
// BN) rows; an MN-major operand [K x rows] in boxes of 64 x BK.
template <int EPI, bool AMN = false, bool BMN = false>
cudaError_t launch_gemm(const CUtensorMap& tmA, const CUtensorMap& tmB, GemmArgs g, cudaStream_t s) {
    static std::once_flag once;
    static cudaError_t attr_err = cudaSuccess;
    std::call_once(once, [] {
        attr_err = cudaFuncSetAttribute(tc_gemm_kernel<EPI, AMN, BMN>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                        (int)GEMM_DYN_SMEM);
    });
    if (attr_err != cudaSuccess) return attr_err;
    g.tiles_m = (g.M + BM - 1) / BM;
    g.tiles_n = (g.N + BN - 1) / BN;
    if (EPI != EPI_LSE) g.tiles_per_unit = 1;
    g.units_n = (g.tiles_n + g.tiles_per_unit - 1) / g.tiles_per_unit;
    g.num_units = (int64_t)g.tiles_m * g.units_n;
    if (g.num_units == 0) return cudaSuccess;
    const int64_t grid = std::min<int64_t>(g.num_units, device_sm_count());
    tc_gemm_kernel<EPI, AMN, BMN><<<(unsigned)grid, GEMM_THREADS, GEMM_DYN_SMEM, s>>>(tmA, tmB, g);
    return cudaGetLastError();
}

size_t al256(size_t b) { return (b + 255) & ~size_t(255); }

struct LmheadWorkspace {
    float2* part;
    float* zy;
    float* rowK;
    float* rowcoef;
    void* loss_ws;
    uint16_t* DL;
    int64_t chunk;
    size_t bytes;
};

LmheadWorkspace lmhead_layout(void* base, int64_t N, int32_t H, int32_t V, bool with_dhidden, bool with_dW) {
    LmheadWorkspace w = {};
    const int64_t tiles_n = ((int64_t)V + BN - 1) / BN;
    const int64_t units_n = (tiles_n + LSE_TILES_PER_UNIT - 1) / LSE_TILES_PER_UNIT;
    const int64_t ldv = ((int64_t)V + 7) & ~int64_t(7);
    char* p = static_cast<char*>(base);
    size_t off = 0;
    auto take = [&](size_t bytes) {
        char* q = p ? p + off : nullptr;
        off += al256(bytes);
        return q;
    };
    w.part = reinterpret_cast<float2*>(take(units_n * N * sizeof(float2)));
    w.zy = reinterpret_cast<float*>(take(N * sizeof(float)));
    w.rowK = reinterpret_cast<float*>(take(N * sizeof(float)));
    w.rowcoef = reinterpret_cast<float*>(take(N * sizeof(float)));
    w.loss_ws = take(loss_workspace_bytes(N));
    w.chunk = std::min<int64_t>(N, DLOGITS_CHUNK_ROWS);
    if (with_dhidden || with_dW) w.DL = reinterpret_cast<uint16_t*>(take((size_t)w.chunk * ldv * 2));
    w.bytes = off;
    return w;
}

bool al16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

// ---- entry points used by leap_api-style validation below ----
}  // namespace leap

using namespace leap;

extern "C" leap_status_t leap_gemm_bf16_nt(const uint16_t* A, int64_t lda, const uint16_t* B, int64_t ldb,
                                           uint16_t* C, int64_t ldc, int32_t M, int32_t N, int32_t K, void* stream) {
    if (M < 0 || N < 0 || K < 1) return LEAP_ERR_INVALID_ARG;
    if (M == 0 || N == 0) return LEAP_OK;
    if (!A || !B || !C || !al16(A) || !al16(B) || !al16(C)) return LEAP_ERR_INVALID_ARG;
    if (lda < K || ldb < K || ldc < N || (lda & 7) || (ldb & 7) || (ldc & 7)) return LEAP_ERR_INVALID_ARG;
    CUtensorMap ta, tb;
    if (!make_tmap(&ta, A, (uint64_t)K, (uint64_t)M, (uint64_t)lda * 2, BM)) return LEAP_ERR_CUDA;
    if (!make_tmap(&tb, B, (uint64_t)K, (uint64_t)N, (uint64_t)ldb * 2, BN)) return LEAP_ERR_CUDA;
    GemmArgs g = {};
    g.M = M;
    g.N = N;
    g.K = K;
    g.tiles_per_unit = 1;
    g.out = C;
    g.ldo = ldc;
    g.group_m = kStGroupM;
    g.status = nullptr;
    const cudaError_t e = launch_gemm<EPI_STORE>(ta, tb, g, static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? LEAP_OK : LEAP_ERR_CUDA;
}

extern "C" leap_status_t leap_gemm_bf16_tn_f32(const uint16_t* A, int64_t lda, const uint16_t* B, int64_t ldb,
                                               float* C, int64_t ldc, int32_t M, int32_t N, int32_t K,
                                               int32_t accumulate, void* stream) {
    if (M < 0 || N < 0 || K < 0) return LEAP_ERR_INVALID_ARG;
    if (M == 0 || N == 0) return LEAP_OK;
    if (!C || !al16(C) || ldc < N || (ldc & 3)) return LEAP_ERR_INVALID_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (K == 0) {   // an empty sum: C = 0 (or unchanged)
        if (accumulate) return LEAP_OK;
        return cudaMemset2DAsync(C, (size_t)ldc * 4, 0, (size_t)N * 4, (size_t)M, s) == cudaSuccess ? LEAP_OK
                                                                                             : LEAP_ERR_CUDA;
    }
    if (!A || !B || !al16(A) || !al16(B)) return LEAP_ERR_INVALID_ARG;
    if (lda < M || ldb < N || (lda & 7) || (ldb & 7)) return LEAP_ERR_INVALID_ARG;
    CUtensorMap ta, tb;
    if (!make_tmap_mn(&ta, A, (uint64_t)M, (uint64_t)K, (uint64_t)lda * 2)) return LEAP_ERR_CUDA;
    if (!make_tmap_mn(&tb, B, (uint64_t)N, (uint64_t)K, (uint64_t)ldb * 2)) return LEAP_ERR_CUDA;
    GemmArgs g = {};
    g.M = M;
    g.N = N;
    g.K = K;
    g.tiles_per_unit = 1;
    g.outf = C;
    g.ldo = ldc;
    g.accumulate = accumulate != 0;
    g.n_fastest = 1;
    g.status = nullptr;
    return launch_gemm<EPI_ACC_F32, true, true>(ta, tb, g, s) == cudaSuccess ? LEAP_OK : LEAP_ERR_CUDA;
}

extern "C" size_t leap_fused_lmhead_workspace_size(int64_t N, int32_t H, int32_t V, int32_t grads) {
    if (N < 0 || H < 1 || V < 1) return 0;
    return lmhead_layout(nullptr, N, H, V, (grads & LEAP_LMHEAD_DHIDDEN) != 0, (grads & LEAP_LMHEAD_DW) != 0).bytes;
}

extern "C" leap_status_t leap_fused_lmhead_logprobs(const leap_loss_params_t* p, const uint16_t* hidden,
                                                    const uint16_t* W, int64_t N, int32_t H, int32_t V,
                                                    const int32_t* ids, const float* old_logp, const float* adv,
                                                    const float* w, float* loss, float* logp, float* lse, float* ell,
                                                    uint16_t* dhidden, float* dW, void* workspace, size_t ws_bytes,
                                                    leap_loss_stats_t* stats, void* stream) {
    if (!p || !isfinite(p->eps_low) || !isfinite(p->eps_high) || p->eps_low < 0.f || p->eps_high < 0.f)
        return LEAP_ERR_INVALID_ARG;
    if (!isfinite(p->inv_temp) || !(p->inv_temp > 0.f) || !isfinite(p->grad_scale)) return LEAP_ERR_INVALID_ARG;
    if (p->flags & ~LEAP_LOSS_ACCUMULATE) return LEAP_ERR_INVALID_ARG;
    if (N < 0 || N > (int64_t)0x7fffffff || H < 1 || V < 1 || (H & 7) != 0 || !loss) return LEAP_ERR_INVALID_ARG;
    if (N > 0 && (!hidden || !W || !ids || !old_logp || !adv || !w || !al16(hidden) || !al16(W)))
        return LEAP_ERR_INVALID_ARG;
    if ((dhidden && !al16(dhidden)) || (dW && !al16(dW))) return LEAP_ERR_INVALID_ARG;
    if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return LEAP_ERR_INVALID_ARG;
    const LmheadWorkspace L = lmhead_layout(workspace, N, H, V, dhidden != nullptr, dW != nullptr);
    if (ws_bytes < L.bytes) return LEAP_ERR_INVALID_ARG;
    unsigned int* status = device_status_ptr();
    if (!status) return LEAP_ERR_CUDA;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const float c1 = p->inv_temp * kLog2e;
    const LossWorkspace lws = carve_loss_workspace(L.loss_ws, N);
    cudaError_t e = cudaSuccess;

    RowArgs ra = {};
    ra.ids = ids;
    ra.old_logp = old_logp;
    ra.adv = adv;
    ra.w = w;
    ra.N = N;
    ra.V = V;
    ra.eps_low = p->eps_low;
    ra.eps_high = p->eps_high;
    ra.inv_temp = p->inv_temp;
    ra.grad_scale = p->grad_scale;
    ra.logp = logp;
    ra.lse = lse;
    ra.ell = ell;
    ra.ws_contrib = lws.contrib;
    ra.ws_rho = lws.rho;
    ra.ws_flag = lws.flag;
    ra.status = status;

    CUtensorMap tH, tW;
    if (N > 0) {
        // Forward: log-sum-exp partials per (vocabulary unit, row) + target logit.
        if (!make_tmap(&tH, hidden, (uint64_t)H, (uint64_t)N, (uint64_t)H * 2, BM)) return LEAP_ERR_CUDA;
        if (!make_tmap(&tW, W, (uint64_t)H, (uint64_t)V, (uint64_t)H * 2, BN)) return LEAP_ERR_CUDA;
        GemmArgs g = {};
        g.M = (int32_t)N;
        g.N = V;
        g.K = H;
        g.tiles_per_unit = LSE_TILES_PER_UNIT;
        g.group_m = kLseGroupM;
        g.part = L.part;
        g.zy = L.zy;
        g.ids = ids;
        g.c1 = c1;
        g.status = status;
        e = launch_gemm<EPI_LSE>(tH, tW, g, s);
        if (e != cudaSuccess) return LEAP_ERR_CUDA;
        const int32_t units_n = (int32_t)((((int64_t)V + BN - 1) / BN + LSE_TILES_PER_UNIT - 1) / LSE_TILES_PER_UNIT);
        lmhead_combine_kernel<<<(unsigned)((N + 255) / 256), 256, 0, s>>>(ra, L.part, L.zy, units_n, L.rowK, L.rowcoef);
        if ((e = cudaGetLastError()) != cudaSuccess) return LEAP_ERR_CUDA;
    }
    e = launch_loss_reduce(lws, N, loss, stats, (p->flags & LEAP_LOSS_ACCUMULATE) != 0, s);
    if (e != cudaSuccess) return LEAP_ERR_CUDA;

    const bool acc = (p->flags & LEAP_LOSS_ACCUMULATE) != 0;
    if (dW && N == 0 && !acc) {   // an empty sum over tokens
        if (cudaMemsetAsync(dW, 0, (size_t)V * H * sizeof(float), s) != cudaSuccess) return LEAP_ERR_CUDA;
    }
    if ((dhidden || dW) && N > 0) {
        // Backward through token chunks of transient bf16 dlogits:
        //   dhidden_chunk = DL . W      (K = V; DL K-major, W read in place MN-major)
        //   dW += DL^T . hidden_chunk   (K = chunk tokens; DL and hidden read MN-major)
        const int64_t ldv = ((int64_t)V + 7) & ~int64_t(7);
        CUtensorMap tWt;
        if (dhidden && !make_tmap_mn(&tWt, W, (uint64_t)H, (uint64_t)V, (uint64_t)H * 2)) return LEAP_ERR_CUDA;
        for (int64_t c0 = 0; c0 < N; c0 += L.chunk) {
            const int64_t cr = std::min<int64_t>(L.chunk, N - c0);
            CUtensorMap tHc;
            if (!make_tmap(&tHc, hidden + c0 * H, (uint64_t)H, (uint64_t)cr, (uint64_t)H * 2, BM)) return LEAP_ERR_CUDA;
            GemmArgs g1 = {};
            g1.M = (int32_t)cr;
            g1.N = V;
            g1.K = H;
            g1.out = L.DL;
            g1.ldo = ldv;
            g1.ids = ids + c0;
            g1.rowK = L.rowK + c0;
            g1.rowcoef = L.rowcoef + c0;
            g1.c1 = c1;
            g1.group_m = kDlGroupM;
            g1.status = status;
            if (launch_gemm<EPI_DLOGITS>(tHc, tW, g1, s) != cudaSuccess) return LEAP_ERR_CUDA;
            if (dhidden) {
                CUtensorMap tDL;
                if (!make_tmap(&tDL, L.DL, (uint64_t)V, (uint64_t)cr, (uint64_t)ldv * 2, BM)) return LEAP_ERR_CUDA;
                GemmArgs g2 = {};
                g2.M = (int32_t)cr;
                g2.N = H;
                g2.K = V;
                g2.out = dhidden + c0 * H;
                g2.ldo = H;
                g2.group_m = kStGroupM;
                g2.status = status;
                if (launch_gemm<EPI_STORE, false, true>(tDL, tWt, g2, s) != cudaSuccess) return LEAP_ERR_CUDA;
            }
            if (dW) {
                CUtensorMap tDLt, tHt;
                if (!make_tmap_mn(&tDLt, L.DL, (uint64_t)V, (uint64_t)cr, (uint64_t)ldv * 2)) return LEAP_ERR_CUDA;
                if (!make_tmap_mn(&tHt, hidden + c0 * H, (uint64_t)H, (uint64_t)cr, (uint64_t)H * 2))
                    return LEAP_ERR_CUDA;
                GemmArgs g3 = {};
                g3.M = V;
                g3.N = H;
                g3.K = (int32_t)cr;
                g3.tiles_per_unit = 1;
                g3.outf = dW;
                g3.ldo = H;
                g3.accumulate = (acc || c0 > 0) ? 1 : 0;
                g3.n_fastest = 1;   // CTAs in flight share dlogits column blocks; hidden stays in L2
                g3.status = status;
                if (launch_gemm<EPI_ACC_F32, true, true>(tDLt, tHt, g3, s) != cudaSuccess) return LEAP_ERR_CUDA;
            }
        }
    }
    return LEAP_OK;
}
