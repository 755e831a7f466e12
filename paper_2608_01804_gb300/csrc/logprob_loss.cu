// Token log-probs, the clipped GRPO surrogate (Eq. 3, KL skipped) with its
// deterministic masked reduction, and the dlogits backward.
//
// Kernels
//   row_stream_kernel  one pass over each logits row with an online
//                      (max, sum) -> log-probs, or the loss forward without
//                      dlogits.  2V bytes read per row.
//   (the default fused forward + backward is fused_loss_pipe_kernel in
//   loss_pipe.cu: two passes per row, pipelined across rows on every SM)
//   fused_loss_kernel  forward + backward with the row split over a cluster
//                      of C CTAs that keep their slices in registers and
//                      exchange one (max, sum) pair through distributed
//                      shared memory: each row is read from HBM exactly once
//                      whatever else uses L2 (LEAP_LOSS_SINGLE_READ).
//   (rows of V <= 32,768 take short_row_kernel in short_rows.cu)
//   split_bwd_kernel   dlogits from a saved lse: 2V read + 2V written.
//   reduce kernels     fixed-order fp64 sum of the per-row loss terms.
#include "../../include/leap.h"
#include "leap_common.cuh"
#include "leap_internal.h"
#include "loss_math.cuh"
#include "row_math.cuh"

#include <algorithm>
#include <math.h>
#include <mutex>

namespace leap {
namespace {

// ---------------------------------------------------------------------------
// Streaming single pass.  TPR threads per row (32: several rows per CTA;
// 512: one row per CTA), U vectors of 8 bf16 in flight per thread.
// mode 0: log-probs (every row read); mode 1: loss forward (w == 0 rows skipped).
// ---------------------------------------------------------------------------
template <int TPR, int U, int MINB>
__global__ void __launch_bounds__(512, MINB) row_stream_kernel(RowArgs a, int mode) {
    __shared__ float2 wpart[16];
    const int t = threadIdx.x % TPR;
    const int64_t row = (int64_t)blockIdx.x * (blockDim.x / TPR) + threadIdx.x / TPR;
    if (row >= a.N) return;  // uniform per row group (one row per CTA when TPR = 512)
    const int V = a.V;
    const float wk = (mode == 1) ? a.w[row] : 1.f;
    const int id = a.ids[row];
    const bool bad = (wk != 0.f) && (id < 0 || id >= V);
    if (mode == 1 && (wk == 0.f || bad)) {
        if (t == 0) {
            write_masked_outputs(a, row);
            if (bad) flag_status(a.status, LEAP_DEV_BAD_ID);
        }
        return;
    }
    const uint16_t* zr = a.logits + row * a.ld;
    float zy = 0.f;
    if (t == 0 && !bad) zy = bf16_at(zr + id);

    const uint4* zrow = reinterpret_cast<const uint4*>(zr);
    const int64_t V8 = ((int64_t)V + 7) >> 3;
    const int tailn = V & 7;
    const float c1 = a.inv_temp * kLog2e;
    float m = -INFINITY, s = 0.f;
    for (int64_t v0 = t; v0 < V8; v0 += (int64_t)TPR * U) {
        uint4 x[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int64_t vi = v0 + (int64_t)u * TPR;
            x[u] = (vi < V8) ? ld_stream(zrow + vi) : neg_inf4();
            if (tailn && vi == V8 - 1) mask_tail(x[u], tailn);
        }
        const float bm = tree_max(x);
        if (bm == -INFINITY) continue;
        const float mn = fmaxf(m, bm);
        const float mc = mn * c1;
        const float acc = tree_exp_sum(x, c1, mc);
        s = (s == 0.f) ? acc : fmaf(s, ex2((m - mn) * c1), acc);
        m = mn;
    }
    warp_lse_merge(m, s, c1);
    if (TPR > 32) {
        const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
        if (lane == 0) wpart[warp] = make_float2(m, s);
        __syncthreads();
        if (warp == 0) {
            const float2 p = (lane < TPR / 32) ? wpart[lane] : make_float2(-INFINITY, 0.f);
            m = p.x;
            s = p.y;
            warp_lse_merge(m, s, c1);
        }
    }
    if (t != 0) return;
    if (mode == 0) {
        const float lnS = logf(s);
        if (a.lse) a.lse[row] = fmaf(m, a.inv_temp, lnS);
        if (bad) {
            a.logp[row] = 0.f;
            flag_status(a.status, LEAP_DEV_BAD_ID);
        } else {
            a.logp[row] = a.inv_temp * (zy - m) - lnS;
        }
        return;
    }
    const TokenLoss r = token_loss(a, m, s, zy, a.old_logp[row], a.adv[row], wk);
    write_row_outputs(a, row, r, wk);
}

// ---------------------------------------------------------------------------
// Fused forward + backward, persistent.  A cluster of C CTAs owns one row at a
// time and walks rows cid, cid + ncl, cid + 2 ncl, ...; CTA c owns 16-byte
// vectors [c * per, (c+1) * per) of every row.  Per CTA:
//   * a producer warp reads the weights / ids of the next 32 rows of the
//     sequence at once and, for each live row, issues a 1-D bulk async copy
//     (TMA) of the CTA's slice plus the 16-byte vector holding the target logit
//     into one of STAGES shared-memory stages (mbarrier full/empty pipeline);
//   * T consumer threads copy a ready stage into registers (NV vectors each),
//     release it at once, reduce it to (max, sum of 2^((z - max) log2e)), push
//     that pair to every CTA of the cluster through distributed shared memory
//     with a remote mbarrier arrive, merge the C pairs, and write the dlogits
//     slice straight from the registers they still hold.
// Logits are read from HBM once and dlogits written once.  Masked rows skip
// the copy and write zeros.  Every wait is bounded (LEAP_DEV_TIMEOUT).
// ---------------------------------------------------------------------------
template <int STAGES, int C>
struct FusedSmem {
    uint64_t full[STAGES];
    uint64_t empty[STAGES];
    uint64_t ex[2];          // exchange barriers (C arrivals each), alternating per live row
    float2 slot[2][C];       // (max, sum) of each CTA of the cluster, alternating per live row
    float2 wpart[32];
    float bc[2];
    uint4 yvec[STAGES];      // the 16-byte vector that holds the target logit
    int abort_flag;          // set once a bounded wait of this CTA gave up
};

template <int C, int T, int NV, int STAGES, int MINB>
__global__ void __launch_bounds__(T + 32, MINB) fused_loss_kernel(RowArgs a, int32_t per, int32_t ncl) {
    extern __shared__ __align__(128) uint4 stage_mem[];  // STAGES * per vectors
    __shared__ __align__(16) FusedSmem<STAGES, C> sm;
    const int t = threadIdx.x;
    const uint32_t crank = (C > 1) ? cluster_ctarank() : 0u;
    const int64_t cid = blockIdx.x / C;
    const int V = a.V;
    const int64_t V8 = ((int64_t)V + 7) >> 3;
    const int64_t vbeg = min((int64_t)crank * per, V8);
    const int64_t vend = min(vbeg + per, V8);
    const uint32_t nvec = (uint32_t)(vend - vbeg);
    const int tailn = V & 7;

    if (t == 0) {
#pragma unroll
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&sm.full[s], 1);
            mbar_init(&sm.empty[s], T / 32);
        }
        mbar_init(&sm.ex[0], C);
        mbar_init(&sm.ex[1], C);
        sm.abort_flag = 0;
        fence_mbar_init();
    }
    __syncthreads();
    if (C > 1) {  // every CTA's barriers are initialised before any remote arrive
        cluster_arrive_release();
        cluster_wait_acquire();
    }

    if (t >= T) {
        // ---------------- producer warp ----------------
        const int lane = t - T;
        uint32_t j = 0;
        for (int64_t k0 = 0; cid + k0 * ncl < a.N; k0 += 32) {
            const int64_t row = cid + (k0 + lane) * ncl;
            bool live = false;
            int id = 0;
            if (row < a.N) {
                const float w = a.w[row];
                id = a.ids[row];
                live = (w != 0.f) && id >= 0 && id < V;
            }
            uint32_t mask = __ballot_sync(0xffffffffu, live);
            while (mask) {
                const int b = __ffs(mask) - 1;
                mask &= mask - 1;
                const int idb = __shfl_sync(0xffffffffu, id, b);
                if (lane == 0) {
                    const int64_t r = cid + (k0 + b) * ncl;
                    const uint32_t s = j % STAGES;
                    if (j >= STAGES) mbar_wait(&sm.empty[s], ((j / STAGES) - 1) & 1u, a.status, &sm.abort_flag);
                    mbar_arrive_expect_tx(&sm.full[s], nvec * 16u + 16u);
                    const uint16_t* zr = a.logits + r * a.ld;
                    if (nvec) bulk_g2s(stage_mem + (size_t)s * per, zr + vbeg * 8, nvec * 16u, &sm.full[s]);
                    bulk_g2s(&sm.yvec[s], zr + (idb & ~7), 16u, &sm.full[s]);
                }
                ++j;
            }
        }
        return;
    }

    // ---------------- consumers ----------------
    const int lane = t & 31, warp = t >> 5;
    const float c1 = a.inv_temp * kLog2e;
    uint32_t j = 0;
    float w_next = 0.f;
    int id_next = 0;
    if (cid < a.N) {
        w_next = a.w[cid];
        id_next = a.ids[cid];
    }
    for (int64_t row = cid; row < a.N; row += ncl) {
        const float wk = w_next;
        const int id = id_next;
        if (row + ncl < a.N) {  // next row's scalars, one row ahead
            w_next = a.w[row + ncl];
            id_next = a.ids[row + ncl];
        }
        const bool bad = (wk != 0.f) && (id < 0 || id >= V);
        uint4* drow = reinterpret_cast<uint4*>(a.dlogits + row * a.ld);
        if (wk == 0.f || bad) {  // masked row: same branch in every CTA of the cluster
#pragma unroll
            for (int k = 0; k < NV; ++k) {
                const int64_t vi = vbeg + t + (int64_t)k * T;
                if (vi < vend) store_vec(drow, vi, make_uint4(0, 0, 0, 0), V8, tailn);
            }
            if (crank == 0 && t == 0) {
                write_masked_outputs(a, row);
                if (bad) flag_status(a.status, LEAP_DEV_BAD_ID);
            }
            continue;
        }
        float old = 0.f, A = 0.f;
        if (t == 0) {
            old = a.old_logp[row];
            A = a.adv[row];
        }
        const uint32_t s = j % STAGES;
        mbar_wait(&sm.full[s], (j / STAGES) & 1u, a.status, &sm.abort_flag);
        const uint4* st = stage_mem + (size_t)s * per;
        uint4 x[NV];
#pragma unroll
        for (int k = 0; k < NV; ++k) {
            const uint32_t li = (uint32_t)(t + k * T);
            x[k] = (li < nvec) ? st[li] : neg_inf4();
            if (tailn && vbeg + (int64_t)li == V8 - 1) mask_tail(x[k], tailn);
        }
        float zy = 0.f;
        if (t == 0) zy = bf16_at(reinterpret_cast<const uint16_t*>(&sm.yvec[s]) + (id & 7));
        __syncwarp();
        if (lane == 0) mbar_arrive(&sm.empty[s]);  // this warp is done with the stage

        float m = tree_max(x);
        float ssum = (m != -INFINITY) ? tree_exp_sum(x, c1, m * c1) : 0.f;
        warp_lse_merge(m, ssum, c1);
        if (lane == 0) sm.wpart[warp] = make_float2(m, ssum);
        named_bar_sync(1, T);
        if (warp == 0) {
            const float2 p = (lane < T / 32) ? sm.wpart[lane] : make_float2(-INFINITY, 0.f);
            m = p.x;
            ssum = p.y;
            warp_lse_merge(m, ssum, c1);
            if (C > 1) {
                const uint32_t e = j & 1u;
                if (lane < C) {
                    st_cluster_f32x2(cluster_map(smem_addr(&sm.slot[e][crank]), (uint32_t)lane), m, ssum);
                    mbar_arrive_remote(cluster_map(smem_addr(&sm.ex[e]), (uint32_t)lane));
                }
                mbar_wait_cluster(&sm.ex[e], (j >> 1) & 1u, a.status, &sm.abort_flag);
                const volatile float2* sl = &sm.slot[e][0];
                float2 q = make_float2(-INFINITY, 0.f);
                if (lane < C) {
                    q.x = sl[lane].x;
                    q.y = sl[lane].y;
                }
                m = q.x;
                ssum = q.y;
                warp_lse_merge(m, ssum, c1);
            }
            if (lane == 0) {
                const TokenLoss r = token_loss(a, m, ssum, zy, old, A, wk);
                sm.bc[0] = fmaf(m, c1, log2f(ssum));            // log2 of the softmax denominator
                sm.bc[1] = a.grad_scale * r.g * a.inv_temp;     // dlogits scale
                if (crank == 0) write_row_outputs(a, row, r, wk);
            }
        }
        named_bar_sync(1, T);
        const float K = sm.bc[0], coef = sm.bc[1];
        const int64_t yv = id >> 3;
        const int ylane = id & 7;
#pragma unroll
        for (int k = 0; k < NV; ++k) {
            const int64_t vi = vbeg + t + (int64_t)k * T;
            if (vi < vend) {
                const uint4 d = (coef == 0.f) ? make_uint4(0, 0, 0, 0)
                                              : dlogit8(x[k], c1, K, coef, vi == yv ? ylane : -1);
                store_vec(drow, vi, d, V8, tailn);
            }
        }
        ++j;
    }
}

// ---------------------------------------------------------------------------
// Split backward from the saved lse.  Every thread recomputes the row's scalar
// coefficient from broadcast loads, so no block synchronisation is needed.
// ---------------------------------------------------------------------------
template <int TPR, int U>
__global__ void __launch_bounds__(512) split_bwd_kernel(RowArgs a) {
    const int t = threadIdx.x % TPR;
    const int64_t row = (int64_t)blockIdx.x * (blockDim.x / TPR) + threadIdx.x / TPR;
    if (row >= a.N) return;
    const int V = a.V;
    const int64_t V8 = ((int64_t)V + 7) >> 3;
    const int tailn = V & 7;
    const float wk = a.w[row];
    const int id = a.ids[row];
    const bool bad = (wk != 0.f) && (id < 0 || id >= V);
    uint4* drow = reinterpret_cast<uint4*>(a.dlogits + row * a.ld);
    float coef = 0.f, K = 0.f;
    if (wk != 0.f && !bad) {
        const float lse = a.lse_in[row];
        const float logp = a.inv_temp * bf16_at(a.logits + row * a.ld + id) - lse;
        const float A = a.adv[row];
        const float rho = expf(logp - a.old_logp[row]);
        const bool active = (A >= 0.f) ? (rho <= 1.f + a.eps_high) : (rho >= 1.f - a.eps_low);
        coef = active ? a.grad_scale * (-wk * A * rho) * a.inv_temp : 0.f;
        K = lse * kLog2e;
    }
    if (bad && t == 0) flag_status(a.status, LEAP_DEV_BAD_ID);
    const uint4* zrow = reinterpret_cast<const uint4*>(a.logits + row * a.ld);
    const float c1 = a.inv_temp * kLog2e;
    const int64_t yv = bad ? -1 : (id >> 3);
    const int ylane = id & 7;
    for (int64_t v0 = t; v0 < V8; v0 += (int64_t)TPR * U) {
        if (coef == 0.f) {
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int64_t vi = v0 + (int64_t)u * TPR;
                if (vi < V8) store_vec(drow, vi, make_uint4(0, 0, 0, 0), V8, tailn);
            }
            continue;
        }
        uint4 x[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int64_t vi = v0 + (int64_t)u * TPR;
            x[u] = (vi < V8) ? ld_stream(zrow + vi) : neg_inf4();
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int64_t vi = v0 + (int64_t)u * TPR;
            if (vi < V8) store_vec(drow, vi, dlogit8(x[u], c1, K, coef, vi == yv ? ylane : -1), V8, tailn);
        }
    }
}

// ---------------------------------------------------------------------------
// Deterministic reduction: block b sums rows [b R, (b+1) R) in a fixed order,
// then one block sums the block partials in a fixed order.
// ---------------------------------------------------------------------------
constexpr int kRedThreads = 256;

// The four sums of the loss reduction, over a block in a fixed order: a
// shuffle tree within each warp, then thread 0 adds the warps' sums in warp
// order (one block barrier).  The result is valid in thread 0.
struct LossSums {
    double loss, rho;
    long long live, clip;
};
__device__ __forceinline__ LossSums block_sums_fixed(LossSums v) {
    __shared__ LossSums sh[kRedThreads / 32];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        v.loss += __shfl_down_sync(0xffffffffu, v.loss, o);
        v.rho += __shfl_down_sync(0xffffffffu, v.rho, o);
        v.live += __shfl_down_sync(0xffffffffu, v.live, o);
        v.clip += __shfl_down_sync(0xffffffffu, v.clip, o);
    }
    if ((threadIdx.x & 31) == 0) sh[threadIdx.x >> 5] = v;
    __syncthreads();
    LossSums t = {0.0, 0.0, 0, 0};
    if (threadIdx.x == 0) {
#pragma unroll
        for (int w = 0; w < kRedThreads / 32; ++w) {
            t.loss += sh[w].loss;
            t.rho += sh[w].rho;
            t.live += sh[w].live;
            t.clip += sh[w].clip;
        }
    }
    return t;
}

// Partial sums of kReduceRowsPerBlock rows per block (2 per thread), so
// that the dependent fp64 additions per thread stay few and the partial
// blocks spread over the SMs.
__global__ void __launch_bounds__(kRedThreads) reduce_partial_kernel(LossWorkspace ws, int64_t N) {
    const int64_t lo = (int64_t)blockIdx.x * kReduceRowsPerBlock;
    const int64_t hi = min(N, lo + kReduceRowsPerBlock);
    LossSums v = {0.0, 0.0, 0, 0};
    for (int64_t i = lo + threadIdx.x; i < hi; i += kRedThreads) {
        v.loss += ws.contrib[i];
        v.rho += (double)ws.rho[i];
        const uint8_t f = ws.flag[i];
        v.live += (f & 1u);
        v.clip += (f >> 1) & 1u;
    }
    const LossSums t = block_sums_fixed(v);
    if (threadIdx.x == 0) {
        ws.part_loss[blockIdx.x] = t.loss;
        ws.part_rho[blockIdx.x] = t.rho;
        ws.part_live[blockIdx.x] = t.live;
        ws.part_clip[blockIdx.x] = t.clip;
    }
}

__global__ void __launch_bounds__(kRedThreads) reduce_final_kernel(LossWorkspace ws, float* loss,
                                                                    leap_loss_stats_t* stats, int accumulate) {
    LossSums v = {0.0, 0.0, 0, 0};
    for (int64_t b = threadIdx.x; b < ws.nblk; b += kRedThreads) {
        v.loss += ws.part_loss[b];
        v.rho += ws.part_rho[b];
        v.live += ws.part_live[b];
        v.clip += ws.part_clip[b];
    }
    const LossSums t = block_sums_fixed(v);
    if (threadIdx.x == 0) {
        loss[0] = accumulate ? loss[0] + (float)t.loss : (float)t.loss;
        if (stats) {
            if (accumulate) {
                stats->loss_sum += t.loss;
                stats->rho_sum += t.rho;
                stats->live_tokens += t.live;
                stats->clipped_tokens += t.clip;
            } else {
                stats->loss_sum = t.loss;
                stats->rho_sum = t.rho;
                stats->live_tokens = t.live;
                stats->clipped_tokens = t.clip;
            }
        }
    }
}

// ---- fused-kernel configurations ------------------------------------------
struct FusedCfg {
    int C, T, NV, STAGES;
};
// The V = 151,936 configuration: one shared-memory stage per CTA and a
// register budget for three CTAs per SM (51 resident clusters).
constexpr int kBigStages = 1;
constexpr int kBigMinBlocks = 3;
// Rows of V <= 32,768 never reach this kernel (they take short_row_kernel).
constexpr FusedCfg kFused[] = {
    {4, 256, 10, 2}, {8, 256, 10, 2}, {8, 256, 16, 2},
};

template <int C, int T, int NV, int STAGES, int MINB = 1>
cudaError_t launch_fused_cfg(const RowArgs& a, cudaStream_t s) {
    auto kern = fused_loss_kernel<C, T, NV, STAGES, MINB>;
    const int64_t V8 = ((int64_t)a.V + 7) >> 3;
    const int per = (int)((V8 + C - 1) / C);
    const size_t dyn = (size_t)STAGES * per * 16;
    // Resident clusters for this shared-memory size (cached per size).
    static std::mutex mu;
    static size_t cached_dyn = 0;
    static int cached_dev = -1;
    static int cached_ncl = 0;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.blockDim = dim3(T + 32, 1, 1);
    cfg.dynamicSmemBytes = dyn;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = C;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    if (C > 1) {
        cfg.attrs = attr;
        cfg.numAttrs = 1;
    }
    int ncl = 0;
    {
        std::lock_guard<std::mutex> lk(mu);
        if (cached_dyn == dyn && cached_dev == dev) {
            ncl = cached_ncl;
        } else {
            e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
            if (e != cudaSuccess) return e;
            cfg.gridDim = dim3(C, 1, 1);
            if (C > 1) {
                e = cudaOccupancyMaxActiveClusters(&ncl, kern, &cfg);
            } else {
                int per_sm = 0;
                e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, T + 32, dyn);
                ncl = per_sm * device_sm_count();
            }
            if (e != cudaSuccess) return e;
            cached_dyn = dyn;
            cached_dev = dev;
            cached_ncl = ncl;
        }
    }
    if (ncl <= 0) return cudaErrorNotSupported;
    if ((int64_t)ncl > a.N) ncl = (int)a.N;
    cfg.gridDim = dim3((unsigned)(ncl * C), 1, 1);
    return cudaLaunchKernelEx(&cfg, kern, a, (int32_t)per, (int32_t)ncl);
}

}  // namespace

size_t loss_workspace_bytes(int64_t N) {
    const int64_t nblk = std::max<int64_t>(1, (N + kReduceRowsPerBlock - 1) / kReduceRowsPerBlock);
    auto al = [](size_t b) { return (b + 255) & ~size_t(255); };
    return al(N * sizeof(double)) + al(N * sizeof(float)) + al(N) + 4 * al(nblk * 8);
}

LossWorkspace carve_loss_workspace(void* base, int64_t N) {
    auto al = [](size_t b) { return (b + 255) & ~size_t(255); };
    LossWorkspace w;
    w.nblk = std::max<int64_t>(1, (N + kReduceRowsPerBlock - 1) / kReduceRowsPerBlock);
    char* p = static_cast<char*>(base);
    w.contrib = reinterpret_cast<double*>(p);
    p += al(N * sizeof(double));
    w.rho = reinterpret_cast<float*>(p);
    p += al(N * sizeof(float));
    w.flag = reinterpret_cast<uint8_t*>(p);
    p += al(N);
    w.part_loss = reinterpret_cast<double*>(p);
    p += al(w.nblk * 8);
    w.part_rho = reinterpret_cast<double*>(p);
    p += al(w.nblk * 8);
    w.part_live = reinterpret_cast<long long*>(p);
    p += al(w.nblk * 8);
    w.part_clip = reinterpret_cast<long long*>(p);
    return w;
}

int64_t fused_max_vocab() {
    const FusedCfg& c = kFused[sizeof(kFused) / sizeof(kFused[0]) - 1];
    return (int64_t)c.C * c.T * c.NV * 8;
}

cudaError_t launch_row_stream(const RowArgs& a, int mode, cudaStream_t s) {
    if (a.N == 0) return cudaSuccess;
    const int64_t V8 = ((int64_t)a.V + 7) >> 3;
    if (V8 <= 128) {
        const int64_t blocks = (a.N + 7) / 8;
        row_stream_kernel<32, 4, 1><<<(unsigned)blocks, 256, 0, s>>>(a, mode);
    } else {
        row_stream_kernel<512, 4, 3><<<(unsigned)a.N, 512, 0, s>>>(a, mode);
    }
    return cudaGetLastError();
}

cudaError_t launch_split_bwd(const RowArgs& a, cudaStream_t s) {
    if (a.N == 0) return cudaSuccess;
    const int64_t V8 = ((int64_t)a.V + 7) >> 3;
    if (V8 <= 128) {
        const int64_t blocks = (a.N + 7) / 8;
        split_bwd_kernel<32, 4><<<(unsigned)blocks, 256, 0, s>>>(a);
    } else {
        split_bwd_kernel<512, 4><<<(unsigned)a.N, 512, 0, s>>>(a);
    }
    return cudaGetLastError();
}

cudaError_t launch_fused_loss(const RowArgs& a, bool single_read, cudaStream_t s) {
    if (a.N == 0) return cudaSuccess;
    if (a.V <= kShortRowMaxV) return launch_short_row_loss(a, s);   // short_rows.cu
    if (!single_read) return launch_pipe_loss(a, s);                  // loss_pipe.cu
    const int64_t V8 = ((int64_t)a.V + 7) >> 3;
    for (const FusedCfg& c : kFused) {
        const int64_t per = (V8 + c.C - 1) / c.C;
        if (per > (int64_t)c.T * c.NV) continue;
        if (c.C == 4) return launch_fused_cfg<4, 256, 10, 2, 2>(a, s);
        if (c.NV == 10) return launch_fused_cfg<8, 256, 10, kBigStages, kBigMinBlocks>(a, s);
        return launch_fused_cfg<8, 256, 16, 2>(a, s);
    }
    return cudaErrorNotSupported;
}

cudaError_t launch_loss_reduce(const LossWorkspace& ws, int64_t N, float* loss, void* stats, bool accumulate,
                               cudaStream_t s) {
    // nblk >= 1: with N == 0 the single block writes zero partials.
    reduce_partial_kernel<<<(unsigned)ws.nblk, kRedThreads, 0, s>>>(ws, N);
    reduce_final_kernel<<<1, kRedThreads, 0, s>>>(ws, loss, static_cast<leap_loss_stats_t*>(stats),
                                                  accumulate ? 1 : 0);
    return cudaGetLastError();
}

}  // namespace leap
