// Token log-probs, the clipped GRPO surrogate (Eq. 3, KL skipped) with its
// deterministic masked reduction, and the dlogits backward.
//
// Kernels
//   row_stream_kernel  one pass over each logits row with an online
//                      (max, sum) -> log-probs, or the loss forward without
//                      dlogits.  2V bytes read per row.
//   fused_loss_l2_kernel  forward + backward, one persistent CTA per SM taking
//                      rows round-robin, two passes per row, the second
//                      served by L2.  2V read + 2V written per row.  A bulk
//                      L2 prefetch puts the whole row's HBM reads in flight
//                      at once, and the head of the CTA's next row is
//                      prefetched while this one writes, so reads and writes
//                      overlap on every SM.
//   fused_loss_kernel  forward + backward with the row split over a cluster
//                      of C CTAs that keep their slices in registers and
//                      exchange one (max, sum) pair through distributed
//                      shared memory: each row is read from HBM exactly once
//                      whatever else uses L2 (LEAP_LOSS_SINGLE_READ).
//   short_row_kernel   forward + backward for V <= 8,192: a group of 1-8
//                      warps holds one row in registers (read once) and
//                      reduces it with warp shuffles; persistent groups load
//                      the next row while they write the current one.
//   split_bwd_kernel   dlogits from a saved lse: 2V read + 2V written.
//   reduce kernels     fixed-order fp64 sum of the per-row loss terms.
#include "../../include/leap.h"
#include "leap_common.cuh"
#include "leap_internal.h"
#include "loss_math.cuh"

#include <algorithm>
#include <math.h>
#include <mutex>

namespace leap {
namespace {

__device__ __forceinline__ uint4 neg_inf4() {
    return make_uint4(kNegInfBf16x2, kNegInfBf16x2, kNegInfBf16x2, kNegInfBf16x2);
}

// Sets elements n..7 of an 8 x bf16 vector to -inf (row tail beyond V).
__device__ __forceinline__ void mask_tail(uint4& x, int n) {
    uint32_t w[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        if (j >= n) {
            if (j & 1) w[j >> 1] = (w[j >> 1] & 0x0000ffffu) | 0xff800000u;
            else       w[j >> 1] = (w[j >> 1] & 0xffff0000u) | 0x0000ff80u;
        }
    }
    x = make_uint4(w[0], w[1], w[2], w[3]);
}

// Stores vector vi of a dlogits row; the row's last vector keeps columns >= V intact.
__device__ __forceinline__ void store_vec(uint4* drow, int64_t vi, uint4 val, int64_t V8, int tailn) {
    if (tailn == 0 || vi != V8 - 1) {
        st_stream(drow + vi, val);
    } else {
        uint16_t* p = reinterpret_cast<uint16_t*>(drow + vi);
        const uint32_t w[4] = {val.x, val.y, val.z, val.w};
#pragma unroll
        for (int j = 0; j < 8; ++j)
            if (j < tailn) p[j] = (uint16_t)((j & 1) ? (w[j >> 1] >> 16) : (w[j >> 1] & 0xffffu));
    }
}

__device__ __forceinline__ float bf16_at(const uint16_t* p) {
    return __uint_as_float(((uint32_t)*p) << 16);
}

// Max of NV vectors of 8 bf16 as a balanced tree of packed maxima (depth
// 2 + log2 NV instead of a 4 NV-long chain).
template <int NV>
__device__ __forceinline__ float tree_max(const uint4 (&x)[NV]) {
    uint32_t v[NV];
#pragma unroll
    for (int k = 0; k < NV; ++k) v[k] = max_bf16x2(max_bf16x2(x[k].x, x[k].y), max_bf16x2(x[k].z, x[k].w));
#pragma unroll
    for (int stride = 1; stride < NV; stride *= 2) {
#pragma unroll
        for (int k = 0; k + stride < NV; k += 2 * stride) v[k] = max_bf16x2(v[k], v[k + stride]);
    }
    return fmaxf(bf16_lo(v[0]), bf16_hi(v[0]));
}

// Sum over NV vectors of 2^(z * c1 - mc), one accumulator per element
// position (8 independent chains of length NV), then a tree.
template <int NV>
__device__ __forceinline__ float tree_exp_sum(const uint4 (&x)[NV], float c1, float mc) {
    float acc[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[j] = 0.f;
#pragma unroll
    for (int k = 0; k < NV; ++k) {
        const uint32_t w[4] = {x[k].x, x[k].y, x[k].z, x[k].w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            acc[2 * q] += ex2(fmaf(bf16_lo(w[q]), c1, -mc));
            acc[2 * q + 1] += ex2(fmaf(bf16_hi(w[q]), c1, -mc));
        }
    }
    return ((acc[0] + acc[1]) + (acc[2] + acc[3])) + ((acc[4] + acc[5]) + (acc[6] + acc[7]));
}

// dlogits of one vector: coef * (1[v = y] - 2^(z c1 - K)); `yl` is the target's
// lane in this vector or -1.
__device__ __forceinline__ uint4 dlogit8(const uint4& x, float c1, float K, float coef, int yl) {
    const uint32_t w[4] = {x.x, x.y, x.z, x.w};
    uint32_t o[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        float lo = -coef * ex2(fmaf(bf16_lo(w[q]), c1, -K));
        float hi = -coef * ex2(fmaf(bf16_hi(w[q]), c1, -K));
        if (yl == 2 * q) lo += coef;
        if (yl == 2 * q + 1) hi += coef;
        o[q] = pack_bf16x2(lo, hi);
    }
    return make_uint4(o[0], o[1], o[2], o[3]);
}

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
// Fused forward + backward (default): one persistent CTA of T threads per SM
// taking rows round-robin, two passes over each row.  A bulk L2 prefetch puts
// the whole row's reads in flight; the first pass reads it (evict_last) and
// reduces it; the second reads it back (evict_first) and writes dlogits with
// streaming stores, while the head of the CTA's next row is prefetched.  With
// one row per SM in flight (152 rows, 46 MB at V = 151,936) the second read is
// an L2 hit: DRAM sees 2V bytes read and 2V written per live row.
// ---------------------------------------------------------------------------
// Measured settings (the alternatives are in the kernel's profile summary):
constexpr int kL2Threads = 1024;           // one CTA per SM (512 x 2 and 256 x 4 overflow L2)
constexpr int kL2U1 = 4;                   // 16-byte vectors in flight per thread, pass 1 (2: 0.850, 8: 0.791)
constexpr int kL2U2 = 6;                   // and pass 2 (2: 0.824, 4: 0.874, 5-8: 0.882-0.883, 10 spills)
constexpr int64_t kPfChunk = 32768;        // bytes per bulk L2 prefetch request
constexpr int64_t kNextBytes = 65536;      // head of the next row prefetched during pass 2
// Warp-wide: bulk L2 prefetch of the first min(cap, row) bytes of a logits row.
__device__ __forceinline__ void prefetch_row_l2(const uint16_t* zr, int V, int64_t cap, uint64_t policy, int lane) {
    int64_t bytes = (int64_t)(V & ~7) * 2;
    if (bytes > cap) bytes = cap & ~int64_t(15);
    for (int64_t off = (int64_t)lane * kPfChunk; off < bytes; off += 32 * kPfChunk)
        bulk_prefetch_l2(reinterpret_cast<const char*>(zr) + off,
                         (uint32_t)(bytes - off < kPfChunk ? bytes - off : kPfChunk), policy);
}
// This CTA's next row (next_stride rows on), if it is live: prefetch its head
// so that its pass 1 overlaps this row's writes.
__device__ __forceinline__ void prefetch_next_row(const RowArgs& a, int64_t row, uint64_t policy, int lane) {
    const int64_t nr = row + a.next_stride;
    if (a.next_stride > 0 && nr < a.N && a.w[nr] != 0.f)
        prefetch_row_l2(a.logits + nr * a.ld, a.V, kNextBytes, policy, lane);
}

// One row of the fused two-pass forward + backward, by the whole CTA.
template <int T, int U1, int U2>
__device__ __forceinline__ void l2_row(const RowArgs& a, const int64_t row, float2* wpart, float* bc) {
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int V = a.V;
    const int64_t V8 = ((int64_t)V + 7) >> 3;
    const int tailn = V & 7;
    const float wk = a.w[row];
    const int id = a.ids[row];
    const bool bad = (wk != 0.f) && (id < 0 || id >= V);
    uint4* drow = reinterpret_cast<uint4*>(a.dlogits + row * a.ld);
    if (wk == 0.f || bad) {
        if (warp == 1) prefetch_next_row(a, row, l2_policy_evict_last(), lane);
        for (int64_t vi = t; vi < V8; vi += T) store_vec(drow, vi, make_uint4(0, 0, 0, 0), V8, tailn);
        if (t == 0) {
            write_masked_outputs(a, row);
            if (bad) flag_status(a.status, LEAP_DEV_BAD_ID);
        }
        return;
    }
    const uint16_t* zr = a.logits + row * a.ld;
    const uint4* zrow = reinterpret_cast<const uint4*>(zr);
    float zy = 0.f, old = 0.f, A = 0.f;
    if (t == 0) {
        zy = bf16_at(zr + id);
        old = a.old_logp[row];
        A = a.adv[row];
    }
    const uint64_t keep = l2_policy_evict_last();
    // Put the whole row's HBM reads in flight at once: pass 1 then waits on
    // L2, not on the few loads each thread can hold in registers.
    if (warp == 0) prefetch_row_l2(zr, V, (int64_t)1 << 40, keep, lane);
    const float c1 = a.inv_temp * kLog2e;
    float m = -INFINITY, s = 0.f;
    for (int64_t v0 = t; v0 < V8; v0 += (int64_t)T * U1) {
        uint4 x[U1];
#pragma unroll
        for (int u = 0; u < U1; ++u) {
            const int64_t vi = v0 + (int64_t)u * T;
            x[u] = (vi < V8) ? ld_stream_hint(zrow + vi, keep) : neg_inf4();
            if (tailn && vi == V8 - 1) mask_tail(x[u], tailn);
        }
        const float bm = tree_max(x);
        if (bm == -INFINITY) continue;
        const float mn = fmaxf(m, bm);
        const float acc = tree_exp_sum(x, c1, mn * c1);
        s = (s == 0.f) ? acc : fmaf(s, ex2((m - mn) * c1), acc);
        m = mn;
    }
    warp_lse_merge(m, s, c1);
    if (lane == 0) wpart[warp] = make_float2(m, s);
    __syncthreads();
    if (warp == 0) {
        const float2 p = (lane < T / 32) ? wpart[lane] : make_float2(-INFINITY, 0.f);
        m = p.x;
        s = p.y;
        warp_lse_merge(m, s, c1);
        if (lane == 0) {
            const TokenLoss r = token_loss(a, m, s, zy, old, A, wk);
            bc[0] = fmaf(m, c1, log2f(s));
            bc[1] = a.grad_scale * r.g * a.inv_temp;
            write_row_outputs(a, row, r, wk);
        }
    }
    __syncthreads();
    if (warp == 1) prefetch_next_row(a, row, keep, lane);
    const float K = bc[0], coef = bc[1];
    const uint64_t drop = l2_policy_evict_first();
    const int64_t yv = id >> 3;
    const int ylane = id & 7;
    for (int64_t v0 = t; v0 < V8; v0 += (int64_t)T * U2) {
        if (coef == 0.f) {
#pragma unroll
            for (int u = 0; u < U2; ++u) {
                const int64_t vi = v0 + (int64_t)u * T;
                if (vi < V8) store_vec(drow, vi, make_uint4(0, 0, 0, 0), V8, tailn);
            }
            continue;
        }
        uint4 x[U2];
#pragma unroll
        for (int u = 0; u < U2; ++u) {
            const int64_t vi = v0 + (int64_t)u * T;
            x[u] = (vi < V8) ? ld_stream_hint(zrow + vi, drop) : neg_inf4();
        }
#pragma unroll
        for (int u = 0; u < U2; ++u) {
            const int64_t vi = v0 + (int64_t)u * T;
            if (vi < V8) store_vec(drow, vi, dlogit8(x[u], c1, K, coef, vi == yv ? ylane : -1), V8, tailn);
        }
    }
}

// One persistent CTA per SM walks rows blockIdx.x, + gridDim.x, ... with no
// CTA launch between rows (the round-robin spreads masked and live rows
// evenly; one CTA per row measured 0.845 of the copy peak against 0.871).
template <int T, int U1, int U2>
__global__ void __launch_bounds__(T, 1) fused_loss_l2_kernel(RowArgs a) {
    __shared__ float2 wpart[T / 32];
    __shared__ float bc[2];
    for (int64_t row = blockIdx.x; row < a.N; row += gridDim.x) l2_row<T, U1, U2>(a, row, wpart, bc);
}

// ---------------------------------------------------------------------------
// Fused forward + backward for short rows (V <= 8,192).  A row group of W
// warps owns one row at a time; warp w of the group owns the contiguous slice
// of 16-byte vectors [128 w, 128 (w + 1)) of the row (2 KB), lane l vectors
// 128 w + l + 32 k (k < 4), so the row is read from HBM once.
//   * Staging: each warp double-buffers its slice in shared memory.  While it
//     works on row i, a 1-D bulk copy (TMA) of its slice of row i + 1 is in
//     flight into the other stage, completing on that stage's mbarrier; every
//     wait is bounded (LEAP_DEV_TIMEOUT).  Registers hold one row only.
//   * Arithmetic: the kernel would otherwise be bound by instruction issue,
//     so the row max is reduced first (packed bf16 maxima, then the warp), the
//     exponentials 2^((z - m) c1) are taken once and kept in registers
//     (32 fp32 per lane), element pairs go through packed fp32x2 FMA / add /
//     multiply, and dlogits is one multiply per element.
//   * W > 1: each warp publishes (max, sum) and, if it holds it, the target
//     logit in shared memory behind one named barrier per live row (two
//     alternating slots); every warp then merges the W pairs directly.
//   * FULL (V a multiple of 1,024): every slice is whole, so the per-vector
//     bounds and tail checks are compiled out.
// Row groups are persistent and walk rows g, g + stride, ...  Masked rows are
// not read.
// ---------------------------------------------------------------------------
constexpr int kShortThreads = 256;        // 8 warps per CTA
constexpr int kShortNV = 4;               // 16-byte vectors per lane and row
constexpr int kShortVPW = 32 * kShortNV;  // vectors per warp slice (2 KB)
constexpr int kShortMinBlocks = 3;        // register budget: 80 per thread

struct ShortSmem {
    uint4 stage[kShortThreads / 32][2][kShortVPW];   // 32 KB: two 2 KB stages per warp
    uint64_t full[kShortThreads / 32][2];            // one mbarrier per stage
    float4 part[2][kShortThreads / 32];              // (max, sum, target logit, holds target) per warp
    int abort_flag;
};

// Packed pairs of fp32 (Blackwell's f32x2 FMA / add / multiply: one
// instruction for two lanes of arithmetic).
__device__ __forceinline__ uint64_t f2_pack(float lo, float hi) {
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}
__device__ __forceinline__ void f2_unpack(uint64_t v, float& lo, float& hi) {
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t f2_fma(uint64_t a, uint64_t b, uint64_t c) {
    uint64_t r;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
    return r;
}
__device__ __forceinline__ uint64_t f2_add(uint64_t a, uint64_t b) {
    uint64_t r;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}
__device__ __forceinline__ uint64_t f2_mul(uint64_t a, uint64_t b) {
    uint64_t r;
    asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}

template <int W, bool FULL>
__global__ void __launch_bounds__(kShortThreads, kShortMinBlocks) short_row_kernel(RowArgs a) {
    constexpr int NV = kShortNV, VPW = kShortVPW, TG = 32 * W, GPB = kShortThreads / TG;
    __shared__ __align__(128) ShortSmem sm;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int gib = warp / W;                  // row group within the block
    const int wig = warp % W;                  // warp within the row group
    // 32-bit row and vector indices (N < 2^31 is checked on the host; V8 <= 1,024).
    const int stride = (int)gridDim.x * GPB;
    const int N = (int)a.N;
    const int V = a.V;
    const int V8 = FULL ? W * VPW : (V + 7) >> 3;
    const int tailn = FULL ? 0 : (V & 7);
    const float c1 = a.inv_temp * kLog2e;
    const int vbase = wig * VPW;                                  // this warp's first vector
    const int nvec = FULL ? VPW : max(0, min(VPW, V8 - vbase));   // vectors in this warp's slice
    const uint32_t slice_bytes = (uint32_t)nvec * 16u;

    if (threadIdx.x == 0) sm.abort_flag = 0;
    if (lane == 0) {
        mbar_init(&sm.full[warp][0], 1);
        mbar_init(&sm.full[warp][1], 1);
        fence_mbar_init();
    }
    __syncthreads();

    auto is_live = [&](float wr, int idr) { return wr != 0.f && idr >= 0 && idr < V; };
    uint32_t phase = 0;     // bit s: parity of the next completion of stage s
    uint32_t pending = 0;   // bit s: a copy into stage s has not been waited for
    // Lane 0 starts the copy of this warp's slice of row r into stage st (none
    // once a wait of this CTA has given up, so at most one copy per stage is
    // ever outstanding).
    auto issue = [&](int r, int st) {
        if (slice_bytes == 0 || *reinterpret_cast<volatile int*>(&sm.abort_flag)) return;
        pending |= 1u << st;
        if (lane == 0) {
            mbar_arrive_expect_tx(&sm.full[warp][st], slice_bytes);
            bulk_g2s(&sm.stage[warp][st][0], a.logits + (int64_t)r * a.ld + (int64_t)vbase * 8, slice_bytes,
                     &sm.full[warp][st]);
        }
    };
    // w and id of the row `k` strides after `r`, or (0, 0) past the end.
    auto scalars = [&](int r, int k, float& wr, int& idr) {
        wr = 0.f;
        idr = 0;
        if (r < N - k * stride) {   // r + k * stride < N without overflow
            wr = a.w[r + k * stride];
            idr = a.ids[r + k * stride];
        }
    };

    int row = (int)blockIdx.x * GPB + gib;
    float w0, w1, w2;
    int id0, id1, id2;
    scalars(row, 0, w0, id0);
    scalars(row, 1, w1, id1);
    scalars(row, 2, w2, id2);
    if (row < N && is_live(w0, id0)) issue(row, 0);
    if (is_live(w1, id1)) issue(row + stride, 1);
    int par = 0;
    const uint64_t c1x2 = f2_pack(c1, c1);

    for (int it = 0; row < N; row += stride, ++it) {
        const int st = it & 1;
        float w3;
        int id3;
        scalars(row, 3, w3, id3);

        const bool bad = (w0 != 0.f) && (id0 < 0 || id0 >= V);
        uint4* drow = reinterpret_cast<uint4*>(a.dlogits + (int64_t)row * a.ld);
        if (w0 == 0.f || bad) {   // masked row: the same branch in every warp of the group
#pragma unroll
            for (int k = 0; k < NV; ++k) {
                const int vi = vbase + lane + 32 * k;
                if (FULL || vi < V8) store_vec(drow, vi, make_uint4(0, 0, 0, 0), V8, tailn);
            }
            if (wig == 0 && lane == 0) {
                write_masked_outputs(a, row);
                if (bad) flag_status(a.status, LEAP_DEV_BAD_ID);
            }
            if (is_live(w2, id2)) issue(row + 2 * stride, st);   // this row left stage st unused
        } else {
            const float old = a.old_logp[row], A = a.adv[row];
            uint4 x[NV];
            if (pending & (1u << st)) {
                if (mbar_wait(&sm.full[warp][st], (phase >> st) & 1u, a.status, &sm.abort_flag)) {
                    phase ^= 1u << st;
                    pending &= ~(1u << st);
                }   // else: results undefined (LEAP_DEV_TIMEOUT); the copy stays pending
            }
#pragma unroll
            for (int k = 0; k < NV; ++k) {
                const int li = lane + 32 * k;
                if (FULL) {
                    x[k] = sm.stage[warp][st][li];
                } else {
                    x[k] = (li < nvec) ? sm.stage[warp][st][li] : neg_inf4();
                    if (tailn && vbase + li == V8 - 1) mask_tail(x[k], tailn);
                }
            }
            // The target logit, if it lies in this warp's slice.
            const int yl = id0 - vbase * 8;
            const bool own_y = yl >= 0 && yl < nvec * 8;
            float zy = own_y ? bf16_at(reinterpret_cast<const uint16_t*>(&sm.stage[warp][st][0]) + yl) : 0.f;
            // Every lane has read the stage: it may take the copy of row i + 2.
            __syncwarp();
            fence_proxy_async_smem();
            if (is_live(w2, id2)) issue(row + 2 * stride, st);
            // Row max: packed maxima, then the warp.
            float m = tree_max(x);
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
            // Exponentials against the warp max, kept (as pairs) for the backward.
            uint64_t e2[NV][4];
            float ssum = 0.f;
            if (m != -INFINITY) {
                const float nmc = -m * c1;
                const uint64_t nmc2 = f2_pack(nmc, nmc);
                uint64_t acc2[2] = {f2_pack(0.f, 0.f), f2_pack(0.f, 0.f)};
#pragma unroll
                for (int k = 0; k < NV; ++k) {
                    const uint32_t wv[4] = {x[k].x, x[k].y, x[k].z, x[k].w};
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        float lo, hi;
                        f2_unpack(f2_fma(f2_pack(bf16_lo(wv[q]), bf16_hi(wv[q])), c1x2, nmc2), lo, hi);
                        e2[k][q] = f2_pack(ex2(lo), ex2(hi));
                        acc2[q & 1] = f2_add(acc2[q & 1], e2[k][q]);
                    }
                }
                float s0, s1, s2, s3;
                f2_unpack(acc2[0], s0, s1);
                f2_unpack(acc2[1], s2, s3);
                ssum = (s0 + s1) + (s2 + s3);
            } else {
#pragma unroll
                for (int k = 0; k < NV; ++k)
#pragma unroll
                    for (int q = 0; q < 4; ++q) e2[k][q] = f2_pack(0.f, 0.f);
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) ssum += __shfl_xor_sync(0xffffffffu, ssum, o);
            // The row's (max, sum), the target logit and this warp's factor 2^((m_warp - m_row) c1).
            float mrow = m, srow = ssum, wscale = 1.f;
            if (W > 1) {
                if (lane == 0) sm.part[par][warp] = make_float4(m, ssum, zy, own_y ? 1.f : 0.f);
                named_bar_sync(1 + gib, TG);
                float4 p[W];
#pragma unroll
                for (int v = 0; v < W; ++v) p[v] = sm.part[par][gib * W + v];
                mrow = p[0].x;
#pragma unroll
                for (int v = 1; v < W; ++v) mrow = fmaxf(mrow, p[v].x);
                srow = 0.f;
#pragma unroll
                for (int v = 0; v < W; ++v) {
                    if (p[v].y != 0.f) srow = fmaf(p[v].y, ex2((p[v].x - mrow) * c1), srow);
                    if (p[v].w != 0.f) zy = p[v].z;
                }
                wscale = (ssum != 0.f) ? ex2((m - mrow) * c1) : 0.f;
                par ^= 1;   // live rows alternate slots: a slot is rewritten only after the
                            // next live row's barrier, which every reader of it has passed
            }
            const TokenLoss r = token_loss(a, mrow, srow, zy, old, A, w0);
            const float coef = a.grad_scale * r.g * a.inv_temp;
            if (wig == 0 && lane == 0) write_row_outputs(a, row, r, w0);
            // dlogits_v = coef (1[v = y] - e_v wscale / s_row); the factor's own
            // rounding (fast reciprocal, ~2 ulp of fp32) is far below bf16's.
            const float nf = -__fdividef(coef * wscale, srow);
            const uint64_t nf2 = f2_pack(nf, nf);
            const int yv = id0 >> 3;
            const int ylane = id0 & 7;
#pragma unroll
            for (int k = 0; k < NV; ++k) {
                const int vi = vbase + lane + 32 * k;
                if (FULL || vi < V8) {
                    uint4 d = make_uint4(0, 0, 0, 0);
                    if (coef != 0.f) {
                        float o8[8];
#pragma unroll
                        for (int q = 0; q < 4; ++q) f2_unpack(f2_mul(e2[k][q], nf2), o8[2 * q], o8[2 * q + 1]);
                        if (vi == yv) {
#pragma unroll
                            for (int j = 0; j < 8; ++j)
                                if (j == ylane) o8[j] += coef;
                        }
                        d = make_uint4(pack_bf16x2(o8[0], o8[1]), pack_bf16x2(o8[2], o8[3]),
                                       pack_bf16x2(o8[4], o8[5]), pack_bf16x2(o8[6], o8[7]));
                    }
                    if (FULL) st_stream(drow + vi, d);
                    else store_vec(drow, vi, d, V8, tailn);
                }
            }
        }
        // Shift the scalar pipeline by one row.
        w0 = w1;
        id0 = id1;
        w1 = w2;
        id1 = id2;
        w2 = w3;
        id2 = id3;
    }
    // Every copy is waited for before its row is used, so one can still be in
    // flight here only after a wait gave up: wait for it (bounded again) so no
    // copy lands in the shared memory of an exited CTA.
    if (pending) {
        volatile int fresh = 0;
        for (int st = 0; st < 2; ++st)
            if (pending & (1u << st)) mbar_wait(&sm.full[warp][st], (phase >> st) & 1u, a.status, &fresh);
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

template <typename Tv>
__device__ __forceinline__ Tv block_sum_fixed(Tv v, Tv* sh) {
    sh[threadIdx.x] = v;
    __syncthreads();
    for (int o = blockDim.x / 2; o > 0; o >>= 1) {
        if ((int)threadIdx.x < o) sh[threadIdx.x] += sh[threadIdx.x + o];
        __syncthreads();
    }
    const Tv r = sh[0];
    __syncthreads();
    return r;
}

__global__ void __launch_bounds__(kRedThreads) reduce_partial_kernel(LossWorkspace ws, int64_t N) {
    __shared__ double shd[kRedThreads];
    __shared__ long long shl[kRedThreads];
    const int64_t lo = (int64_t)blockIdx.x * kReduceRowsPerBlock;
    const int64_t hi = min(N, lo + kReduceRowsPerBlock);
    double l = 0.0, rs = 0.0;
    long long live = 0, clip = 0;
    for (int64_t i = lo + threadIdx.x; i < hi; i += kRedThreads) {
        l += ws.contrib[i];
        rs += (double)ws.rho[i];
        const uint8_t f = ws.flag[i];
        live += (f & 1u);
        clip += (f >> 1) & 1u;
    }
    l = block_sum_fixed(l, shd);
    rs = block_sum_fixed(rs, shd);
    live = block_sum_fixed(live, shl);
    clip = block_sum_fixed(clip, shl);
    if (threadIdx.x == 0) {
        ws.part_loss[blockIdx.x] = l;
        ws.part_rho[blockIdx.x] = rs;
        ws.part_live[blockIdx.x] = live;
        ws.part_clip[blockIdx.x] = clip;
    }
}

__global__ void __launch_bounds__(kRedThreads) reduce_final_kernel(LossWorkspace ws, float* loss,
                                                                    leap_loss_stats_t* stats, int accumulate) {
    __shared__ double shd[kRedThreads];
    __shared__ long long shl[kRedThreads];
    double l = 0.0, rs = 0.0;
    long long live = 0, clip = 0;
    for (int64_t b = threadIdx.x; b < ws.nblk; b += kRedThreads) {
        l += ws.part_loss[b];
        rs += ws.part_rho[b];
        live += ws.part_live[b];
        clip += ws.part_clip[b];
    }
    l = block_sum_fixed(l, shd);
    rs = block_sum_fixed(rs, shd);
    live = block_sum_fixed(live, shl);
    clip = block_sum_fixed(clip, shl);
    if (threadIdx.x == 0) {
        loss[0] = accumulate ? loss[0] + (float)l : (float)l;
        if (stats) {
            if (accumulate) {
                stats->loss_sum += l;
                stats->rho_sum += rs;
                stats->live_tokens += live;
                stats->clipped_tokens += clip;
            } else {
                stats->loss_sum = l;
                stats->rho_sum = rs;
                stats->live_tokens = live;
                stats->clipped_tokens = clip;
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
// Rows of V <= 8,192 never reach this kernel (they take short_row_kernel).
constexpr FusedCfg kFused[] = {
    {2, 256, 8, 2}, {4, 256, 10, 2}, {8, 256, 10, 2}, {8, 256, 16, 2},
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

// Persistent grid of the short-row kernel: the CTAs that fit at once (cached
// per device), at most one row group per row.
template <int W, bool FULL>
cudaError_t launch_short_rows(const RowArgs& a, cudaStream_t s) {
    static std::mutex mu;
    static int cached_dev = -1, cached_resident = 0;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    int resident = 0;   // CTAs resident at once on the whole device
    {
        std::lock_guard<std::mutex> lk(mu);
        if (cached_dev != dev) {
            int per_sm = 0;
            e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, short_row_kernel<W, FULL>, kShortThreads, 0);
            if (e != cudaSuccess) return e;
            cached_dev = dev;
            cached_resident = per_sm * device_sm_count();
        }
        resident = cached_resident;
    }
    if (resident <= 0) return cudaErrorNotSupported;
    constexpr int GPB = kShortThreads / (32 * W);
    const int64_t blocks = std::min<int64_t>((a.N + GPB - 1) / GPB, (int64_t)resident);
    short_row_kernel<W, FULL><<<(unsigned)blocks, kShortThreads, 0, s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_fused_loss(const RowArgs& a, bool single_read, cudaStream_t s) {
    if (a.N == 0) return cudaSuccess;
    const int64_t V8s = ((int64_t)a.V + 7) >> 3;
    if (V8s <= (int64_t)8 * 32 * kShortNV) {   // V <= 8,192: the row lives in one row group's registers
        const int W = V8s <= kShortVPW ? 1 : V8s <= 2 * kShortVPW ? 2 : V8s <= 4 * kShortVPW ? 4 : 8;
        // Whole 2 KB slices for every warp (V = 1,024 W): no per-vector bounds checks.
        const bool full = a.V == W * 8 * kShortVPW;
        switch (W) {
            case 1: return full ? launch_short_rows<1, true>(a, s) : launch_short_rows<1, false>(a, s);
            case 2: return full ? launch_short_rows<2, true>(a, s) : launch_short_rows<2, false>(a, s);
            case 4: return full ? launch_short_rows<4, true>(a, s) : launch_short_rows<4, false>(a, s);
            default: return full ? launch_short_rows<8, true>(a, s) : launch_short_rows<8, false>(a, s);
        }
    }
    if (!single_read) {
        RowArgs b = a;
        const int64_t grid = std::min<int64_t>(a.N, (int64_t)device_sm_count());
        b.next_stride = (int32_t)grid;   // exactly the CTA's next row
        fused_loss_l2_kernel<kL2Threads, kL2U1, kL2U2><<<(unsigned)grid, kL2Threads, 0, s>>>(b);
        return cudaGetLastError();
    }
    const int64_t V8 = ((int64_t)a.V + 7) >> 3;
    for (const FusedCfg& c : kFused) {
        const int64_t per = (V8 + c.C - 1) / c.C;
        if (per > (int64_t)c.T * c.NV) continue;
        if (c.C == 2) return launch_fused_cfg<2, 256, 8, 2, 2>(a, s);
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
