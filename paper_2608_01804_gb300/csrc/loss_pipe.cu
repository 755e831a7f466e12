// Fused forward + backward of the clipped surrogate (Eq. 3, KL skipped) with
// the two passes over a row pipelined across consecutive rows of one SM.
//
// One persistent CTA per SM takes its share of the rows: a balanced list
// (build_row_list: equal live and masked row counts per CTA; RowSeq: order)
// or rows c, c + G, ... (G = grid size).  Its warps have five roles:
//   producer A  (one lane)  bulk-copies (TMA, 1-D) each 16 KB chunk of the
//                           CTA's next live row into ring A (3 stages), an L2
//                           evict_last policy on the copy so the row stays
//                           for pass 2;
//   group A     (4 warps)   pass 1: reduces each chunk of ring A to per-warp
//                           (max, sum of exponentials) and goes straight on
//                           to the next live row;
//   finishing   (one warp)  merges group A's partials of a row, evaluates the
//                           token's loss and outputs, and hands (K, coef) for
//                           the backward to group B through a two-slot queue;
//   producer B  (one lane)  bulk-copies the same live rows again, from L2
//                           (evict_first), into ring B (11 stages);
//   group B     (8 warps)   pass 2: walks every row of the CTA in order,
//                           writing zeros for masked rows and dlogits from
//                           ring B for live ones.
// So on every SM pass 1 of row j (HBM reads) runs beside pass 2 of row j - 1
// (L2 re-reads and HBM writes), with up to 14 16 KB copies in flight
// independent of the threads' registers, and each role loads the next row's
// weight and id a row ahead (the finishing warp also the row's loss inputs
// before it waits for the row's partials), so no chain of dependent global
// loads and no block-wide barrier sits between two rows; group A starts a
// row only once group B has finished the row two before it, which keeps the
// rows between the passes in L2.
// HBM sees 2V bytes read and 2V written per live row, 2V written per masked
// row.
//
// Every wait is on an mbarrier and bounded (2 s, LEAP_DEV_TIMEOUT): after a
// give-up the CTA's abort flag stops every role, and each producer waits
// (bounded again) for its copies still in flight before the CTA exits.
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

// 1-D bulk copy global -> own shared memory with an L2 cache policy,
// completing on `bar` (addresses and size multiples of 16).
__device__ __forceinline__ void bulk_g2s_hint(void* smem_dst, const void* gsrc, uint32_t bytes, uint64_t* bar,
                                              uint64_t policy) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], "
        "%4;" ::"r"(smem_addr(smem_dst)),
        "l"(gsrc), "r"(bytes), "r"(smem_addr(bar)), "l"(policy)
        : "memory");
}

constexpr int kPipeListMax = 576;   // rows per CTA the balanced list holds (fits the shared memory left)

template <int NA, int SA, int SB, int CVA, int CVB>
struct PipeSmem {
    uint4 ringA[SA][CVA];
    uint4 ringB[SB][CVB];
    uint64_t fullA[SA], emptyA[SA], fullB[SB], emptyB[SB];
    uint64_t kcfull[2], kcempty[2];
    float2 kc[2];            // (K = log2 of the row's normaliser in c1 units, coef) per queue slot
    float2 wpart[2][NA];     // per-warp (max, sum) of group A, by row parity
    uint64_t wfull[2], wempty[2];   // group A -> finishing warp, by row parity
    int32_t list[kPipeListMax];     // this CTA's rows (balanced assignment; RowSeq walks it)
    int32_t wcnt[32];               // live rows per warp block while the list is built
    int32_t nlist, nlive;           // the list's rows, the live ones first
    int abort_flag;
};

// The order in which every role of a CTA visits its n rows.  With the CTA's
// list (the balanced assignment below) and P = 1: the list's order, the
// stream's.  With the list and P = 2 (the list then holds the CTA's nl live
// rows, then its masked ones, each in stream order): the live rows spread
// evenly over the walk, visit j live iff floor((j + 1) nl / n) > floor(j nl /
// n), so that on every SM masked rows (dlogits zeros, no reads) sit between
// the live ones instead of the stream's long runs of either (the packed
// multi-turn workload: 0.934 -> 0.949 of the copy peak; the padded single-turn
// batch, with short runs, keeps the stream order: 0.951 against 0.945).
// Without a list: rows c, c + G, ... (c = blockIdx.x, G = gridDim.x), walked
// as P interleaved streams, stream p holding the p-th run of ceil(n / P)
// rows, so that row j of the walk is row ((j mod P) ceil(n / P) + j div P) of
// the CTA, or none past the end.
template <int P>
struct RowSeq {
    int64_t c, G, n, np, nl;
    const int32_t* list;
    __device__ __forceinline__ RowSeq(int64_t N, const int32_t* lst, int32_t nlst, int32_t nlv)
        : c(blockIdx.x), G(gridDim.x), nl(nlv), list(lst) {
        n = lst ? nlst : (N - c + G - 1) / G;
        np = (n + P - 1) / P;
    }
    __device__ __forceinline__ int64_t len() const { return np * P; }
    __device__ __forceinline__ int64_t row(int64_t j) const {
        if (j >= np * P) return -1;
        if (list) {
            if (j >= n) return -1;
            if (P == 1) return (int64_t)list[j];
            const int64_t lo = j * nl / n, hi = (j + 1) * nl / n;
            return hi > lo ? (int64_t)list[lo] : (int64_t)list[nl + j - lo];
        }
        const int64_t idx = (j % P) * np + j / P;
        if (idx >= n) return -1;
        return c + idx * G;
    }
};

// Balanced assignment of the rows to the G CTAs, built by every CTA from w
// alone: a live row (w != 0) moves 4V bytes and a masked one 2V, so CTA c
// takes the live rows of live rank = c (mod G) and the masked rows of masked
// rank = G - 1 - c (mod G) (the CTAs short of a live row are the ones given an
// extra masked row), in stream order: every CTA is within one live and one
// masked row of the average work, where taking rows c, c + G, ... left the
// busiest CTA 2.5 % above it on the single-turn workload.  Warp k counts the
// live rows of its block of rows (coalesced loads, ballots), the warps' counts
// give each block its first live rank, and each warp walks its block again
// placing this CTA's rows at their index in the list: the number of this
// CTA's rows of either kind before them, or with SPLIT its live rows first
// (at their index among its live rows) and its masked rows after them (at
// their index among its masked rows).  Needs G >= 32.
template <int NW, bool SPLIT>
__device__ __forceinline__ void build_row_list(const RowArgs& a, int32_t* list, int32_t* wcnt, int32_t* nlist,
                                               int32_t* nlive) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t N = a.N;
    const int G = (int)gridDim.x, c = (int)blockIdx.x;
    const int64_t per = ((N + NW * 32 - 1) / (NW * 32)) * 32;   // rows per warp block, a multiple of 32
    const int64_t r0 = (int64_t)warp * per, r1 = r0 + per < N ? r0 + per : N;
    int cnt = 0;
    for (int64_t b = r0; b < r1; b += 32 * 8) {
        float x[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int64_t r = b + 32 * u + lane;
            x[u] = r < r1 ? a.w[r] : 0.f;
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) cnt += __popc(__ballot_sync(0xffffffffu, x[u] != 0.f));
    }
    if (lane == 0) wcnt[warp] = cnt;
    __syncthreads();
    int64_t lbefore = 0, ltot = 0;
    for (int k = 0; k < NW; ++k) {
        const int v = wcnt[k];
        ltot += v;
        if (k < warp) lbefore += v;
    }
    const int64_t ncl = (ltot + G - 1 - c) / G;   // this CTA's live rows
    // Ranks of the block's first row and their residues mod G, kept up to date
    // per 32 rows (an increment below 32 <= G needs one conditional subtraction).
    int64_t lr = lbefore, mr = (r0 < r1 ? r0 : 0) - lbefore;
    int lrm = (int)(lr % G), mrm = (int)(mr % G);
    const unsigned lt = (1u << lane) - 1u;
    for (int64_t b = r0; b < r1; b += 32) {
        const int64_t r = b + lane;
        const bool in = r < r1;
        const bool live = in && a.w[r] != 0.f;
        const unsigned bal = __ballot_sync(0xffffffffu, live);
        const int pl = __popc(bal & lt), pm = lane - pl;   // live / masked rows of this chunk before the lane
        if (in) {
            int ml = lrm + pl, mm = mrm + pm;
            if (ml >= G) ml -= G;
            if (mm >= G) mm -= G;
            const int64_t my_lr = lr + pl, my_mr = mr + pm;
            if (live && ml == c)
                list[SPLIT ? (my_lr - c) / G : (my_lr - c) / G + (my_mr + c) / G] = (int32_t)r;
            else if (!live && mm == G - 1 - c)
                list[SPLIT ? ncl + (my_mr - (G - 1 - c)) / G
                           : (my_mr - (G - 1 - c)) / G + (my_lr + G - 1 - c) / G] = (int32_t)r;
        }
        const int nin = r1 - b < 32 ? (int)(r1 - b) : 32;
        const int nl = __popc(bal), nm = nin - nl;
        lr += nl;
        mr += nm;
        lrm += nl;
        if (lrm >= G) lrm -= G;
        mrm += nm;
        if (mrm >= G) mrm -= G;
    }
    if (threadIdx.x == 0) {
        const int64_t mtot = N - ltot;
        *nlist = (int32_t)(ncl + (mtot + c) / G);
        *nlive = (int32_t)ncl;
    }
}

// One producer: copies every chunk of the CTA's live rows, in the CTA's row
// order, into a ring of S stages; then waits for whatever of its copies is
// still in flight.
template <int S, int CV, int P>
__device__ __forceinline__ void pipe_produce(const RowArgs& a, uint4 (*ring)[CV], uint64_t* full,
                                             uint64_t* empty, uint64_t policy, volatile int* abort_flag,
                                             const int32_t* list, int32_t nlist, int32_t nlive) {
    constexpr int64_t kPipeChunk = CV * 16;
    const int64_t rowbytes = (int64_t)(a.V & ~7) * 2;
    const int64_t nch = (rowbytes + kPipeChunk - 1) / kPipeChunk;
    uint32_t cnt = 0;
    bool go = true;
    const RowSeq<P> seq(a.N, list, nlist, nlive);
    int64_t rn = seq.row(0);
    float w_next = a.w[rn];     // the next row's weight and id, a row ahead
    int id_next = a.ids[rn];
    for (int64_t j = 0; go && j < seq.len(); ++j) {
        const int64_t row = rn;
        const float wk = w_next;
        const int id = id_next;
        rn = seq.row(j + 1);
        if (rn >= 0) {
            w_next = a.w[rn];
            id_next = a.ids[rn];
        }
        if (row < 0 || !(wk != 0.f && id >= 0 && id < a.V)) continue;
        const char* src = reinterpret_cast<const char*>(a.logits + row * a.ld);
        for (int64_t k = 0; k < nch; ++k) {
            const uint32_t s = cnt % S, ph = (cnt / S) & 1u;
            if (!mbar_wait(&empty[s], ph ^ 1u, a.status, abort_flag)) {
                go = false;
                break;
            }
            fence_proxy_async_smem();
            const uint32_t bytes = (uint32_t)min((int64_t)kPipeChunk, rowbytes - k * kPipeChunk);
            mbar_arrive_expect_tx(&full[s], bytes);
            bulk_g2s_hint(&ring[s][0], src + k * kPipeChunk, bytes, &full[s], policy);
            ++cnt;
        }
    }
    // Copies the consumers have not waited for may still be landing: wait
    // for the last copy of every stage (returns at once for consumed ones).
    for (uint32_t s = 0; s < (uint32_t)S && s < cnt; ++s) {
        const uint32_t last = cnt - 1 - ((cnt - 1 - s) % S);   // last copy into stage s
        mbar_wait_bounded<false>(&full[s], (last / S) & 1u, a.status, abort_flag);
    }
    if (*abort_flag) {
        // After a give-up the waits above return at once: spin (bounded) on
        // the stages directly so no copy outlives the CTA.
        for (uint32_t s = 0; s < (uint32_t)S && s < cnt; ++s) {
            const uint32_t last = cnt - 1 - ((cnt - 1 - s) % S);
            const uint64_t t0 = globaltimer_ns();
            while (!mbar_try_wait(&full[s], (last / S) & 1u) && globaltimer_ns() - t0 < kWaitLimitNs) {
            }
        }
    }
}

template <int NA, int NB, int SA, int SB, int CVA, int CVB, int P>
__global__ void __launch_bounds__(32 * (3 + NA + NB), 1) fused_loss_pipe_kernel(RowArgs a) {
    extern __shared__ __align__(128) unsigned char pipe_smem_raw[];
    PipeSmem<NA, SA, SB, CVA, CVB>& sm = *reinterpret_cast<PipeSmem<NA, SA, SB, CVA, CVB>*>(pipe_smem_raw);
    constexpr int TA = 32 * NA, TB = 32 * NB;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    volatile int* abort_flag = &sm.abort_flag;

    if (threadIdx.x == 0) {
        sm.abort_flag = 0;
        for (int s = 0; s < SA; ++s) {
            mbar_init(&sm.fullA[s], 1);
            mbar_init(&sm.emptyA[s], NA);
        }
        for (int s = 0; s < SB; ++s) {
            mbar_init(&sm.fullB[s], 1);
            mbar_init(&sm.emptyB[s], NB);
        }
        for (int q = 0; q < 2; ++q) {
            mbar_init(&sm.kcfull[q], 1);
            mbar_init(&sm.kcempty[q], NB);
            mbar_init(&sm.wfull[q], NA);
            mbar_init(&sm.wempty[q], 1);
        }
        fence_mbar_init();
    }
    // The balanced row list when the grid is wide and the list fits (single-
    // turn workload, in stream order: 0.932 -> 0.936 of the copy peak against
    // rows c, c + G, ...; live rows spread evenly, P = 2: above).
    const bool listed = gridDim.x >= 32 && (a.N + gridDim.x - 1) / gridDim.x + 2 <= kPipeListMax;
    if (listed) build_row_list<3 + NA + NB, P == 2>(a, sm.list, sm.wcnt, &sm.nlist, &sm.nlive);
    __syncthreads();
    const int32_t* list = listed ? sm.list : nullptr;
    const int32_t nlist = listed ? sm.nlist : 0;
    const int32_t nlive = listed ? sm.nlive : 0;

    const int V = a.V;
    const int64_t V8 = ((int64_t)V + 7) >> 3;
    const int tailn = V & 7;
    const int64_t V8f = (int64_t)(V >> 3);             // whole vectors, all bulk-copied
    const int64_t rowbytes = V8f * 16;
    const float c1 = a.inv_temp * kLog2e;

    if (warp == 0) {
        if (lane == 0) pipe_produce<SA, CVA, P>(a, sm.ringA, sm.fullA, sm.emptyA, l2_policy_evict_last(), abort_flag, list,
                                                 nlist, nlive);
        return;
    }
    if (warp == 1) {
        if (lane == 0) pipe_produce<SB, CVB, P>(a, sm.ringB, sm.fullB, sm.emptyB, l2_policy_evict_first(), abort_flag, list,
                                                 nlist, nlive);
        return;
    }

    constexpr int A0 = 3;   // first warp of group A
    if (warp == 2) {
        // ---- finishing warp: merges group A's partials, evaluates the token's
        // loss and hands (K, coef) to group B, while group A goes on to the
        // next row.
        uint32_t li = 0;
        const RowSeq<P> seq(a.N, list, nlist, nlive);
        int64_t rn = seq.row(0);
        float w_next = a.w[rn];
        int id_next = a.ids[rn];
        for (int64_t j = 0; j < seq.len(); ++j) {
            const int64_t row = rn;
            const float wk = w_next;
            const int id = id_next;
            rn = seq.row(j + 1);
            if (rn >= 0) {
                w_next = a.w[rn];
                id_next = a.ids[rn];
            }
            if (row < 0 || !(wk != 0.f && id >= 0 && id < V)) continue;
            float zy = 0.f, old = 0.f, Adv = 0.f;
            if (lane == 0) {
                zy = bf16_at(a.logits + row * a.ld + id);
                old = a.old_logp[row];
                Adv = a.adv[row];
            }
            const uint32_t q = li & 1u;
            if (!mbar_wait(&sm.wfull[q], (li >> 1) & 1u, a.status, abort_flag)) break;
            const float2 p = (lane < NA) ? sm.wpart[q][lane] : make_float2(-INFINITY, 0.f);
            float m = p.x, s = p.y;
            warp_lse_merge(m, s, c1);
            if (lane == 0) {
                const TokenLoss r = token_loss(a, m, s, zy, old, Adv, wk);
                write_row_outputs(a, row, r, wk);
                if (mbar_wait(&sm.kcempty[q], ((li >> 1) & 1u) ^ 1u, a.status, abort_flag)) {
                    sm.kc[q] = make_float2(fmaf(m, c1, log2f(s)), a.grad_scale * r.g * a.inv_temp);
                    mbar_arrive(&sm.kcfull[q]);
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&sm.wempty[q]);
            ++li;
        }
        return;
    }
    if (warp < A0 + NA) {
        // ---- group A: pass 1 -------------------------------------------------
        const int ta = threadIdx.x - 32 * A0, wa = warp - A0;
        constexpr int64_t kPipeChunk = CVA * 16;
        constexpr int kPipeChunkVec = CVA;
        const int64_t nch = (rowbytes + kPipeChunk - 1) / kPipeChunk;
        uint32_t cnt = 0, li = 0;
        // The next row's weight and id are loaded a row ahead (every role does;
        // with the finishing warp's early loads of the loss inputs, measured
        // 0.914 -> 0.928 of the copy peak).
        const RowSeq<P> seq(a.N, list, nlist, nlive);
        int64_t rn = seq.row(0);
        float w_next = a.w[rn];
        int id_next = a.ids[rn];
        for (int64_t j = 0; j < seq.len(); ++j) {
            const int64_t row = rn;
            const float wk = w_next;
            const int id = id_next;
            rn = seq.row(j + 1);
            if (rn >= 0) {
                w_next = a.w[rn];
                id_next = a.ids[rn];
            }
            if (row < 0 || !(wk != 0.f && id >= 0 && id < V)) continue;
            const uint16_t* zr = a.logits + row * a.ld;
            // The row's last, partial vector (not bulk-copied) is loaded now,
            // so its latency hides behind the row's chunks.
            uint4 tailx = make_uint4(0, 0, 0, 0);
            if (tailn && ta == 0) tailx = ld_stream(reinterpret_cast<const uint4*>(zr) + V8f);
            // Start live row li once group B has finished row li - 2 (the
            // queue slot's release): pass 1 stays at most about one row
            // ahead of pass 2, so the rows between them still sit in L2 when
            // pass 2 re-reads them (long masked runs would otherwise let it
            // run three rows ahead and the re-reads miss).
            if (li >= 2) {
                if (lane == 0) mbar_wait(&sm.kcempty[li & 1u], ((li >> 1) & 1u) ^ 1u, a.status, abort_flag);
                __syncwarp();
            }
            float m = -INFINITY, s = 0.f;
            bool ok = true;
            for (int64_t k = 0; k < nch && ok; ++k) {
                const uint32_t st = cnt % SA, ph = (cnt / SA) & 1u;
                ok = mbar_wait(&sm.fullA[st], ph, a.status, abort_flag);
                if (ok) {
                    const int nvec = (int)(min((int64_t)kPipeChunk, rowbytes - k * kPipeChunk) >> 4);
                    constexpr int U = (kPipeChunkVec + TA - 1) / TA;
                    uint4 x[U];
#pragma unroll
                    for (int u = 0; u < U; ++u) {
                        const int v = ta + u * TA;
                        x[u] = v < nvec ? sm.ringA[st][v] : neg_inf4();
                    }
                    __syncwarp();                   // the stage is in registers: hand it back
                    if (lane == 0) mbar_arrive(&sm.emptyA[st]);
                    const float bm = tree_max(x);
                    if (bm != -INFINITY) {
                        const float mn = fmaxf(m, bm);
                        const float acc = tree_exp_sum(x, c1, mn * c1);
                        s = (s == 0.f) ? acc : fmaf(s, ex2((m - mn) * c1), acc);
                        m = mn;
                    }
                } else {
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&sm.emptyA[st]);
                }
                ++cnt;
            }
            if (ok && tailn && ta == 0) {   // the last, partial vector
                uint4 x[1] = {tailx};
                mask_tail(x[0], tailn);
                const float bm = tree_max(x);
                const float mn = fmaxf(m, bm);
                const float acc = tree_exp_sum(x, c1, mn * c1);
                s = (s == 0.f) ? acc : fmaf(s, ex2((m - mn) * c1), acc);
                m = mn;
            }
            warp_lse_merge(m, s, c1);
            // Hand the warp's partial to the finishing warp (its slot of this
            // row parity is free once that warp merged the row two rows back).
            if (!ok) break;
            if (lane == 0) {
                const uint32_t q = li & 1u;
                if (mbar_wait(&sm.wempty[q], ((li >> 1) & 1u) ^ 1u, a.status, abort_flag)) {
                    sm.wpart[q][wa] = make_float2(m, s);
                    mbar_arrive(&sm.wfull[q]);
                }
            }
            __syncwarp();
            ++li;
        }
        return;
    }

    // ---- group B: pass 2 over every row of the CTA, in order ------------------
    const int tb = threadIdx.x - 32 * (A0 + NA);
    constexpr int64_t kPipeChunk = CVB * 16;
    constexpr int kPipeChunkVec = CVB;
    const int64_t nch = (rowbytes + kPipeChunk - 1) / kPipeChunk;
    uint32_t cnt = 0, li = 0;
    const RowSeq<P> seq(a.N, list, nlist, nlive);
    int64_t rn = seq.row(0);
    float w_next = a.w[rn];
    int id_next = a.ids[rn];
    for (int64_t j = 0; j < seq.len(); ++j) {
        const int64_t row = rn;
        const float wk = w_next;
        const int id = id_next;
        rn = seq.row(j + 1);
        if (rn >= 0) {
            w_next = a.w[rn];
            id_next = a.ids[rn];
        }
        if (row < 0) continue;
        uint4* drow = reinterpret_cast<uint4*>(a.dlogits + row * a.ld);
        if (!(wk != 0.f && id >= 0 && id < V)) {
            for (int64_t vi = tb; vi < V8; vi += TB) store_vec(drow, vi, make_uint4(0, 0, 0, 0), V8, tailn);
            if (tb == 0) {
                write_masked_outputs(a, row);
                if (wk != 0.f) flag_status(a.status, LEAP_DEV_BAD_ID);
            }
            continue;
        }
        uint4 tailx = make_uint4(0, 0, 0, 0);   // the partial last vector, loaded ahead of its use
        if (tailn && tb == 0) tailx = ld_stream(reinterpret_cast<const uint4*>(a.logits + row * a.ld) + V8f);
        const uint32_t q = li & 1u;
        if (!mbar_wait(&sm.kcfull[q], (li >> 1) & 1u, a.status, abort_flag)) break;
        const float2 kc = sm.kc[q];
        const float K = kc.x, coef = kc.y;
        const int64_t yv = id >> 3;
        const int ylane = id & 7;
        bool ok = true;
        for (int64_t k = 0; k < nch && ok; ++k) {
            const uint32_t st = cnt % SB, ph = (cnt / SB) & 1u;
            ok = mbar_wait(&sm.fullB[st], ph, a.status, abort_flag);
            if (ok) {
                const int nvec = (int)(min((int64_t)kPipeChunk, rowbytes - k * kPipeChunk) >> 4);
                constexpr int U = (kPipeChunkVec + TB - 1) / TB;
                const int64_t g0 = k * kPipeChunkVec;
                uint4 x[U];
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    const int v = tb + u * TB;
                    x[u] = v < nvec ? sm.ringB[st][v] : make_uint4(0, 0, 0, 0);
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(&sm.emptyB[st]);
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    const int v = tb + u * TB;
                    if (v < nvec) {
                        const int64_t gv = g0 + v;
                        const uint4 d = (coef == 0.f) ? make_uint4(0, 0, 0, 0)
                                                      : dlogit8(x[u], c1, K, coef, gv == yv ? ylane : -1);
                        st_stream(drow + gv, d);
                    }
                }
            } else {
                __syncwarp();
                if (lane == 0) mbar_arrive(&sm.emptyB[st]);
            }
            ++cnt;
        }
        if (ok && tailn && tb == 0) {
            const uint4 d = (coef == 0.f) ? make_uint4(0, 0, 0, 0)
                                          : dlogit8(tailx, c1, K, coef, yv == V8f ? ylane : -1);
            store_vec(drow, V8f, d, V8, tailn);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&sm.kcempty[q]);
        if (!ok) break;
        ++li;
    }
}

template <int NA, int NB, int SA, int SB, int CVA, int CVB, int P = 1>
cudaError_t launch_pipe_cfg(const RowArgs& a, cudaStream_t s) {
    auto kern = fused_loss_pipe_kernel<NA, NB, SA, SB, CVA, CVB, P>;
    const size_t dyn = sizeof(PipeSmem<NA, SA, SB, CVA, CVB>);
    static_assert(sizeof(PipeSmem<NA, SA, SB, CVA, CVB>) <= 232448, "dynamic shared memory above 227 KB");
    static std::mutex mu;
    static int done_dev = -1;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    {
        std::lock_guard<std::mutex> lk(mu);
        if (done_dev != dev) {
            e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
            if (e != cudaSuccess) return e;
            done_dev = dev;
        }
    }
    const int64_t grid = std::min<int64_t>(a.N, (int64_t)device_sm_count());
    kern<<<(unsigned)grid, 32 * (3 + NA + NB), dyn, s>>>(a);
    return cudaGetLastError();
}

// Measured on the single-turn workload (32,768 rows, V = 151,936; fraction of
// the copy peak; the two-pass kernel without the pipeline 0.882 beside it).
// Before the per-row scalars were loaded a row ahead:
//   ring B depth (A 4 stages): 8 -> 0.835, 9 -> 0.853; (A 3 stages) 10 -> 0.906,
//   11 -> 0.910: pass 2's re-reads want the deep ring;
//   ring A depth (B 10-11): 2 -> 0.824, 3 -> 0.906-0.910, 4 -> 0.867: three
//   16 KB copies in flight per SM keep pass 1 at its share of HBM, more only
//   crowd pass 2's copies;
//   chunks of 8 / 12 / 20 KB at the same ring bytes: 0.81-0.87 / 0.87-0.90 / 0.874;
//   group A of 4 / 8 warps: 0.914 / 0.910; group B of 4 / 8 / 12 / 16 warps
//   (A 4-8): 0.734 / 0.910-0.914 / 0.911 / 0.900;
//   L2 policy of the pass-1 copies evict_last / normal: 0.910 / 0.909; of
//   the pass-2 copies evict_first / normal: 0.910 / 0.891;
//   pass 2 loading its row from L2 into registers (16-24 warps, 4-8 vectors
//   in flight each) instead of through ring B: 0.69-0.77.
// With them (this configuration 0.928-0.930):
//   A / B stages 4 / 10, 2 / 12, 5 / 9: 0.891, 0.836, 0.825; A of 8 warps
//   0.922, B of 12 warps 0.923; ring A of 8 KB x 5-6 or 32 KB x 2 chunks:
//   0.867-0.896; ring B of 24 KB x 7 chunks: 0.927.
// A finishing warp taking the row-end merge and loss off group A (which no
// longer meets at a block barrier per row): 0.926 -> 0.931 (4 / 10 stages
// with it 0.840, group A of 8 warps 0.918), but the multi-turn step (long
// masked runs) 0.904 -> 0.890 as pass 1 ran further ahead of pass 2; with
// pass 1's lead bounded to two rows of queue: 0.933 and 0.910.
// Rows visited as P interleaved streams (RowSeq): P = 1 / 2 / 4 single-turn
// 0.933 / 0.930 / 0.922, multi-turn 0.907 / 0.923 / 0.923; P = 2 is the
// LEAP_LOSS_INTERLEAVED_ROWS hint, P = 1 the default.
constexpr int kPipeWarpsA = 4, kPipeWarpsB = 8, kPipeStagesA = 3, kPipeStagesB = 11;
constexpr int kPipeChunkVectors = 1024;   // 16 KB per staged chunk

}  // namespace

cudaError_t launch_pipe_loss(const RowArgs& a, cudaStream_t s) {
    if (a.N == 0) return cudaSuccess;
    if (a.row_streams == 2)
        return launch_pipe_cfg<kPipeWarpsA, kPipeWarpsB, kPipeStagesA, kPipeStagesB, kPipeChunkVectors,
                               kPipeChunkVectors, 2>(a, s);
    return launch_pipe_cfg<kPipeWarpsA, kPipeWarpsB, kPipeStagesA, kPipeStagesB, kPipeChunkVectors,
                           kPipeChunkVectors>(a, s);
}

}  // namespace leap
