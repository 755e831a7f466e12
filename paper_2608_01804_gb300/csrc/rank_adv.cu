// Rank-based advantages (Sec. 3.1 Eqs. 1-2, Sec. 3.2 Eqs. 4-6 + GRPO step,
// Sec. 3.3 discount) and the per-token scatter of the turn advantages.
//
// One warp per rollout group.  In the generic kernel lane l owns rollouts
// l, l + 32, ...; in the pair kernel (the paper's comparator, G even and at
// most 64) it owns 2l and 2l + 1.  Because the paper's comparator looks only
// at the tier r in [0, M], the O(G^2) tournament of Eq. 5 collapses to a walk
// over the M + 1 tiers: N_worse = #peers in lower tiers, N_better = #peers in
// higher tiers, each tier counted with warp ballots, so the whole group stays
// in registers.
#include "leap_common.cuh"
#include "leap_internal.h"

#include <algorithm>
#include <math.h>

namespace leap {
namespace {

constexpr int kMaxM = 8;

// Sum over aligned segments of W lanes (W = 32: the warp; W = 16: each half).
template <int W = 32>
__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
    for (int o = W / 2; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Per-warp running counters (lane 0), reduced per block then added atomically;
// the order of leap_rank_stats_t: 9 scalars, passes by turn, the rollout
// composition [bucket][type][sign], groups per bucket.
constexpr int kPassBuckets = 10;
constexpr int kCompBase = 9 + kMaxM;
constexpr int kBucketBase = kCompBase + kPassBuckets * 6;
constexpr int kNumStats = kBucketBase + kPassBuckets;

// Eq. 6 and the advantage of every rollout the lane holds: the tournament
// reward with the GRPO step, or the static-scalar baseline reward.  A group
// spans W aligned lanes (32, or 16 when a warp holds two groups).
template <int J, int W = 32>
__device__ __forceinline__ void group_reward(const RankArgs& a, int G, int M, const int (&d)[J], const int (&r)[J],
                                             const bool (&valid)[J], int dd, float (&Rv)[J], float (&Av)[J]) {
    const float gm1 = (float)(G - 1);
    const float den = a.std_unbiased ? gm1 : (float)G;
    if (a.reward == 0) {
        // GRPO standardisation of the tournament reward.  mean_g R = 0
        // exactly (every strict pair adds +1 and -1 to the net scores), so
        // A_i = d_i / ((G - 1)(std + eps)) with (G - 1) std = sqrt(sum d^2 / den).
        // fp32 with IEEE division and square root: at most ~3.5 ulp on A.
        float inv_scale = 0.f;  // all-tied group: no preference signal, A = 0
        if (a.norm == 0 && dd != 0) inv_scale = 1.f / (sqrtf((float)dd / den) + gm1 * a.eps_std);
#pragma unroll
        for (int j = 0; j < J; ++j) {
            Rv[j] = (float)d[j] / gm1;  // correctly rounded
            Av[j] = (a.norm == 1) ? Rv[j] : (float)d[j] * inv_scale;
        }
    } else {
        // Static-scalar baseline reward, standard GRPO with its own mean.
        float sum = 0.f, lo = 2.f, hi = -1.f;
#pragma unroll
        for (int j = 0; j < J; ++j) {
            Rv[j] = (r[j] == M) ? 1.f : ((r[j] > 0) ? a.static_c : 0.f);
            if (valid[j]) {
                sum += Rv[j];
                lo = fminf(lo, Rv[j]);
                hi = fmaxf(hi, Rv[j]);
            }
        }
        const float mean = warp_sum_f<W>(sum) / (float)G;
#pragma unroll
        for (int o = W / 2; o > 0; o >>= 1) {
            lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
            hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
        }
        float ss = 0.f;
#pragma unroll
        for (int j = 0; j < J; ++j)
            if (valid[j]) ss += (Rv[j] - mean) * (Rv[j] - mean);
        const float stdv = sqrtf(warp_sum_f<W>(ss) / den);
#pragma unroll
        for (int j = 0; j < J; ++j)
            Av[j] = (a.norm == 1) ? Rv[j] : ((hi == lo) ? 0.f : (Rv[j] - mean) / (stdv + a.eps_std));
    }
}

// Training-observability counters of one group (Table 5, Sec. 4.3; Table 2,
// Sec. 4.2) and its rollout composition (Fig. 4, Sec. 4.5), added to the
// warp's row of shared-memory counters by lane 0.  MB: a bound on M known at
// compile time (passes at turns above it cannot occur).  The composition
// bucket is the group's first-turn pass rate, min(9, 10 (G - N_fail) div G);
// a rollout with A != 0 counts by type (r = M immediate pass, 0 < r < M
// debug-assisted pass, r = 0 failure) and by the sign of A.
template <int J, int MB = kMaxM>
__device__ __forceinline__ void group_stats(long long* cnt, int G, int M, bool gate, int n_fail,
                                            const bool (&valid)[J], const bool (&bad)[J], const int (&pt0)[J],
                                            const int (&T)[J], const int (&r)[J], const float (&Av)[J],
                                            int lane) {
    int nonzero = 0, first = 0, later = 0, failed_on = 0, turns = 0;
    int by_turn[kMaxM];
    int comp[6];
#pragma unroll
    for (int m = 0; m < kMaxM; ++m) by_turn[m] = 0;
#pragma unroll
    for (int c = 0; c < 6; ++c) comp[c] = 0;
#pragma unroll
    for (int j = 0; j < J; ++j) {
        const bool ok = valid[j] && !bad[j];
        const int pt = pt0[j];
        nonzero += __popc(__ballot_sync(0xffffffffu, valid[j] && Av[j] != 0.f));
        first += __popc(__ballot_sync(0xffffffffu, ok && pt == 1));
        later += __popc(__ballot_sync(0xffffffffu, ok && gate && pt >= 2));
        failed_on += __popc(__ballot_sync(0xffffffffu, ok && gate && pt != 1));
        turns += __reduce_add_sync(0xffffffffu, valid[j] ? T[j] : 0);
#pragma unroll
        for (int m = 1; m < MB; ++m)
            by_turn[m] += __popc(__ballot_sync(0xffffffffu, ok && gate && pt == m + 1));
        // Composition category (type * 2 + sign), -1 for A == 0.
        const int kind = (r[j] == M) ? 0 : ((r[j] > 0) ? 1 : 2);
        const int cat = (valid[j] && Av[j] != 0.f) ? kind * 2 + (Av[j] < 0.f ? 1 : 0) : -1;
#pragma unroll
        for (int c = 0; c < 6; ++c) comp[c] += __popc(__ballot_sync(0xffffffffu, cat == c));
    }
    if (lane == 0) {
        long long* c = cnt;
        c[0] += 1;
        c[1] += gate;
        c[2] += G;
        c[3] += nonzero;
        c[4] += first;
        c[5] += later;
        c[6] += (later > 0);
        c[7] += failed_on;
        c[8] += turns;
        c[9] += first;
#pragma unroll
        for (int m = 1; m < kMaxM; ++m) c[9 + m] += by_turn[m];
        const int bucket = min(kPassBuckets - 1, (kPassBuckets * (G - n_fail)) / G);
#pragma unroll
        for (int k = 0; k < 6; ++k) c[kCompBase + bucket * 6 + k] += comp[k];
        c[kBucketBase + bucket] += 1;
    }
    __syncwarp();
}

// group_stats for a warp holding two groups of 64 (lanes 0-15 the first,
// 16-31 the second; J = 4 rollouts per lane): each lane counts its own
// rollouts, and one warp reduction adds two counters for both groups at once
// (8-bit fields: a group holds at most 64), so a counter costs half a
// reduction instead of J ballots.  The running totals stay in registers:
// the scalar counters in every lane (warp-uniform), the Fig. 4 counters of
// pass-rate bucket b in lane b; quad_stats_flush writes them to the warp's
// shared-memory row once.  A warp sees at most 2^31 / (4 x 64) groups per
// launch, so 32-bit totals cannot overflow.
template <int MB>
struct QuadStats {
    uint32_t sc[9 + MB];   // leap_rank_stats_t's scalar counters, in its order (passes at turns <= MB)
    uint32_t bk[7];        // this lane's bucket: composition [type][sign], then groups
};

template <int MB>
__device__ __forceinline__ void group_stats_quad(QuadStats<MB>& q, int M, bool gate, int n_fail, bool own,
                                                 const bool (&valid)[4], const bool (&bad)[4], const int (&pt0)[4],
                                                 const int (&T)[4], const int (&r)[4], const float (&Av)[4],
                                                 int lane) {
    constexpr int G = 64;
    constexpr int NC = 10 + (MB - 1);   // nonzero, first, later, failed_on, comp[6], by_turn[1..MB-1]
    int loc[NC];
#pragma unroll
    for (int c = 0; c < NC; ++c) loc[c] = 0;
    int turns = 0;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const bool ok = valid[j] && !bad[j];
        const int pt = pt0[j];
        const bool nz = valid[j] && Av[j] != 0.f;
        loc[0] += nz;
        loc[1] += ok && pt == 1;
        loc[2] += ok && gate && pt >= 2;
        loc[3] += ok && gate && pt != 1;
        const int kind = (r[j] == M) ? 0 : ((r[j] > 0) ? 1 : 2);
        const int cat = nz ? kind * 2 + (Av[j] < 0.f ? 1 : 0) : -1;
#pragma unroll
        for (int c = 0; c < 6; ++c) loc[4 + c] += (cat == c);
#pragma unroll
        for (int m = 1; m < MB; ++m) loc[9 + m] += ok && gate && pt == m + 1;
        turns += valid[j] ? T[j] : 0;
    }
    const int half = lane >> 4;
    int tot[2][NC];
#pragma unroll
    for (int c = 0; c < NC; c += 2) {
        const unsigned v = ((unsigned)loc[c] << (8 * half)) |
                           (c + 1 < NC ? ((unsigned)loc[c + 1] << (16 + 8 * half)) : 0u);
        const unsigned s2 = __reduce_add_sync(0xffffffffu, v);
        tot[0][c] = (int)(s2 & 0xffu);
        tot[1][c] = (int)((s2 >> 8) & 0xffu);
        if (c + 1 < NC) {
            tot[0][c + 1] = (int)((s2 >> 16) & 0xffu);
            tot[1][c + 1] = (int)(s2 >> 24);
        }
    }
    const unsigned ts = __reduce_add_sync(0xffffffffu, (unsigned)turns << (16 * half));
    const bool gate1 = __shfl_sync(0xffffffffu, gate, 16);
    const int n_fail1 = __shfl_sync(0xffffffffu, n_fail, 16);
    const bool own1 = __shfl_sync(0xffffffffu, own, 16);
    const bool gate0 = __shfl_sync(0xffffffffu, gate, 0);
    const int n_fail0 = __shfl_sync(0xffffffffu, n_fail, 0);
    const bool own0 = __shfl_sync(0xffffffffu, own, 0);
#pragma unroll
    for (int g = 0; g < 2; ++g) {
        if (!(g ? own1 : own0)) continue;
        const bool gt = g ? gate1 : gate0;
        const int nf = g ? n_fail1 : n_fail0;
        const int* t = tot[g];
        q.sc[0] += 1;
        q.sc[1] += gt;
        q.sc[2] += G;
        q.sc[3] += t[0];
        q.sc[4] += t[1];
        q.sc[5] += t[2];
        q.sc[6] += (t[2] > 0);
        q.sc[7] += t[3];
        q.sc[8] += g ? (ts >> 16) : (ts & 0xffffu);
        q.sc[9] += t[1];
#pragma unroll
        for (int m = 1; m < MB; ++m) q.sc[9 + m] += t[9 + m];
        if (lane == min(kPassBuckets - 1, (kPassBuckets * (G - nf)) / G)) {
#pragma unroll
            for (int k = 0; k < 6; ++k) q.bk[k] += t[4 + k];
            q.bk[6] += 1;
        }
    }
}

// The warp's running counters into its row of shared-memory counters.
template <int MB>
__device__ __forceinline__ void quad_stats_flush(const QuadStats<MB>& q, long long* cnt, int lane) {
    if (lane == 0)
        for (int k = 0; k < kCompBase; ++k) cnt[k] = k < 9 + MB ? (long long)q.sc[k] : 0;
    if (lane < kPassBuckets) {
        for (int k = 0; k < 6; ++k) cnt[kCompBase + lane * 6 + k] = q.bk[k];
        cnt[kBucketBase + lane] = q.bk[6];
    }
    __syncwarp();
}

// One rollout's outcome fields: malformed (pass_turn outside [0, M], turns
// outside [1, M], a pass after the last generated turn) or well formed, and
// whether it failed its first turn (Eq. 1; a malformed outcome counts as
// failed).  pt0 is the pass turn with malformed outcomes mapped to 0.
__device__ __forceinline__ void decode_outcome(int pt, int nt, int M, bool valid, bool& bad, bool& fail1, int& pt0) {
    bad = valid && (pt < 0 || pt > M || nt < 1 || nt > M || (pt >= 1 && pt > nt));
    fail1 = valid && (bad || pt != 1);
    pt0 = (valid && !bad) ? pt : 0;
}

// Tier rule of Sec. 3.2 (r = M - m + 1 for a pass at turn m, 0 for a fail)
// and the turns that count; gated-off groups ran turn 1 only.
__device__ __forceinline__ void tier_rule(int pt, int nt, bool valid, bool bad, bool gate, int M, int& r, int& T) {
    if (!valid || bad) {
        r = 0;
        T = 0;
    } else if (!gate) {
        r = (pt == 1) ? M : 0;
        T = 1;
    } else {
        r = (pt >= 1) ? (M - pt + 1) : 0;
        T = nt;
    }
}

// Adds the block's shared-memory counters to the caller's leap_rank_stats_t.
__device__ __forceinline__ void flush_stats(const RankArgs& a, long long (*sst)[kNumStats]) {
    __syncthreads();
    if (threadIdx.x < kNumStats) {
        long long v = 0;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) v += sst[w][threadIdx.x];
        if (v) atomicAdd(reinterpret_cast<unsigned long long*>(a.stats) + threadIdx.x, (unsigned long long)v);
    }
}

// Blocks of 256 threads per SM the register budget is cut for (measured: 4
// for the generic kernel with J <= 2, 6 for the pair kernel).
constexpr int kRankMinBlocks = 4;
constexpr int kPairMinBlocks = 6;
constexpr int kPairLexiMinBlocks = 4;   // the tie-broken comparator: keys and peer loops need registers
template <int J, bool LEXI>  // rollouts per lane: G <= 32 * J; tie-broken comparator
__global__ void __launch_bounds__(256, (J <= 2 ? kRankMinBlocks : 1)) rank_adv_kernel(RankArgs a) {
    const int lane = threadIdx.x & 31;
    const int wib = threadIdx.x >> 5;
    const int G = a.G, M = a.M;
    constexpr bool lexi = LEXI;
    const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
    __shared__ long long sst[8][kNumStats];  // per-warp counters (only with a.stats)
    if (a.stats) {
        for (int k = lane; k < kNumStats; k += 32) sst[wib][k] = 0;
        __syncwarp();
    }

    for (int64_t group = (int64_t)blockIdx.x * (blockDim.x >> 5) + wib; group < a.num_groups; group += warps) {
        const int64_t base = group * G;
        int r[J], T[J], pt0[J], tk[J];
        float sp[J];
        bool valid[J], bad[J];
        int n_fail = 0;
#pragma unroll
        for (int j = 0; j < J; ++j) {
            const int i = lane + 32 * j;
            valid[j] = i < G;
            int pt = 0, nt = 1;
            sp[j] = 0.f;
            tk[j] = 0;
            if (valid[j]) {
                pt = a.pass_turn[base + i];
                nt = a.num_turns[base + i];
                if (lexi) {
                    sp[j] = a.speedup[base + i];
                    tk[j] = a.ntokens[base + i];
                }
            }
            bool fail1;
            decode_outcome(pt, nt, M, valid[j], bad[j], fail1, pt0[j]);
            n_fail += __popc(__ballot_sync(0xffffffffu, fail1));
            T[j] = nt;
        }
        // Eq. 2 (or the recorded gate).
        const bool gate = a.gate_in ? (a.gate_in[group] != 0) : (a.tau_min <= n_fail && n_fail <= a.tau_max);

#pragma unroll
        for (int j = 0; j < J; ++j) {
            tier_rule(pt0[j], T[j], valid[j], bad[j], gate, M, r[j], T[j]);
            if (bad[j]) flag_status(a.status, 2u);
        }

        // Eq. 5: N_worse / N_better.
        int nw[J], nb[J];
        if constexpr (!lexi) {
            // The paper's comparator looks only at r: walk the M + 1 tiers in
            // order, counting each tier's members with ballots; a rollout of
            // tier b has `below` peers strictly worse and c - 1 tied.
            int eq[J];
#pragma unroll
            for (int j = 0; j < J; ++j) nw[j] = eq[j] = 0;
            int below = 0;
            for (int b = 0; b <= M; ++b) {
                int c = 0;
#pragma unroll
                for (int j = 0; j < J; ++j) c += __popc(__ballot_sync(0xffffffffu, valid[j] && r[j] == b));
#pragma unroll
                for (int j = 0; j < J; ++j) {
                    if (r[j] == b) {
                        nw[j] = below;
                        eq[j] = c;
                    }
                }
                below += c;
            }
#pragma unroll
            for (int j = 0; j < J; ++j) nb[j] = below - nw[j] - eq[j];  // below == G here
        } else {
            // Tie-broken comparator: every rollout against every peer.  The
            // keys of 32 peers at a time are staged in the warp's slice of
            // shared memory and read back as broadcasts.
            __shared__ int4 lkeys[8][32];
#pragma unroll
            for (int j = 0; j < J; ++j) nw[j] = nb[j] = 0;
            bool keyed = false;
            if constexpr (J <= 8) {  // larger groups keep their registers for the peer loop
                bool nan_key = false;
#pragma unroll
                for (int j = 0; j < J; ++j) nan_key |= valid[j] && r[j] > 0 && isnan(sp[j]);
                keyed = !__any_sync(0xffffffffu, nan_key);
            }
            if (keyed) {
                // Without NaN the order within a tier is total: each passing
                // rollout gets one 64-bit key (speedup, -tokens) that orders
                // exactly as the comparator's tie-breaks.  Peers in other
                // tiers are counted from the tier histogram (failures tie
                // whatever their speedup and tokens); the keys of a tier are
                // gathered into consecutive slots of the warp's shared memory,
                // so each passing rollout compares itself only with its own
                // tier (strict comparisons skip itself).
                if constexpr (J <= 8) {
                    __shared__ unsigned long long tkeys[8][32 * J];
                    unsigned long long key[J];
#pragma unroll
                    for (int j = 0; j < J; ++j) {
                        const unsigned b = __float_as_uint(sp[j] + 0.f);   // -0 -> +0, equal as floats
                        const unsigned o = (b & 0x80000000u) ? ~b : (b | 0x80000000u);
                        key[j] = ((unsigned long long)o << 32) | ~((unsigned)tk[j] ^ 0x80000000u);
                    }
                    const unsigned lt = (1u << lane) - 1u;
                    int lo[J], cnt[J], pos[J];
#pragma unroll
                    for (int j = 0; j < J; ++j) lo[j] = cnt[j] = pos[j] = 0;
                    int below = 0;
                    for (int b = 0; b <= M; ++b) {   // tiers in order: slots below_b .. below_b + c_b
                        int pre = 0;
#pragma unroll
                        for (int j = 0; j < J; ++j) {
                            const bool in = valid[j] && r[j] == b;
                            const unsigned bal = __ballot_sync(0xffffffffu, in);
                            if (in) {
                                pos[j] = below + pre + __popc(bal & lt);
                                lo[j] = below;
                            }
                            pre += __popc(bal);
                        }
#pragma unroll
                        for (int j = 0; j < J; ++j)
                            if (valid[j] && r[j] == b) cnt[j] = pre;
                        below += pre;
                    }
                    __syncwarp();
#pragma unroll
                    for (int j = 0; j < J; ++j)
                        if (valid[j] && r[j] > 0) tkeys[wib][pos[j]] = key[j];
                    __syncwarp();
#pragma unroll
                    for (int j = 0; j < J; ++j) {
                        int win = 0, loss = 0;
                        if (valid[j] && r[j] > 0) {
                            for (int p = lo[j]; p < lo[j] + cnt[j]; ++p) {
                                const unsigned long long kp = tkeys[wib][p];
                                win += key[j] > kp;
                                loss += kp > key[j];
                            }
                        }
                        nw[j] = lo[j] + win;                       // every lower tier, then wins in the tier
                        nb[j] = (below - lo[j] - cnt[j]) + loss;   // every higher tier, then losses
                    }
                }
            } else {
                // A NaN speedup compares false both ways, and G > 256 keeps
                // the registers: the comparator itself, peer by peer.
#pragma unroll
                for (int sidx = 0; sidx < J; ++sidx) {
                    const int npeer = min(32, G - 32 * sidx);
                    if (npeer <= 0) break;
                    __syncwarp();
                    lkeys[wib][lane] = make_int4(r[sidx], __float_as_int(sp[sidx]), tk[sidx], 0);
                    __syncwarp();
                    for (int l = 0; l < npeer; ++l) {
                        const int4 kj = lkeys[wib][l];
                        const int rj = kj.x, tkj = kj.z;
                        const float spj = __int_as_float(kj.y);
                        const int jj = 32 * sidx + l;
#pragma unroll
                        for (int q = 0; q < J; ++q) {
                            if (!valid[q] || lane + 32 * q == jj) continue;
                            const bool tie_r = r[q] == rj && rj > 0;
                            nw[q] += (r[q] > rj) || (tie_r && (sp[q] > spj || (sp[q] == spj && tk[q] < tkj)));
                            nb[q] += (rj > r[q]) || (tie_r && (spj > sp[q] || (spj == sp[q] && tkj < tk[q])));
                        }
                    }
                }
            }
        }

        // Eq. 6 and the sum of squared net scores (exact: at most G (G - 1)^2 < 2^31).
        int d[J];
        int dd = 0;
#pragma unroll
        for (int j = 0; j < J; ++j) {
            d[j] = nw[j] - nb[j];
            if (valid[j]) {
                dd += d[j] * d[j];
                const int64_t i = base + lane + 32 * j;
                if (a.n_worse) a.n_worse[i] = nw[j];
                if (a.n_better) a.n_better[i] = nb[j];
                if (a.r_out) a.r_out[i] = (uint8_t)r[j];
                a.T_eff[i] = (uint8_t)T[j];
            }
        }
        dd = __reduce_add_sync(0xffffffffu, dd);

        float Rv[J], Av[J];
        group_reward<J>(a, G, M, d, r, valid, dd, Rv, Av);

#pragma unroll
        for (int j = 0; j < J; ++j) {
            if (!valid[j]) continue;
            const int64_t i = base + lane + 32 * j;
            if (a.R) a.R[i] = Rv[j];
            if (a.A) a.A[i] = Av[j];
            // Sec. 3.3: beta = gamma for A >= 0, else 1; last turn keeps A.
            const float beta = (Av[j] >= 0.f) ? a.gamma : 1.f;
            float* ta = a.turn_adv + i * M;
            float p = Av[j];
            for (int t = M - 1; t >= 0; --t) {
                if (t < T[j]) {
                    ta[t] = p;
                    p *= beta;
                } else {
                    ta[t] = 0.f;
                }
            }
        }
        if (lane == 0 && a.gate_out) a.gate_out[group] = gate ? 1 : 0;

        if (a.stats) group_stats<J>(sst[wib], G, M, gate, n_fail, valid, bad, pt0, T, r, Av, lane);
    }

    if (a.stats) flush_stats(a, sst);
}

// The common case as its own kernel: the paper's comparator, G even and at
// most 64, M known at compile time.  Lane l holds rollouts 2l and 2l + 1, so
// it reads both outcomes with one 2-byte load and writes every output of the
// pair with one vector store (the turn advantages as M float2), and the tier
// walk and the discount loops unroll.
template <int MC, bool LEXI = false>
__global__ void __launch_bounds__(256, LEXI ? kPairLexiMinBlocks : kPairMinBlocks) rank_pair_kernel(RankArgs a) {
    constexpr int J = 2, M = MC;
    const int lane = threadIdx.x & 31;
    const int wib = threadIdx.x >> 5;
    const int G = a.G;
    const bool own = 2 * lane < G;
    const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
    __shared__ long long sst[8][kNumStats];
    if (a.stats) {
        for (int k = lane; k < kNumStats; k += 32) sst[wib][k] = 0;
        __syncwarp();
    }

    for (int64_t group = (int64_t)blockIdx.x * (blockDim.x >> 5) + wib; group < a.num_groups; group += warps) {
        const int64_t i0 = group * G + 2 * lane;
        int pt[J] = {0, 0}, T[J] = {1, 1};
        float sp[J] = {0.f, 0.f};
        int tk[J] = {0, 0};
        if (own) {
            const unsigned p2 = *reinterpret_cast<const uint16_t*>(a.pass_turn + i0);
            const unsigned n2 = *reinterpret_cast<const uint16_t*>(a.num_turns + i0);
            pt[0] = (int8_t)(p2 & 0xffu);
            pt[1] = (int8_t)(p2 >> 8);
            T[0] = (int8_t)(n2 & 0xffu);
            T[1] = (int8_t)(n2 >> 8);
            if (LEXI) {
                const float2 s2 = *reinterpret_cast<const float2*>(a.speedup + i0);
                const int2 t2 = *reinterpret_cast<const int2*>(a.ntokens + i0);
                sp[0] = s2.x;
                sp[1] = s2.y;
                tk[0] = t2.x;
                tk[1] = t2.y;
            }
        }
        bool valid[J] = {own, own}, bad[J];
        int pt0[J], r[J];
        int fails = 0;
#pragma unroll
        for (int j = 0; j < J; ++j) {
            bool fail1;
            decode_outcome(pt[j], T[j], M, valid[j], bad[j], fail1, pt0[j]);
            fails += fail1;
        }
        const int n_fail = __reduce_add_sync(0xffffffffu, fails);
        const bool gate = a.gate_in ? (a.gate_in[group] != 0) : (a.tau_min <= n_fail && n_fail <= a.tau_max);
#pragma unroll
        for (int j = 0; j < J; ++j) {
            tier_rule(pt0[j], T[j], valid[j], bad[j], gate, M, r[j], T[j]);
            if (bad[j]) flag_status(a.status, 2u);
        }

        // Eq. 5 for the paper's comparator: the tier histogram as 8-bit
        // counters packed four to a word (a group holds at most 64), summed
        // over the warp with one reduction per word; the byte-wise prefix
        // (multiplication by 0x01010101) gives each tier its count of peers
        // in lower tiers.
        constexpr int W = (M + 4) / 4;   // words for the M + 1 tiers
        unsigned hist[W], pre[W];
#pragma unroll
        for (int w = 0; w < W; ++w) {
            unsigned mine = 0;
#pragma unroll
            for (int j = 0; j < J; ++j)
                if (own && (r[j] >> 2) == w) mine += 1u << (8 * (r[j] & 3));
            hist[w] = __reduce_add_sync(0xffffffffu, mine);
        }
        unsigned carry = 0;   // peers in the tiers of earlier words
#pragma unroll
        for (int w = 0; w < W; ++w) {
            pre[w] = hist[w] * 0x01010101u + carry * 0x01010101u;   // inclusive prefix per byte
            carry = pre[w] >> 24;
        }
        const int below = (int)carry;   // == G
        int nw[J], nb[J], d[J];
#pragma unroll
        for (int j = 0; j < J; ++j) {
            const int w = r[j] >> 2, k = r[j] & 3;
            unsigned hw = hist[0], pw = pre[0];
#pragma unroll
            for (int q = 1; q < W; ++q)
                if (w == q) {
                    hw = hist[q];
                    pw = pre[q];
                }
            const int eq = (int)((hw >> (8 * k)) & 0xffu);
            const int incl = (int)((pw >> (8 * k)) & 0xffu);   // peers in tiers <= r (this one included)
            nw[j] = incl - eq;
            nb[j] = below - incl;
            d[j] = nw[j] - nb[j];
        }
        if constexpr (LEXI) {
            // Tie-broken comparator (r, then speedup higher, then tokens
            // fewer): the counts above already hold every peer of another
            // tier; failures tie among themselves; within a passing tier the
            // keys decide.
            __shared__ unsigned long long tkeys[8][64];
            __shared__ int4 lkeys[8][64];
            bool nan_key = false;
#pragma unroll
            for (int j = 0; j < J; ++j) nan_key |= own && r[j] > 0 && isnan(sp[j]);
            if (!__any_sync(0xffffffffu, nan_key)) {
                // Without NaN the order within a tier is total: one 64-bit key
                // (speedup, -tokens) per passing rollout orders exactly as the
                // tie-breaks (-0 folded into +0); the keys of tier b fill its
                // slots [lower, lower + size) in the warp's shared memory.
                unsigned long long key[J];
#pragma unroll
                for (int j = 0; j < J; ++j) {
                    const unsigned b = __float_as_uint(sp[j] + 0.f);
                    const unsigned o = (b & 0x80000000u) ? ~b : (b | 0x80000000u);
                    key[j] = ((unsigned long long)o << 32) | ~((unsigned)tk[j] ^ 0x80000000u);
                }
                const unsigned lt = (1u << lane) - 1u;
                int lo[J] = {0, 0}, cnt[J] = {0, 0};
#pragma unroll
                for (int b = 1; b <= M; ++b) {
                    const unsigned b0 = __ballot_sync(0xffffffffu, own && r[0] == b);
                    const unsigned b1 = __ballot_sync(0xffffffffu, own && r[1] == b);
                    if (own && (r[0] == b || r[1] == b)) {
                        const int lower = r[0] == b ? nw[0] : nw[1];   // peers in lower tiers
                        const int size = __popc(b0) + __popc(b1);
                        if (r[0] == b) {
                            tkeys[wib][lower + __popc(b0 & lt)] = key[0];
                            lo[0] = lower;
                            cnt[0] = size;
                        }
                        if (r[1] == b) {
                            tkeys[wib][lower + __popc(b0) + __popc(b1 & lt)] = key[1];
                            lo[1] = lower;
                            cnt[1] = size;
                        }
                    }
                }
                __syncwarp();
#pragma unroll
                for (int j = 0; j < J; ++j) {
                    int win = 0, loss = 0;
                    if (own && r[j] > 0) {
                        for (int p = lo[j]; p < lo[j] + cnt[j]; ++p) {
                            const unsigned long long kp = tkeys[wib][p];
                            win += key[j] > kp;
                            loss += kp > key[j];
                        }
                    }
                    nw[j] += win;
                    nb[j] += loss;
                }
                __syncwarp();
            } else {
                // A NaN speedup compares false both ways: the comparator itself,
                // peer by peer, over the group's (tier, speedup, tokens).
#pragma unroll
                for (int j = 0; j < J; ++j) lkeys[wib][2 * lane + j] = make_int4(r[j], __float_as_int(sp[j]), tk[j], 0);
                __syncwarp();
#pragma unroll
                for (int j = 0; j < J; ++j) nw[j] = nb[j] = 0;
                for (int p = 0; p < G; ++p) {
                    const int4 kp = lkeys[wib][p];
                    const int rj = kp.x, tkj = kp.z;
                    const float spj = __int_as_float(kp.y);
#pragma unroll
                    for (int j = 0; j < J; ++j) {
                        if (!own || 2 * lane + j == p) continue;
                        const bool tie_r = r[j] == rj && rj > 0;
                        nw[j] += (r[j] > rj) || (tie_r && (sp[j] > spj || (sp[j] == spj && tk[j] < tkj)));
                        nb[j] += (rj > r[j]) || (tie_r && (spj > sp[j] || (spj == sp[j] && tkj < tk[j])));
                    }
                }
                __syncwarp();
            }
#pragma unroll
            for (int j = 0; j < J; ++j) d[j] = nw[j] - nb[j];
        }
        const int dd = __reduce_add_sync(0xffffffffu, own ? d[0] * d[0] + d[1] * d[1] : 0);

        float Rv[J], Av[J];
        group_reward<J>(a, G, M, d, r, valid, dd, Rv, Av);

        if (own) {
            if (a.n_worse) *reinterpret_cast<int2*>(a.n_worse + i0) = make_int2(nw[0], nw[1]);
            if (a.n_better) *reinterpret_cast<int2*>(a.n_better + i0) = make_int2(nb[0], nb[1]);
            if (a.r_out) *reinterpret_cast<uint16_t*>(a.r_out + i0) = (uint16_t)(r[0] | (r[1] << 8));
            *reinterpret_cast<uint16_t*>(a.T_eff + i0) = (uint16_t)(T[0] | (T[1] << 8));
            if (a.R) *reinterpret_cast<float2*>(a.R + i0) = make_float2(Rv[0], Rv[1]);
            if (a.A) *reinterpret_cast<float2*>(a.A + i0) = make_float2(Av[0], Av[1]);
            // Sec. 3.3: beta = gamma for A >= 0, else 1; the last counted turn keeps A.
            float tv[J][M];
#pragma unroll
            for (int j = 0; j < J; ++j) {
                const float beta = (Av[j] >= 0.f) ? a.gamma : 1.f;
                float p = Av[j];
#pragma unroll
                for (int t = M - 1; t >= 0; --t) {
                    tv[j][t] = (t < T[j]) ? p : 0.f;
                    if (t < T[j]) p *= beta;
                }
            }
            float2* ta = reinterpret_cast<float2*>(a.turn_adv + i0 * M);
#pragma unroll
            for (int q = 0; q < M; ++q)
                ta[q] = make_float2(tv[(2 * q) / M][(2 * q) % M], tv[(2 * q + 1) / M][(2 * q + 1) % M]);
        }
        if (lane == 0 && a.gate_out) a.gate_out[group] = gate ? 1 : 0;

        if (a.stats) group_stats<J, M>(sst[wib], G, M, gate, n_fail, valid, bad, pt0, T, r, Av, lane);
    }
    if (a.stats) flush_stats(a, sst);
}

// G = 64 with the paper's comparator (either reward, with or without the
// training counters): a warp takes two groups per iteration (128 consecutive
// rollouts), lane l holding rollouts 4l .. 4l + 3 (lanes 0-15 the first group,
// 16-31 the second).  Each outcome array is one 4-byte load and each output
// array one 16-byte store per lane (the turn advantages as M float4), and the
// two groups' sums share warp reductions (the failure counts packed in 16-bit
// halves, the tier histograms and squared net scores one reduction per group,
// the static reward's sums over half-warps, the counters two per reduction):
// half the memory instructions and loop overhead of the pair kernel per
// rollout.
// Blocks of 256 per SM the register budget is cut for: 4 without counters
// (64 registers); with them (the running totals take 9 + M + 7 registers) 3.
constexpr int kQuadMinBlocks = 4, kQuadStatsMinBlocks = 3;
template <int MC, bool STATS>
__global__ void __launch_bounds__(256, STATS ? kQuadStatsMinBlocks : kQuadMinBlocks) rank_quad_kernel(RankArgs a) {
    constexpr int J = 4, M = MC, G = 64;
    const int lane = threadIdx.x & 31;
    const int half = lane >> 4;

    const int64_t npairs = ((int64_t)a.num_groups + 1) / 2;
    const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
    const int wib = threadIdx.x >> 5;
    __shared__ long long sst[8][kNumStats];
    QuadStats<MC> qs;
    if (STATS) {
#pragma unroll
        for (int k = 0; k < 9 + MC; ++k) qs.sc[k] = 0;
#pragma unroll
        for (int k = 0; k < 7; ++k) qs.bk[k] = 0;
    }
    for (int64_t pr = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); pr < npairs; pr += warps) {
        const int64_t group = 2 * pr + half;
        const bool own = group < a.num_groups;   // the last pair may hold one group
        const int64_t i0 = group * G + 4 * (lane & 15);
        int pt[J], T[J];
        {
            unsigned p4 = 0u, n4 = 0x01010101u;
            if (own) {
                p4 = *reinterpret_cast<const uint32_t*>(a.pass_turn + i0);
                n4 = *reinterpret_cast<const uint32_t*>(a.num_turns + i0);
            }
#pragma unroll
            for (int j = 0; j < J; ++j) {
                pt[j] = (int8_t)((p4 >> (8 * j)) & 0xffu);
                T[j] = (int8_t)((n4 >> (8 * j)) & 0xffu);
            }
        }
        bool valid[J], bad[J];
        int pt0[J], r[J];
        int fails = 0;
#pragma unroll
        for (int j = 0; j < J; ++j) {
            valid[j] = own;
            bool fail1;
            decode_outcome(pt[j], T[j], M, valid[j], bad[j], fail1, pt0[j]);
            fails += fail1;
        }
        const unsigned both = __reduce_add_sync(0xffffffffu, (unsigned)fails << (16 * half));
        const int n_fail = (int)(half ? (both >> 16) : (both & 0xffffu));
        const bool gate = a.gate_in ? (own && a.gate_in[group] != 0) : (a.tau_min <= n_fail && n_fail <= a.tau_max);
#pragma unroll
        for (int j = 0; j < J; ++j) {
            tier_rule(pt0[j], T[j], valid[j], bad[j], gate, M, r[j], T[j]);
            if (bad[j]) flag_status(a.status, 2u);
        }

        // Eq. 5: the tier histogram of each group (8-bit counters, four tiers
        // to a word), then the byte-wise prefix as in the pair kernel.
        constexpr int W = (M + 4) / 4;
        unsigned hist[W], pre[W];
#pragma unroll
        for (int w = 0; w < W; ++w) {
            unsigned mine = 0;
#pragma unroll
            for (int j = 0; j < J; ++j)
                if (own && (r[j] >> 2) == w) mine += 1u << (8 * (r[j] & 3));
            const unsigned h0 = __reduce_add_sync(0xffffffffu, half ? 0u : mine);
            const unsigned h1 = __reduce_add_sync(0xffffffffu, half ? mine : 0u);
            hist[w] = half ? h1 : h0;
        }
        unsigned carry = 0;
#pragma unroll
        for (int w = 0; w < W; ++w) {
            pre[w] = hist[w] * 0x01010101u + carry * 0x01010101u;
            carry = pre[w] >> 24;
        }
        const int below = (int)carry;   // == G
        int nw[J], nb[J], d[J];
        int dsq = 0;
#pragma unroll
        for (int j = 0; j < J; ++j) {
            const int w = r[j] >> 2, k = r[j] & 3;
            unsigned hw = hist[0], pw = pre[0];
#pragma unroll
            for (int q = 1; q < W; ++q)
                if (w == q) {
                    hw = hist[q];
                    pw = pre[q];
                }
            const int eq = (int)((hw >> (8 * k)) & 0xffu);
            const int incl = (int)((pw >> (8 * k)) & 0xffu);
            nw[j] = incl - eq;
            nb[j] = below - incl;
            d[j] = nw[j] - nb[j];
            dsq += d[j] * d[j];
        }
        if (!own) dsq = 0;
        const int dd0 = __reduce_add_sync(0xffffffffu, half ? 0 : dsq);
        const int dd1 = __reduce_add_sync(0xffffffffu, half ? dsq : 0);
        const int dd = half ? dd1 : dd0;

        float Rv[J], Av[J];
        group_reward<J, 16>(a, G, M, d, r, valid, dd, Rv, Av);

        if (own) {
            if (a.n_worse) *reinterpret_cast<int4*>(a.n_worse + i0) = make_int4(nw[0], nw[1], nw[2], nw[3]);
            if (a.n_better) *reinterpret_cast<int4*>(a.n_better + i0) = make_int4(nb[0], nb[1], nb[2], nb[3]);
            if (a.r_out)
                *reinterpret_cast<uint32_t*>(a.r_out + i0) =
                    (uint32_t)r[0] | ((uint32_t)r[1] << 8) | ((uint32_t)r[2] << 16) | ((uint32_t)r[3] << 24);
            *reinterpret_cast<uint32_t*>(a.T_eff + i0) =
                (uint32_t)T[0] | ((uint32_t)T[1] << 8) | ((uint32_t)T[2] << 16) | ((uint32_t)T[3] << 24);
            if (a.R) *reinterpret_cast<float4*>(a.R + i0) = make_float4(Rv[0], Rv[1], Rv[2], Rv[3]);
            if (a.A) *reinterpret_cast<float4*>(a.A + i0) = make_float4(Av[0], Av[1], Av[2], Av[3]);
            // Sec. 3.3: beta = gamma for A >= 0, else 1; the last counted turn keeps A.
            float tv[J * M];
#pragma unroll
            for (int j = 0; j < J; ++j) {
                const float beta = (Av[j] >= 0.f) ? a.gamma : 1.f;
                float p = Av[j];
#pragma unroll
                for (int t = M - 1; t >= 0; --t) {
                    tv[j * M + t] = (t < T[j]) ? p : 0.f;
                    if (t < T[j]) p *= beta;
                }
            }
            float4* ta = reinterpret_cast<float4*>(a.turn_adv + i0 * M);
#pragma unroll
            for (int q = 0; q < M; ++q) ta[q] = make_float4(tv[4 * q], tv[4 * q + 1], tv[4 * q + 2], tv[4 * q + 3]);
            if ((lane & 15) == 0 && a.gate_out) a.gate_out[group] = gate ? 1 : 0;
        }
        if (STATS) group_stats_quad<M>(qs, M, gate, n_fail, own, valid, bad, pt0, T, r, Av, lane);
    }
    if (STATS) {
        quad_stats_flush(qs, sst[wib], lane);
        flush_stats(a, sst);
    }
}

template <int MC>
cudaError_t launch_quad(const RankArgs& a, cudaStream_t s) {
    const int warps = 8;
    const int64_t pairs = ((int64_t)a.num_groups + 1) / 2;
    const int per_sm = a.stats ? kQuadStatsMinBlocks : kQuadMinBlocks;
    const int64_t blocks = std::min<int64_t>((pairs + warps - 1) / warps, (int64_t)device_sm_count() * per_sm);
    if (a.stats) rank_quad_kernel<MC, true><<<(unsigned)blocks, warps * 32, 0, s>>>(a);
    else rank_quad_kernel<MC, false><<<(unsigned)blocks, warps * 32, 0, s>>>(a);
    return cudaGetLastError();
}

template <int J>
cudaError_t launch_rank_j(const RankArgs& a, cudaStream_t s) {
    const int warps = 8;
    int64_t blocks = ((int64_t)a.num_groups + warps - 1) / warps;
    // With counters, fewer blocks loop over the groups: one atomic set per block.
    if (a.stats) blocks = std::min<int64_t>(blocks, (int64_t)device_sm_count() * 16);
    if (a.cmp == 1) rank_adv_kernel<J, true><<<(unsigned)blocks, warps * 32, 0, s>>>(a);
    else rank_adv_kernel<J, false><<<(unsigned)blocks, warps * 32, 0, s>>>(a);
    return cudaGetLastError();
}

// ---- per-rollout token counts --------------------------------------------

__global__ void zero_counts_kernel(int32_t* L, int32_t n, int64_t* totals) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        L[i] = 0;
    if (blockIdx.x == 0 && threadIdx.x < 2) totals[threadIdx.x] = 0;
}

// Validates segment s; returns false (and flags) when it is malformed.
__device__ __forceinline__ bool segment_ok(const SegArgs& a, int64_t s, int32_t& lo, int32_t& hi,
                                           int32_t& i, int32_t& t) {
    lo = a.seg_offsets[s];
    hi = a.seg_offsets[s + 1];
    t = a.seg_turn[s];
    i = a.seg_rollout[s];
    const bool ok = lo >= 0 && hi >= lo && (int64_t)hi <= a.N && t < a.M &&
                    (t < 0 || (i >= 0 && i < a.n_rollouts));
    return ok;
}

__global__ void segment_count_kernel(SegArgs a) {
    const int64_t s = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (s >= a.num_segs) return;
    int32_t lo, hi, i, t;
    if (!segment_ok(a, s, lo, hi, i, t)) {
        flag_status(a.status, 4u);
        return;
    }
    if (t < 0 || hi == lo) return;
    if (t < (int)a.T_eff[i]) atomicAdd(&a.L_out[i], hi - lo);
}

// The whole count in one launch when the per-rollout counters fit in shared
// memory: one block zeroes them there, adds every segment with shared-memory
// atomics, then writes L and the two totals (block barriers instead of three
// dependent launches).
constexpr int kCountThreads = 1024;
constexpr int kCountSmemRollouts = 12000;   // int32 counters within the 48 KB of static shared memory

__global__ void __launch_bounds__(kCountThreads) counts_one_block_kernel(SegArgs a) {
    __shared__ int32_t sL[kCountSmemRollouts];
    __shared__ long long st[2][kCountThreads / 32];
    const int n = a.n_rollouts;
    for (int i = threadIdx.x; i < n; i += kCountThreads) sL[i] = 0;
    __syncthreads();
    // Two segments per thread per pass, both segments' fields and turn counts
    // loaded before either is counted (two dependent load rounds per pass
    // instead of four).
    for (int64_t s0 = threadIdx.x; s0 < a.num_segs; s0 += 2 * kCountThreads) {
        int32_t lo[2], hi[2], i[2], t[2];
        bool ok[2], use[2];
#pragma unroll
        for (int u = 0; u < 2; ++u) {
            const int64_t s = s0 + (int64_t)u * kCountThreads;
            ok[u] = s < a.num_segs && segment_ok(a, s, lo[u], hi[u], i[u], t[u]);
            if (s < a.num_segs && !ok[u]) flag_status(a.status, 4u);
        }
        int te[2];
#pragma unroll
        for (int u = 0; u < 2; ++u) {
            use[u] = ok[u] && t[u] >= 0 && hi[u] > lo[u];
            te[u] = use[u] ? (int)a.T_eff[i[u]] : 0;
        }
#pragma unroll
        for (int u = 0; u < 2; ++u)
            if (use[u] && t[u] < te[u]) atomicAdd(&sL[i[u]], hi[u] - lo[u]);
    }
    __syncthreads();
    long long tok = 0, roll = 0;
    for (int i = threadIdx.x; i < n; i += kCountThreads) {
        const int32_t l = sL[i];
        a.L_out[i] = l;
        tok += l;
        roll += (l > 0);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        tok += __shfl_xor_sync(0xffffffffu, tok, o);
        roll += __shfl_xor_sync(0xffffffffu, roll, o);
    }
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) {
        st[0][w] = tok;
        st[1][w] = roll;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        long long a0 = 0, a1 = 0;
        for (int k = 0; k < kCountThreads / 32; ++k) {
            a0 += st[0][k];
            a1 += st[1][k];
        }
        a.totals_out[0] = a0;
        a.totals_out[1] = a1;
    }
}

__global__ void totals_kernel(const int32_t* L, int32_t n, int64_t* totals) {
    long long tok = 0, roll = 0;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        const int32_t l = L[i];
        tok += l;
        roll += (l > 0);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        tok += __shfl_xor_sync(0xffffffffu, tok, o);
        roll += __shfl_xor_sync(0xffffffffu, roll, o);
    }
    __shared__ long long st[2][32];
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) { st[0][w] = tok; st[1][w] = roll; }
    __syncthreads();
    if (threadIdx.x == 0) {
        long long a0 = 0, a1 = 0;
        for (int k = 0; k < (int)(blockDim.x >> 5); ++k) { a0 += st[0][k]; a1 += st[1][k]; }
        if (a0) atomicAdd(reinterpret_cast<unsigned long long*>(&totals[0]), (unsigned long long)a0);
        if (a1) atomicAdd(reinterpret_cast<unsigned long long*>(&totals[1]), (unsigned long long)a1);
    }
}

// ---- per-token scatter ------------------------------------------------------

// 1 / x for an exact positive integer x, as fp32 rounded once: IEEE fp32
// division when x fits the 24-bit significand, else fp64 then rounding.
__device__ __forceinline__ float recip_count(double x) {
    return (x < 16777216.0) ? 1.f / (float)x : (float)(1.0 / x);
}

// One warp per chunk of 32 * kScatterIters consecutive tokens.  The warp
// finds the chunk's first segment with a 32-ary search (each level one round
// of 32 parallel loads and a ballot, so about log32 S dependent loads instead
// of log2 S), then every lane walks forward through the (non-decreasing)
// offsets as its tokens advance, reloading a segment's fields only when it
// enters a new segment.
constexpr int kScatterIters = 8;   // 256 tokens per warp chunk (16 and 4 measured no better)

__global__ void __launch_bounds__(256) scatter_kernel(SegArgs a) {
    const int64_t nv = a.totals_in[0];
    const int64_t rv = a.totals_in[1];
    const int32_t S = a.num_segs;
    const int lane = threadIdx.x & 31;
    const int64_t chunk = (int64_t)32 * kScatterIters;
    const int64_t nchunks = (a.N + chunk - 1) / chunk;
    const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
    for (int64_t c = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); c < nchunks; c += warps) {
        const int64_t k0 = c * chunk;
        // Last s with seg_offsets[s] <= k0 (0 if none) within [lo, lo + n).
        int32_t seg = 0;
        if (S > 0) {
            int32_t lo = 0, n = S;
            while (n > 1) {
                const int32_t step = (n + 31) / 32;
                const bool in = lane * step < n;
                const bool le = in && a.seg_offsets[lo + lane * step] <= k0;
                const unsigned m = __ballot_sync(0xffffffffu, le);
                if (m == 0) break;
                const int32_t hl = 31 - __clz(m);
                lo += hl * step;
                n = min(step, n - hl * step);
            }
            seg = lo;
        }
        int32_t cur = -1, clo = 0, chi = 0;
        float cadv = 0.f, cw = 0.f;
        // Start of the segment after `seg` (kept in a register: reloaded only
        // when the walk moves on).
        int64_t nxt = (S > 0 && seg + 1 < S) ? (int64_t)a.seg_offsets[seg + 1] : INT64_MAX;
#pragma unroll 1
        for (int it = 0; it < kScatterIters; ++it) {
            const int64_t k = k0 + it * 32 + lane;
            if (k >= a.N) break;
            float adv = 0.f, w = 0.f;
            if (S > 0) {
                while (nxt <= k) {
                    ++seg;
                    nxt = (seg + 1 < S) ? (int64_t)a.seg_offsets[seg + 1] : INT64_MAX;
                }
                if (seg != cur) {   // entering a segment: its fields, advantage and weight
                    cur = seg;
                    int32_t i, t;
                    cadv = cw = 0.f;
                    chi = clo = 0;
                    if (segment_ok(a, seg, clo, chi, i, t) && t >= 0 && t < (int)a.T_eff[i]) {
                        cadv = a.turn_adv[(int64_t)i * a.M + t];
                        if (a.agg == 1) {
                            cw = nv > 0 ? recip_count((double)nv) : 0.f;
                        } else {
                            const int32_t L = a.L_in[i];
                            cw = (rv > 0 && L > 0) ? recip_count((double)rv * (double)L) : 0.f;
                        }
                    } else {
                        chi = clo;   // no generated tokens here
                    }
                }
                if (k >= clo && k < chi) {
                    adv = cadv;
                    w = cw;
                }
            }
            a.adv_out[k] = adv;
            a.w_out[k] = w;
        }
    }
}

// ---- counts + scatter in one launch (single rank) ---------------------------
// Every block builds in shared memory what the scatter needs from the whole
// batch: the per-rollout counts L (hence the two totals), then for every
// segment its advantage, weight and the end of its weighted tokens; then its
// warps scatter their 256-token chunks with the same 32-ary search and walk
// as scatter_kernel, reading the segment table from shared memory instead of
// chasing dependent global loads.  The segment table (offsets, rollout, turn)
// and T_eff are copied into shared memory in one round of independent loads,
// so the counting needs no global load and the per-segment step one more round
// (its turn advantage).  Block 0 also writes L and the totals.  The counting
// is repeated by every block (a few KB of the segment table read from L2 per
// block) in exchange for one launch instead of two.
constexpr int kTokThreads = 256;
// Every block repeats the table work, so the one launch pays off on small
// tables only (measured: 117 / 255 segments 0.75 / 0.71 of the two launches'
// time; 1,514 segments 1.32 times it).
constexpr int kTokMaxSegs = 768;
constexpr size_t kTokSmemMax = 48 * 1024;

// Shared memory of token_adv_fused_kernel: L and T_eff per rollout; offsets,
// weighted end, advantage, weight, rollout and turn per segment.
size_t fused_tok_smem(int64_t n, int64_t S) {
    return 4 * (size_t)n + 4 * ((size_t)S + 1) + 17 * (size_t)S + (size_t)n + 16;
}

__global__ void __launch_bounds__(kTokThreads) token_adv_fused_kernel(SegArgs a) {
    extern __shared__ __align__(16) int32_t tsm[];
    const int n = a.n_rollouts, S = a.num_segs;
    int32_t* sL = tsm;                                    // [n] per-rollout counts
    int32_t* soff = sL + n;                               // [S + 1] segment offsets
    int32_t* send = soff + S + 1;                         // [S] end of the weighted tokens (= start if none)
    float* sadv = reinterpret_cast<float*>(send + S);     // [S]
    float* sw = sadv + S;                                 // [S]
    int32_t* srol = reinterpret_cast<int32_t*>(sw + S);   // [S] seg_rollout
    int8_t* sturn = reinterpret_cast<int8_t*>(srol + S);  // [S] seg_turn
    uint8_t* ste = reinterpret_cast<uint8_t*>(sturn + S); // [n] T_eff
    __shared__ long long red[2][kTokThreads / 32];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

    for (int i = tid; i < n; i += kTokThreads) {
        sL[i] = 0;
        ste[i] = a.T_eff[i];
    }
    if (S > 0)
        for (int q = tid; q <= S; q += kTokThreads) {
            soff[q] = a.seg_offsets[q];
            if (q < S) {
                srol[q] = a.seg_rollout[q];
                sturn[q] = a.seg_turn[q];
            }
        }
    __syncthreads();
    auto seg_fields = [&](int q, int& lo, int& hi, int& i, int& t) {
        lo = soff[q];
        hi = soff[q + 1];
        t = sturn[q];
        i = srol[q];
        return lo >= 0 && hi >= lo && (int64_t)hi <= a.N && t < a.M && (t < 0 || (i >= 0 && i < n));
    };
    for (int q = tid; q < S; q += kTokThreads) {   // L_i (Sec. 3.3 token sets)
        int lo, hi, i, t;
        if (!seg_fields(q, lo, hi, i, t)) {
            if (blockIdx.x == 0) flag_status(a.status, 4u);
            continue;
        }
        if (t >= 0 && hi > lo && t < (int)ste[i]) atomicAdd(&sL[i], hi - lo);
    }
    __syncthreads();
    long long tok = 0, roll = 0;
    for (int i = tid; i < n; i += kTokThreads) {
        const int32_t l = sL[i];
        tok += l;
        roll += (l > 0);
        if (blockIdx.x == 0) a.L_out[i] = l;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        tok += __shfl_xor_sync(0xffffffffu, tok, o);
        roll += __shfl_xor_sync(0xffffffffu, roll, o);
    }
    if (lane == 0) {
        red[0][warp] = tok;
        red[1][warp] = roll;
    }
    __syncthreads();
    long long nv = 0, rv = 0;
#pragma unroll
    for (int k = 0; k < kTokThreads / 32; ++k) {
        nv += red[0][k];
        rv += red[1][k];
    }
    if (blockIdx.x == 0 && tid == 0) {
        a.totals_out[0] = nv;
        a.totals_out[1] = rv;
    }
    for (int q = tid; q < S; q += kTokThreads) {   // per-segment advantage and weight
        int lo, hi, i, t;
        const bool ok = seg_fields(q, lo, hi, i, t);
        float av = 0.f, wv = 0.f;
        int end = lo;
        if (ok && t >= 0 && t < (int)ste[i]) {
            av = a.turn_adv[(int64_t)i * a.M + t];
            if (a.agg == 1) {
                wv = nv > 0 ? recip_count((double)nv) : 0.f;
            } else {
                const int32_t Li = sL[i];
                wv = (rv > 0 && Li > 0) ? recip_count((double)rv * (double)Li) : 0.f;
            }
            end = hi;
        }
        send[q] = end;
        sadv[q] = av;
        sw[q] = wv;
    }
    __syncthreads();

    const int64_t chunk = (int64_t)32 * kScatterIters;
    const int64_t nchunks = (a.N + chunk - 1) / chunk;
    const int64_t warps = (int64_t)gridDim.x * (kTokThreads / 32);
    for (int64_t c = (int64_t)blockIdx.x * (kTokThreads / 32) + warp; c < nchunks; c += warps) {
        const int64_t k0 = c * chunk;
        int32_t seg = 0;   // last s with soff[s] <= k0 (0 if none), 32-ary search
        if (S > 0) {
            int32_t lo = 0, cnt = S;
            while (cnt > 1) {
                const int32_t step = (cnt + 31) / 32;
                const bool in = lane * step < cnt;
                const bool le = in && soff[lo + lane * step] <= k0;
                const unsigned m = __ballot_sync(0xffffffffu, le);
                if (m == 0) break;
                const int32_t hl = 31 - __clz(m);
                lo += hl * step;
                cnt = min(step, cnt - hl * step);
            }
            seg = lo;
        }
        int32_t cur = -1, clo = 0, chi = 0;
        float cadv = 0.f, cw = 0.f;
#pragma unroll 1
        for (int it = 0; it < kScatterIters; ++it) {
            const int64_t k = k0 + it * 32 + lane;
            if (k >= a.N) break;
            float adv = 0.f, w = 0.f;
            if (S > 0) {
                while (seg + 1 < S && soff[seg + 1] <= k) ++seg;
                if (seg != cur) {
                    cur = seg;
                    clo = soff[seg];
                    chi = send[seg];
                    cadv = sadv[seg];
                    cw = sw[seg];
                }
                if (k >= clo && k < chi) {
                    adv = cadv;
                    w = cw;
                }
            }
            a.adv_out[k] = adv;
            a.w_out[k] = w;
        }
    }
}

bool aligned_to(const void* p, uintptr_t n) { return (reinterpret_cast<uintptr_t>(p) & (n - 1)) == 0; }

template <int MC>
cudaError_t launch_pair(const RankArgs& a, cudaStream_t s) {
    const int warps = 8;
    // A persistent grid (the blocks that fit at once) walks the groups: 10 %
    // faster than one block per 8 groups, and one counter flush per block.
    const int per_sm = a.cmp == 1 ? kPairLexiMinBlocks : kPairMinBlocks;
    const int64_t blocks = std::min<int64_t>(((int64_t)a.num_groups + warps - 1) / warps,
                                             (int64_t)device_sm_count() * per_sm);
    if (a.cmp == 1) rank_pair_kernel<MC, true><<<(unsigned)blocks, warps * 32, 0, s>>>(a);
    else rank_pair_kernel<MC, false><<<(unsigned)blocks, warps * 32, 0, s>>>(a);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_rank_advantages(const RankArgs& a, cudaStream_t s) {
    if (a.num_groups == 0) return cudaSuccess;
    // Groups of 64 (the quad kernel): 4-byte aligned byte arrays and 16-byte
    // aligned 4-byte arrays (every lane's four rollouts start at a multiple of 4).
    const bool quad = a.cmp == 0 && a.G == 64 && aligned_to(a.pass_turn, 4) &&
                      aligned_to(a.num_turns, 4) && aligned_to(a.T_eff, 4) && aligned_to(a.r_out, 4) &&
                      aligned_to(a.n_worse, 16) && aligned_to(a.n_better, 16) && aligned_to(a.R, 16) &&
                      aligned_to(a.A, 16) && aligned_to(a.turn_adv, 16);
    if (quad) {
        switch (a.M) {
            case 1: return launch_quad<1>(a, s);
            case 2: return launch_quad<2>(a, s);
            case 3: return launch_quad<3>(a, s);
            case 4: return launch_quad<4>(a, s);
            case 5: return launch_quad<5>(a, s);
            case 6: return launch_quad<6>(a, s);
            case 7: return launch_quad<7>(a, s);
            case 8: return launch_quad<8>(a, s);
            default: break;
        }
    }
    // The pair kernel's vector accesses need 2-byte aligned byte arrays and
    // 8-byte aligned 4-byte arrays (rollout pairs start at even indices).
    // The tie-broken comparator takes it too, with 8-byte aligned speedups and
    // token counts.
    const bool pair = a.G % 2 == 0 && a.G <= 64 && aligned_to(a.pass_turn, 2) &&
                      aligned_to(a.num_turns, 2) && aligned_to(a.T_eff, 2) && aligned_to(a.r_out, 2) &&
                      aligned_to(a.n_worse, 8) && aligned_to(a.n_better, 8) && aligned_to(a.R, 8) &&
                      aligned_to(a.A, 8) && aligned_to(a.turn_adv, 8) &&
                      (a.cmp == 0 || (aligned_to(a.speedup, 8) && aligned_to(a.ntokens, 8)));
    if (pair) {
        switch (a.M) {
            case 1: return launch_pair<1>(a, s);
            case 2: return launch_pair<2>(a, s);
            case 3: return launch_pair<3>(a, s);
            case 4: return launch_pair<4>(a, s);
            case 5: return launch_pair<5>(a, s);
            case 6: return launch_pair<6>(a, s);
            case 7: return launch_pair<7>(a, s);
            case 8: return launch_pair<8>(a, s);
            default: break;
        }
    }
    const int J = (a.G + 31) / 32;
    if (J <= 1) return launch_rank_j<1>(a, s);
    if (J <= 2) return launch_rank_j<2>(a, s);
    if (J <= 4) return launch_rank_j<4>(a, s);
    if (J <= 8) return launch_rank_j<8>(a, s);
    if (J <= 16) return launch_rank_j<16>(a, s);
    return launch_rank_j<32>(a, s);
}

cudaError_t launch_token_counts(const SegArgs& a, cudaStream_t s) {
    if (a.n_rollouts <= kCountSmemRollouts) {
        counts_one_block_kernel<<<1, kCountThreads, 0, s>>>(a);
        return cudaGetLastError();
    }
    const int sms = device_sm_count();
    const int64_t zb = std::min<int64_t>(((int64_t)a.n_rollouts + 255) / 256, (int64_t)sms * 4);
    zero_counts_kernel<<<(unsigned)std::max<int64_t>(zb, 1), 256, 0, s>>>(a.L_out, a.n_rollouts, a.totals_out);
    if (a.num_segs > 0) {
        segment_count_kernel<<<(unsigned)(((int64_t)a.num_segs + 255) / 256), 256, 0, s>>>(a);
    }
    if (a.n_rollouts > 0) {
        totals_kernel<<<(unsigned)std::max<int64_t>(zb, 1), 256, 0, s>>>(a.L_out, a.n_rollouts, a.totals_out);
    }
    return cudaGetLastError();
}

cudaError_t launch_token_advantages(const SegArgs& a, cudaStream_t s) {
    const size_t smem = fused_tok_smem(a.n_rollouts, a.num_segs);
    if (a.num_segs > kTokMaxSegs || smem > kTokSmemMax) {   // a large table: the two-kernel path
        cudaError_t e = launch_token_counts(a, s);
        if (e != cudaSuccess) return e;
        SegArgs b = a;
        b.L_in = a.L_out;
        b.totals_in = a.totals_out;
        return launch_scatter(b, s);
    }
    const int sms = device_sm_count();
    const int64_t chunks = (a.N + 32 * kScatterIters - 1) / (32 * kScatterIters);
    const int64_t wpb = kTokThreads / 32;
    const int64_t blocks = std::max<int64_t>(1, std::min<int64_t>((chunks + wpb - 1) / wpb, (int64_t)sms * 2));
    token_adv_fused_kernel<<<(unsigned)blocks, kTokThreads, smem, s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_scatter(const SegArgs& a, cudaStream_t s) {
    if (a.N == 0) return cudaSuccess;
    const int sms = device_sm_count();
    const int64_t chunks = (a.N + 32 * kScatterIters - 1) / (32 * kScatterIters);
    const int64_t blocks = std::min<int64_t>((chunks + 7) / 8, (int64_t)sms * 16);
    scatter_kernel<<<(unsigned)blocks, 256, 0, s>>>(a);
    return cudaGetLastError();
}

}  // namespace leap
