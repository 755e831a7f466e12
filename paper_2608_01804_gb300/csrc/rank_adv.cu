// Rank-based advantages (Sec. 3.1 Eqs. 1-2, Sec. 3.2 Eqs. 4-6 + GRPO step,
// Sec. 3.3 discount) and the per-token scatter of the turn advantages.
//
// One warp per rollout group.  Lane l owns rollouts l, l + 32, ...  Because
// the paper's comparator looks only at the tier r in [0, M], the O(G^2)
// tournament of Eq. 5 collapses to a histogram of r: N_worse = #peers with a
// lower tier, N_better = #peers with a higher tier.  The histogram is built
// with warp ballots, so the whole group stays in registers.
#include "leap_common.cuh"
#include "leap_internal.h"

#include <algorithm>
#include <math.h>

namespace leap {
namespace {

constexpr int kMaxM = 8;

__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Per-warp running counters (lane 0), reduced per block then added atomically.
constexpr int kNumStats = 9 + kMaxM;

template <int J, bool LEXI>  // rollouts per lane: G <= 32 * J; tie-broken comparator
__global__ void __launch_bounds__(256) rank_adv_kernel(RankArgs a) {
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
            bad[j] = valid[j] && (pt < 0 || pt > M || nt < 1 || nt > M || (pt >= 1 && pt > nt));
            // Eq. 1 over first-turn outcomes; a malformed outcome counts as failed.
            const bool fail1 = valid[j] && (bad[j] || pt != 1);
            n_fail += __popc(__ballot_sync(0xffffffffu, fail1));
            pt0[j] = (valid[j] && !bad[j]) ? pt : 0;
            T[j] = nt;
        }
        // Eq. 2 (or the recorded gate).
        const bool gate = a.gate_in ? (a.gate_in[group] != 0) : (a.tau_min <= n_fail && n_fail <= a.tau_max);

        // Tier rule of Sec. 3.2; gated-off groups ran turn 1 only.
#pragma unroll
        for (int j = 0; j < J; ++j) {
            const int pt = pt0[j];
            if (!valid[j] || bad[j]) {
                r[j] = 0;
                T[j] = 0;
            } else if (!gate) {
                r[j] = (pt == 1) ? M : 0;
                T[j] = 1;
            } else {
                r[j] = (pt >= 1) ? (M - pt + 1) : 0;
            }
            if (bad[j]) flag_status(a.status, 2u);
        }

        // Eq. 5: N_worse / N_better.
        int nw[J], nb[J];
        if constexpr (!lexi) {
            // The paper's comparator looks only at r: a histogram of tiers via ballots.
            int hist[kMaxM + 1];
#pragma unroll
            for (int b = 0; b <= kMaxM; ++b) {
                int c = 0;
                if (b <= M) {
#pragma unroll
                    for (int j = 0; j < J; ++j) c += __popc(__ballot_sync(0xffffffffu, valid[j] && r[j] == b));
                }
                hist[b] = c;
            }
#pragma unroll
            for (int j = 0; j < J; ++j) {
                nw[j] = 0;
                nb[j] = 0;
#pragma unroll
                for (int b = 0; b <= kMaxM; ++b) {
                    nw[j] += (b < r[j]) ? hist[b] : 0;
                    nb[j] += (b > r[j]) ? hist[b] : 0;
                }
            }
        } else {
            // Tie-broken comparator: every rollout against every peer, keys
            // broadcast from the lane that holds them.
#pragma unroll
            for (int j = 0; j < J; ++j) nw[j] = nb[j] = 0;
#pragma unroll
            for (int sidx = 0; sidx < J; ++sidx) {
                for (int l = 0; l < 32; ++l) {
                    const int jj = 32 * sidx + l;
                    if (jj >= G) break;  // uniform across the warp
                    const int rj = __shfl_sync(0xffffffffu, r[sidx], l);
                    const float spj = __shfl_sync(0xffffffffu, sp[sidx], l);
                    const int tkj = __shfl_sync(0xffffffffu, tk[sidx], l);
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

        // Eq. 6 and the sum of squared net scores (exact).
        int d[J];
        long long dd = 0;
#pragma unroll
        for (int j = 0; j < J; ++j) {
            d[j] = nw[j] - nb[j];
            if (valid[j]) {
                dd += (long long)d[j] * d[j];
                const int64_t i = base + lane + 32 * j;
                if (a.n_worse) a.n_worse[i] = nw[j];
                if (a.n_better) a.n_better[i] = nb[j];
                if (a.r_out) a.r_out[i] = (uint8_t)r[j];
                a.T_eff[i] = (uint8_t)T[j];
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) dd += __shfl_xor_sync(0xffffffffu, dd, o);

        const float gm1 = (float)(G - 1);
        const float den = a.std_unbiased ? gm1 : (float)G;
        float Rv[J], Av[J];
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
            const float mean = warp_sum_f(sum) / (float)G;
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
                hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
            }
            float ss = 0.f;
#pragma unroll
            for (int j = 0; j < J; ++j)
                if (valid[j]) ss += (Rv[j] - mean) * (Rv[j] - mean);
            const float stdv = sqrtf(warp_sum_f(ss) / den);
#pragma unroll
            for (int j = 0; j < J; ++j)
                Av[j] = (a.norm == 1) ? Rv[j] : ((hi == lo) ? 0.f : (Rv[j] - mean) / (stdv + a.eps_std));
        }

        int nonzero = 0;
#pragma unroll
        for (int j = 0; j < J; ++j) {
            nonzero += __popc(__ballot_sync(0xffffffffu, valid[j] && Av[j] != 0.f));
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

        if (a.stats) {  // training-observability counters (Table 5, Sec. 4.2)
            int first = 0, later = 0, failed_on = 0, turns = 0;
            int by_turn[kMaxM];
#pragma unroll
            for (int m = 0; m < kMaxM; ++m) by_turn[m] = 0;
#pragma unroll
            for (int j = 0; j < J; ++j) {
                const bool ok = valid[j] && !bad[j];
                const int pt = pt0[j];
                first += __popc(__ballot_sync(0xffffffffu, ok && pt == 1));
                later += __popc(__ballot_sync(0xffffffffu, ok && gate && pt >= 2));
                failed_on += __popc(__ballot_sync(0xffffffffu, ok && gate && pt != 1));
                int tsum = valid[j] ? T[j] : 0;
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) tsum += __shfl_xor_sync(0xffffffffu, tsum, o);
                turns += tsum;
#pragma unroll
                for (int m = 1; m < kMaxM; ++m)
                    by_turn[m] += __popc(__ballot_sync(0xffffffffu, ok && gate && pt == m + 1));
            }
            if (lane == 0) {
                long long* c = sst[wib];
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
            }
            __syncwarp();
        }
    }

    if (a.stats) {
        __syncthreads();
        if (threadIdx.x < kNumStats) {
            long long v = 0;
            for (int w = 0; w < (int)(blockDim.x >> 5); ++w) v += sst[w][threadIdx.x];
            if (v) atomicAdd(reinterpret_cast<unsigned long long*>(a.stats) + threadIdx.x, (unsigned long long)v);
        }
    }
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

// One warp per chunk of 32 * kScatterIters consecutive tokens: lane 0 finds
// the chunk's first segment by binary search, then every lane walks forward
// through the (non-decreasing) offsets as its tokens advance.
constexpr int kScatterIters = 8;

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
        int32_t seg = 0;
        if (lane == 0 && S > 0) {  // last s with seg_offsets[s] <= k0 (0 if none)
            int32_t lo = 0, hi = S;
            while (hi - lo > 1) {
                const int32_t mid = (lo + hi) >> 1;
                if (a.seg_offsets[mid] <= k0) lo = mid; else hi = mid;
            }
            seg = lo;
        }
        seg = __shfl_sync(0xffffffffu, seg, 0);
#pragma unroll 1
        for (int it = 0; it < kScatterIters; ++it) {
            const int64_t k = k0 + it * 32 + lane;
            if (k >= a.N) break;
            float adv = 0.f, w = 0.f;
            if (S > 0) {
                while (seg + 1 < S && a.seg_offsets[seg + 1] <= k) ++seg;
                int32_t lo, hi, i, t;
                if (segment_ok(a, seg, lo, hi, i, t) && k >= lo && k < hi && t >= 0 && t < (int)a.T_eff[i]) {
                    adv = a.turn_adv[(int64_t)i * a.M + t];
                    if (a.agg == 1) {
                        w = nv > 0 ? recip_count((double)nv) : 0.f;
                    } else {
                        const int32_t L = a.L_in[i];
                        w = (rv > 0 && L > 0) ? recip_count((double)rv * (double)L) : 0.f;
                    }
                }
            }
            a.adv_out[k] = adv;
            a.w_out[k] = w;
        }
    }
}

}  // namespace

cudaError_t launch_rank_advantages(const RankArgs& a, cudaStream_t s) {
    if (a.num_groups == 0) return cudaSuccess;
    const int J = (a.G + 31) / 32;
    if (J <= 1) return launch_rank_j<1>(a, s);
    if (J <= 2) return launch_rank_j<2>(a, s);
    if (J <= 4) return launch_rank_j<4>(a, s);
    if (J <= 8) return launch_rank_j<8>(a, s);
    if (J <= 16) return launch_rank_j<16>(a, s);
    return launch_rank_j<32>(a, s);
}

cudaError_t launch_token_counts(const SegArgs& a, cudaStream_t s) {
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

cudaError_t launch_scatter(const SegArgs& a, cudaStream_t s) {
    if (a.N == 0) return cudaSuccess;
    const int sms = device_sm_count();
    const int64_t chunks = (a.N + 32 * kScatterIters - 1) / (32 * kScatterIters);
    const int64_t blocks = std::min<int64_t>((chunks + 7) / 8, (int64_t)sms * 16);
    scatter_kernel<<<(unsigned)blocks, 256, 0, s>>>(a);
    return cudaGetLastError();
}

}  // namespace leap
