// Fused forward + backward of the clipped surrogate (Eq. 3) for short and
// mid-size rows (V <= 32,768): every leap_grpo_loss_fwd call with dlogits and
// such a vocabulary lands here (logprob_loss.cu routes it).
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

// 1-D bulk copy own shared memory -> global (bytes and both addresses
// multiples of 16) in the issuing thread's bulk-async group, with an L2 cache
// policy; bulk_commit closes the group.
__device__ __forceinline__ void bulk_s2g(void* gdst, const void* smem_src, uint32_t bytes, uint64_t policy) {
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group.L2::cache_hint [%0], [%1], %2, %3;" ::"l"(gdst),
                 "r"(smem_addr(smem_src)), "r"(bytes), "l"(policy)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// Waits until the issuing thread's bulk groups have read their shared-memory
// sources (all but the newest N groups).
template <int N>
__device__ __forceinline__ void bulk_wait_read() {
    asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}
// Waits until the issuing thread's bulk groups have completed (all but the
// newest N).
template <int N>
__device__ __forceinline__ void bulk_wait_all() {
    asm volatile("cp.async.bulk.wait_group %0;" ::"n"(N) : "memory");
}

// ---------------------------------------------------------------------------
// Fused forward + backward for rows of V <= 32,768.  A row group of W warps
// owns one row at a time; warp w of the group owns the contiguous slice of
// 16-byte vectors [32 NV w, 32 NV (w + 1)) of the row (512 NV bytes), lane l
// vectors 32 NV w + l + 32 k (k < NV), so the row is read from HBM once.
// Shapes (W warps per row, NV vectors per lane, CTA threads, CTAs per SM):
//   V <= 8,192:   W = 1, 2, 4 or 8, NV = 4, 256 threads, 3 per SM;
//   V <= 16,384:  W = 8,  NV = 8, 256 threads, 2 per SM;
//   V <= 32,768:  W = 16, NV = 8, 512 threads, 1 per SM.
//   * Staging: each warp double-buffers its slice in shared memory.  While it
//     works on row i, a 1-D bulk copy (TMA) of its slice of row i + 1 is in
//     flight into the other stage, completing on that stage's mbarrier; every
//     wait is bounded (LEAP_DEV_TIMEOUT).  Registers hold one row only.  The
//     dlogits slice goes back the same way: the lanes write it to a shared
//     buffer and one bulk copy stores it (zeros for masked rows come from a
//     shared zero slice).  Stage entries past a warp's slice hold -inf and the
//     row's partial last vector is masked in shared memory, so neither the
//     loads nor the stores carry per-vector bounds checks.
//   * Arithmetic: the kernel would otherwise be bound by instruction issue,
//     so the row max is reduced first (packed bf16 maxima, then the warp), the
//     exponentials 2^((z - m) c1) are taken once and kept in registers
//     (8 NV fp32 per lane), element pairs go through packed fp32x2 FMA / add /
//     multiply, and dlogits is one multiply per element.
//   * W > 1: each warp publishes (max, sum) and, if it holds it, the target
//     logit in shared memory behind one named barrier per live row (two
//     alternating slots); every warp then merges the W pairs directly.
//   * FULL (V = 256 NV W): every slice is whole, with no tail.
// Row groups are persistent and walk rows g, g + stride, ...  Masked rows are
// not read.
// ---------------------------------------------------------------------------
// Shared memory of a CTA of NW warps (dynamic: 50 KB at NV = 4, 100 KB at
// NV = 8 with 8 warps, 197 KB with 16).
template <int NW, int NV>
struct ShortSmem {
    uint4 stage[NW][2][32 * NV];   // two stages per warp
    uint4 out[NW][32 * NV];        // the warp's dlogits slice on its way to HBM
    uint4 zeros[32 * NV];          // source of the masked rows' slices
    uint64_t full[NW][2];          // one mbarrier per stage
    float4 part[2][NW];            // (max, sum, target logit, holds target) per warp
    int abort_flag;
};

template <int W, int NV, int THREADS, int MINB, bool FULL>
__global__ void __launch_bounds__(THREADS, MINB) short_row_kernel(RowArgs a) {
    constexpr int NW = THREADS / 32, VPW = 32 * NV, TG = 32 * W, GPB = THREADS / TG;
    extern __shared__ __align__(128) unsigned char short_smem_raw[];
    ShortSmem<NW, NV>& sm = *reinterpret_cast<ShortSmem<NW, NV>*>(short_smem_raw);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int gib = warp / W;                  // row group within the block
    const int wig = warp % W;                  // warp within the row group
    // 32-bit row and vector indices (N < 2^31 is checked on the host; V8 <= 4,096).
    const int stride = (int)gridDim.x * GPB;
    const int N = (int)a.N;
    const int V = a.V;
    const int V8 = FULL ? W * VPW : (V + 7) >> 3;
    const int tailn = FULL ? 0 : (V & 7);
    const float c1 = a.inv_temp * kLog2e;
    const int vbase = wig * VPW;                                  // this warp's first vector
    const int nvec = FULL ? VPW : max(0, min(VPW, V8 - vbase));   // vectors in this warp's slice
    const uint32_t slice_bytes = (uint32_t)nvec * 16u;
    // The row's partial last vector (V not a multiple of 8) is stored element
    // by element, the whole vectors before it by one bulk copy.
    const bool owns_tail = !FULL && tailn != 0 && nvec > 0 && vbase + nvec == V8;
    const uint32_t store_bytes = (uint32_t)(nvec - (owns_tail ? 1 : 0)) * 16u;
    const uint64_t policy = l2_policy_evict_first();

    if (threadIdx.x == 0) sm.abort_flag = 0;
    if (lane == 0) {
        mbar_init(&sm.full[warp][0], 1);
        mbar_init(&sm.full[warp][1], 1);
        fence_mbar_init();
    }
    if (!FULL) {   // never written by a copy: reads as -inf
        for (int li = nvec + lane; li < VPW; li += 32) {
            sm.stage[warp][0][li] = neg_inf4();
            sm.stage[warp][1][li] = neg_inf4();
        }
    }
    for (int i = threadIdx.x; i < VPW; i += THREADS) sm.zeros[i] = make_uint4(0, 0, 0, 0);
    fence_proxy_async_smem();   // the zero slice is read by bulk copies
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
            if (lane == 0) {
                if (store_bytes) {
                    bulk_s2g(drow + vbase, &sm.zeros[0], store_bytes, policy);
                    bulk_commit();
                }
                if (owns_tail) store_vec(drow, V8 - 1, make_uint4(0, 0, 0, 0), V8, tailn);
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
            if (owns_tail) {   // columns >= V of the last vector read as -inf
                if (lane == 0) mask_tail(sm.stage[warp][st][nvec - 1], tailn);
                __syncwarp();
            }
#pragma unroll
            for (int k = 0; k < NV; ++k) x[k] = sm.stage[warp][st][lane + 32 * k];
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
                const float4* p = &sm.part[par][gib * W];
                if (W <= 8) {
                    float4 q[W];
#pragma unroll
                    for (int v = 0; v < W; ++v) q[v] = p[v];
                    mrow = q[0].x;
#pragma unroll
                    for (int v = 1; v < W; ++v) mrow = fmaxf(mrow, q[v].x);
                    srow = 0.f;
#pragma unroll
                    for (int v = 0; v < W; ++v) {
                        if (q[v].y != 0.f) srow = fmaf(q[v].y, ex2((q[v].x - mrow) * c1), srow);
                        if (q[v].w != 0.f) zy = q[v].z;
                    }
                } else {   // 16 partials: read twice rather than held in registers
                    mrow = p[0].x;
#pragma unroll
                    for (int v = 1; v < W; ++v) mrow = fmaxf(mrow, p[v].x);
                    srow = 0.f;
#pragma unroll 4
                    for (int v = 0; v < W; ++v) {
                        const float4 q = p[v];
                        if (q.y != 0.f) srow = fmaf(q.y, ex2((q.x - mrow) * c1), srow);
                        if (q.w != 0.f) zy = q.z;
                    }
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
            if (lane == 0) bulk_wait_read<0>();   // the previous slice has left the buffer
            __syncwarp();
#pragma unroll
            for (int k = 0; k < NV; ++k) {
                const int vi = vbase + lane + 32 * k;
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
                sm.out[warp][lane + 32 * k] = d;
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
                if (store_bytes) {
                    bulk_s2g(drow + vbase, &sm.out[warp][0], store_bytes, policy);
                    bulk_commit();
                }
                if (owns_tail) store_vec(drow, V8 - 1, sm.out[warp][nvec - 1], V8, tailn);
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
    if (lane == 0) bulk_wait_all<0>();   // the dlogits stores have completed
    // Every copy is waited for before its row is used, so one can still be in
    // flight here only after a wait gave up: wait for it (bounded again) so no
    // copy lands in the shared memory of an exited CTA.
    if (pending) {
        volatile int fresh = 0;
        for (int st = 0; st < 2; ++st)
            if (pending & (1u << st)) mbar_wait(&sm.full[warp][st], (phase >> st) & 1u, a.status, &fresh);
    }
}

// Persistent grid of the short-row kernel: the CTAs that fit at once (cached
// per device, with the shared-memory opt-in), at most one row group per row.
template <int W, int NV, int THREADS, int MINB, bool FULL>
cudaError_t launch_short_rows(const RowArgs& a, cudaStream_t s) {
    constexpr size_t smem = sizeof(ShortSmem<THREADS / 32, NV>);
    static_assert(smem <= 232448, "short-row shared memory exceeds the per-CTA limit");
    static std::mutex mu;
    static int cached_dev = -1, cached_resident = 0;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    int resident = 0;   // CTAs resident at once on the whole device
    {
        std::lock_guard<std::mutex> lk(mu);
        if (cached_dev != dev) {
            e = cudaFuncSetAttribute(short_row_kernel<W, NV, THREADS, MINB, FULL>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            if (e != cudaSuccess) return e;
            int per_sm = 0;
            e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, short_row_kernel<W, NV, THREADS, MINB, FULL>,
                                                              THREADS, smem);
            if (e != cudaSuccess) return e;
            cached_dev = dev;
            cached_resident = per_sm * device_sm_count();
        }
        resident = cached_resident;
    }
    if (resident <= 0) return cudaErrorNotSupported;
    constexpr int GPB = THREADS / (32 * W);
    const int64_t blocks = std::min<int64_t>((a.N + GPB - 1) / GPB, (int64_t)resident);
    short_row_kernel<W, NV, THREADS, MINB, FULL><<<(unsigned)blocks, THREADS, smem, s>>>(a);
    return cudaGetLastError();
}

template <int W, int NV, int THREADS, int MINB>
cudaError_t launch_short_shape(const RowArgs& a, cudaStream_t s) {
    // Whole slices for every warp (V = 256 NV W): no per-vector bounds checks.
    if (a.V == W * 256 * NV) return launch_short_rows<W, NV, THREADS, MINB, true>(a, s);
    return launch_short_rows<W, NV, THREADS, MINB, false>(a, s);
}

}  // namespace

cudaError_t launch_short_row_loss(const RowArgs& a, cudaStream_t s) {
    if (a.N == 0) return cudaSuccess;
    const int64_t V8s = ((int64_t)a.V + 7) >> 3;   // 16-byte vectors per row
    if (V8s <= 128) return launch_short_shape<1, 4, 256, 3>(a, s);
    if (V8s <= 256) return launch_short_shape<2, 4, 256, 3>(a, s);
    if (V8s <= 512) return launch_short_shape<4, 4, 256, 3>(a, s);
    if (V8s <= 1024) return launch_short_shape<8, 4, 256, 3>(a, s);
    if (V8s <= 2048) return launch_short_shape<8, 8, 256, 2>(a, s);
    return launch_short_shape<16, 8, 512, 1>(a, s);
}

}  // namespace leap
