// Vector helpers of the row kernels (logprob_loss.cu, loss_pipe.cu, short_rows.cu): bf16
// vectors of 8 logits as uint4, their masked tail, stores that keep the
// columns past V, and the per-vector max / exponential-sum / dlogits
// arithmetic, and the packed fp32x2 instructions (FMA / add / multiply) they use.
#pragma once

#include "leap_common.cuh"

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
// position (8 independent chains of length NV), then a tree.  Element pairs
// go through the packed fp32x2 FMA and add (each lane rounds as the scalar
// instruction would, so the result is the same bits as element by element).
template <int NV>
__device__ __forceinline__ float tree_exp_sum(const uint4 (&x)[NV], float c1, float mc) {
    uint64_t acc[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) acc[q] = f2_pack(0.f, 0.f);
    const uint64_t c12 = f2_pack(c1, c1), nmc2 = f2_pack(-mc, -mc);
#pragma unroll
    for (int k = 0; k < NV; ++k) {
        const uint32_t w[4] = {x[k].x, x[k].y, x[k].z, x[k].w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            float lo, hi;
            f2_unpack(f2_fma(f2_pack(bf16_lo(w[q]), bf16_hi(w[q])), c12, nmc2), lo, hi);
            acc[q] = f2_add(acc[q], f2_pack(ex2(lo), ex2(hi)));
        }
    }
    float a[8];
#pragma unroll
    for (int q = 0; q < 4; ++q) f2_unpack(acc[q], a[2 * q], a[2 * q + 1]);
    return ((a[0] + a[1]) + (a[2] + a[3])) + ((a[4] + a[5]) + (a[6] + a[7]));
}

// dlogits of one vector: coef * (1[v = y] - 2^(z c1 - K)); `yl` is the target's
// lane in this vector or -1.  Element pairs through the packed fp32x2 FMA and
// multiply (the same bits as element by element).
__device__ __forceinline__ uint4 dlogit8(const uint4& x, float c1, float K, float coef, int yl) {
    const uint32_t w[4] = {x.x, x.y, x.z, x.w};
    const uint64_t c12 = f2_pack(c1, c1), nK2 = f2_pack(-K, -K), nc2 = f2_pack(-coef, -coef);
    uint32_t o[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        float lo, hi;
        f2_unpack(f2_fma(f2_pack(bf16_lo(w[q]), bf16_hi(w[q])), c12, nK2), lo, hi);
        f2_unpack(f2_mul(nc2, f2_pack(ex2(lo), ex2(hi))), lo, hi);
        if (yl == 2 * q) lo += coef;
        if (yl == 2 * q + 1) hi += coef;
        o[q] = pack_bf16x2(lo, hi);
    }
    return make_uint4(o[0], o[1], o[2], o[3]);
}

}  // namespace
}  // namespace leap
