// twk_df.cuh -- double-float arithmetic (an unevaluated sum of two floats) and the one
// dot-product routine behind every exact similarity value of the TwinKV pass: bf16 x
// bf16 products are exact in fp32 and are accumulated with Knuth's TwoSum, four lanes
// per dot product, each over every fourth 16-byte chunk, combined in a fixed tree.  Every
// dot product (norms included) goes through group_dot_df, so identical keys give
// identical values and the value of k_i . k_j equals that of k_j . k_i bit for bit.
#pragma once
#include <cstdint>
#include <cuda_runtime.h>

namespace twk {

__device__ __forceinline__ void two_sum_acc(float& hi, float& lo, float p)
{
    const float s = __fadd_rn(hi, p);
    const float bp = __fsub_rn(s, hi);
    const float e = __fadd_rn(__fsub_rn(hi, __fsub_rn(s, bp)), __fsub_rn(p, bp));
    hi = s;
    lo = __fadd_rn(lo, e);
}

// An unevaluated sum hi + lo of two floats (a double-float).
struct DFPair {
    float h, l;
};

// (hi, lo) + (hi2, lo2) as a double-float sum.  TwoSum gives the exact rounding error
// whatever the operand order, so the result does not depend on which side is which.
__device__ __forceinline__ void df_add(float& hi, float& lo, float hi2, float lo2)
{
    const float s = __fadd_rn(hi, hi2);
    const float bp = __fsub_rn(s, hi);
    float e = __fadd_rn(__fsub_rn(hi, __fsub_rn(s, bp)), __fsub_rn(hi2, bp));
    e = __fadd_rn(e, __fadd_rn(lo, lo2));
    hi = __fadd_rn(s, e);
    lo = __fsub_rn(e, __fsub_rn(hi, s));
}

constexpr int kParts = 4;   // threads per dot product, each over every fourth 16-byte chunk

// One lane's part of a . b for two bf16 rows of length D: the 16-byte chunks part,
// part + kParts, part + 2 kParts, ... (so that the kParts lanes of a dot product read
// kParts * 16 contiguous bytes per load), terms in increasing t.
template <int D>
__device__ __forceinline__ void quarter_dot(const uint16_t* __restrict__ a,
                                            const uint16_t* __restrict__ b, int part,
                                            float& hi, float& lo)
{
    constexpr int Q = D / 8 / kParts;   // 16-byte chunks per lane
    const uint4* a4 = reinterpret_cast<const uint4*>(a) + part;
    const uint4* b4 = reinterpret_cast<const uint4*>(b) + part;
    hi = 0.f;
    lo = 0.f;
#pragma unroll
    for (int q = 0; q < Q; ++q) {
        const uint4 va = __ldg(a4 + q * kParts);
        const uint4 vb = __ldg(b4 + q * kParts);
        const uint32_t wa[4] = {va.x, va.y, va.z, va.w};
        const uint32_t wb[4] = {vb.x, vb.y, vb.z, vb.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            // element 2k (low half) then 2k+1 (high half) of this 16-byte chunk
            two_sum_acc(hi, lo, __fmul_rn(__uint_as_float(wa[k] << 16), __uint_as_float(wb[k] << 16)));
            two_sum_acc(hi, lo, __fmul_rn(__uint_as_float(wa[k] & 0xFFFF0000u),
                                          __uint_as_float(wb[k] & 0xFFFF0000u)));
        }
    }
}

// a . b by the kParts consecutive lanes of a group (every lane passes its part): the
// lanes' parts are summed as ((q0 + q1) + (q2 + q3)), and every lane of the group returns
// the same double-float.  All dot products, norms included, go through this routine.
template <int D>
__device__ __forceinline__ DFPair group_dot_df(const uint16_t* __restrict__ a,
                                             const uint16_t* __restrict__ b, int part)
{
    float hi, lo;
    quarter_dot<D>(a, b, part, hi, lo);
#pragma unroll
    for (int o = 1; o < kParts; o <<= 1) {
        const float h2 = __shfl_xor_sync(0xFFFFFFFFu, hi, o);
        const float l2 = __shfl_xor_sync(0xFFFFFFFFu, lo, o);
        df_add(hi, lo, h2, l2);
    }
    return DFPair{hi, lo};
}

// The same two dot products a . b0 and a . b1 at once, one in each half of paired
// (f32x2) instructions: each half performs exactly the scalar sequence of
// group_dot_df, with the same rounding, term order and combine tree, so each result
// equals group_dot_df's bit for bit.
__device__ __forceinline__ float2 neg2(float2 a) { return make_float2(-a.x, -a.y); }

__device__ __forceinline__ void two_sum_acc2(float2& hi, float2& lo, float2 p)
{
    const float2 s = __fadd2_rn(hi, p);
    const float2 bp = __fadd2_rn(s, neg2(hi));
    const float2 e = __fadd2_rn(__fadd2_rn(hi, neg2(__fadd2_rn(s, neg2(bp)))),
                                __fadd2_rn(p, neg2(bp)));
    hi = s;
    lo = __fadd2_rn(lo, e);
}

__device__ __forceinline__ void df_add2(float2& hi, float2& lo, float2 hi2, float2 lo2)
{
    const float2 s = __fadd2_rn(hi, hi2);
    const float2 bp = __fadd2_rn(s, neg2(hi));
    float2 e = __fadd2_rn(__fadd2_rn(hi, neg2(__fadd2_rn(s, neg2(bp)))), __fadd2_rn(hi2, neg2(bp)));
    e = __fadd2_rn(e, __fadd2_rn(lo, lo2));
    hi = __fadd2_rn(s, e);
    lo = __fadd2_rn(e, neg2(__fadd2_rn(hi, neg2(s))));
}

// b1 is read only where use1 (elsewhere its terms are zero and r1 is meaningless).
template <int D>
__device__ __forceinline__ void group_dot2_df(const uint16_t* __restrict__ a,
                                              const uint16_t* __restrict__ b0,
                                              const uint16_t* __restrict__ b1, bool use1,
                                              int part, DFPair& r0, DFPair& r1)
{
    constexpr int Q = D / 8 / kParts;
    const uint4* a4 = reinterpret_cast<const uint4*>(a) + part;
    const uint4* c4 = reinterpret_cast<const uint4*>(b0) + part;
    const uint4* d4 = reinterpret_cast<const uint4*>(b1) + part;
    float2 hi = make_float2(0.f, 0.f), lo = make_float2(0.f, 0.f);
#pragma unroll
    for (int q = 0; q < Q; ++q) {
        const uint4 va = __ldg(a4 + q * kParts);
        const uint4 vc = __ldg(c4 + q * kParts);
        const uint4 vd = use1 ? __ldg(d4 + q * kParts) : make_uint4(0u, 0u, 0u, 0u);
        const uint32_t wa[4] = {va.x, va.y, va.z, va.w};
        const uint32_t wc[4] = {vc.x, vc.y, vc.z, vc.w};
        const uint32_t wd[4] = {vd.x, vd.y, vd.z, vd.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const float lo_a = __uint_as_float(wa[k] << 16);
            const float hi_a = __uint_as_float(wa[k] & 0xFFFF0000u);
            two_sum_acc2(hi, lo, __fmul2_rn(make_float2(lo_a, lo_a),
                                            make_float2(__uint_as_float(wc[k] << 16),
                                                        __uint_as_float(wd[k] << 16))));
            two_sum_acc2(hi, lo, __fmul2_rn(make_float2(hi_a, hi_a),
                                            make_float2(__uint_as_float(wc[k] & 0xFFFF0000u),
                                                        __uint_as_float(wd[k] & 0xFFFF0000u))));
        }
    }
#pragma unroll
    for (int o = 1; o < kParts; o <<= 1) {
        const float2 h2 = make_float2(__shfl_xor_sync(0xFFFFFFFFu, hi.x, o),
                                      __shfl_xor_sync(0xFFFFFFFFu, hi.y, o));
        const float2 l2 = make_float2(__shfl_xor_sync(0xFFFFFFFFu, lo.x, o),
                                      __shfl_xor_sync(0xFFFFFFFFu, lo.y, o));
        df_add2(hi, lo, h2, l2);
    }
    r0 = DFPair{hi.x, lo.x};
    r1 = DFPair{hi.y, lo.y};
}

// ---- double-float (unevaluated fp32 pair) helpers --------------------------------

using DF = DFPair;

// a * b as a double-float.  The cross terms are summed as (a.h * b.l + a.l * b.h), so
// the result does not depend on the operand order.
__device__ __forceinline__ DF df_mul(DF a, DF b)
{
    const float p = __fmul_rn(a.h, b.h);
    float e = __fmaf_rn(a.h, b.h, -p);
    e = __fadd_rn(e, __fadd_rn(__fmul_rn(a.h, b.l), __fmul_rn(a.l, b.h)));
    const float h = __fadd_rn(p, e);
    return DF{h, __fsub_rn(e, __fsub_rn(h, p))};
}

// 1/sqrt(s) for s > 0 (about 2^-44 relative): one Newton step around rsqrtf, with the
// residual 1 - s r^2 formed in double-float.
__device__ __forceinline__ DF df_rsqrt(DF s)
{
    const float r = rsqrtf(s.h);
    const float r2h = __fmul_rn(r, r);
    const float r2l = __fmaf_rn(r, r, -r2h);
    const float th = __fmul_rn(s.h, r2h);
    const float tl = __fadd_rn(__fmaf_rn(s.h, r2h, -th),
                               __fadd_rn(__fmul_rn(s.h, r2l), __fmul_rn(s.l, r2h)));
    const float e = __fsub_rn(__fsub_rn(1.0f, th), tl);   // 1 - th is exact (th ~ 1)
    const float c = __fmul_rn(__fmul_rn(r, e), 0.5f);
    const float h = __fadd_rn(r, c);
    return DF{h, __fsub_rn(c, __fsub_rn(h, r))};
}

__device__ __forceinline__ double df_to_double(DF a)
{
    return static_cast<double>(a.h) + static_cast<double>(a.l);
}

}  // namespace twk
