// twk_refine.cu -- exact value of the winning similarity (TwinKV, arXiv 2608.27128,
// Sec. 3.2 Eq. 1).
//
// The audit kernel picks each row's twin from fp32 tensor-core dot products whose low
// mantissa bits carry the column index, so its own score is only good to ~2^-16.  This
// pass recomputes, for the chosen twin j of every row i,
//     sim(i, j) = (k_i . k_j) / sqrt((k_i . k_i) (k_j . k_j))
// with every dot product formed as a double-float sum: each bf16 x bf16 product is
// exact in fp32, and the running sum is an unevaluated pair (hi, lo) updated with
// Knuth's TwoSum, so its error is of order 2^-48 of the sum of |products|.  Four lanes
// share a dot product (a contiguous quarter each, combined in a fixed tree).  The
// cosine is then (k_i . k_j) * (1/||k_i|| * 1/||k_j||) in double-float arithmetic
// (relative error below 1e-12; fp64 square roots and quotients are slow on this GPU),
// except within 2^-20 of +-1, where the exact fp64 form is used.  All dot products
// (norms included) use the same routine and term order, and the product of the two
// inverse norms is formed symmetrically, so the result is symmetric in (i, j) bit for
// bit and exactly 1 for a duplicate.
#include "twk_internal.h"

namespace twk {
namespace {

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

constexpr int kParts = 4;   // threads per dot product, each over a contiguous quarter

// One quarter of a . b for two bf16 rows of length D: terms in increasing t.
template <int D>
__device__ __forceinline__ void quarter_dot(const uint16_t* __restrict__ a,
                                            const uint16_t* __restrict__ b, int part,
                                            float& hi, float& lo)
{
    constexpr int Q = D / 8 / kParts;   // 16-byte chunks per quarter
    const uint4* a4 = reinterpret_cast<const uint4*>(a) + part * Q;
    const uint4* b4 = reinterpret_cast<const uint4*>(b) + part * Q;
    hi = 0.f;
    lo = 0.f;
#pragma unroll
    for (int q = 0; q < Q; ++q) {
        const uint4 va = __ldg(a4 + q);
        const uint4 vb = __ldg(b4 + q);
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
// quarters are summed as ((q0 + q1) + (q2 + q3)), and every lane of the group returns
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

// Per key: its squared norm k . k and 1/||k||, both as double-floats, in one float4
// {k.k hi, k.k lo, rinv hi, rinv lo}; kParts threads per key.
template <int D>
__global__ void norms_kernel(const uint16_t* __restrict__ keys, int64_t n,
                             float4* __restrict__ norms)
{
    const int part = threadIdx.x % kParts;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * (blockDim.x / kParts);
    const int64_t first = blockIdx.x * static_cast<int64_t>(blockDim.x / kParts) + threadIdx.x / kParts;
    // every group iterates the same number of times, so the shuffles stay converged
    const int64_t iters = (n + stride - 1) / stride;
    for (int64_t it = 0; it < iters; ++it) {
        const int64_t r = first + it * stride;
        const int64_t rr = r < n ? r : n - 1;
        const uint16_t* k = keys + rr * D;
        const DF sq = group_dot_df<D>(k, k, part);
        if (part == 0 && r < n) {
            const DF rn = sq.h > 0.f ? df_rsqrt(sq) : DF{0.f, 0.f};
            norms[r] = make_float4(sq.h, sq.l, rn.h, rn.l);
        }
    }
}

// sim(i, j) of Eq. 1 from the dot product and the two keys' norm records.
__device__ __forceinline__ double cosine(DF dot, float4 ni, float4 nj)
{
    if (ni.x == 0.f || nj.x == 0.f) return 0.0;   // a zero key has similarity 0
    const DF c = df_mul(dot, df_mul(DF{ni.z, ni.w}, DF{nj.z, nj.w}));
    if (fabsf(c.h) < 1.0f - 0x1p-20f) return df_to_double(c);
    // Within 2^-20 of +-1: the exact fp64 form, which gives exactly +-1 when the keys
    // are parallel (a duplicate, or a copy scaled by a power of two).
    const double si = df_to_double(DF{ni.x, ni.y});
    const double sj = df_to_double(DF{nj.x, nj.y});
    return df_to_double(dot) / sqrt(si * sj);
}

constexpr int kRefineThreads = 256;
constexpr int kRowsPerBlock = kRefineThreads / kParts;

// For every row (u, i): b0 = sim(i, twin0), -1 where twin0 is -1 (empty candidate
// set, Eq. 4).  With twin1 (the best evicted column, -1 when the evicted columns do not
// reach the retained best) given, the best over all columns is the larger of
// sim(i, twin0) and sim(i, twin1), the lower position on an exact tie; twin1 is
// overwritten with it and b1 (if given) receives its value.  Grid: (row blocks, units),
// kParts threads per row.
template <int D>
__global__ void __launch_bounds__(kRefineThreads)
    refine_kernel(const uint16_t* __restrict__ keys, int N, const float4* __restrict__ norms,
                  const int* __restrict__ twin0, int* __restrict__ twin1,
                  double* __restrict__ b0, double* __restrict__ b1)
{
    const int part = threadIdx.x % kParts;
    const int i = blockIdx.x * kRowsPerBlock + threadIdx.x / kParts;
    const bool live = i < N;
    const int64_t base = static_cast<int64_t>(blockIdx.y) * N;
    const int64_t r = base + (live ? i : N - 1);
    const uint16_t* ki = keys + r * D;
    const int j0 = twin0[r];
    const int j1 = twin1 ? twin1[r] : -1;
    // Every lane of the warp takes part in the shuffled dot products; a missing twin is
    // stood in for by the row itself and its value discarded.
    const int64_t s0 = base + (j0 >= 0 ? j0 : r - base);
    const DF d0 = group_dot_df<D>(ki, keys + s0 * D, part);
    DF d1{0.f, 0.f};
    int64_t s1 = s0;
    if (__any_sync(0xFFFFFFFFu, j1 >= 0)) {
        s1 = base + (j1 >= 0 ? j1 : r - base);
        d1 = group_dot_df<D>(ki, keys + s1 * D, part);
    }
    // lane 0 of the group evaluates the first cosine, lane 1 the second
    double v = -1.0;
    if (part == 0 && j0 >= 0) v = cosine(d0, norms[r], norms[s0]);
    if (part == 1 && j1 >= 0) v = cosine(d1, norms[r], norms[s1]);
    const double v0 = v;
    const double v1 = __shfl_down_sync(0xFFFFFFFFu, v, 1);
    if (part == 0 && live) {
        b0[r] = v0;
        if (twin1) {
            const bool take1 = j1 >= 0 && (j0 < 0 || v1 > v0 || (v1 == v0 && j1 < j0));
            twin1[r] = take1 ? j1 : j0;
            if (b1) b1[r] = take1 ? v1 : v0;
        }
    }
}

int blocks_for(int64_t n, int threads)
{
    int64_t b = (n + threads - 1) / threads;
    if (b > 65535LL * 16) b = 65535LL * 16;
    return static_cast<int>(b < 1 ? 1 : b);
}

}  // namespace

cudaError_t launch_norms(const uint16_t* keys, int64_t n, int d, float4* norms, cudaStream_t st)
{
    const int blocks = blocks_for(n * kParts, 256);
    if (d == 128)
        norms_kernel<128><<<blocks, 256, 0, st>>>(keys, n, norms);
    else
        norms_kernel<64><<<blocks, 256, 0, st>>>(keys, n, norms);
    return cudaGetLastError();
}

cudaError_t launch_refine(const uint16_t* keys, int U, int N, int d, const float4* norms,
                          const int* twin0, int* twin1, double* b0, double* b1,
                          cudaStream_t st)
{
    const dim3 grid((N + kRowsPerBlock - 1) / kRowsPerBlock, U);
    if (d == 128)
        refine_kernel<128><<<grid, kRefineThreads, 0, st>>>(keys, N, norms, twin0, twin1, b0, b1);
    else
        refine_kernel<64><<<grid, kRefineThreads, 0, st>>>(keys, N, norms, twin0, twin1, b0, b1);
    return cudaGetLastError();
}

}  // namespace twk
