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
// share a dot product (every fourth 16-byte chunk each, combined in a fixed tree).  The
// cosine is then (k_i . k_j) * (1/||k_i|| * 1/||k_j||) in double-float arithmetic
// (relative error below 1e-12; fp64 square roots and quotients are slow on this GPU),
// except within 2^-20 of +-1, where the exact fp64 form is used.  All dot products
// (norms included) use the same routine and term order (the paired version used when a
// row has two candidates computes each dot exactly as the single one), and the product
// of the two inverse norms is formed symmetrically, so the result is symmetric in
// (i, j) bit for bit and exactly 1 for a duplicate.
#include "twk_df.cuh"
#include "twk_internal.h"

namespace twk {
namespace {

// This GPU's FP64 pipe runs at a small fraction of its FP32 rate, so the values stay
// double-floats until each output is written: comparisons are made on the pairs, and a
// pair becomes a double by widening both floats with integer operations and one fp64
// addition (exact: the pair's 48 significant bits fit in a double).

// A float as a double, for zero and normal floats by moving its bits (the conversion
// instruction for the rest, which similarity values do not reach).
__device__ __forceinline__ double widen(float f)
{
    const uint32_t u = __float_as_uint(f);
    const uint32_t e = (u >> 23) & 0xFFu;
    const uint64_t sign = static_cast<uint64_t>(u & 0x80000000u) << 32;
    if ((u & 0x7FFFFFFFu) == 0u) return __longlong_as_double(static_cast<long long>(sign));
    if (e == 0u || e == 0xFFu) return static_cast<double>(f);
    return __longlong_as_double(static_cast<long long>(
        sign | (static_cast<uint64_t>(e + 896u) << 52) | (static_cast<uint64_t>(u & 0x7FFFFFu) << 29)));
}

__device__ __forceinline__ double to_double(DF a) { return widen(a.h) + widen(a.l); }

// a > b and a == b for normalised pairs (|l| at most half an ulp of h).
__device__ __forceinline__ bool df_gt(DF a, DF b) { return a.h > b.h || (a.h == b.h && a.l > b.l); }
__device__ __forceinline__ bool df_eq(DF a, DF b) { return a.h == b.h && a.l == b.l; }

// sim(i, j) of Eq. 1 from the dot product and the two keys' norm records, as a
// double-float.
__device__ __forceinline__ DF cosine(DF dot, float4 ni, float4 nj)
{
    if (ni.x == 0.f || nj.x == 0.f) return DF{0.f, 0.f};   // a zero key has similarity 0
    const DF c = df_mul(dot, df_mul(DF{ni.z, ni.w}, DF{nj.z, nj.w}));
    if (fabsf(c.h) < 1.0f - 0x1p-20f) return c;
    // Within 2^-20 of +-1: the exact fp64 form, which gives exactly +-1 when the keys
    // are parallel (a duplicate, or a copy scaled by a power of two), split back into a
    // pair (its leading 48 bits).
    const double si = to_double(DF{ni.x, ni.y});
    const double sj = to_double(DF{nj.x, nj.y});
    const double x = to_double(dot) / sqrt(si * sj);
    const float h = static_cast<float>(x);
    return DF{h, static_cast<float>(x - static_cast<double>(h))};
}

constexpr int kRefineThreads = 256;
constexpr int kRowsPerBlock = kRefineThreads / kParts;

// For every row (u, i): b0 = sim(i, twin0), -1 where twin0 is -1 (empty candidate
// set, Eq. 4).  With twin1 (the best evicted column, -1 when the evicted columns do not
// reach the retained best) given, the best over all columns is the larger of
// sim(i, twin0) and sim(i, twin1), the lower position on an exact tie; twin1 is
// overwritten with it and b1 (if given) receives its value.  Grid: (row blocks, units),
// kParts threads per row.  kMinBlocks = 5 (at most 51 registers) is the standalone
// launch; 6 caps the registers at 40 so that a block fits on an SM beside a persistent
// audit CTA.
template <int D, int kMinBlocks>
__global__ void __launch_bounds__(kRefineThreads, kMinBlocks)
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
    const int64_t s1 = base + (j1 >= 0 ? j1 : r - base);
    // The standalone launch loads the norm records the cosine needs (the row's, and
    // the twin's this lane evaluates) beside the keys rather than after the dot
    // product; the launch beside the audit has no registers to hold them.
    constexpr bool kEarly = kMinBlocks < 6;
    float4 nr{}, nt{};
    if constexpr (kEarly) {
        nr = norms[r];
        nt = norms[part == 1 ? s1 : s0];
    }
    DF d0, d1{0.f, 0.f};
    if (__any_sync(0xFFFFFFFFu, j1 >= 0))   // both dots at once, one per f32x2 half
        group_dot2_df<D>(ki, keys + s0 * D, keys + s1 * D, j1 >= 0, part, d0, d1);
    else
        d0 = group_dot_df<D>(ki, keys + s0 * D, part);
    // lane 0 of the group evaluates the first cosine, lane 1 the second
    DF v{-1.f, 0.f};
    if (part == 0 && j0 >= 0) v = cosine(d0, kEarly ? nr : norms[r], kEarly ? nt : norms[s0]);
    if (part == 1 && j1 >= 0) v = cosine(d1, kEarly ? nr : norms[r], kEarly ? nt : norms[s1]);
    const DF v0 = v;
    const DF v1{__shfl_down_sync(0xFFFFFFFFu, v.h, 1), __shfl_down_sync(0xFFFFFFFFu, v.l, 1)};
    if (part == 0 && live) {
        b0[r] = to_double(v0);
        if (twin1) {
            const bool take1 =
                j1 >= 0 && (j0 < 0 || df_gt(v1, v0) || (df_eq(v1, v0) && j1 < j0));
            twin1[r] = take1 ? j1 : j0;
            if (b1) b1[r] = to_double(take1 ? v1 : v0);
        }
    }
}


}  // namespace

cudaError_t launch_refine(const uint16_t* keys, int U, int N, int d, const float4* norms,
                          const int* twin0, int* twin1, double* b0, double* b1,
                          cudaStream_t st, bool beside_audit)
{
    const dim3 grid((N + kRowsPerBlock - 1) / kRowsPerBlock, U);
    if (d == 128 && beside_audit)
        refine_kernel<128, 6><<<grid, kRefineThreads, 0, st>>>(keys, N, norms, twin0, twin1, b0, b1);
    else if (d == 128)
        refine_kernel<128, 5><<<grid, kRefineThreads, 0, st>>>(keys, N, norms, twin0, twin1, b0, b1);
    else if (beside_audit)
        refine_kernel<64, 6><<<grid, kRefineThreads, 0, st>>>(keys, N, norms, twin0, twin1, b0, b1);
    else
        refine_kernel<64, 5><<<grid, kRefineThreads, 0, st>>>(keys, N, norms, twin0, twin1, b0, b1);
    return cudaGetLastError();
}

}  // namespace twk
