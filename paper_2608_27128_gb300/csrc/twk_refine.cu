// twk_refine.cu -- exact value of the winning similarity (TwinKV, arXiv 2608.27128,
// Sec. 3.2 Eq. 1).
//
// The audit kernel picks each row's twin from fp32 tensor-core dot products whose low
// mantissa bits carry the column index, so its own score is only good to ~2^-16.  This
// pass recomputes, for the chosen twin j of every row i,
//     sim(i, j) = (k_i . k_j) / sqrt((k_i . k_i) (k_j . k_j))
// with every dot product formed as a double-float sum: each bf16 x bf16 product is
// exact in fp32, and the running sum is an unevaluated pair (hi, lo) updated with
// Knuth's TwoSum, so its error is of order 2^-48 of the sum of |products|.  The final
// product, square root and quotient are rounded once each in fp64.  All dot products
// (norms included) use the same routine and term order, so the result is symmetric in
// (i, j) bit for bit and exactly 1 for a duplicate.
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

// sum over t in increasing order of a[t] * b[t] for two bf16 rows of length D.
template <int D>
__device__ __forceinline__ double exact_dot(const uint16_t* __restrict__ a,
                                            const uint16_t* __restrict__ b)
{
    const uint4* a4 = reinterpret_cast<const uint4*>(a);
    const uint4* b4 = reinterpret_cast<const uint4*>(b);
    float hi = 0.f, lo = 0.f;
#pragma unroll 2
    for (int q = 0; q < D / 8; ++q) {
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
    return static_cast<double>(hi) + static_cast<double>(lo);
}

// norm2[u][p] = k_p . k_p, one thread per key.
template <int D>
__global__ void norm2_kernel(const uint16_t* __restrict__ keys, int64_t n, double* __restrict__ norm2)
{
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t r = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; r < n; r += stride) {
        const uint16_t* k = keys + r * D;
        norm2[r] = exact_dot<D>(k, k);
    }
}

__device__ __forceinline__ double cosine(double dot, double si, double sj)
{
    if (si == 0.0 || sj == 0.0) return 0.0;
    return dot / sqrt(si * sj);
}

// For every row (u, i): b0 = sim(i, twin0), -1 where twin0 is -1 (empty candidate
// set, Eq. 4).  With twin1 (the best evicted column) given, the best over all columns
// is the larger of sim(i, twin0) and sim(i, twin1), the lower position on an exact tie;
// twin1 is overwritten with it and b1 (if given) receives its value.
template <int D>
__global__ void refine_kernel(const uint16_t* __restrict__ keys, int U, int N,
                              const double* __restrict__ norm2, const int* __restrict__ twin0,
                              int* __restrict__ twin1, double* __restrict__ b0,
                              double* __restrict__ b1)
{
    const int64_t n = static_cast<int64_t>(U) * N;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t r = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; r < n; r += stride) {
        const int64_t base = (r / N) * N;
        const uint16_t* ki = keys + r * D;
        const double si = norm2[r];
        const int j0 = twin0[r];
        const double v0 = j0 < 0 ? -1.0
                                 : cosine(exact_dot<D>(ki, keys + (base + j0) * D), si,
                                          norm2[base + j0]);
        b0[r] = v0;
        if (twin1) {
            const int j1 = twin1[r];
            int jb = j0;
            double vb = v0;
            if (j1 >= 0) {
                const double v1 =
                    cosine(exact_dot<D>(ki, keys + (base + j1) * D), si, norm2[base + j1]);
                if (j0 < 0 || v1 > v0 || (v1 == v0 && j1 < j0)) {
                    jb = j1;
                    vb = v1;
                }
            }
            twin1[r] = jb;
            if (b1) b1[r] = vb;
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

cudaError_t launch_norm2(const uint16_t* keys, int64_t n, int d, double* norm2, cudaStream_t st)
{
    if (d == 128)
        norm2_kernel<128><<<blocks_for(n, 256), 256, 0, st>>>(keys, n, norm2);
    else
        norm2_kernel<64><<<blocks_for(n, 256), 256, 0, st>>>(keys, n, norm2);
    return cudaGetLastError();
}

cudaError_t launch_refine(const uint16_t* keys, int U, int N, int d, const double* norm2,
                          const int* twin0, int* twin1, double* b0, double* b1,
                          cudaStream_t st)
{
    const int64_t n = static_cast<int64_t>(U) * N;
    if (d == 128)
        refine_kernel<128><<<blocks_for(n, 128), 128, 0, st>>>(keys, U, N, norm2, twin0, twin1,
                                                               b0, b1);
    else
        refine_kernel<64><<<blocks_for(n, 128), 128, 0, st>>>(keys, U, N, norm2, twin0, twin1,
                                                              b0, b1);
    return cudaGetLastError();
}

}  // namespace twk
