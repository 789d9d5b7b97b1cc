// twk_prep.cu -- O(N d) preparation for the audit (TwinKV, arXiv 2608.27128):
//   * float32 keys -> bf16 (round to nearest even),
//   * per key k . k and 1/||k|| (the l2 normalisation of Sec. 3.2 Eq. 1, applied later
//     as a scale; a zero key gets 0, so it has similarity 0 with every key),
//   * the retained-first column layout used by the repair audit: retained keys in
//     position order, padded to a 256-column tile, then evicted keys in position order,
//     with per-column 1/||k|| (NaN on padding columns, which the audit then ignores)
//     and per-column original position.
#include <cuda_bf16.h>

#include "twk_df.cuh"
#include "twk_internal.h"

namespace twk {
namespace {

__device__ __forceinline__ float nan_f() { return __uint_as_float(0x7FFFFFFFu); }

__global__ void round_bf16_kernel(const float* __restrict__ in, uint16_t* __restrict__ out,
                                  int64_t n)
{
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
         i += stride)
        out[i] = __bfloat16_as_ushort(__float2bfloat16_rn(in[i]));
}

constexpr int kPrepThreads = 256;
constexpr int kKeysPerBlock = kPrepThreads / kParts;   // NP is a multiple of this

// The norm record of one key, computed by its kParts-lane group: k.k and 1/||k|| as
// double-floats (for the exact similarity values) and 1/||k|| in fp32 (for the audit).
template <int D>
__device__ __forceinline__ float4 key_norms(const uint16_t* key, int part, float& rinv32)
{
    const DF sq = group_dot_df<D>(key, key, part);
    const DF rn = sq.h > 0.f ? df_rsqrt(sq) : DF{0.f, 0.f};
    rinv32 = rn.h;
    return make_float4(sq.h, sq.l, rn.h, rn.l);
}

// The largest k.k of unit u so far, as float bits (k.k >= 0, so the unsigned order of
// the bits is the float order): one atomic per block (hundreds of blocks share a unit's
// word, so per-warp atomics queue up).  Every thread of the block calls it; lanes pass
// 0 for nothing.
__device__ __forceinline__ void unit_max_kk(unsigned* unit_kk, int64_t u, float kk)
{
    __shared__ unsigned wmax[kPrepThreads / 32];
    const unsigned m = __reduce_max_sync(0xFFFFFFFFu, __float_as_uint(kk));
    if ((threadIdx.x & 31) == 0) wmax[threadIdx.x >> 5] = m;
    __syncthreads();
    if (threadIdx.x == 0) {
        unsigned t = 0u;
#pragma unroll
        for (int w = 0; w < kPrepThreads / 32; ++w) t = max(t, wmax[w]);
        if (t != 0u) atomicMax(unit_kk + u, t);
    }
}

// Mode 0 (keys as given): per column p of unit blockIdx.y, colrinv = rscale/||k_p||
// (rscale a power of two, so the scaling is exact) and colpos = p, NaN / -1 on the
// padding columns [N, NP); norms[u][p] = the norm record; unit_kk[u] (if given) =
// the unit's largest k.k.  Grid (NP / kKeysPerBlock, U), kParts lanes per column.
template <int D>
__global__ void __launch_bounds__(kPrepThreads)
    norms_identity_kernel(const uint16_t* __restrict__ keys, int N, int64_t NP,
                          float* __restrict__ colrinv, int* __restrict__ colpos,
                          float4* __restrict__ norms, float rscale, unsigned* unit_kk)
{
    const int part = threadIdx.x % kParts;
    const int p = blockIdx.x * kKeysPerBlock + threadIdx.x / kParts;
    const int64_t u = blockIdx.y;
    // every lane takes part in the shuffles of group_dot_df: padding columns use key 0
    const int pk = p < N ? p : 0;
    float r32;
    const float4 nr = key_norms<D>(keys + (u * N + pk) * D, part, r32);
    if (part == 0) {
        colrinv[u * NP + p] = p < N ? r32 * rscale : nan_f();
        colpos[u * NP + p] = p < N ? p : -1;
        if (p < N) norms[u * N + p] = nr;
    }
    if (unit_kk) unit_max_kk(unit_kk, u, (part == 0 && p < N) ? nr.x : 0.f);
}

// Mode 1, step 1: cnt[u][p] = number of retained positions before p; kb[u] = |S0|.
// One block per unit; a mask byte counts as retained when non-zero.
__global__ void scan_kernel(const uint8_t* __restrict__ mask, int N, int* __restrict__ cnt,
                            int* __restrict__ kb)
{
    __shared__ int warp_tot[32];
    __shared__ int carry;
    const int u = blockIdx.x;
    const uint8_t* m = mask + static_cast<int64_t>(u) * N;
    int* c = cnt + static_cast<int64_t>(u) * N;
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = blockDim.x >> 5;
    if (threadIdx.x == 0) carry = 0;
    __syncthreads();
    for (int base = 0; base < N; base += blockDim.x) {
        const int p = base + threadIdx.x;
        const int f = (p < N && m[p] != 0) ? 1 : 0;
        int x = f;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xFFFFFFFFu, x, o);
            if (lane >= o) x += y;
        }
        if (lane == 31) warp_tot[wid] = x;
        __syncthreads();
        if (wid == 0) {
            int t = lane < nw ? warp_tot[lane] : 0;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int y = __shfl_up_sync(0xFFFFFFFFu, t, o);
                if (lane >= o) t += y;
            }
            if (lane < nw) warp_tot[lane] = t;   // inclusive prefix of warp totals
        }
        __syncthreads();
        const int before = carry + (wid > 0 ? warp_tot[wid - 1] : 0) + (x - f);
        if (p < N) c[p] = before;
        __syncthreads();
        if (threadIdx.x == 0) carry += warp_tot[nw - 1];
        __syncthreads();
    }
    if (threadIdx.x == 0) kb[u] = carry;
}

// Mode 1, step 2: slot p < N of unit blockIdx.y is key p: its kParts-lane group copies
// it to its column of the retained-first layout (retained keys in position order, then
// from the next tile boundary the evicted ones), with 1/||k_p|| (fp32) and p as column
// metadata, and writes its norm record.  Slots p >= N are the padding columns
// [K, Kpad) and [Kpad + N - K, NP): zero keys, NaN, -1.  unit_kk[u] = the unit's
// largest k.k.  Grid (NP / kKeysPerBlock, U).
template <int D>
__global__ void __launch_bounds__(kPrepThreads)
    gather_kernel(const uint16_t* __restrict__ keys, const uint8_t* __restrict__ mask,
                  const int* __restrict__ cnt, const int* __restrict__ kb, int N, int64_t NP,
                  uint16_t* __restrict__ kp, float* __restrict__ colrinv,
                  int* __restrict__ colpos, float4* __restrict__ norms, unsigned* unit_kk)
{
    constexpr int Q = D / 8 / kParts;   // 16-byte chunks per lane
    const int part = threadIdx.x % kParts;
    const int p = blockIdx.x * kKeysPerBlock + threadIdx.x / kParts;
    const int64_t u = blockIdx.y;
    const int k = kb[u];
    const int kpad = ((k + kBN - 1) / kBN) * kBN;
    const int pk = p < N ? p : 0;   // every lane takes part in the shuffles
    const uint16_t* key = keys + (u * N + pk) * D;
    float r32;
    const float4 nr = key_norms<D>(key, part, r32);
    int col;
    if (p < N) {
        const int before = cnt[u * N + p];
        col = mask[u * N + p] ? before : kpad + (p - before);
    } else {
        const int r = p - N;
        col = r < kpad - k ? k + r : kpad + (N - k) + (r - (kpad - k));
    }
    // the lane's 16-byte chunks part, part + kParts, ... (those its dot product read)
    const uint4* src = reinterpret_cast<const uint4*>(key) + part;
    uint4* dst = reinterpret_cast<uint4*>(kp + (u * NP + col) * D) + part;
#pragma unroll
    for (int q = 0; q < Q; ++q)
        dst[q * kParts] = p < N ? __ldg(src + q * kParts) : make_uint4(0u, 0u, 0u, 0u);
    if (part == 0) {
        colrinv[u * NP + col] = p < N ? r32 : nan_f();
        colpos[u * NP + col] = p < N ? p : -1;
        if (p < N) norms[u * N + p] = nr;
    }
    unit_max_kk(unit_kk, u, (part == 0 && p < N) ? nr.x : 0.f);
}

// colrinv[u][c] *= 2^-e_u, the power of two with 2^e_u >= the largest ||k|| of unit u
// (from unit_kk), so that every scaled similarity x_ij * colrinv_j = sim(i,j) ||k_i||
// 2^-e_u lies in [-1, 1].  Exact (a power of two); NaN padding stays NaN.  A unit of
// zero keys keeps its scale.  Grid (NP / kPrepThreads, U).
__global__ void __launch_bounds__(kPrepThreads)
    scale_columns_kernel(float* __restrict__ colrinv, int64_t NP,
                         const unsigned* __restrict__ unit_kk)
{
    const int64_t u = blockIdx.y;
    const int64_t c = static_cast<int64_t>(blockIdx.x) * kPrepThreads + threadIdx.x;
    const float kk = __uint_as_float(unit_kk[u]);
    if (c >= NP || !(kk > 0.f)) return;
    int E;
    (void)frexpf(kk, &E);               // kk < 2^E, so ||k|| < 2^ceil(E / 2)
    const int e = (E + 1) >> 1;          // ceil(E / 2), also for E <= 0
    colrinv[u * NP + c] = ldexpf(colrinv[u * NP + c], -e);
}


}  // namespace

cudaError_t launch_round_bf16(const float* in, uint16_t* out, int64_t n, cudaStream_t st)
{
    int64_t blocks = (n + 255) / 256;
    if (blocks > 65535LL * 16) blocks = 65535LL * 16;
    if (blocks < 1) blocks = 1;
    round_bf16_kernel<<<static_cast<int>(blocks), 256, 0, st>>>(in, out, n);
    return cudaGetLastError();
}

cudaError_t launch_norms_identity(const uint16_t* keys, int U, int N, int d, int64_t NP,
                                  float* colrinv, int* colpos, float4* norms, cudaStream_t st,
                                  float rscale, unsigned* unit_kk)
{
    const dim3 grid(static_cast<unsigned>(NP / kKeysPerBlock), U);
    if (d == 128)
        norms_identity_kernel<128><<<grid, kPrepThreads, 0, st>>>(keys, N, NP, colrinv, colpos,
                                                                   norms, rscale, unit_kk);
    else
        norms_identity_kernel<64><<<grid, kPrepThreads, 0, st>>>(keys, N, NP, colrinv, colpos,
                                                                  norms, rscale, unit_kk);
    return cudaGetLastError();
}

cudaError_t launch_scale_columns(float* colrinv, int U, int64_t NP, const unsigned* unit_kk,
                                 cudaStream_t st)
{
    const dim3 grid(static_cast<unsigned>((NP + kPrepThreads - 1) / kPrepThreads), U);
    scale_columns_kernel<<<grid, kPrepThreads, 0, st>>>(colrinv, NP, unit_kk);
    return cudaGetLastError();
}

cudaError_t launch_scan(const uint8_t* mask, int U, int N, int* cnt, int* kb, cudaStream_t st)
{
    scan_kernel<<<U, 1024, 0, st>>>(mask, N, cnt, kb);
    return cudaGetLastError();
}

cudaError_t launch_gather(const uint16_t* keys, const uint8_t* mask, const int* cnt,
                          const int* kb, int U, int N, int d, int64_t NP, uint16_t* kp,
                          float* colrinv, int* colpos, float4* norms, unsigned* unit_kk,
                          cudaStream_t st)
{
    const dim3 grid(static_cast<unsigned>(NP / kKeysPerBlock), U);
    if (d == 128)
        gather_kernel<128><<<grid, kPrepThreads, 0, st>>>(keys, mask, cnt, kb, N, NP, kp,
                                                           colrinv, colpos, norms, unit_kk);
    else
        gather_kernel<64><<<grid, kPrepThreads, 0, st>>>(keys, mask, cnt, kb, N, NP, kp,
                                                          colrinv, colpos, norms, unit_kk);
    return cudaGetLastError();
}

}  // namespace twk
