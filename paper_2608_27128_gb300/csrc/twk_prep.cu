// twk_prep.cu -- O(N d) preparation for the audit (TwinKV, arXiv 2608.27128):
//   * float32 keys -> bf16 (round to nearest even),
//   * 1/||k|| per key, the l2 normalisation of Sec. 3.2 Eq. 1, applied later as a scale
//     (a zero key gets 0, so it has similarity 0 with every key),
//   * the retained-first column layout used by the repair audit: retained keys in
//     position order, padded to a 256-column tile, then evicted keys in position order,
//     with per-column 1/||k|| (NaN on padding columns, which the audit then ignores)
//     and per-column original position.
#include <cuda_bf16.h>

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

// Sum of squares of one bf16 key row by a full warp; returns 1/||k|| (0 for k = 0).
template <int D>
__device__ __forceinline__ float warp_rinv(const uint16_t* row, uint32_t (&v)[D / 64])
{
    float sq = 0.f;
    const uint32_t* r32 = reinterpret_cast<const uint32_t*>(row);
#pragma unroll
    for (int k = 0; k < D / 64; ++k) {
        v[k] = r32[k * 32 + (threadIdx.x & 31)];
        const float lo = __uint_as_float(v[k] << 16);
        const float hi = __uint_as_float(v[k] & 0xFFFF0000u);
        sq = fmaf(lo, lo, sq);
        sq = fmaf(hi, hi, sq);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xFFFFFFFFu, sq, o);
    return sq > 0.f ? 1.0f / sqrtf(sq) : 0.f;
}

// Mode 0 (keys as given): colrinv[u][p] = 1/||k_p||, colpos[u][p] = p; padding columns
// p in [N, NP) get NaN / -1.  One warp per column.
template <int D>
__global__ void norms_identity_kernel(const uint16_t* __restrict__ keys, int U, int N,
                                      int64_t NP, float* __restrict__ colrinv,
                                      int* __restrict__ colpos)
{
    const int64_t total = static_cast<int64_t>(U) * NP;
    const int64_t wstride = static_cast<int64_t>(gridDim.x) * (blockDim.x >> 5);
    for (int64_t c = blockIdx.x * static_cast<int64_t>(blockDim.x >> 5) + (threadIdx.x >> 5);
         c < total; c += wstride) {
        const int64_t u = c / NP;
        const int p = static_cast<int>(c - u * NP);
        float r = nan_f();
        if (p < N) {
            uint32_t v[D / 64];
            r = warp_rinv<D>(keys + (u * N + p) * D, v);
        }
        if ((threadIdx.x & 31) == 0) {
            colrinv[c] = r;
            colpos[c] = p < N ? p : -1;
        }
    }
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

// Mode 1, step 2: one warp per position p of unit u copies key p to its column of the
// retained-first layout and records 1/||k_p||; one warp per padding column writes NaN.
template <int D>
__global__ void gather_kernel(const uint16_t* __restrict__ keys, const uint8_t* __restrict__ mask,
                              const int* __restrict__ cnt, const int* __restrict__ kb, int U,
                              int N, int64_t NP, uint16_t* __restrict__ kp,
                              float* __restrict__ colrinv, int* __restrict__ colpos)
{
    const int64_t total = static_cast<int64_t>(U) * NP;   // N positions + NP-N padding per unit
    const int64_t wstride = static_cast<int64_t>(gridDim.x) * (blockDim.x >> 5);
    const int lane = threadIdx.x & 31;
    for (int64_t g = blockIdx.x * static_cast<int64_t>(blockDim.x >> 5) + (threadIdx.x >> 5);
         g < total; g += wstride) {
        const int64_t u = g / NP;
        const int p = static_cast<int>(g - u * NP);
        const int k = kb[u];
        const int kpad = ((k + kBN - 1) / kBN) * kBN;
        uint32_t* dst32;
        if (p < N) {
            const int before = cnt[u * N + p];
            const int col = mask[u * N + p] ? before : kpad + (p - before);
            uint32_t v[D / 64];
            const float r = warp_rinv<D>(keys + (u * N + p) * D, v);
            dst32 = reinterpret_cast<uint32_t*>(kp + (u * NP + col) * D);
#pragma unroll
            for (int t = 0; t < D / 64; ++t) dst32[t * 32 + lane] = v[t];
            if (lane == 0) {
                colrinv[u * NP + col] = r;
                colpos[u * NP + col] = p;
            }
        } else {
            // padding columns: [k, kpad) and [kpad + N - k, NP)
            const int r = p - N;
            const int col = r < kpad - k ? k + r : kpad + (N - k) + (r - (kpad - k));
            dst32 = reinterpret_cast<uint32_t*>(kp + (u * NP + col) * D);
#pragma unroll
            for (int t = 0; t < D / 64; ++t) dst32[t * 32 + lane] = 0u;
            if (lane == 0) {
                colrinv[u * NP + col] = nan_f();
                colpos[u * NP + col] = -1;
            }
        }
    }
}

int grid_for(int64_t warps, int per_block_warps)
{
    int64_t blocks = (warps + per_block_warps - 1) / per_block_warps;
    if (blocks > 65535LL * 16) blocks = 65535LL * 16;
    if (blocks < 1) blocks = 1;
    return static_cast<int>(blocks);
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
                                  float* colrinv, int* colpos, cudaStream_t st)
{
    const int grid = grid_for(static_cast<int64_t>(U) * NP, 8);
    if (d == 128)
        norms_identity_kernel<128><<<grid, 256, 0, st>>>(keys, U, N, NP, colrinv, colpos);
    else
        norms_identity_kernel<64><<<grid, 256, 0, st>>>(keys, U, N, NP, colrinv, colpos);
    return cudaGetLastError();
}

cudaError_t launch_scan(const uint8_t* mask, int U, int N, int* cnt, int* kb, cudaStream_t st)
{
    scan_kernel<<<U, 1024, 0, st>>>(mask, N, cnt, kb);
    return cudaGetLastError();
}

cudaError_t launch_gather(const uint16_t* keys, const uint8_t* mask, const int* cnt,
                          const int* kb, int U, int N, int d, int64_t NP, uint16_t* kp,
                          float* colrinv, int* colpos, cudaStream_t st)
{
    const int grid = grid_for(static_cast<int64_t>(U) * NP, 8);
    if (d == 128)
        gather_kernel<128><<<grid, 256, 0, st>>>(keys, mask, cnt, kb, U, N, NP, kp, colrinv,
                                                 colpos);
    else
        gather_kernel<64><<<grid, 256, 0, st>>>(keys, mask, cnt, kb, U, N, NP, kp, colrinv,
                                                colpos);
    return cudaGetLastError();
}

}  // namespace twk
