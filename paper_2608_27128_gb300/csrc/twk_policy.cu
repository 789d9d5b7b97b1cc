// twk_policy.cu -- selection of the standalone TwinKV policy (arXiv 2608.27128, Sec. 3.2,
// Eq. 3).
//
// The score of position i is s_i = -r_i / n (Eq. 3) with r_i the redundancy count of
// Eq. 2; the sink and recent regions get the maximum score; the budget's worth of
// highest scores is kept.  Ranking by s descending is ranking by r ascending, so each
// position gets the 32-bit key
//     key_i = 0 for a protected position, r_i + 1 otherwise,
// and the K smallest keys are kept, equal keys in position order (lower first).
//
// One 1024-thread block per unit:
//   1. a radix select over the key bytes from the top finds the cut: the key value c
//      and how many items equal to c are still to be kept (stopping early when every
//      item sharing the selected prefix is kept);
//   2. one ordered pass keeps every key below the cut and the first `need` keys equal
//      to it, in position order (warp ballots + a block scan), writing the mask.
// Counts are read from global memory (N int32 per pass); nothing else is stored.
#include "twk_internal.h"

namespace twk {
namespace {

constexpr int kPT = 1024;
constexpr int kPW = kPT / 32;

struct PolicyShared {
    int hist[256];
    int wsum[kPW];
    int sel_digit, sel_before, sel_count;
};

__device__ __forceinline__ uint32_t policy_key(const int* count, int i, int N, int n_sink,
                                               int n_recent)
{
    const bool prot = i < n_sink || i >= N - n_recent;
    return prot ? 0u : static_cast<uint32_t>(count[i]) + 1u;
}

// Exclusive block prefix of a 0/1 flag over the current chunk; returns the prefix and
// the chunk total.
__device__ __forceinline__ int block_scan(PolicyShared& s, int f, int& total)
{
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    const uint32_t bal = __ballot_sync(0xFFFFFFFFu, f);
    if (lane == 0) s.wsum[wid] = __popc(bal);
    __syncthreads();
    if (wid == 0) {
        int v = s.wsum[lane];   // kPW == 32
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xFFFFFFFFu, v, o);
            if (lane >= o) v += y;
        }
        s.wsum[lane] = v;       // inclusive
    }
    __syncthreads();
    const int pre = (wid ? s.wsum[wid - 1] : 0) + __popc(bal & ((1u << lane) - 1u));
    total = s.wsum[kPW - 1];
    __syncthreads();
    return pre;
}

__global__ void __launch_bounds__(kPT, 1)
    policy_select_kernel(const int* __restrict__ count_all, int N, const int* __restrict__ budget,
                         int n_sink, int n_recent, uint8_t* __restrict__ mask_all,
                         int* __restrict__ status)
{
    static_assert(kPW == 32, "one warp holds the per-warp totals");
    __shared__ PolicyShared s;
    const int u = blockIdx.x;
    const int* count = count_all + static_cast<int64_t>(u) * N;
    uint8_t* mask = mask_all + static_cast<int64_t>(u) * N;
    const int K = budget[u];
    const int lane = threadIdx.x & 31;

    if (K < 0 || K > N) {
        for (int i = threadIdx.x; i < N; i += kPT) mask[i] = 0;
        if (status && threadIdx.x == 0) status[u] = 1;   // TWINKV_ERR_INVALID_ARG
        return;
    }
    if (status && threadIdx.x == 0) status[u] = 0;
    if (K == 0 || K == N) {
        for (int i = threadIdx.x; i < N; i += kPT) mask[i] = K == N ? 1 : 0;
        return;
    }

    // 1. radix select of the cut, byte by byte from the top
    uint32_t prefix = 0, pmask = 0;
    int need = K;
    bool whole = false;
    for (int shift = 24; shift >= 0 && !whole; shift -= 8) {
        for (int d = threadIdx.x; d < 256; d += kPT) s.hist[d] = 0;
        __syncthreads();
        for (int c0 = 0; c0 < N; c0 += kPT) {
            const int i = c0 + threadIdx.x;
            int dg = 256;
            if (i < N) {
                const uint32_t key = policy_key(count, i, N, n_sink, n_recent);
                if ((key & pmask) == prefix) dg = static_cast<int>((key >> shift) & 255u);
            }
            const uint32_t peers = __match_any_sync(0xFFFFFFFFu, dg);
            if (dg < 256 && lane == __ffs(peers) - 1) atomicAdd(&s.hist[dg], __popc(peers));
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            int run = 0, d = 0;
            for (; d < 255 && run + s.hist[d] < need; ++d) run += s.hist[d];
            s.sel_digit = d;
            s.sel_before = run;
            s.sel_count = s.hist[d];
        }
        __syncthreads();
        need -= s.sel_before;
        prefix |= static_cast<uint32_t>(s.sel_digit) << shift;
        pmask |= 255u << shift;
        whole = s.sel_count == need;
        __syncthreads();
    }

    // 2. keep the keys below the cut and the first `need` equal to it
    int seen_eq = 0;
    for (int c0 = 0; c0 < N; c0 += kPT) {
        const int i = c0 + threadIdx.x;
        int lt = 0, eq = 0;
        if (i < N) {
            const uint32_t km = policy_key(count, i, N, n_sink, n_recent) & pmask;
            lt = km < prefix || (whole && km == prefix);
            eq = !whole && km == prefix;
        }
        int te = 0;
        const int pe = block_scan(s, eq, te);
        if (i < N) mask[i] = (lt || (eq && seen_eq + pe < need)) ? 1 : 0;
        seen_eq += te;
    }
}

}  // namespace

cudaError_t launch_policy_select(const int* count, int U, int N, const int* budget, int n_sink,
                                 int n_recent, uint8_t* out_mask, int* out_status,
                                 cudaStream_t st)
{
    policy_select_kernel<<<U, kPT, 0, st>>>(count, N, budget, n_sink, n_recent, out_mask,
                                            out_status);
    return cudaGetLastError();
}

}  // namespace twk
