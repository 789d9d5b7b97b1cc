// twk_repair.cu -- budget-exact repair swap of TwinKV (arXiv 2608.27128, Sec. 3.4).
//
// Per unit (layer, KV head):
//   classify  orphan = i not in S0 and b_i < tau,
//             donor  = j in S0, outside [0, n_sink) and [N - n_recent, N), b_j >= tau,
//   each entry a (severity key, position) pair: orphans keyed by b ascending, donors by
//   b descending, through an order-preserving fp64 -> u64 map (-0 folded into +0);
//   m = min(|O|, |D|); the m most severe orphans and donors, ordered by (key, position)
//   so that equal severities keep position order (lower position first);
//   S1 = S0 with the m donors cleared and the m orphans set; swaps[k] = (donor k,
//   orphan k); a unit whose mask has a byte > 1 or whose popcount differs from its
//   budget gets status, nswaps = -1 and S1 = S0.
//
// The literal rule (select_kernel<C>) runs each unit on a cluster of C CTAs (C = 1, 2,
// 4, 8 or 16, chosen so that every SM has work): see "cluster selection" below.  Its
// scratch is caller workspace ([U][N] keys and positions, twice) and 48 KB of dynamic
// shared memory per CTA.
//
// Dedup variant (dedup_kernel, given the twin of every position; one 512-thread block
// per unit): evicting a donor keeps its twin, so a twin pair never loses both members.
// All donors are sorted; each gets the donor rank of its twin (through a position ->
// rank table in the workspace); one thread then walks the ranks in severity order with
// two bits of state per rank in shared memory (evicted, pinned): a donor is skipped
// when it is pinned (the twin of an evicted donor) or its twin is evicted, and the
// walk stops after |O| evictions.  The ranks it needs are staged in shared memory
// chunk by chunk, so the walk itself touches shared memory only.  m = the evictions;
// the m most severe orphans are then selected with a radix select (byte histograms
// from the top) and sorted: up to 4096 items by a bitonic network in shared memory,
// more by a stable LSD radix sort (8-bit digits, warp match + per-warp digit counts; a
// digit position shared by every key is skipped).
#include <cooperative_groups.h>

#include "twk_internal.h"

namespace twk {
namespace {

constexpr int kT = 512;   // two blocks per SM: every unit of a prefill in one wave
constexpr int kW = kT / 32;

// Order-preserving map of an fp64 value to a u64 key (-0 folded into +0), in integer
// operations only: fp64 comparisons run on this GPU's narrow FP64 pipe.
__device__ __forceinline__ uint64_t ordered(double b)
{
    uint64_t u = static_cast<uint64_t>(__double_as_longlong(b));
    if (u == 0x8000000000000000ull) u = 0ull;
    return (u >> 63) ? ~u : (u | 0x8000000000000000ull);
}

__device__ __forceinline__ bool is_nan_bits(double b)
{
    return (static_cast<uint64_t>(__double_as_longlong(b)) & 0x7FFFFFFFFFFFFFFFull) >
           0x7FF0000000000000ull;
}

struct Shared {
    int warp_cnt[kW][256];   // per-warp digit counts, then their prefix over warps
    int base[256];           // running output offset of each digit
    int chunk_tot[256];
    int wsum[2][kW];         // block-scan scratch for the two lists
    int red[4];
    int flag;
    int sel_digit, sel_before, sel_count;
};

// Block-wide exclusive scan of two 0/1 flags; returns the prefixes and the chunk totals.
__device__ __forceinline__ void scan2(Shared& s, int fo, int fd, int& po, int& pd, int& to,
                                      int& td)
{
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    const uint32_t bo = __ballot_sync(0xFFFFFFFFu, fo);
    const uint32_t bd = __ballot_sync(0xFFFFFFFFu, fd);
    const uint32_t lt = (1u << lane) - 1u;
    if (lane == 0) {
        s.wsum[0][wid] = __popc(bo);
        s.wsum[1][wid] = __popc(bd);
    }
    __syncthreads();
    if (wid == 0) {
        int a = lane < kW ? s.wsum[0][lane] : 0, b = lane < kW ? s.wsum[1][lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int ya = __shfl_up_sync(0xFFFFFFFFu, a, o);
            const int yb = __shfl_up_sync(0xFFFFFFFFu, b, o);
            if (lane >= o) {
                a += ya;
                b += yb;
            }
        }
        if (lane < kW) {
            s.wsum[0][lane] = a;   // inclusive
            s.wsum[1][lane] = b;
        }
    }
    __syncthreads();
    po = (wid ? s.wsum[0][wid - 1] : 0) + __popc(bo & lt);
    pd = (wid ? s.wsum[1][wid - 1] : 0) + __popc(bd & lt);
    to = s.wsum[0][kW - 1];
    td = s.wsum[1][kW - 1];
    __syncthreads();
}

// Called by warp 0 only: the 256 digit counts in cnt become their exclusive prefix
// (eight digits per lane and a shuffle scan); returns whether one digit holds all n.
__device__ __forceinline__ bool digit_prefix(int* cnt, int n)
{
    const int lane = threadIdx.x & 31;
    int c[8], t = 0;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        c[j] = cnt[lane * 8 + j];
        t += c[j];
    }
    int incl = t;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
        if (lane >= o) incl += y;
    }
    int run = incl - t;
    bool one = false;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        one |= c[j] == n;
        cnt[lane * 8 + j] = run;
        run += c[j];
    }
    return __any_sync(0xFFFFFFFFu, one);
}

// Called by warp 0 only: the smallest digit d whose counts up to and including d reach
// `need` (255 at most), the count before it and its own count, into s.
__device__ __forceinline__ void digit_cut(const int* cnt, int need, int& sel_digit,
                                          int& sel_before, int& sel_count)
{
    const int lane = threadIdx.x & 31;
    int c[8], t = 0;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        c[j] = cnt[lane * 8 + j];
        t += c[j];
    }
    int incl = t;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
        if (lane >= o) incl += y;
    }
    const uint32_t reach = __ballot_sync(0xFFFFFFFFu, incl >= need);
    const int L = reach ? __ffs(reach) - 1 : 31;
    if (lane == L) {
        // the first of the lane's digits whose running count reaches need (its last
        // digit otherwise: digit 255 for lane 31); constant indices keep c in registers
        int run = incl - t, sel = 7, before = 0, count = c[7];
        bool found = false;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            if (!found && (j == 7 || run + c[j] >= need)) {
                sel = j;
                before = run;
                count = c[j];
                found = true;
            }
            if (!found) run += c[j];
        }
        sel_digit = L * 8 + sel;
        sel_before = before;
        sel_count = count;
    }
}

// Block-wide exclusive scan of two per-thread counts; returns each thread's prefixes
// and the totals.
__device__ __forceinline__ void scan2n(Shared& s, int co, int cd, int& po, int& pd, int& to,
                                       int& td)
{
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    int io = co, id = cd;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int yo = __shfl_up_sync(0xFFFFFFFFu, io, o);
        const int yd = __shfl_up_sync(0xFFFFFFFFu, id, o);
        if (lane >= o) {
            io += yo;
            id += yd;
        }
    }
    if (lane == 31) {
        s.wsum[0][wid] = io;
        s.wsum[1][wid] = id;
    }
    __syncthreads();
    if (wid == 0) {
        int x = lane < kW ? s.wsum[0][lane] : 0, y = lane < kW ? s.wsum[1][lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int xo = __shfl_up_sync(0xFFFFFFFFu, x, o);
            const int yo = __shfl_up_sync(0xFFFFFFFFu, y, o);
            if (lane >= o) {
                x += xo;
                y += yo;
            }
        }
        if (lane < kW) {
            s.wsum[0][lane] = x;   // inclusive
            s.wsum[1][lane] = y;
        }
    }
    __syncthreads();
    po = (wid ? s.wsum[0][wid - 1] : 0) + io - co;
    pd = (wid ? s.wsum[1][wid - 1] : 0) + id - cd;
    to = s.wsum[0][kW - 1];
    td = s.wsum[1][kW - 1];
    __syncthreads();
}

constexpr int kE = 4;   // consecutive positions per thread in the streaming passes
constexpr int kH = 4;   // items per thread per round of a digit histogram

// One stable counting pass on digit (key >> shift) & 255 of n items; returns false
// (and moves nothing) when every item has the same digit.
__device__ bool radix_pass(Shared& s, const uint64_t* kin, const int* iin, uint64_t* kout,
                           int* iout, int n, int shift)
{
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    for (int i = threadIdx.x; i < kW * 256; i += kT) (&s.warp_cnt[0][0])[i] = 0;
    if (threadIdx.x < 256) s.base[threadIdx.x] = 0;
    __syncthreads();
    for (int c0 = 0; c0 < n; c0 += kT * kH) {
        int dg[kH];
#pragma unroll
        for (int e = 0; e < kH; ++e) {   // the loads first: kH in flight per thread
            const int i = c0 + e * kT + threadIdx.x;
            dg[e] = i < n ? static_cast<int>((kin[i] >> shift) & 255) : 256;
        }
#pragma unroll
        for (int e = 0; e < kH; ++e) {
            const uint32_t peers = __match_any_sync(0xFFFFFFFFu, dg[e]);
            if (dg[e] < 256 && lane == __ffs(peers) - 1) atomicAdd(&s.base[dg[e]], __popc(peers));
        }
    }
    __syncthreads();
    if (threadIdx.x < 32) {
        const bool single = digit_prefix(s.base, n);
        if (threadIdx.x == 0) s.flag = single;
    }
    __syncthreads();
    if (s.flag) return false;
    for (int c0 = 0; c0 < n; c0 += kT) {
        const int i = c0 + threadIdx.x;
        const bool valid = i < n;
        const uint64_t key = valid ? kin[i] : 0ull;
        const int dg = valid ? static_cast<int>((key >> shift) & 255) : 256;
        const uint32_t peers = __match_any_sync(0xFFFFFFFFu, dg);
        const int rank = __popc(peers & ((1u << lane) - 1u));
        if (valid && rank == 0) s.warp_cnt[wid][dg] = __popc(peers);
        __syncthreads();
        if (threadIdx.x < 256) {
            int run = 0;
            for (int w = 0; w < kW; ++w) {
                const int t = s.warp_cnt[w][threadIdx.x];
                s.warp_cnt[w][threadIdx.x] = run;
                run += t;
            }
            s.chunk_tot[threadIdx.x] = run;
        }
        __syncthreads();
        if (valid) {
            const int dst = s.base[dg] + s.warp_cnt[wid][dg] + rank;
            kout[dst] = key;
            iout[dst] = iin[i];
        }
        __syncthreads();
        if (threadIdx.x < 256) {
            s.base[threadIdx.x] += s.chunk_tot[threadIdx.x];
            for (int w = 0; w < kW; ++w) s.warp_cnt[w][threadIdx.x] = 0;
        }
        __syncthreads();
    }
    return true;
}

// Sorts n (key, position) items held at offset `off` of buffer 0; returns the buffer
// (0 or 1) that holds the sorted result.
__device__ int radix_sort(Shared& s, uint64_t* k0, int* i0, uint64_t* k1, int* i1, int n)
{
    int cur = 0;
    for (int shift = 0; shift < 64; shift += 8) {
        const bool moved = cur == 0 ? radix_pass(s, k0, i0, k1, i1, n, shift)
                                    : radix_pass(s, k1, i1, k0, i0, n, shift);
        if (moved) cur ^= 1;
        __syncthreads();
    }
    return cur;
}

// Moves the m smallest of the n (key, position) items in (kin, iin) to (kout, iout),
// keeping their order (position order), so that ties at the cut go to the lower
// positions.  The cut is found byte by byte from the top (a radix select: one
// histogram per byte over the items that still share the selected prefix), stopping
// early once the whole boundary bucket is selected.  Requires 0 < m <= n.
__device__ void select_smallest(Shared& s, const uint64_t* kin, const int* iin, uint64_t* kout,
                                int* iout, int n, int m)
{
    const int lane = threadIdx.x & 31;
    uint64_t prefix = 0, pmask = 0;
    int need = m;                 // items still to take among those matching the prefix
    bool whole = false;           // every item matching the prefix is taken
    for (int shift = 56; shift >= 0 && !whole; shift -= 8) {
        if (threadIdx.x < 256) s.base[threadIdx.x] = 0;
        __syncthreads();
        for (int c0 = 0; c0 < n; c0 += kT * kH) {
            int dg[kH];
#pragma unroll
            for (int e = 0; e < kH; ++e) {   // the loads first: kH in flight per thread
                const int i = c0 + e * kT + threadIdx.x;
                dg[e] = 256;
                if (i < n) {
                    const uint64_t key = kin[i];
                    if ((key & pmask) == prefix) dg[e] = static_cast<int>((key >> shift) & 255);
                }
            }
#pragma unroll
            for (int e = 0; e < kH; ++e) {
                const uint32_t peers = __match_any_sync(0xFFFFFFFFu, dg[e]);
                if (dg[e] < 256 && lane == __ffs(peers) - 1)
                    atomicAdd(&s.base[dg[e]], __popc(peers));
            }
        }
        __syncthreads();
        if (threadIdx.x < 32) digit_cut(s.base, need, s.sel_digit, s.sel_before, s.sel_count);
        __syncthreads();
        need -= s.sel_before;
        prefix |= static_cast<uint64_t>(s.sel_digit) << shift;
        pmask |= 255ull << shift;
        whole = s.sel_count == need;
        __syncthreads();
    }
    // Ordered compaction: items below the prefix, then those equal to it (all of them
    // when `whole`, else the first `need` in position order).
    int base = 0, seen_eq = 0;
    for (int c0 = 0; c0 < n; c0 += kT) {
        const int i = c0 + threadIdx.x;
        int fl = 0, fe = 0;
        uint64_t key = 0;
        if (i < n) {
            key = kin[i];
            const uint64_t km = key & pmask;
            fl = km < prefix || (whole && km == prefix);
            fe = !whole && km == prefix;
        }
        int pl, pe, tl, te;
        scan2(s, fl, fe, pl, pe, tl, te);
        const int k_eq = max(0, min(te, need - seen_eq));   // eq items taken in this chunk
        if (fl || (fe && pe < k_eq)) {
            const int dst = base + pl + min(pe, k_eq);
            kout[dst] = key;
            iout[dst] = iin[i];
        }
        base += tl + k_eq;
        seen_eq += te;
    }
    __syncthreads();
}

// Lists of at most kSortMax items are sorted in shared memory (kSortMax * 12 bytes of
// dynamic shared memory), longer ones by the radix passes over the workspace.
constexpr int kSortMax = 4096;

// Sorts the n <= kSortMax items (kin, iin) ascending by (key, position) into (kout,
// iout), with a bitonic network in shared memory (sk, si) padded to a power of two by
// items that sort last.  Positions are distinct, so the order equals that of a stable
// sort by key of a list in position order.
__device__ void smem_sort(uint64_t* sk, int* si, const uint64_t* kin, const int* iin, int n,
                          uint64_t* kout, int* iout)
{
    int P = 1;
    while (P < n) P <<= 1;
    for (int t = threadIdx.x; t < P; t += kT) {
        sk[t] = t < n ? kin[t] : ~0ull;
        si[t] = t < n ? iin[t] : 0x7FFFFFFF;
    }
    __syncthreads();
    for (int size = 2; size <= P; size <<= 1) {
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            for (int t = threadIdx.x; t < P / 2; t += kT) {
                const int lo = 2 * t - (t & (stride - 1));
                const int hi = lo + stride;
                const uint64_t ka = sk[lo], kb = sk[hi];
                const int pa = si[lo], pb = si[hi];
                const bool gt = ka > kb || (ka == kb && pa > pb);
                if (gt == ((lo & size) == 0)) {   // ascending blocks swap a greater first
                    sk[lo] = kb;
                    sk[hi] = ka;
                    si[lo] = pb;
                    si[hi] = pa;
                }
            }
            __syncthreads();
        }
    }
    for (int t = threadIdx.x; t < n; t += kT) {
        kout[t] = sk[t];
        iout[t] = si[t];
    }
    __syncthreads();
}

// The m most severe items of one list, in severity order: (key, position) pairs at
// (k, i) with scratch (kx, ix) of the same extent; returns the position array holding
// them.  (sk, si): kSortMax items of shared memory.
__device__ const int* most_severe(Shared& s, uint64_t* k, int* i, uint64_t* kx, int* ix, int n,
                                  int m, uint64_t* sk, int* si)
{
    if (n > m) {
        select_smallest(s, k, i, kx, ix, n, m);
        if (m <= kSortMax) {
            smem_sort(sk, si, kx, ix, m, k, i);
            return i;
        }
        return radix_sort(s, kx, ix, k, i, m) ? i : ix;
    }
    if (n <= kSortMax) {
        smem_sort(sk, si, k, i, n, kx, ix);
        return ix;
    }
    return radix_sort(s, k, i, kx, ix, n) ? ix : i;
}

constexpr int kWalkChunk = 4096;   // twin ranks staged per step of the dedup walk

// Dynamic shared memory of the dedup variant: 2 state bits per donor rank (n_d <= N),
// then one chunk of staged twin ranks (the sort buffers follow, 16-byte aligned).
__host__ __device__ inline size_t dedup_smem_bytes(int N)
{
    return static_cast<size_t>((N + 15) / 16) * 4 + kWalkChunk * 4;
}

// Offset of the shared-memory sort buffers (kSortMax keys, then kSortMax positions) in
// the dynamic shared memory, and the total dynamic bytes.
__host__ __device__ inline size_t sort_smem_offset(int N)
{
    return (dedup_smem_bytes(N) + 15) / 16 * 16;
}

__host__ __device__ inline size_t dedup_kernel_smem_bytes(int N)
{
    return sort_smem_offset(N) + static_cast<size_t>(kSortMax) * 12;
}

// ---------------------------------------------------------------- cluster selection
//
// The literal repair (Sec. 3.4) of one unit on a cluster of C CTAs (C = 1: one CTA).
// CTA r of the cluster owns the slice [r S, (r + 1) S) of the unit's positions.
//   A. One pass over the slice: S1 = S0, validation counts, and the slice's orphans
//      (forward from the slice start) and donors (backward from the slice end) as
//      (severity key, position) pairs in keys0/idx0.  n_o + n_d never exceeds the
//      slice length, so the two lists never meet.
//   B. Counts through distributed shared memory: totals, this CTA's offsets, status,
//      m = min(|O|, |D|).  The side with more than m items is cut by a radix select
//      whose digit histograms are summed over the cluster (each CTA histograms its own
//      items; the sums, and so every decision, are identical in every CTA); the other
//      side is taken whole; each CTA's own counts below and at the cut come from its
//      own histograms.  An ordered compaction writes the m items of each side, in
//      position order, to keys1/idx1 (orphans at [0, m), donors at [N/2, N/2 + m)).
//   C. Each CTA sorts its share of both lists by (key, position) with a bitonic
//      network held in registers (eight slots per thread; warp shuffles for strides up
//      to 128, shared memory beyond): both sides at once for shares of up to kChunk
//      items, one side after the other for shares of up to 2 kChunk.  An item's place
//      in the swap list is its rank in its own share plus, for every other share, the
//      number of that share's items ordered before it (binary search in the other
//      CTA's shared memory).  Larger shares are sorted by one CTA per side with the
//      stable radix passes over the workspace.
// Every CTA of a cluster runs the same sequence of cluster barriers: each branch and
// loop bound that leads to one depends only on values that are identical in every CTA.
namespace cg = cooperative_groups;

constexpr int kChunk = 2048;   // items per side a CTA sorts at once (both sides)

template <int C>
__device__ __forceinline__ void cluster_sync()
{
    if constexpr (C == 1) __syncthreads();
    else cg::this_cluster().sync();
}

// The same shared-memory object in CTA `rank` of the cluster.
template <int C, typename T>
__device__ __forceinline__ T* peer(T* p, int rank)
{
    if constexpr (C == 1) return p;
    else return cg::this_cluster().map_shared_rank(p, rank);
}

struct ClusterShared {
    int cnt[4];          // this CTA's orphans, donors, retained count, invalid-byte flag
    int lcnt[2];         // compaction: this CTA's items below the cut and at it
    int hist[2][256];    // this CTA's digit histogram, alternating between passes
    int tot[8];          // cluster-wide values derived by thread 0
};

__device__ __forceinline__ bool before(uint64_t ka, int pa, uint64_t kb, int pb)
{
    return ka < kb || (ka == kb && pa < pb);
}

// Number of entries of the sorted (key, position) array of P = 2^k entries that order
// before (k, p).
__device__ __forceinline__ int count_before(const uint64_t* sk, const int* si, int P, uint64_t k,
                                            int p)
{
    int pos = 0;
    for (int half = P >> 1; half > 0; half >>= 1)
        if (before(sk[pos + half - 1], si[pos + half - 1], k, p)) pos += half;
    if (before(sk[pos], si[pos], k, p)) ++pos;
    return pos;
}

constexpr int kR = 8;   // items per thread in the share sort's registers

// Compare-exchange of two items: afterwards a orders before b when `up`, after it
// otherwise.
__device__ __forceinline__ void cx(uint64_t& ka, int& pa, uint64_t& kb, int& pb, bool up)
{
    const bool sw = before(kb, pb, ka, pa) == up;
    const uint64_t k0 = sw ? kb : ka, k1 = sw ? ka : kb;
    const int p0 = sw ? pb : pa, p1 = sw ? pa : pb;
    ka = k0;
    kb = k1;
    pa = p0;
    pb = p1;
}

// kR items between registers and the shared-memory slots [at, at + kR) (16-byte
// aligned: at is a multiple of kR).
__device__ __forceinline__ void store_run(uint64_t* sk, int* si, int at, const uint64_t* kx,
                                          const int* px)
{
#pragma unroll
    for (int e = 0; e < kR; e += 2)
        *reinterpret_cast<ulonglong2*>(sk + at + e) = make_ulonglong2(kx[e], kx[e + 1]);
#pragma unroll
    for (int e = 0; e < kR; e += 4)
        *reinterpret_cast<int4*>(si + at + e) = make_int4(px[e], px[e + 1], px[e + 2], px[e + 3]);
}

__device__ __forceinline__ void load_run(const uint64_t* sk, const int* si, int at, uint64_t* kx,
                                         int* px)
{
#pragma unroll
    for (int e = 0; e < kR; e += 2) {
        const ulonglong2 v = *reinterpret_cast<const ulonglong2*>(sk + at + e);
        kx[e] = v.x;
        kx[e + 1] = v.y;
    }
#pragma unroll
    for (int e = 0; e < kR; e += 4) {
        const int4 v = *reinterpret_cast<const int4*>(si + at + e);
        px[e] = v.x;
        px[e + 1] = v.y;
        px[e + 2] = v.z;
        px[e + 3] = v.w;
    }
}

constexpr int kEA = 8;   // consecutive positions per thread in the classification pass

// Slice length: ceil(N / C) rounded up to a multiple of kEA.
__host__ __device__ inline int slice_len(int N, int C)
{
    const int q = (N + C - 1) / C;
    return (q + kEA - 1) / kEA * kEA;
}

template <int C>
__global__ void __launch_bounds__(kT, 2) select_kernel(const RepairArgs a)
{
    __shared__ Shared s;
    __shared__ ClusterShared cs;
    extern __shared__ __align__(16) uint32_t dyn[];
    uint64_t* sk_o = reinterpret_cast<uint64_t*>(dyn);   // [kChunk] orphans' keys
    uint64_t* sk_d = sk_o + kChunk;                      // [kChunk] donors' keys
    int* si_o = reinterpret_cast<int*>(sk_d + kChunk);   // [kChunk] positions
    int* si_d = si_o + kChunk;

    const int tid = threadIdx.x, lane = tid & 31;
    int r = 0;
    if constexpr (C > 1) r = static_cast<int>(cg::this_cluster().block_rank());
    const int u = static_cast<int>(blockIdx.x / C);
    const int N = a.N;
    const int64_t off = static_cast<int64_t>(u) * N;
    const uint8_t* S0 = a.mask + off;
    const double* b = a.b + off;
    uint8_t* S1 = a.out_mask + off;
    int* swaps = a.out_swaps + static_cast<int64_t>(u) * 2 * (N / 2);
    uint64_t* K0 = a.keys0 + off;
    int* I0 = a.idx0 + off;
    uint64_t* K1 = a.keys1 + off;
    int* I1 = a.idx1 + off;
    const int S = slice_len(N, C);
    const int lo = min(N, r * S), hi = min(N, lo + S);
    const uint64_t ktau = ordered(a.tau);

    // A. S1 = S0, counts, and the slice's lists (orphans forward from lo, donors
    // backward from hi: donor k in position order sits at hi - 1 - k).  A thread takes
    // kEA consecutive positions: one 8-byte mask load and four 16-byte b loads when
    // every unit's rows are aligned for them (N a multiple of 8, aligned base
    // pointers), else one at a time.
    int bad = 0, cnt = 0, my_o = 0, my_d = 0;
    const bool vec = (N % kEA) == 0 && (reinterpret_cast<uintptr_t>(a.mask) & 7) == 0 &&
                     (reinterpret_cast<uintptr_t>(a.out_mask) & 7) == 0 &&
                     (reinterpret_cast<uintptr_t>(a.b) & 15) == 0;
    for (int c0 = lo; c0 < hi; c0 += kT * kEA) {
        const int i0 = c0 + tid * kEA;
        uint32_t mv[kEA];
        double bv[kEA];
        if (vec && i0 + kEA <= hi) {
            const uint2 m8 = *reinterpret_cast<const uint2*>(S0 + i0);
            *reinterpret_cast<uint2*>(S1 + i0) = m8;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                mv[j] = (m8.x >> (8 * j)) & 255u;
                mv[4 + j] = (m8.y >> (8 * j)) & 255u;
            }
            const double2* b2 = reinterpret_cast<const double2*>(b + i0);
#pragma unroll
            for (int j = 0; j < kEA / 2; ++j) {
                const double2 t = b2[j];
                bv[2 * j] = t.x;
                bv[2 * j + 1] = t.y;
            }
        } else {
#pragma unroll
            for (int j = 0; j < kEA; ++j) {
                const int i = i0 + j;
                mv[j] = 0u;
                bv[j] = 0.0;
                if (i < hi) {
                    mv[j] = S0[i];
                    bv[j] = b[i];
                    S1[i] = static_cast<uint8_t>(mv[j]);
                }
            }
        }
        // b < tau and b >= tau decided on the order-preserving keys (a NaN b is
        // neither an orphan nor a donor, as in fp64 comparisons)
        int fo[kEA], fd[kEA], co = 0, cd = 0;
        uint64_t kv[kEA];
#pragma unroll
        for (int j = 0; j < kEA; ++j) {
            const int i = i0 + j;
            const bool in = i < hi && !is_nan_bits(bv[j]);
            kv[j] = ordered(bv[j]);
            bad |= mv[j] > 1u;
            cnt += mv[j] != 0u;
            const bool prot = i < a.n_sink || i >= N - a.n_recent;
            fo[j] = in && mv[j] == 0u && kv[j] < ktau;
            fd[j] = in && mv[j] != 0u && !prot && kv[j] >= ktau;
            co += fo[j];
            cd += fd[j];
        }
        int po, pd, to, td;
        scan2n(s, co, cd, po, pd, to, td);
#pragma unroll
        for (int j = 0; j < kEA; ++j) {
            const int i = i0 + j;
            if (fo[j]) {
                K0[lo + my_o + po] = kv[j];
                I0[lo + my_o + po] = i;
                ++po;
            }
            if (fd[j]) {
                K0[hi - 1 - (my_d + pd)] = ~kv[j];
                I0[hi - 1 - (my_d + pd)] = i;
                ++pd;
            }
        }
        my_o += to;
        my_d += td;
    }
    if (tid < 4) s.red[tid] = 0;
    __syncthreads();
    bad = __reduce_or_sync(0xFFFFFFFFu, bad);
    cnt = __reduce_add_sync(0xFFFFFFFFu, cnt);
    if (lane == 0) {
        atomicOr(&s.red[0], bad);
        atomicAdd(&s.red[1], cnt);
    }
    __syncthreads();
    if (tid == 0) {
        cs.cnt[0] = my_o;
        cs.cnt[1] = my_d;
        cs.cnt[2] = s.red[1];
        cs.cnt[3] = s.red[0];
    }
    cluster_sync<C>();

    // B. totals, offsets, status and m (identical in every CTA of the cluster)
    if (tid == 0) {
        int n_o = 0, n_d = 0, tc = 0, tb = 0, bo = 0, bd = 0;
        for (int q = 0; q < C; ++q) {
            const int* rc = peer<C>(cs.cnt, q);
            if (q == r) {
                bo = n_o;
                bd = n_d;
            }
            n_o += rc[0];
            n_d += rc[1];
            tc += rc[2];
            tb |= rc[3];
        }
        int status = 0;
        if (tb) status = 1;                                  // TWINKV_ERR_INVALID_ARG
        else if (a.budget && a.budget[u] != tc) status = 3;  // TWINKV_ERR_BUDGET
        cs.tot[0] = n_o;
        cs.tot[1] = n_d;
        cs.tot[2] = bo;
        cs.tot[3] = bd;
        cs.tot[4] = status;
        cs.tot[5] = status ? 0 : min(n_o, n_d);
    }
    __syncthreads();
    const int n_o = cs.tot[0], n_d = cs.tot[1], bo = cs.tot[2], bd = cs.tot[3];
    const int status = cs.tot[4], m = cs.tot[5];
    if (status != 0 || m == 0) {
        cluster_sync<C>();   // every CTA has read the counts before any CTA exits
        if (r == 0 && tid == 0) {
            a.out_nswaps[u] = status ? -1 : 0;
            if (a.out_status) a.out_status[u] = status;
        }
        return;
    }

    // The side with more than m items is cut (at most one: m = min(n_o, n_d)); the
    // other is taken whole.  Item k (position order) of this CTA's list on side x:
    auto item_key = [&](int x, int k) { return x == 0 ? K0[lo + k] : K0[hi - 1 - k]; };
    auto item_pos = [&](int x, int k) { return x == 0 ? I0[lo + k] : I0[hi - 1 - k]; };
    const int half = N / 2;
    for (int x = 0; x < 2; ++x) {
        const int mine = x == 0 ? my_o : my_d;
        const int my_before = x == 0 ? bo : bd;
        const int dst0 = x == 0 ? 0 : half;
        if ((x == 0 ? n_o : n_d) == m) {
            for (int k = tid; k < mine; k += kT) {
                K1[dst0 + my_before + k] = item_key(x, k);
                I1[dst0 + my_before + k] = item_pos(x, k);
            }
            continue;
        }
        // radix select of the m smallest keys over the cluster, a byte at a time from
        // the top, stopping once the boundary bucket is taken whole
        uint64_t prefix = 0, pmask = 0;
        int need = m;
        bool whole = false;
        int pass = 0;
        int below = 0, at_cut = 0;   // this CTA's items below the cut and at it, per digit
        for (int shift = 56; shift >= 0 && !whole; shift -= 8, ++pass) {
            int* h = cs.hist[pass & 1];
            if (tid < 256) h[tid] = 0;
            __syncthreads();
            for (int c0 = 0; c0 < mine; c0 += kT * kH) {
                int dg[kH];
#pragma unroll
                for (int e = 0; e < kH; ++e) {
                    const int k = c0 + e * kT + tid;
                    dg[e] = 256;
                    if (k < mine) {
                        const uint64_t key = item_key(x, k);
                        if ((key & pmask) == prefix) dg[e] = static_cast<int>((key >> shift) & 255);
                    }
                }
#pragma unroll
                for (int e = 0; e < kH; ++e) {
                    const uint32_t peers = __match_any_sync(0xFFFFFFFFu, dg[e]);
                    if (dg[e] < 256 && lane == __ffs(peers) - 1) atomicAdd(&h[dg[e]], __popc(peers));
                }
            }
            cluster_sync<C>();   // every CTA's histogram of this pass is complete
            int own = 0;
            if (tid < 256) {
                int t = 0;
                for (int q = 0; q < C; ++q) t += peer<C>(h, q)[tid];
                s.base[tid] = t;
                own = h[tid];
            }
            __syncthreads();
            if (tid < 32) digit_cut(s.base, need, s.sel_digit, s.sel_before, s.sel_count);
            __syncthreads();
            need -= s.sel_before;
            prefix |= static_cast<uint64_t>(s.sel_digit) << shift;
            pmask |= 255ull << shift;
            whole = s.sel_count == need;
            // digit tid of this CTA's own histogram: below the selected digit, or at it
            below += tid < s.sel_digit ? own : 0;
            at_cut = tid == s.sel_digit ? own : 0;
            __syncthreads();
        }
        // ordered compaction: every item below the cut (and at it when `whole`), then
        // the first `need` items at the cut in position order over the cluster
        int nl = below + (whole ? at_cut : 0), ne = whole ? 0 : at_cut;
        if (tid < 2) s.red[tid] = 0;
        __syncthreads();
        nl = __reduce_add_sync(0xFFFFFFFFu, nl);
        ne = __reduce_add_sync(0xFFFFFFFFu, ne);
        if (lane == 0) {
            atomicAdd(&s.red[0], nl);
            atomicAdd(&s.red[1], ne);
        }
        __syncthreads();
        if (tid == 0) {
            cs.lcnt[0] = s.red[0];
            cs.lcnt[1] = s.red[1];
        }
        cluster_sync<C>();
        if (tid == 0) {
            int sel_before = 0, eq_before = 0;
            for (int q = 0; q < r; ++q) {
                const int* lc = peer<C>(cs.lcnt, q);
                sel_before += lc[0] + max(0, min(lc[1], need - eq_before));
                eq_before += lc[1];
            }
            cs.tot[6] = sel_before;
            cs.tot[7] = eq_before;
        }
        __syncthreads();
        int base = cs.tot[6], seen_eq = cs.tot[7];
        for (int c0 = 0; c0 < mine; c0 += kT * kEA) {
            // a thread takes kEA consecutive items; fl: below the cut (or at it when
            // `whole`), fe: at the cut
            const int k0 = c0 + tid * kEA;
            uint64_t kk[kEA];
            int pp[kEA];
            uint32_t fl = 0, fe = 0;
#pragma unroll
            for (int j = 0; j < kEA; ++j) {
                kk[j] = 0;
                pp[j] = 0;
                if (k0 + j < mine) {
                    kk[j] = item_key(x, k0 + j);
                    pp[j] = item_pos(x, k0 + j);
                    const uint64_t km = kk[j] & pmask;
                    fl |= static_cast<uint32_t>(km < prefix || (whole && km == prefix)) << j;
                    fe |= static_cast<uint32_t>(!whole && km == prefix) << j;
                }
            }
            int pl, pe, tl, te;
            scan2n(s, __popc(fl), __popc(fe), pl, pe, tl, te);
            const int k_eq = max(0, min(te, need - seen_eq));   // taken at the cut here
#pragma unroll
            for (int j = 0; j < kEA; ++j) {
                const int l = (fl >> j) & 1, e = (fe >> j) & 1;
                if (l || (e && pe < k_eq)) {
                    const int dst = base + pl + min(pe, k_eq);
                    K1[dst0 + dst] = kk[j];
                    I1[dst0 + dst] = pp[j];
                }
                pl += l;
                pe += e;
            }
            base += tl + k_eq;
            seen_eq += te;
        }
    }
    cluster_sync<C>();   // both lists of m items are in keys1/idx1, in position order

    // C. the swap list: m items per side in severity order
    const int q = (m + C - 1) / C;
    if (q <= 2 * kChunk) {
        // Each CTA sorts its share of both lists by (key, position) with a bitonic
        // network over P = 2^k >= max(q, kR) slots per side; padding sorts last.  Thread
        // tt of a side holds the slots [kR*tt, kR*tt + kR) in registers: strides below
        // kR are exchanged inside the thread, strides up to 16*kR between the lanes of
        // a warp by shuffles, and longer ones through shared memory.  Shares of up to
        // kChunk items sort both sides at once (half of the threads and of the buffer
        // each); longer ones (up to 2*kChunk) sort one side after the other, each over
        // all threads and the whole buffer (sk_o..sk_d and si_o..si_d are contiguous).
        const bool both = q <= kChunk;
        const int nside = both ? 2 : 1;
        int P = kR;
        while (P < q) P <<= 1;
        const int TP = P / kR;   // threads per side; threads from nside*TP on hold padding
        const int c_lo = min(m, r * q), c_n = min(m, c_lo + q) - c_lo;
        for (int pass = 0; pass < 3 - nside; ++pass) {
            const int sd = both && tid >= TP;     // the thread's side among those sorted
            const int side = both ? sd : pass;    // 0: orphans, 1: donors
            const int tt = tid - sd * TP;
            const bool live = tid < nside * TP;
            uint64_t* sk = sd ? sk_d : sk_o;
            int* si = sd ? si_d : si_o;
            uint64_t kx[kR];
            int px[kR];
#pragma unroll
            for (int e = 0; e < kR; ++e) {
                const int t = tt * kR + e;
                const bool in = live && t < c_n;
                kx[e] = in ? K1[side * half + c_lo + t] : ~0ull;
                px[e] = in ? I1[side * half + c_lo + t] : 0x7FFFFFFF;
            }
            for (int size = 2; size <= P; size <<= 1) {
                const bool up_t = ((tt * kR) & size) == 0;   // the direction once size >= kR
                if (size >= 64 * kR) {
                    if (live) store_run(sk, si, tt * kR, kx, px);
                    __syncthreads();
                    for (int stride = size >> 1; stride >= 32 * kR; stride >>= 1) {
                        for (int t = tid; t < nside * (P / 2); t += kT) {
                            const int s2 = t >= P / 2;   // pairs of the second side (both)
                            const int ts = s2 ? t - P / 2 : t;
                            uint64_t* k2 = s2 ? sk_d : sk_o;
                            int* i2 = s2 ? si_d : si_o;
                            const int lo2 = 2 * ts - (ts & (stride - 1));
                            const int hi2 = lo2 + stride;
                            uint64_t ka = k2[lo2], kb = k2[hi2];
                            int pa = i2[lo2], pb = i2[hi2];
                            cx(ka, pa, kb, pb, (lo2 & size) == 0);
                            k2[lo2] = ka;
                            k2[hi2] = kb;
                            i2[lo2] = pa;
                            i2[hi2] = pb;
                        }
                        __syncthreads();
                    }
                    if (live) load_run(sk, si, tt * kR, kx, px);
                }
                for (int stride = min(size >> 1, 16 * kR); stride >= kR; stride >>= 1) {
                    const int lm = stride / kR;
                    const bool keep_first = ((tt & lm) == 0) == up_t;
#pragma unroll
                    for (int e = 0; e < kR; ++e) {
                        const uint64_t ok = __shfl_xor_sync(0xFFFFFFFFu, kx[e], lm);
                        const int op = __shfl_xor_sync(0xFFFFFFFFu, px[e], lm);
                        if (before(ok, op, kx[e], px[e]) == keep_first) {
                            kx[e] = ok;
                            px[e] = op;
                        }
                    }
                }
#pragma unroll
                for (int stride = kR / 2; stride > 0; stride >>= 1) {
                    if (stride >= size) continue;
#pragma unroll
                    for (int e = 0; e < kR; ++e)
                        if ((e & stride) == 0)
                            cx(kx[e], px[e], kx[e + stride], px[e + stride],
                               (((tt * kR) | e) & size) == 0);
                }
            }
            if (live) store_run(sk, si, tt * kR, kx, px);
            cluster_sync<C>();   // every share of the sides sorted in this pass is sorted
            for (int t = tid; t < nside * c_n; t += kT) {
                const int s2 = t >= c_n;
                const int ts = s2 ? t - c_n : t;
                const int sdx = both ? s2 : pass;   // 0: orphans, 1: donors
                const uint64_t* k2 = s2 ? sk_d : sk_o;
                const int* i2 = s2 ? si_d : si_o;
                const uint64_t key = k2[ts];
                const int pos = i2[ts];
                // its rank: its place in its own share plus, in every other share, the
                // number of items ordered before it
                int rank = ts;
                for (int qq = 0; qq < C; ++qq)
                    if (qq != r)
                        rank += count_before(peer<C>(const_cast<uint64_t*>(k2), qq),
                                             peer<C>(const_cast<int*>(i2), qq), P, key, pos);
                swaps[2 * rank + (sdx ? 0 : 1)] = pos;
                S1[pos] = sdx ? 0 : 1;
            }
            cluster_sync<C>();   // every lookup into this CTA's shares is done
        }
    } else {
        // long lists: one CTA per side sorts its m items with the stable radix passes
        // (keys0/idx0, free by now, as the second buffer)
        for (int x = 0; x < 2; ++x) {
            if (r != (C > 1 ? x : 0)) continue;
            const int o = x == 0 ? 0 : half;
            const int cur = radix_sort(s, K1 + o, I1 + o, K0 + o, I0 + o, m);
            const int* ip = (cur == 0 ? I1 : I0) + o;
            for (int k = tid; k < m; k += kT) {
                const int pos = ip[k];
                swaps[2 * k + (x == 0 ? 1 : 0)] = pos;
                S1[pos] = x == 0 ? 1 : 0;
            }
            __syncthreads();
        }
    }
    if (r == 0 && tid == 0) {
        a.out_nswaps[u] = m;
        if (a.out_status) a.out_status[u] = 0;
    }
}

__global__ void __launch_bounds__(kT, 2) dedup_kernel(const RepairArgs a)   // 2 blocks/SM
{
    __shared__ Shared s;
    const int u = blockIdx.x;
    const int N = a.N;
    const int64_t off = static_cast<int64_t>(u) * N;
    const uint8_t* S0 = a.mask + off;
    const double* b = a.b + off;
    uint8_t* S1 = a.out_mask + off;
    int* swaps = a.out_swaps + static_cast<int64_t>(u) * 2 * (N / 2);

    // 1. validation, counts, and S1 = S0 (also the answer for a failed unit or m = 0)
    int bad = 0, cnt = 0, no = 0, nd = 0;
    // b < tau and b >= tau decided on the order-preserving keys (integer operations;
    // a NaN b is neither an orphan nor a donor, as in fp64 comparisons)
    const uint64_t ktau = ordered(a.tau);
    for (int c0 = 0; c0 < N; c0 += kT * kE) {
#pragma unroll
        for (int j = 0; j < kE; ++j) {
            const int i = c0 + threadIdx.x * kE + j;
            if (i < N) {
                const uint8_t v = S0[i];
                const double bi = b[i];
                const uint64_t ki = ordered(bi);
                const bool num = !is_nan_bits(bi);
                S1[i] = v;
                bad |= v > 1;
                cnt += v != 0;
                const bool prot = i < a.n_sink || i >= N - a.n_recent;
                no += (v == 0 && num && ki < ktau);
                nd += (v != 0 && !prot && num && ki >= ktau);
            }
        }
    }
    if (threadIdx.x < 4) s.red[threadIdx.x] = 0;
    __syncthreads();
    bad = __reduce_or_sync(0xFFFFFFFFu, bad);
    cnt = __reduce_add_sync(0xFFFFFFFFu, cnt);
    no = __reduce_add_sync(0xFFFFFFFFu, no);
    nd = __reduce_add_sync(0xFFFFFFFFu, nd);
    if ((threadIdx.x & 31) == 0) {
        atomicOr(&s.red[0], bad);
        atomicAdd(&s.red[1], cnt);
        atomicAdd(&s.red[2], no);
        atomicAdd(&s.red[3], nd);
    }
    __syncthreads();
    int status = 0;
    if (s.red[0]) status = 1;                                   // TWINKV_ERR_INVALID_ARG
    else if (a.budget && a.budget[u] != s.red[1]) status = 3;   // TWINKV_ERR_BUDGET
    const int n_o = s.red[2], n_d = s.red[3];
    const int m = status ? 0 : min(n_o, n_d);

    if (status != 0 || m == 0) {
        if (threadIdx.x == 0) {
            a.out_nswaps[u] = status ? -1 : 0;
            if (a.out_status) a.out_status[u] = status;
        }
        return;
    }

    // 2-3. classify and compact: orphans at [0, n_o), donors at [n_o, n_o + n_d)
    uint64_t* k0 = a.keys0 + off;
    int* i0 = a.idx0 + off;
    uint64_t* k1 = a.keys1 + off;
    int* i1 = a.idx1 + off;
    int base_o = 0, base_d = n_o;
    for (int c0 = 0; c0 < N; c0 += kT * kE) {
        int fo[kE], fd[kE], co = 0, cd = 0;
        double bv[kE];
#pragma unroll
        for (int j = 0; j < kE; ++j) {
            const int i = c0 + threadIdx.x * kE + j;
            fo[j] = fd[j] = 0;
            bv[j] = 0.0;
            if (i < N) {
                const uint8_t v = S0[i];
                bv[j] = b[i];
                const bool prot = i < a.n_sink || i >= N - a.n_recent;
                const uint64_t kj = ordered(bv[j]);
                const bool num = !is_nan_bits(bv[j]);
                fo[j] = (v == 0 && num && kj < ktau);
                fd[j] = (v != 0 && !prot && num && kj >= ktau);
            }
            co += fo[j];
            cd += fd[j];
        }
        int po, pd, to, td;
        scan2n(s, co, cd, po, pd, to, td);
#pragma unroll
        for (int j = 0; j < kE; ++j) {
            const int i = c0 + threadIdx.x * kE + j;
            if (fo[j]) {
                k0[base_o + po] = ordered(bv[j]);
                i0[base_o + po] = i;
                ++po;
            }
            if (fd[j]) {
                k0[base_d + pd] = ~ordered(bv[j]);
                i0[base_d + pd] = i;
                ++pd;
            }
        }
        base_o += to;
        base_d += td;
    }
    __syncthreads();

    // 4. the m most severe orphans and donors, in severity order
    extern __shared__ __align__(16) uint32_t dyn[];
    uint64_t* sk = reinterpret_cast<uint64_t*>(
        reinterpret_cast<unsigned char*>(dyn) + sort_smem_offset(N));
    int* si = reinterpret_cast<int*>(sk + kSortMax);
    const int* orph;
    const int* don;
    int m_eff = m;
    {
        uint32_t* state = dyn;                                   // 2 bits per rank
        int* trs = reinterpret_cast<int*>(dyn + (N + 15) / 16);  // staged twin ranks
        // every donor in severity order; the other position buffer and the key
        // buffers' donor regions are free afterwards
        const int* spos =
            most_severe(s, k0 + n_o, i0 + n_o, k1 + n_o, i1 + n_o, n_d, n_d, sk, si);
        int* tr = spos == i0 + n_o ? i1 + n_o : i0 + n_o;
        int* dlist = reinterpret_cast<int*>(k0 + n_o);
        int* R = a.rank_of + off;
        for (int i = threadIdx.x; i < N; i += kT) R[i] = -1;
        for (int w = threadIdx.x; w < (n_d + 15) / 16; w += kT) state[w] = 0;
        __syncthreads();
        for (int k = threadIdx.x; k < n_d; k += kT) R[spos[k]] = k;
        __syncthreads();
        const int* tw = a.twin + off;
        for (int k = threadIdx.x; k < n_d; k += kT) {
            const int t = tw[spos[k]];
            tr[k] = (t >= 0 && t < N) ? R[t] : -1;
        }
        __syncthreads();
        int acc = 0;
        for (int c0 = 0; c0 < n_d && acc < n_o; c0 += kWalkChunk) {
            const int len = min(kWalkChunk, n_d - c0);
            for (int j = threadIdx.x; j < len; j += kT) trs[j] = tr[c0 + j];
            __syncthreads();
            if (threadIdx.x == 0) {
                for (int j = 0; j < len && acc < n_o; ++j) {
                    const int k = c0 + j;
                    if ((state[k >> 4] >> ((k & 15) * 2)) & 2u) continue;          // pinned
                    const int t = trs[j];
                    if (t >= 0 && ((state[t >> 4] >> ((t & 15) * 2)) & 1u)) continue;  // twin out
                    state[k >> 4] |= 1u << ((k & 15) * 2);
                    if (t >= 0) state[t >> 4] |= 2u << ((t & 15) * 2);
                    dlist[acc++] = k;
                }
                s.flag = acc;
            }
            __syncthreads();
            acc = s.flag;
            __syncthreads();
        }
        m_eff = acc;
        for (int j = threadIdx.x; j < m_eff; j += kT) dlist[j] = spos[dlist[j]];
        __syncthreads();
        orph = most_severe(s, k0, i0, k1, i1, n_o, m_eff, sk, si);
        don = dlist;
    }
    __syncthreads();

    // 5. swap
    for (int k = threadIdx.x; k < m_eff; k += kT) {
        const int out_ = don[k], in_ = orph[k];
        S1[out_] = 0;
        S1[in_] = 1;
        swaps[2 * k] = out_;
        swaps[2 * k + 1] = in_;
    }
    if (threadIdx.x == 0) {
        a.out_nswaps[u] = m_eff;
        if (a.out_status) a.out_status[u] = 0;
    }
}

}  // namespace

namespace {

template <int C>
cudaError_t config_select(const RepairArgs& a, cudaStream_t st, cudaLaunchConfig_t& cfg,
                          cudaLaunchAttribute* at)
{
    const size_t bytes = 2 * static_cast<size_t>(kChunk) * 12;   // the two shares
    cudaError_t e = cudaFuncSetAttribute(select_kernel<C>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(bytes));
    if (e != cudaSuccess) return e;
    if (C > 8) {
        e = cudaFuncSetAttribute(select_kernel<C>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        if (e != cudaSuccess) return e;
    }
    cfg = cudaLaunchConfig_t{};
    cfg.gridDim = dim3(static_cast<unsigned>(a.U) * C);
    cfg.blockDim = dim3(kT);
    cfg.dynamicSmemBytes = bytes;
    cfg.stream = st;
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = C;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = C > 1 ? 1 : 0;   // one CTA per unit: a plain launch
    return cudaSuccess;
}

// Launches select_kernel<C> if a cluster of C CTAs can be resident; *launched says
// whether it was.
template <int C>
cudaError_t try_select(const RepairArgs& a, cudaStream_t st, bool* launched)
{
    *launched = false;
    cudaLaunchConfig_t cfg;
    cudaLaunchAttribute at[1];
    cudaError_t e = config_select<C>(a, st, cfg, at);
    if (e != cudaSuccess) return e;
    if (C > 1) {
        int clusters = 0;
        e = cudaOccupancyMaxActiveClusters(&clusters, select_kernel<C>, &cfg);
        if (e != cudaSuccess || clusters < 1) {
            cudaGetLastError();   // not resident: the caller tries a smaller cluster
            return cudaSuccess;
        }
    }
    e = cudaLaunchKernelEx(&cfg, select_kernel<C>, a);
    *launched = e == cudaSuccess;
    return e;
}

}  // namespace

int select_cluster_size(int U, int N, int sms)
{
    // the largest cluster that keeps every unit in one wave of two CTAs per SM (more
    // CTAs than that queue behind each other), slices of at least 256 positions, at
    // most 16 CTAs
    int C = 1;
    while (C < 16 && static_cast<int64_t>(U) * (2 * C) <= 2LL * sms && N / (2 * C) >= 256)
        C <<= 1;
    return C;
}

cudaError_t launch_repair(const RepairArgs& a, cudaStream_t st)
{
    if (!a.twin) {
        int C = a.cluster;
        cudaError_t e = cudaSuccess;
        bool done = false;
        while (!done) {
            switch (C) {
            case 16: e = try_select<16>(a, st, &done); break;
            case 8: e = try_select<8>(a, st, &done); break;
            case 4: e = try_select<4>(a, st, &done); break;
            case 2: e = try_select<2>(a, st, &done); break;
            default: e = try_select<1>(a, st, &done); C = 1; break;
            }
            if (e != cudaSuccess) return e;
            if (!done && C == 1) return cudaErrorLaunchFailure;
            C >>= 1;
        }
        return cudaSuccess;
    }
    if (a.N > kDedupMaxN) return cudaErrorInvalidValue;
    const size_t bytes = dedup_kernel_smem_bytes(a.N);
    const cudaError_t e = cudaFuncSetAttribute(
        dedup_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(bytes));
    if (e != cudaSuccess) return e;
    dedup_kernel<<<a.U, kT, bytes, st>>>(a);
    return cudaGetLastError();
}

}  // namespace twk
