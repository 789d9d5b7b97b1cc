// twk_audit.cu -- fused redundancy audit for sm_103a (TwinKV, arXiv 2608.27128).
//
// For every key i of every unit it computes, without materialising the N x N matrix,
//   Sec. 3.2 Eq. 1   sim(i,j) = k_i . k_j / (||k_i|| ||k_j||)
//   Sec. 3.2         only j with |i - j| > w count (this also drops j = i)
//   Sec. 3.4 Eq. 4   b_i(S0) = max over retained j, -1 if none; and its argmax
//   (b_i(all))       the same over every j
//
// Design (one persistent CTA per SM, 64 + 32 * kEpiWarps threads, warp-specialised):
//   warp 0      TMA producer: the 128-row A block of keys i (once per work item), then
//               per 256-column tile the B tile of keys j (in 64-wide K chunks) and the
//               tile's column metadata (1/||k_j|| and original positions).
//   warp 1      owns TMEM (512 columns = two 128x256 fp32 accumulators) and issues
//               tcgen05.mma (M=128, N=256, K=16, bf16 -> fp32) from one thread.
//   warps 2..   epilogue: four warps per column group g (kGW columns of each tile); a
//               thread owns one row (TMEM lane) and keeps its running maximum.
// Keys enter the tensor cores un-normalised (bf16 products are exact in fp32);
// 1/||k_j|| (times a power of two per unit) is applied per element in fp32.
// 1/||k_i|| > 0 does not change the argmax over j, so it is never applied: this kernel
// outputs the twin positions, and the exact similarity of each chosen twin is computed
// afterwards (twk_refine.cu).
//
// Max and argmax: each 32-column chunk is scaled (the column scales carry a power of
// two per unit that brings every value into [-1, 1]), offset to be positive and
// reduced with 3-input maxima.  When a row of the warp improves its best, the chunk's
// column is resolved by replacing the low 5 mantissa bits of each value with (31 - c)
// and taking one more maximum, which returns the lowest column among values equal at
// 2^-18 relative (near-equal candidates only; exact ties go to the lowest column
// whatever their sign, as the values are never negative).  Columns to ignore carry NaN
// (max skips
// NaN): padding columns have 1/||k_j|| = NaN, and window columns (|i - j| <= w) are
// set to NaN on the few tiles that intersect the window band of the row block.
//
// Count mode (Sec. 3.2 Eq. 2, the standalone scorer): instead of the maximum, each row i
// counts the columns j outside the window with sim(i,j) > tau.  With x_ij the raw dot
// product, that is x_ij * (1/||k_j||) > tau * ||k_i||.  The column scales arrive
// multiplied by S = 2^32 (exact), so one fused multiply-add with saturation,
// sat(x_ij * S/||k_j|| - S tau ||k_i||), is 1 when the pair counts and 0 when it does
// not (NaN, for masked and padding columns, saturates to 0); only a pair within
// 2^-32 of the threshold could give a fraction.  The product is never rounded before
// the comparison, the count accumulates in fp32 (exact below 2^24), and all of it
// runs on the FMA pipe.
//
// Column layout: in repair mode the columns of a unit are stored retained-first
// (retained keys in position order, padded to a tile, then evicted keys in position
// order), so every tile belongs to exactly one of the two maxima.  The kernel writes
// both winners; the maximum over all columns is the larger of the two, taken on the
// exact similarities computed afterwards.
#include <cfloat>

#include "twk_internal.h"
#include "twk_ptx.cuh"

namespace twk {
namespace {

constexpr int kEpiWarps = 8;                  // epilogue warps: 2 per SM sub-partition
constexpr int kGroups = kEpiWarps / 4;        // column groups per tile
constexpr int kGW = kBN / kGroups;            // columns per group (a multiple of 32)
constexpr int kThreads = 64 + 32 * kEpiWarps; // + TMA warp + MMA warp
constexpr uint32_t kTmemCols = 512;

template <int D, bool kSym = false>
struct AuditCfg {
    static constexpr int KC = D / 64;                 // 128-byte K chunks per key row
    static constexpr int A_CHUNK = kBM * 128;         // 16 KB
    static constexpr int A_BYTES = KC * A_CHUNK;
    static constexpr int B_STAGE = kBN * 128;         // 32 KB: one K chunk of a tile
    static constexpr int STAGES = (D == 128) ? 4 : 5;
    static constexpr int MSLOTS = 8;
    static constexpr int META = kBN * 8;              // rinv[256] + pos[256]
    static constexpr int OFF_A = 0;
    static constexpr int OFF_B = OFF_A + 2 * A_BYTES;
    static constexpr int OFF_META = OFF_B + STAGES * B_STAGE;
    static constexpr int OFF_X = OFF_META + MSLOTS * META;   // 2 x (groups-1) x 128 x 16 B
    // symmetric mode: each group's four warps exchange their per-column maxima here
    // (two tile parities x groups x 4 lane quarters x 128 columns)
    static constexpr int OFF_CB = OFF_X + 2 * (kGroups - 1) * kBM * 16;
    static constexpr int CB_BYTES = kSym ? 2 * kGroups * 4 * kBM * 4 : 0;
    static constexpr int OFF_BAR = OFF_CB + CB_BYTES;
    static constexpr int NBAR = 2 + 2 + 2 * STAGES + 2 * MSLOTS + 2 + 2 + 2 + 2 + 1 +
                                (kSym ? 2 * kGroups : 0);
    static constexpr int OFF_MISC = OFF_BAR + NBAR * 8;
    static constexpr int BYTES = OFF_MISC + 16 + 1024;       // + 1024 for alignment
};

__device__ __forceinline__ float fmax3(float a, float b, float c)
{
    float r;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
    return r;
}

// (v with its lowest mantissa bits replaced by idx); mask (0xFFFFFFE0) is a kernel
// argument, held in a register, so that idx can be the instruction's immediate.
__device__ __forceinline__ float pack(float v, uint32_t idx, uint32_t mask)
{
    return __uint_as_float((__float_as_uint(v) & mask) | idx);
}

__device__ __forceinline__ float nan_f() { return __uint_as_float(0x7FFFFFFFu); }

// Orders every later use of x after the preceding tcgen05.wait::ld: the registers
// written by tcgen05.ld are only valid after the wait, which the compiler cannot see.
__device__ __forceinline__ void reg_fence(uint32_t (&x)[32])
{
    asm volatile(""
                 : "+r"(x[0]), "+r"(x[1]), "+r"(x[2]), "+r"(x[3]), "+r"(x[4]), "+r"(x[5]),
                   "+r"(x[6]), "+r"(x[7]), "+r"(x[8]), "+r"(x[9]), "+r"(x[10]), "+r"(x[11]),
                   "+r"(x[12]), "+r"(x[13]), "+r"(x[14]), "+r"(x[15]), "+r"(x[16]),
                   "+r"(x[17]), "+r"(x[18]), "+r"(x[19]), "+r"(x[20]), "+r"(x[21]),
                   "+r"(x[22]), "+r"(x[23]), "+r"(x[24]), "+r"(x[25]), "+r"(x[26]),
                   "+r"(x[27]), "+r"(x[28]), "+r"(x[29]), "+r"(x[30]), "+r"(x[31]));
}

// Maximum of 32 values as a tree of 3-input maxima (depth 4); NaN entries are skipped.
__device__ __forceinline__ float tree32(const float (&p)[32])
{
    float q[11];
#pragma unroll
    for (int j = 0; j < 10; ++j) q[j] = fmax3(p[3 * j], p[3 * j + 1], p[3 * j + 2]);
    q[10] = fmaxf(p[30], p[31]);
    const float r0 = fmax3(q[0], q[1], q[2]);
    const float r1 = fmax3(q[3], q[4], q[5]);
    const float r2 = fmax3(q[6], q[7], q[8]);
    const float r3 = fmaxf(q[9], q[10]);
    return fmax3(r0, r1, fmaxf(r2, r3));
}

// Running best of one row over one segment: the scaled similarity x_ij / ||k_j|| in
// fp32 and its column.
struct Best {
    float v;
    int col;
};

// The offset added to every scaled similarity.  The column scales of a unit are
// 2^-e_u / ||k_j||, 2^e_u above every key norm of the unit, so x_ij times the scale is
// sim(i,j) ||k_i|| 2^-e_u, in [-1, 1]; with the offset (a little above 1, for the fp32
// error of x_ij) every value is positive.  A compile-time constant: the fused
// multiply-add then needs no register for it.
constexpr float kOffset = 1.0f + 0x1p-10f;

// Folds 32 columns [col0, col0 + 32) into the running best.  Each accumulator value is
// scaled and offset, v = x_ij 2^-e_u/||k_j|| + kOffset > 0, in one fused multiply-add
// (NaN where the window drops the column, or where the column scale is NaN on
// padding), and the chunk's maximum is taken.  Only when some row of the warp improves
// on its best (strictly, so an earlier column keeps a tie) is the column resolved: each
// value's 5 lowest mantissa bits are replaced by (31 - column) and one more maximum
// returns the lowest column among the values equal to the maximum at 2^-18 relative.
// The values are positive, where a larger low-bit code means a larger float, so ties
// go to the lowest column whatever the sign of the similarity.  Most chunks cost one
// fused multiply-add and one max tree.
template <bool kMasked, bool kEager = false>
__device__ __forceinline__ void fold32(const uint32_t (&x)[32], const float* rinv,
                                       const int* pos, int rw, uint32_t w2, uint32_t mask,
                                       int col0, Best& b)
{
    const float2 ofs = make_float2(kOffset, kOffset);
    float v[32];
#pragma unroll
    for (int k = 0; k < 32; k += 4) {
        const float4 r = *reinterpret_cast<const float4*>(rinv + k);
        const float2 p01 = __ffma2_rn(make_float2(__uint_as_float(x[k]), __uint_as_float(x[k + 1])),
                                      make_float2(r.x, r.y), ofs);
        const float2 p23 = __ffma2_rn(
            make_float2(__uint_as_float(x[k + 2]), __uint_as_float(x[k + 3])),
            make_float2(r.z, r.w), ofs);
        v[k] = p01.x;
        v[k + 1] = p01.y;
        v[k + 2] = p23.x;
        v[k + 3] = p23.y;
        if (kMasked) {
            // column j is dropped when |pos_j - row| <= w, i.e. (unsigned)(pos_j - (row - w)) <= 2w
            const int4 q = *reinterpret_cast<const int4*>(pos + k);
            v[k] = (static_cast<uint32_t>(q.x - rw) > w2) ? v[k] : nan_f();
            v[k + 1] = (static_cast<uint32_t>(q.y - rw) > w2) ? v[k + 1] : nan_f();
            v[k + 2] = (static_cast<uint32_t>(q.z - rw) > w2) ? v[k + 2] : nan_f();
            v[k + 3] = (static_cast<uint32_t>(q.w - rw) > w2) ? v[k + 3] : nan_f();
        }
    }
    if constexpr (kEager) {
        // Where some row of the warp improves in most chunks the vote only adds a
        // branch: every value is packed, one tree gives the lowest column among the
        // values equal to the maximum at 2^-18 relative, and the running best moves at
        // that resolution (an earlier column keeps a tie).
        float p[32];
#pragma unroll
        for (int k = 0; k < 32; ++k) p[k] = pack(v[k], 31u - static_cast<uint32_t>(k), mask);
        const uint32_t mp = __float_as_uint(tree32(p));
        const float m = __uint_as_float(mp & mask);
        if (m > b.v) {
            b.v = m;
            b.col = col0 + 31 - static_cast<int>(mp & 31u);
        }
        return;
    }
    const float m = tree32(v);
    const bool up = m > b.v;
    if (__any_sync(0xFFFFFFFFu, up)) {
        float p[32];
#pragma unroll
        for (int k = 0; k < 32; ++k) p[k] = pack(v[k], 31u - static_cast<uint32_t>(k), mask);
        const int c = 31 - static_cast<int>(__float_as_uint(tree32(p)) & 31u);
        if (up) {
            b.v = m;
            b.col = col0 + c;
        }
    }
}

// The thread's kGW accumulator columns of one tile, loaded into registers (after this,
// the accumulator may be released: the MMA can overwrite it while x is reduced).
__device__ __forceinline__ void load_group(uint32_t taddr, uint32_t (&x0)[32], uint32_t (&x1)[32],
                                           uint32_t (&x2)[32], uint32_t (&x3)[32])
{
    static_assert(kGW == 128, "one 128-column group per warp");
    tmem_ld_32x32b_x32(taddr, x0);
    tmem_ld_32x32b_x32(taddr + 32, x1);
    tmem_ld_32x32b_x32(taddr + 64, x2);
    tmem_ld_32x32b_x32(taddr + 96, x3);
    tmem_wait_ld();
    reg_fence(x0);
    reg_fence(x1);
    reg_fence(x2);
    reg_fence(x3);
}

// Folds the loaded group into the running best, 32 columns at a time in column order.
template <bool kMasked, bool kEager>
__device__ __forceinline__ void reduce_group(const uint32_t (&x0)[32], const uint32_t (&x1)[32],
                                             const uint32_t (&x2)[32], const uint32_t (&x3)[32],
                                             const float* rinv, const int* pos, int rw,
                                             uint32_t w2, uint32_t mask, int col0, Best& b)
{
    fold32<kMasked, kEager>(x0, rinv, pos, rw, w2, mask, col0, b);
    fold32<kMasked, kEager>(x1, rinv + 32, pos + 32, rw, w2, mask, col0 + 32, b);
    fold32<kMasked, kEager>(x2, rinv + 64, pos + 64, rw, w2, mask, col0 + 64, b);
    fold32<kMasked, kEager>(x3, rinv + 96, pos + 96, rw, w2, mask, col0 + 96, b);
}

// Folds one tile's group, eagerly (every chunk resolved, no vote) or vote-gated.
template <bool kEager>
__device__ __forceinline__ void reduce_tile(bool band, const uint32_t (&x0)[32],
                                            const uint32_t (&x1)[32], const uint32_t (&x2)[32],
                                            const uint32_t (&x3)[32], const float* rinv,
                                            const int* pos, int rw, uint32_t w2, uint32_t mask,
                                            int col0, Best& b)
{
    if (band) reduce_group<true, kEager>(x0, x1, x2, x3, rinv, pos, rw, w2, mask, col0, b);
    else reduce_group<false, kEager>(x0, x1, x2, x3, rinv, pos, rw, w2, mask, col0, b);
}

// The argmax modes fold eagerly at d = 64 only.  There a tile's epilogue is twice its
// tensor-core time and, with fewer columns per row, the running best improves in most
// chunks: the eager fold measured 661 TFLOP/s against 617 at the Llama-3.2-1B shape.  It
// compares candidates of different chunks at the packed resolution, so more near ties
// (within 2^-18 relative of the maximum) go to the earlier column; at d = 128 it gained
// nothing measurable (16 eager tiles per row block: 1275 against 1271 TFLOP/s), and the
// vote-gated fold keeps the exact comparison across chunks there.
template <int D>
__device__ __forceinline__ constexpr bool eager_fold()
{
    return D == 64;
}

// sat(a * b + c): fp32 fused multiply-add clamped to [0, 1], NaN to 0.
__device__ __forceinline__ float fma_sat(float a, float b, float c)
{
    float r;
    asm("fma.rn.sat.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
    return r;
}

// Eq. 2 over 32 columns: how many x_j * S/||k_j|| exceed ts = S tau ||k_i||, as two
// partial sums.
template <bool kMasked>
__device__ __forceinline__ float2 count32(const uint32_t (&x)[32], const float* rinv,
                                          const int* pos, int rw, uint32_t w2, float ts)
{
    float2 ca = make_float2(0.f, 0.f), cb = make_float2(0.f, 0.f);
#pragma unroll
    for (int k = 0; k < 32; k += 4) {
        const float4 r = *reinterpret_cast<const float4*>(rinv + k);
        float v0 = __uint_as_float(x[k]), v1 = __uint_as_float(x[k + 1]);
        float v2 = __uint_as_float(x[k + 2]), v3 = __uint_as_float(x[k + 3]);
        if (kMasked) {
            const int4 q = *reinterpret_cast<const int4*>(pos + k);
            v0 = (static_cast<uint32_t>(q.x - rw) > w2) ? v0 : nan_f();
            v1 = (static_cast<uint32_t>(q.y - rw) > w2) ? v1 : nan_f();
            v2 = (static_cast<uint32_t>(q.z - rw) > w2) ? v2 : nan_f();
            v3 = (static_cast<uint32_t>(q.w - rw) > w2) ? v3 : nan_f();
        }
        ca = __fadd2_rn(ca, make_float2(fma_sat(v0, r.x, -ts), fma_sat(v1, r.y, -ts)));
        cb = __fadd2_rn(cb, make_float2(fma_sat(v2, r.z, -ts), fma_sat(v3, r.w, -ts)));
    }
    return __fadd2_rn(ca, cb);
}

template <bool kMasked>
__device__ __forceinline__ float count_group(const uint32_t (&x0)[32], const uint32_t (&x1)[32],
                                             const uint32_t (&x2)[32], const uint32_t (&x3)[32],
                                             const float* rinv, const int* pos, int rw,
                                             uint32_t w2, float ts)
{
    const float2 a = __fadd2_rn(count32<kMasked>(x0, rinv, pos, rw, w2, ts),
                                count32<kMasked>(x1, rinv + 32, pos + 32, rw, w2, ts));
    const float2 b = __fadd2_rn(count32<kMasked>(x2, rinv + 64, pos + 64, rw, w2, ts),
                                count32<kMasked>(x3, rinv + 96, pos + 96, rw, w2, ts));
    const float2 c = __fadd2_rn(a, b);
    return c.x + c.y;
}

__device__ __forceinline__ uint32_t redux_max(uint32_t v)
{
    uint32_t r;
    asm volatile("redux.sync.max.u32 %0, %1, 0xffffffff;" : "=r"(r) : "r"(v));
    return r;
}

// Symmetric mode, the column direction of one 32-column chunk: for every column j of
// the chunk the largest x_ij s_i + kOffset over the warp's 32 rows i (s_i = the row's
// own column scale, so the value is that of row j's candidate i), its low 5 bits
// replaced by (31 - lane) so that a tie goes to the lowest row.  Masked: window pairs
// and rows past the end give 0, below every candidate.  Lane l returns column l's.
template <bool kMasked>
__device__ __forceinline__ uint32_t colpass32(const uint32_t (&x)[32], const int* pos, int rw,
                                              uint32_t w2, float si, bool row_ok)
{
    const int lane = threadIdx.x & 31;
    const uint32_t code = 31u - static_cast<uint32_t>(lane);
    uint32_t keep = 0u;
#pragma unroll
    for (int k = 0; k < 32; k += 4) {
        int4 q = make_int4(0, 0, 0, 0);
        if (kMasked) q = *reinterpret_cast<const int4*>(pos + k);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            float v = fmaf(__uint_as_float(x[k + e]), si, kOffset);
            if (kMasked) {
                const int pj = e == 0 ? q.x : e == 1 ? q.y : e == 2 ? q.z : q.w;
                v = (row_ok && static_cast<uint32_t>(pj - rw) > w2) ? v : 0.f;
            }
            const uint32_t r = redux_max((__float_as_uint(v) & 0xFFFFFFE0u) | code);
            keep = lane == k + e ? r : keep;
        }
    }
    return keep;
}

struct Tiles {
    int tr;   // tiles of segment 0 (retained, or every column in mode 0)
    int te;   // tiles of segment 1 (evicted; 0 unless b_all is wanted)
    int t0;   // the first tile (symmetric mode: the tile holding column 128 rb - 0..128)
};

// Symmetric mode: row block rb takes the tiles from the one holding its own first
// column, rb / 2, to the last; the pairs left of them reach rb's rows through the
// column maxima of the row blocks before it.
template <bool kSym>
__device__ __forceinline__ Tiles unit_tiles(const AuditArgs& a, int u, int rb)
{
    if (kSym) {
        const int t0 = rb >> 1;
        return {(a.N + kBN - 1) / kBN - t0, 0, t0};
    }
    if (!a.repair_mode) return {(a.N + kBN - 1) / kBN, 0, 0};
    const int kb = a.kb[u];
    return {(kb + kBN - 1) / kBN, a.need_all ? (a.N - kb + kBN - 1) / kBN : 0, 0};
}

// Lane 0 waits, the warp follows its verdict.
__device__ __forceinline__ bool lane0_wait(uint64_t* bar, uint32_t parity, const WaitCtl& w,
                                           int where)
{
    int ok = 1;
    if ((threadIdx.x & 31) == 0) ok = mbar_wait(bar, parity, w, where) ? 1 : 0;
    return __shfl_sync(0xFFFFFFFFu, ok, 0) != 0;
}

// Every lane waits (each needs the acquire), the warp agrees on the verdict.
__device__ __forceinline__ bool all_wait(uint64_t* bar, uint32_t parity, const WaitCtl& w,
                                         int where)
{
    const bool ok = mbar_wait(bar, parity, w, where);
    return __all_sync(0xFFFFFFFFu, ok);
}

// Bounded wait that ignores the abort flag (used to drain in-flight copies and MMAs
// after a give-up), never shorter than kDrainFloorNs whatever the caller's limit.
__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity, uint64_t limit_ns)
{
    const uint64_t limit = limit_ns > kDrainFloorNs ? limit_ns : kDrainFloorNs;
    const uint32_t a = smem_u32(bar);
    const uint64_t t0 = globaltimer_ns();
    while (!mbar_try_wait_sleep(a, parity, 1000000u))
        if (globaltimer_ns() - t0 > limit) return;
}

// Parity of the last arming of slot s after `total` armings of a ring of `n` slots,
// or -1 if slot s was never armed.
__device__ __forceinline__ int last_parity(long long total, int n, int s)
{
    if (total <= s) return -1;
    const long long k = s + (long long)n * ((total - 1 - s) / n);
    return static_cast<int>((k / n) & 1);
}

// Registers are per sub-partition (16384 each): with W warps a sub-partition holds
// ceil(W / 4) of them, which bounds the registers per thread.
template <int D, bool kCount, bool kSym>
__global__ void __launch_bounds__(kThreads, 1)
    audit_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                 const __grid_constant__ AuditArgs a)
{
    using C = AuditCfg<D, kSym>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    uint8_t* sA = smem + C::OFF_A;
    uint8_t* sB = smem + C::OFF_B;
    uint8_t* sMeta = smem + C::OFF_META;
    float4* sX = reinterpret_cast<float4*>(smem + C::OFF_X);
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
    uint64_t* a_full = bars;
    uint64_t* a_empty = a_full + 2;
    uint64_t* b_full = a_empty + 2;
    uint64_t* b_empty = b_full + C::STAGES;
    uint64_t* m_full = b_empty + C::STAGES;
    uint64_t* m_empty = m_full + C::MSLOTS;
    uint64_t* t_full = m_empty + C::MSLOTS;
    uint64_t* t_empty = t_full + 2;
    uint64_t* x_full = t_empty + 2;
    uint64_t* x_empty = x_full + 2;
    uint64_t* drain = x_empty + 2;
    uint64_t* cbar = drain + 1;   // symmetric mode: [tile parity][group], 128 arrivals
    uint32_t* sCB = reinterpret_cast<uint32_t*>(smem + C::OFF_CB);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_MISC);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::OFF_MISC + 4);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int i = 0; i < 2; ++i) {
            mbar_init(&a_full[i], 1);
            mbar_init(&a_empty[i], 1);
            mbar_init(&t_full[i], 1);
            mbar_init(&t_empty[i], kEpiWarps);
            mbar_init(&x_full[i], (kGroups - 1) * kBM);
            mbar_init(&x_empty[i], kBM);
        }
        for (int i = 0; i < C::STAGES; ++i) {
            mbar_init(&b_full[i], 1);
            mbar_init(&b_empty[i], 1);
        }
        for (int i = 0; i < C::MSLOTS; ++i) {
            mbar_init(&m_full[i], 1);
            mbar_init(&m_empty[i], kEpiWarps);
        }
        mbar_init(drain, 1);
        if (kSym)
            for (int i = 0; i < 2 * kGroups; ++i) mbar_init(&cbar[i], 4 * 32);
        *abort_flag = 0;
        fence_mbarrier_init();
    }
    if (warp == 0 && lane == 0) {
        prefetch_tensormap(&tmA);
        prefetch_tensormap(&tmB);
    }
    if (warp == 1) tmem_alloc(tmem_slot, kTmemCols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    WaitCtl wc;
    wc.limit_ns = a.timeout_ns;
    wc.abort_flag = abort_flag;
    wc.err = a.err;
    wc.where = 0;
    const int n_items = a.U * a.RB;

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        long long n_a = 0, n_b = 0, n_m = 0;
        bool ok = true;
        for (int item = blockIdx.x; item < n_items && ok; item += gridDim.x) {
            const int u = item / a.RB;
            const int rb = item - u * a.RB;
            const Tiles ut = unit_tiles<kSym>(a, u, rb);
            const int ab = static_cast<int>(n_a & 1);
            ok = lane0_wait(&a_empty[ab], static_cast<uint32_t>(((n_a >> 1) & 1) ^ 1), wc, 1);
            if (!ok) break;
            if (lane == 0) {
                mbar_arrive_expect_tx(&a_full[ab], C::A_BYTES);
                const int y = u * a.N + rb * kBM;
#pragma unroll
                for (int kc = 0; kc < C::KC; ++kc)
                    tma_load_2d(sA + ab * C::A_BYTES + kc * C::A_CHUNK, &tmA, &a_full[ab],
                                kc * 64, y);
            }
            __syncwarp();
            ++n_a;
            const int nt = ut.tr + ut.te;
            for (int t = 0; t < nt && ok; ++t) {
                const int col0 = (ut.t0 + t) * kBN;
                const int ms = static_cast<int>(n_m % C::MSLOTS);
                ok = lane0_wait(&m_empty[ms],
                                static_cast<uint32_t>(((n_m / C::MSLOTS) & 1) ^ 1), wc, 2);
                if (!ok) break;
                if (lane == 0) {
                    mbar_arrive_expect_tx(&m_full[ms], C::META);
                    const int64_t off = static_cast<int64_t>(u) * a.NP + col0;
                    bulk_load(sMeta + ms * C::META, a.colrinv + off, kBN * 4, &m_full[ms]);
                    bulk_load(sMeta + ms * C::META + kBN * 4, a.colpos + off, kBN * 4,
                              &m_full[ms]);
                }
                __syncwarp();
                ++n_m;
                const int yb = static_cast<int>(u * a.b_rows_per_unit + col0);
                for (int kc = 0; kc < C::KC; ++kc) {
                    const int s = static_cast<int>(n_b % C::STAGES);
                    ok = lane0_wait(&b_empty[s],
                                    static_cast<uint32_t>(((n_b / C::STAGES) & 1) ^ 1), wc, 3);
                    if (!ok) break;
                    if (lane == 0) {
                        mbar_arrive_expect_tx(&b_full[s], C::B_STAGE);
                        tma_load_2d(sB + s * C::B_STAGE, &tmB, &b_full[s], kc * 64, yb);
                    }
                    __syncwarp();
                    ++n_b;
                }
            }
        }
        if (!ok && lane == 0) {
            // Let every copy this warp started land before the block exits.
            for (int s = 0; s < 2; ++s) {
                const int p = last_parity(n_a, 2, s);
                if (p >= 0) drain_wait(&a_full[s], p, a.timeout_ns);
            }
            for (int s = 0; s < C::STAGES; ++s) {
                const int p = last_parity(n_b, C::STAGES, s);
                if (p >= 0) drain_wait(&b_full[s], p, a.timeout_ns);
            }
            for (int s = 0; s < C::MSLOTS; ++s) {
                const int p = last_parity(n_m, C::MSLOTS, s);
                if (p >= 0) drain_wait(&m_full[s], p, a.timeout_ns);
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        constexpr uint32_t idesc = umma_idesc_bf16_f32(kBM, kBN);
        long long n_a = 0, n_b = 0, n_t = 0;
        bool ok = true;
        for (int item = blockIdx.x; item < n_items && ok; item += gridDim.x) {
            const int u = item / a.RB;
            const Tiles ut = unit_tiles<kSym>(a, u, item - u * a.RB);
            const int ab = static_cast<int>(n_a & 1);
            ok = lane0_wait(&a_full[ab], static_cast<uint32_t>((n_a >> 1) & 1), wc, 4);
            if (!ok) break;
            tc_fence_after();
            const uint32_t a_base = smem_u32(sA + ab * C::A_BYTES);
            const int nt = ut.tr + ut.te;
            for (int t = 0; t < nt && ok; ++t) {
                const int acc = static_cast<int>(n_t & 1);
                ok = lane0_wait(&t_empty[acc], static_cast<uint32_t>(((n_t >> 1) & 1) ^ 1), wc,
                                5);
                if (!ok) break;
                tc_fence_after();
                const uint32_t d_tmem = tmem + static_cast<uint32_t>(acc * kBN);
                for (int kc = 0; kc < C::KC; ++kc) {
                    const int s = static_cast<int>(n_b % C::STAGES);
                    ok = lane0_wait(&b_full[s], static_cast<uint32_t>((n_b / C::STAGES) & 1), wc,
                                    6);
                    if (!ok) break;
                    tc_fence_after();
                    if (lane == 0) {
                        const uint64_t ad = umma_desc_sw128(a_base + kc * C::A_CHUNK);
                        const uint64_t bd = umma_desc_sw128(smem_u32(sB + s * C::B_STAGE));
#pragma unroll
                        for (int k = 0; k < 4; ++k)
                            umma_bf16(d_tmem, ad + 2u * k, bd + 2u * k, idesc,
                                      (kc | k) != 0 ? 1u : 0u);
                        umma_commit(&b_empty[s]);
                    }
                    __syncwarp();
                    ++n_b;
                }
                if (!ok) break;
                if (lane == 0) umma_commit(&t_full[acc]);
                __syncwarp();
                ++n_t;
            }
            if (!ok) break;
            if (lane == 0) umma_commit(&a_empty[ab]);
            __syncwarp();
            ++n_a;
        }
        // Every MMA this thread issued completes before TMEM is released.
        if (lane == 0) {
            umma_commit(drain);
            drain_wait(drain, 0, a.timeout_ns);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ epilogue
        const int ew = warp - 2;
        const int h = ew >> 2;            // column group of the tile
        const int q = warp & 3;           // TMEM lane quarter this warp may read
        const int row_local = q * 32 + lane;
        const uint32_t lane_base = static_cast<uint32_t>(q * 32) << 16;
        const int w = a.window;
        const uint32_t w2 = 2u * static_cast<uint32_t>(w);
        const uint32_t mask = a.mant_mask;
        uint32_t ms = 0, mph = 0;    // meta ring slot and phase
        uint32_t acc = 0, tph = 0;   // accumulator buffer and phase
        uint32_t n_x = 0;
        uint32_t n_c = 0;   // symmetric mode: tiles whose column maxima were merged
        bool ok = true;
        for (int item = blockIdx.x; item < n_items && ok; item += gridDim.x) {
            const int u = item / a.RB;
            const int rb = item - u * a.RB;
            const Tiles ut = unit_tiles<kSym>(a, u, rb);
            const int nt = ut.tr + ut.te;
            const int r0 = rb * kBM;
            const int row = r0 + row_local;
            // symmetric mode: the row's own column scale (the value of row j's candidate
            // i is x_ij s_i), and whether this row block runs past the end of the unit
            const bool row_ok = row < a.N;
            const float si = (kSym && row_ok) ? a.colrinv[static_cast<int64_t>(u) * a.NP + row] : 0.f;
            const bool pad_item = r0 + kBM > a.N;

            // Column ranges that meet the window band [r0 - w, r0 + 128 + w) of this
            // row block: only tiles meeting them need the per-element window test.
            const int lo = max(r0 - w, 0);
            const int hi = min(r0 + kBM + w, a.N);
            int s0a, s0b, s1a = 0, s1b = 0;
            if (!a.repair_mode) {
                s0a = lo;
                s0b = hi;
            } else {
                const int kb = a.kb[u];
                const int* cnt = a.cnt + static_cast<int64_t>(u) * a.N;
                const int clo = lo < a.N ? cnt[lo] : kb;
                const int chi = hi < a.N ? cnt[hi] : kb;
                const int kpad = ut.tr * kBN;
                s0a = clo;
                s0b = chi;
                s1a = kpad + lo - clo;
                s1b = kpad + hi - chi;
            }

            Best b0{-INFINITY, -1}, b1{-INFINITY, -1};   // retained (or all) / evicted
            const int rw = row - w;

            float cnt = 0.f;                               // count mode: r_i so far
            float thr = 0.f;                               // count mode: S tau ||k_i||
            if (kCount)
                thr = (a.count_tau /
                       (a.colrinv[static_cast<int64_t>(u) * a.NP + row] * (1.0f / kCountScale))) *
                      kCountScale;
            for (int t = 0; t < nt; ++t) {
                ok = all_wait(&m_full[ms], mph, wc, 7);
                if (ok) ok = all_wait(&t_full[acc], tph, wc, 8);
                if (!ok) break;
                tc_fence_after();
                const float* rinv = reinterpret_cast<const float*>(sMeta + ms * C::META) + h * kGW;
                const int* pos =
                    reinterpret_cast<const int*>(sMeta + ms * C::META + kBN * 4) + h * kGW;
                const int c_lo = (ut.t0 + t) * kBN + h * kGW;
                const bool band = (c_lo < s0b && c_lo + kGW > s0a) ||
                                  (c_lo < s1b && c_lo + kGW > s1a);
                const uint32_t taddr = tmem + lane_base + acc * kBN + static_cast<uint32_t>(h * kGW);
                uint32_t x0[32], x1[32], x2[32], x3[32];
                load_group(taddr, x0, x1, x2, x3);
                // The tile is in registers: hand the accumulator back to the MMA warp now,
                // so it can compute the next-but-one tile while this one is reduced.
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&t_empty[acc]);
                if (kSym) {
                    // row maxima (the eager fold: the column pass already costs more than
                    // the vote saves) and each chunk's column maxima over this warp's 32
                    // rows right after it (while its registers are live)
                    uint32_t cr[4];
                    if (band) {
                        fold32<true, true>(x0, rinv, pos, rw, w2, mask, c_lo, b0);
                        cr[0] = colpass32<true>(x0, pos, rw, w2, si, row_ok);
                        fold32<true, true>(x1, rinv + 32, pos + 32, rw, w2, mask, c_lo + 32, b0);
                        cr[1] = colpass32<true>(x1, pos + 32, rw, w2, si, row_ok);
                        fold32<true, true>(x2, rinv + 64, pos + 64, rw, w2, mask, c_lo + 64, b0);
                        cr[2] = colpass32<true>(x2, pos + 64, rw, w2, si, row_ok);
                        fold32<true, true>(x3, rinv + 96, pos + 96, rw, w2, mask, c_lo + 96, b0);
                        cr[3] = colpass32<true>(x3, pos + 96, rw, w2, si, row_ok);
                    } else if (pad_item) {
                        fold32<false, true>(x0, rinv, pos, rw, w2, mask, c_lo, b0);
                        cr[0] = colpass32<true>(x0, pos, rw, w2, si, row_ok);
                        fold32<false, true>(x1, rinv + 32, pos + 32, rw, w2, mask, c_lo + 32, b0);
                        cr[1] = colpass32<true>(x1, pos + 32, rw, w2, si, row_ok);
                        fold32<false, true>(x2, rinv + 64, pos + 64, rw, w2, mask, c_lo + 64, b0);
                        cr[2] = colpass32<true>(x2, pos + 64, rw, w2, si, row_ok);
                        fold32<false, true>(x3, rinv + 96, pos + 96, rw, w2, mask, c_lo + 96, b0);
                        cr[3] = colpass32<true>(x3, pos + 96, rw, w2, si, row_ok);
                    } else {
                        fold32<false, true>(x0, rinv, pos, rw, w2, mask, c_lo, b0);
                        cr[0] = colpass32<false>(x0, pos, rw, w2, si, row_ok);
                        fold32<false, true>(x1, rinv + 32, pos + 32, rw, w2, mask, c_lo + 32, b0);
                        cr[1] = colpass32<false>(x1, pos + 32, rw, w2, si, row_ok);
                        fold32<false, true>(x2, rinv + 64, pos + 64, rw, w2, mask, c_lo + 64, b0);
                        cr[2] = colpass32<false>(x2, pos + 64, rw, w2, si, row_ok);
                        fold32<false, true>(x3, rinv + 96, pos + 96, rw, w2, mask, c_lo + 96, b0);
                        cr[3] = colpass32<false>(x3, pos + 96, rw, w2, si, row_ok);
                    }
                    // merge the four lane quarters of this group: the warps exchange their
                    // 128 column maxima, then warp q takes columns 32q .. 32q + 31
                    const int par = static_cast<int>(n_c & 1);
                    uint32_t* cb = sCB + (par * kGroups + h) * 4 * kBM;
#pragma unroll
                    for (int k = 0; k < 4; ++k) cb[q * kBM + 32 * k + lane] = cr[k];
                    mbar_arrive(&cbar[par * kGroups + h]);
                    ok = all_wait(&cbar[par * kGroups + h], (n_c >> 1) & 1, wc, 11);
                    ++n_c;
                    if (!ok) break;
                    const int c = q * 32 + lane;
                    uint32_t best = cb[c];
                    int bq = 0;
#pragma unroll
                    for (int qq = 1; qq < 4; ++qq) {
                        const uint32_t vq = cb[qq * kBM + c];
                        if ((vq & 0xFFFFFFE0u) > (best & 0xFFFFFFE0u)) {
                            best = vq;
                            bq = qq;
                        }
                    }
                    const int gcol = c_lo + c;
                    if (gcol < a.N && (best & 0xFFFFFFE0u) != 0u) {
                        const uint32_t win = static_cast<uint32_t>(r0 + 32 * bq + 31) - (best & 31u);
                        atomicMax(a.slots + static_cast<int64_t>(u) * a.N + gcol,
                                  (static_cast<unsigned long long>(best & 0xFFFFFFE0u) << 32) |
                                      (0xFFFFFFFFull - win));
                    }
                } else if (kCount) {
                    cnt += band ? count_group<true>(x0, x1, x2, x3, rinv, pos, rw, w2, thr)
                                : count_group<false>(x0, x1, x2, x3, rinv, pos, rw, w2, thr);
                } else if (t < ut.tr) {
                    reduce_tile<eager_fold<D>()>(band, x0, x1, x2, x3, rinv, pos, rw, w2, mask,
                                                 c_lo, b0);
                } else {
                    if (t == ut.tr) {
                        // The evicted segment matters only where it reaches the retained
                        // one: start its running best just below this group's retained
                        // best (exact similarities decide between the two later; the
                        // FLT_MIN keeps an exact tie at 0 in play).
                        b1.v = b0.v - (fabsf(b0.v) * 0x1p-13f + FLT_MIN);
                    }
                    reduce_tile<eager_fold<D>()>(band, x0, x1, x2, x3, rinv, pos, rw, w2, mask,
                                                 c_lo, b1);
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(&m_empty[ms]);
                if (++ms == C::MSLOTS) {
                    ms = 0;
                    mph ^= 1;
                }
                acc ^= 1;
                tph ^= acc == 0 ? 1u : 0u;
            }
            if (!ok) break;
            const float bv0 = b0.v, bv1 = b1.v;
            const int bc0 = b0.col, bc1 = b1.col;

            // Merge the column groups of every row through shared memory: groups
            // 1.. hand their (value, column) pairs to group 0.
            const int xb = static_cast<int>(n_x & 1);
            float4* X = sX + xb * (kGroups - 1) * kBM;
            if (h != 0) {
                ok = all_wait(&x_empty[xb], ((n_x >> 1) & 1) ^ 1, wc, 9);
                if (!ok) break;
                X[(h - 1) * kBM + row_local] =
                    kCount ? make_float4(cnt, 0.f, 0.f, 0.f)
                           : make_float4(bv0, __int_as_float(bc0), bv1, __int_as_float(bc1));
                mbar_arrive(&x_full[xb]);
            } else if (kCount) {
                ok = all_wait(&x_full[xb], (n_x >> 1) & 1, wc, 10);
                if (!ok) break;
                float total = cnt;
#pragma unroll
                for (int g = 1; g < kGroups; ++g) total += X[(g - 1) * kBM + row_local].x;
                mbar_arrive(&x_empty[xb]);
                if (row < a.N)
                    a.out_count[static_cast<int64_t>(u) * a.N + row] = __float2int_rn(total);
            } else {
                ok = all_wait(&x_full[xb], (n_x >> 1) & 1, wc, 10);
                if (!ok) break;
                float v0 = bv0, v1 = bv1;
                int c0 = bc0, c1 = bc1;
#pragma unroll
                for (int g = 1; g < kGroups; ++g) {
                    const float4 o = X[(g - 1) * kBM + row_local];
                    const int oc0 = __float_as_int(o.y), oc1 = __float_as_int(o.w);
                    if (oc0 >= 0 && (c0 < 0 || o.x > v0 || (o.x == v0 && oc0 < c0))) {
                        v0 = o.x;
                        c0 = oc0;
                    }
                    if (oc1 >= 0 && (c1 < 0 || o.z > v1 || (o.z == v1 && oc1 < c1))) {
                        v1 = o.z;
                        c1 = oc1;
                    }
                }
                mbar_arrive(&x_empty[xb]);
                if (kSym) {
                    // the row direction's best joins the column maxima of earlier row
                    // blocks in the row's slot: value (low 5 bits cleared) then lowest
                    // position
                    if (row < a.N && c0 >= 0)
                        atomicMax(a.slots + static_cast<int64_t>(u) * a.N + row,
                                  (static_cast<unsigned long long>(__float_as_uint(v0) &
                                                                   0xFFFFFFE0u) << 32) |
                                      (0xFFFFFFFFull - static_cast<uint32_t>(c0)));
                } else if (row < a.N) {
                    const int64_t o_idx = static_cast<int64_t>(u) * a.N + row;
                    const int64_t cbase = static_cast<int64_t>(u) * a.NP;
                    const int p0 = c0 < 0 ? -1 : (a.repair_mode ? a.colpos[cbase + c0] : c0);
                    a.out_t0[o_idx] = p0;
                    if (a.repair_mode && a.need_all)
                        a.out_t1[o_idx] = c1 < 0 ? -1 : a.colpos[cbase + c1];
                }
            }
            ++n_x;
        }
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem, kTmemCols);
}

}  // namespace

size_t audit_smem_bytes(int d)
{
    return d == 128 ? AuditCfg<128>::BYTES : AuditCfg<64>::BYTES;
}

template <int D, bool kCount, bool kSym>
cudaError_t launch_audit_t(const CUtensorMap& tmA, const CUtensorMap& tmB, const AuditArgs& a,
                           int grid, cudaStream_t st)
{
    const int bytes = AuditCfg<D, kSym>::BYTES;
    cudaError_t e = cudaFuncSetAttribute(audit_kernel<D, kCount, kSym>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e != cudaSuccess) return e;
    audit_kernel<D, kCount, kSym><<<grid, kThreads, bytes, st>>>(tmA, tmB, a);
    return cudaGetLastError();
}

cudaError_t launch_audit(int d, AuditMode mode, const CUtensorMap& tmA, const CUtensorMap& tmB,
                         const AuditArgs& a, int grid, cudaStream_t st)
{
    if (d == 128) {
        if (mode == AuditMode::kCount) return launch_audit_t<128, true, false>(tmA, tmB, a, grid, st);
        if (mode == AuditMode::kSymmetric)
            return launch_audit_t<128, false, true>(tmA, tmB, a, grid, st);
        return launch_audit_t<128, false, false>(tmA, tmB, a, grid, st);
    }
    if (mode == AuditMode::kCount) return launch_audit_t<64, true, false>(tmA, tmB, a, grid, st);
    if (mode == AuditMode::kSymmetric) return launch_audit_t<64, false, true>(tmA, tmB, a, grid, st);
    return launch_audit_t<64, false, false>(tmA, tmB, a, grid, st);
}

namespace {
// twin of every row from its slot: the low word holds 0xFFFFFFFF - position; an empty
// slot (no candidate beyond the window) gives -1
__global__ void slots_to_twins_kernel(const unsigned long long* __restrict__ slots, int64_t n,
                                      int* __restrict__ twin)
{
    const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (i >= n) return;
    const unsigned long long sv = slots[i];
    twin[i] = sv == 0ull ? -1 : static_cast<int>(0xFFFFFFFFull - (sv & 0xFFFFFFFFull));
}
}  // namespace

cudaError_t launch_slots_to_twins(const unsigned long long* slots, int64_t n, int* twin,
                                  cudaStream_t st)
{
    const int64_t blocks = (n + 255) / 256;
    slots_to_twins_kernel<<<static_cast<unsigned>(blocks), 256, 0, st>>>(slots, n, twin);
    return cudaGetLastError();
}

// ---------------------------------------------------------------- wait probe

namespace {
__global__ void wait_probe_kernel(int* err, unsigned long long timeout_ns)
{
    __shared__ uint64_t bar;
    __shared__ uint32_t slot;
    __shared__ int abort_flag;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        abort_flag = 0;
        fence_mbarrier_init();
    }
    if (threadIdx.x < 32) tmem_alloc(&slot, 32);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    WaitCtl wc;
    wc.limit_ns = timeout_ns;
    wc.abort_flag = &abort_flag;
    wc.err = err;
    wc.where = 0;
    // Nothing ever arrives on `bar`: its phase 0 never completes.
    (void)mbar_wait(&bar, 0, wc, 99);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (threadIdx.x < 32) tmem_dealloc(slot, 32);
}
}  // namespace

cudaError_t launch_wait_probe(int* err, unsigned long long timeout_ns, cudaStream_t st)
{
    wait_probe_kernel<<<1, 64, 0, st>>>(err, timeout_ns);
    return cudaGetLastError();
}

}  // namespace twk
