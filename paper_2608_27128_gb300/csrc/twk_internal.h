// twk_internal.h -- kernel argument blocks and launchers shared by the translation
// units of libtwinkv (host-side declarations only).
#pragma once
#include <cstddef>
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

namespace twk {

constexpr int kBM = 128;       // rows (keys i) per work item: the UMMA M
constexpr int kBN = 256;       // columns (keys j) per tile: the UMMA N

// Bounded waits.  A wait on work that another role of the block has to do gives up
// after the caller's limit (twinkv_set_wait_timeout_ns, never below kMinWaitLimitNs).
// After a give-up, the copies and MMAs a CTA already started are drained before it
// frees its tensor memory and exits; those drain waits use at least kDrainFloorNs,
// whatever the caller's limit, since in-flight copies and MMAs complete in
// microseconds unless the device itself is failing.
constexpr unsigned long long kMinWaitLimitNs = 10000000ull;    // 10 ms
constexpr unsigned long long kDrainFloorNs = 200000000ull;     // 200 ms

// Column stride of the per-unit column arrays (a multiple of kBN with room for the
// padding of both the retained and the evicted segment).
inline int64_t column_stride(int N) { return ((int64_t)(N + kBN - 1) / kBN) * kBN + kBN; }

struct AuditArgs {
    int U, N, NP, RB;           // units, keys per unit, column stride, row blocks per unit
    int window;                 // w, clamped to [0, N]
    int repair_mode;            // 0: one segment over the keys as given; 1: retained-first
    int need_all;               // repair mode: also scan the evicted segment
    int64_t b_rows_per_unit;    // row stride of a unit in the B tensor map
    const float* colrinv;       // [U][NP]  1/||k|| per column, NaN on padding columns
    const int* colpos;          // [U][NP]  original position of each column
    const int* cnt;             // [U][N]   retained positions before p (repair mode)
    const int* kb;              // [U]      |S0| (repair mode)
    int* out_t0;                // [U][N]   argmax of segment 0 (retained, or all in mode 0)
    int* out_t1;                // [U][N]   argmax of segment 1, the evicted columns
                                //          (repair mode with need_all), -1 if none
    int* err;
    unsigned long long timeout_ns;
    uint32_t mant_mask;         // 0xFFFFFFE0: clears the 5 mantissa bits that carry the
                                // column; a runtime value, so the compiler keeps it in a
                                // register and the pack is a single 3-input logic op
    // count mode (Eq. 2): mode 0 columns only, colrinv scaled by kCountScale;
    // out_t0/out_t1 unused
    float count_tau;            // tau, compared strictly
    int* out_count;             // [U][N] r_i
    // symmetric mode (mode 0 columns, upper-triangle tiles): per row, the best
    // candidate as (value bits with the 5 low bits cleared) << 32 | (0xFFFFFFFF - pos),
    // combined with atomicMax from both directions; zero-initialised by the caller
    unsigned long long* slots;  // [U][N]
};

enum class AuditMode { kArgmax, kCount, kSymmetric };

struct RepairArgs {
    int U, N;
    const double* b;            // [U][N] b_i(S0)
    const uint8_t* mask;        // [U][N]
    const int* budget;          // [U] or null
    double tau;                 // threshold rounded to float, widened
    int n_sink, n_recent;
    uint8_t* out_mask;          // [U][N]
    int* out_swaps;             // [U][N/2][2]
    int* out_nswaps;            // [U]
    int* out_status;            // [U] or null
    uint64_t* keys0;            // [U][N] sort buffers (ping-pong)
    int* idx0;
    uint64_t* keys1;
    int* idx1;
    // dedup variant (twin != null): a donor is not evicted together with its twin
    const int* twin;            // [U][N] argmax position of b_i(S0), or null
    int* rank_of;               // [U][N] scratch: donor rank of each position
    int cluster;                // literal variant: CTAs per unit (1, 2, 4, 8 or 16)
};

// CTAs per unit of the literal repair's selection: the largest power of two that keeps
// all units in one wave of two CTAs per SM, slices of at least 256 positions, at most
// 16.
int select_cluster_size(int U, int N, int sms);

// The count mode's column scales are 1/||k|| times this power of two: one saturated
// fused multiply-add per pair then gives exactly 1 or 0 (see twk_audit.cu).
constexpr float kCountScale = 0x1p32f;

// Largest N the dedup variant accepts: its walk keeps 2 bits per donor in shared memory.
constexpr int kDedupMaxN = 1 << 19;

// prep kernels
cudaError_t launch_round_bf16(const float* in, uint16_t* out, int64_t n, cudaStream_t st);
// NP must be a multiple of 64 (column_stride gives a multiple of 256).
// rscale: a power of two that multiplies every colrinv (1 except for the count mode)
// unit_kk (zeroed by the caller, or null): receives each unit's largest k.k.
cudaError_t launch_norms_identity(const uint16_t* keys, int U, int N, int d, int64_t NP,
                                  float* colrinv, int* colpos, float4* norms, cudaStream_t st,
                                  float rscale = 1.0f, unsigned* unit_kk = nullptr);
cudaError_t launch_scan(const uint8_t* mask, int U, int N, int* cnt, int* kb, cudaStream_t st);
cudaError_t launch_gather(const uint16_t* keys, const uint8_t* mask, const int* cnt,
                          const int* kb, int U, int N, int d, int64_t NP, uint16_t* kp,
                          float* colrinv, int* colpos, float4* norms, unsigned* unit_kk,
                          cudaStream_t st);
// colrinv of every unit times 2^-e_u, 2^e_u the smallest power of two >= the unit's
// largest ||k|| (unit_kk as written by the kernels above), so that the audit's scaled
// similarities lie in [-1, 1] (argmax mode; not for the count mode's scales).
cudaError_t launch_scale_columns(float* colrinv, int U, int64_t NP, const unsigned* unit_kk,
                                 cudaStream_t st);

// exact similarity of the chosen twins
// norms[r] = {k.k hi, k.k lo, 1/||k|| hi, 1/||k|| lo} (double-float pairs) per key, as
// written by the prep kernels.
// b0 = sim(i, twin0); with twin1 given (the evicted-segment winner), twin1 is
// overwritten with the overall winner and b1 (nullable) receives its similarity.
cudaError_t launch_refine(const uint16_t* keys, int U, int N, int d, const float4* norms,
                          const int* twin0, int* twin1, double* b0, double* b1,
                          cudaStream_t st,
                          bool beside_audit = false);

// audit kernel (tensor maps built by the caller)
size_t audit_smem_bytes(int d);
// kArgmax: max/argmax (Eq. 1, Eq. 4); kCount: redundancy counts (Eq. 2); kSymmetric:
// max/argmax from the upper-triangle tiles only, into a.slots
cudaError_t launch_audit(int d, AuditMode mode, const CUtensorMap& tmA, const CUtensorMap& tmB,
                         const AuditArgs& a, int grid, cudaStream_t st);
// slots [n] (as the symmetric audit leaves them) -> twin positions, -1 for an empty slot
cudaError_t launch_slots_to_twins(const unsigned long long* slots, int64_t n, int* twin,
                                  cudaStream_t st);

// standalone policy selection (Sec. 3.2, Eq. 3): per unit, keep budget[u] positions
// ordered by (protected first, count ascending, position ascending)
cudaError_t launch_policy_select(const int* count, int U, int N, const int* budget, int n_sink,
                                 int n_recent, uint8_t* out_mask, int* out_status,
                                 cudaStream_t st);

// repair kernel
cudaError_t launch_repair(const RepairArgs& a, cudaStream_t st);

// wait probe (exercises the bounded-wait give-up path)
cudaError_t launch_wait_probe(int* err, unsigned long long timeout_ns, cudaStream_t st);

}  // namespace twk
