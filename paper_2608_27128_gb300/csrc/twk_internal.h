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
constexpr int kHalf = kBN / 2; // columns per epilogue warpgroup

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
    const float* rowrinv;       // [U][rowrinv_stride]  1/||k_i|| per row
    int64_t rowrinv_stride;
    const int* cnt;             // [U][N]  retained positions before p (repair mode)
    const int* kb;              // [U]     |S0| (repair mode)
    float* out_b0;              // [U][N]  segment-0 best (b_ret, or b_all in mode 0)
    int* out_t0;                // nullable
    float* out_ball;            // [U][N]  repair mode, nullable
    int* out_tall;              // nullable
    int* err;
    unsigned long long timeout_ns;
};

struct RepairArgs {
    int U, N;
    const float* b;             // [U][N] b_i(S0)
    const uint8_t* mask;        // [U][N]
    const int* budget;          // [U] or null
    float tau;
    int n_sink, n_recent;
    uint8_t* out_mask;          // [U][N]
    int* out_swaps;             // [U][N/2][2]
    int* out_nswaps;            // [U]
    int* out_status;            // [U] or null
    uint32_t* keys0;            // [U][N] sort buffers (ping-pong)
    int* idx0;
    uint32_t* keys1;
    int* idx1;
};

// prep kernels
cudaError_t launch_round_bf16(const float* in, uint16_t* out, int64_t n, cudaStream_t st);
cudaError_t launch_norms_identity(const uint16_t* keys, int U, int N, int d, int64_t NP,
                                  float* colrinv, int* colpos, cudaStream_t st);
cudaError_t launch_scan(const uint8_t* mask, int U, int N, int* cnt, int* kb, cudaStream_t st);
cudaError_t launch_gather(const uint16_t* keys, const uint8_t* mask, const int* cnt,
                          const int* kb, int U, int N, int d, int64_t NP, uint16_t* kp,
                          float* colrinv, int* colpos, float* rowrinv, cudaStream_t st);

// audit kernel (tensor maps built by the caller)
size_t audit_smem_bytes(int d);
cudaError_t launch_audit(int d, const CUtensorMap& tmA, const CUtensorMap& tmB,
                         const AuditArgs& a, int grid, cudaStream_t st);

// repair kernel
cudaError_t launch_repair(const RepairArgs& a, cudaStream_t st);

// wait probe (exercises the bounded-wait give-up path)
cudaError_t launch_wait_probe(int* err, unsigned long long timeout_ns, cudaStream_t st);

}  // namespace twk
