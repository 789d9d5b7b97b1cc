/*
 * twinkv.h -- C ABI of the GB300 (sm_103a) TwinKV key-redundancy audit and repair
 * pass (arXiv 2608.27128, "TwinKV: A Composable Repair Pass for KV Cache Eviction via
 * Pairwise Key Redundancy").
 *
 * Terms, after the paper:
 *   unit        one (layer, KV head); the pass runs on every unit independently
 *               (Sec. 3.1, problem setup).
 *   keys        k_1..k_N of a unit, post-RoPE as stored in the cache (Sec. 3.2).
 *   sim(i,j)    cosine similarity of keys i and j (Sec. 3.2, Eq. 1).
 *   window w    positions with |i-j| <= w never count as twins (Sec. 3.2).
 *   S0          the retained set a wrapped eviction policy produced, K = |S0|
 *               (Sec. 3.4).
 *   b_i(S0)     best surviving twin similarity: max of sim(i,j) over j in S0 with
 *               |i-j| > w, or -1 if no such j (Sec. 3.4, Eq. 4).
 *   b_i(all)    the same maximum over every position j.
 *   orphan      i not in S0 with b_i(S0) < tau (Sec. 3.4).
 *   donor       j in S0, outside the protected sink and recent regions (Sec. 3.2),
 *               with b_j(S0) >= tau (Sec. 3.4).
 *   repair      m = min(|orphans|, |donors|); evict the m donors of largest b,
 *               admit the m orphans of smallest b; |S1| = |S0| (Sec. 3.4).
 *
 * Readings of points the paper leaves open, applied by every call:
 *   - equal similarities: the lowest position j is the twin;
 *   - equal severities: the lower position ranks first, for orphans and donors;
 *   - the k-th donor (by severity) is paired with the k-th orphan in the swap list;
 *   - b is computed once on S0; nothing is recomputed after a swap;
 *   - a key of zero norm has similarity 0 with every key;
 *   - float32 keys are rounded to bf16 (nearest, ties to even) before anything else.
 *
 * Memory.  Every pointer argument except `params` (host) is a DEVICE pointer owned by
 * the caller.  The library allocates nothing: calls that need scratch memory take a
 * caller-owned device `workspace` of at least twinkv_workspace_size() bytes (256-byte
 * aligned).  Tensors are dense, row-major, innermost dimension last:
 *   keys        [L][H][N][d]   bf16 (raw 16-bit patterns) or float32
 *   masks       [L][H][N]      uint8, 0 = evicted, 1 = retained
 *   scores      [L][H][N]      float64 (b values, see "Precision" below)
 *   twins       [L][H][N]      int32 position in 0..N-1, or -1
 *   per-unit    [L*H]          int32
 *   swaps       [L*H][N/2][2]  int32 pairs (evicted donor, admitted orphan); unit u's
 *                              list starts at element u*2*(N/2); twinkv_swaps_capacity()
 *                              gives the total element count
 *
 * Streams.  `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 * Every call only enqueues work on it and returns; outputs are valid once the stream
 * has completed.
 *
 * Per-device state.  The first call on a device records its properties, the device
 * addresses of the library's own device variables (its error word, the fixed scratch
 * of twinkv_repair_select_noalloc) and, for twinkv_repair_host, three streams; they
 * are kept until the process exits.  cudaDeviceReset on a device after the library
 * has been called there is not supported: the recorded addresses would be stale.
 *
 * CUDA graphs.  Once a first call has run on a device outside stream capture, the
 * device-side calls (all but twinkv_repair_host) may be captured in a CUDA graph: they
 * only enqueue kernels and memsets on the given stream, and whatever depends on the
 * data (retained counts, the split of the work, the selection's cut) is computed on the
 * device, so a replay computes on the buffers' contents at replay time.  The captured
 * pointers (inputs, outputs, workspace) must stay valid for the graph's lifetime.
 *
 * Errors.  Argument errors that the host can see (null pointers, sizes, d, dtype,
 * window, threshold, a too-small workspace) are returned at once and nothing is
 * enqueued.  Per-unit data errors are found on the device and reported in
 * out_status[u]: TWINKV_ERR_BUDGET when the popcount of the unit's mask differs from
 * budget[u], TWINKV_ERR_INVALID_ARG when a mask byte is neither 0 nor 1; such a unit
 * gets out_nswaps[u] = -1 and out_mask equal to its input mask.  A device-side wait
 * that gives up (TWINKV_ERR_TIMEOUT) and asynchronous CUDA errors are reported by
 * twinkv_get_last_error().  No call throws, traps or aborts the process.
 *
 * Precision.  The twin of each key is the argmax of fp32 tensor-core similarities
 * (bf16 products, fp32 accumulation), the lowest position on a tie; candidates within
 * about 8e-6 in similarity of the maximum (for a key of its unit's largest norm, more
 * for smaller keys in proportion) count as tied, within each 32-column chunk at
 * d = 128 and across all columns at d = 64, so such a near tie can go to a lower
 * position than the exact argmax.  The band is about 2^-17 * max||k|| / ||k_i|| in
 * similarity (max over the key's unit): keys down to 1/100 of their unit's longest
 * stay well inside a 2e-3 tolerance; at d = 64, keys 1000 times shorter than an outlier
 * key of their unit measured deviations up to 8e-3.  The reported b of that twin is then
 * recomputed as
 * (k_i . k_j) / sqrt((k_i . k_i)(k_j . k_j)) with double-float dot products (relative
 * error ~1e-13) and fp64 rounding, so it is symmetric in (i, j) and exactly 1 for a
 * duplicate; orphan/donor decisions and the severity ranking use these fp64 values.
 *
 * Limits: d in {64, 128}; 1 <= N <= 1048576; L*H <= 65535; L*H*N*d < 2^31 elements
 * per tensor coordinate; L*H*(N rounded up to 256, plus 256) < 2^31 rows.
 */
#ifndef TWINKV_H
#define TWINKV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define TWINKV_ABI_VERSION 1

typedef enum {
    TWINKV_OK = 0,
    TWINKV_ERR_INVALID_ARG = 1,   /* a host-visible argument is wrong, or a mask byte > 1 */
    TWINKV_ERR_UNSUPPORTED = 2,   /* valid request this build does not cover (d, device) */
    TWINKV_ERR_BUDGET = 3,        /* popcount(mask of unit u) != budget[u] */
    TWINKV_ERR_CUDA = 4,          /* a CUDA runtime/driver call failed */
    TWINKV_ERR_TIMEOUT = 5,       /* a device-side wait gave up; outputs are undefined */
    TWINKV_ERR_WORKSPACE = 6,     /* workspace missing, misaligned or too small */
    TWINKV_ERR_TOO_LARGE = 7      /* more than TWINKV_NOALLOC_MAX_POSITIONS positions were
                                     given to twinkv_repair_select_noalloc */
} twinkv_status;

typedef enum { TWINKV_BF16 = 0, TWINKV_F32 = 1 } twinkv_dtype;

/* keys[L][H][N][d] of element type `dtype` (a twinkv_dtype value). */
typedef struct {
    int32_t L, H, N, d;
    int32_t dtype;
} twinkv_shape;

/* Scorer parameters (Sec. 3.2): threshold tau, local window w, protected regions. */
typedef struct {
    float threshold;     /* tau; twinkv_repair's own `threshold` argument overrides it */
    int32_t window;      /* w >= 0 */
    int32_t n_sink;      /* positions i < n_sink are protected (never donors) */
    int32_t n_recent;    /* positions i >= N - n_recent are protected */
} twinkv_params;

/* Operations, for twinkv_workspace_size(). */
typedef enum {
    TWINKV_OP_REDUNDANCY = 0,
    TWINKV_OP_REPAIR = 1,
    TWINKV_OP_REPAIR_SELECT = 2,
    TWINKV_OP_POLICY = 3,
    TWINKV_OP_REPAIR_SELECT_DEDUP = 4,
    TWINKV_OP_REDUNDANCY_SYMMETRIC = 5
} twinkv_op;

/* Kernels, for the profiling hooks. */
typedef enum {
    TWINKV_KERNEL_PREP = 0,      /* bf16 rounding, norms, retained-first column gather */
    TWINKV_KERNEL_AUDIT = 1,     /* fused similarity + masked max/argmax (Eq. 1, Eq. 4) */
    TWINKV_KERNEL_REPAIR = 2,    /* classify, rank, select and swap (Sec. 3.4); the
                                    standalone policy's selection (Sec. 3.2, Eq. 3) */
    TWINKV_KERNEL_REFINE = 3,    /* exact value of each chosen twin's similarity (Eq. 1) */
    TWINKV_KERNEL_COUNT = 4
} twinkv_kernel;

/* Paper defaults: tau = 0.85, w = 32, 4 sink and 64 recent positions (Sec. 3.2). */
twinkv_params twinkv_default_params(void);

/* Number of int32 elements out_swaps must hold: L*H*(N/2)*2.  0 on a bad shape. */
size_t twinkv_swaps_capacity(twinkv_shape s);

/* Workspace bytes `op` needs for shape s (0 on a bad shape or op). */
size_t twinkv_workspace_size(twinkv_shape s, int32_t op);

/*
 * Best twin of every key over all other keys (Sec. 3.2, Eq. 1 and the twin window;
 * the maximum b_i(all) behind the redundancy count of Eq. 2: r_i > 0 iff
 * b_i(all) > tau).
 *   keys       [L][H][N][d] device, dtype per s.dtype, 16-byte aligned
 *   window     w >= 0
 *   out_score  [L][H][N] float64: b_i(all), or -1 when no position lies beyond w
 *   out_twin   [L][H][N] int32: its position (lowest on ties), or -1
 */
twinkv_status twinkv_redundancy(const void* keys, twinkv_shape s, int32_t window,
                                double* out_score, int32_t* out_twin, void* workspace,
                                size_t workspace_bytes, void* stream);

/*
 * twinkv_redundancy computed from half the similarity tiles (Sec. 3.5: the audit costs
 * O(n^2 d) per head; Eq. 1 is symmetric, sim(i,j) = sim(j,i)).  Row block rb (rows
 * [128 rb, 128 rb + 128)) computes only the 256-column tiles from the one holding
 * column 128 rb on; each tile's similarities serve both its rows (maxima over its
 * columns) and its columns (maxima over its rows, the candidates of the rows those
 * columns stand for).  The two directions meet per row in a packed (value,
 * position) word combined with atomic maxima: the larger value, the lower position
 * on a tie, with values that agree to 2^-18 relative counting as tied.  Same
 * arguments and outputs as twinkv_redundancy; workspace
 * twinkv_workspace_size(s, TWINKV_OP_REDUNDANCY_SYMMETRIC).  About half the tensor-core
 * work of twinkv_redundancy, but more work per tile after it (the column maxima are
 * reduced across the threads that hold the rows).
 */
twinkv_status twinkv_redundancy_symmetric(const void* keys, twinkv_shape s, int32_t window,
                                          double* out_score, int32_t* out_twin,
                                          void* workspace, size_t workspace_bytes,
                                          void* stream);

/*
 * Audit of a retained set and the budget-exact repair swap (Sec. 3.4, Eq. 4 and the
 * orphan/donor rule), all units in one pass.
 *   keys           [L][H][N][d] device, 16-byte aligned
 *   retained_mask  [L][H][N] uint8, S0
 *   budget         [L*H] int32 expected |S0| per unit, or NULL (no check)
 *   threshold      tau (finite); overrides params->threshold
 *   params         host pointer, or NULL for twinkv_default_params(); its window,
 *                  n_sink and n_recent are used
 *   out_mask       [L][H][N] uint8: S1
 *   out_swaps      [L*H][N/2][2] int32: (evicted donor, admitted orphan), most severe
 *                  first; entries past out_nswaps[u] are left untouched
 *   out_nswaps     [L*H] int32: m, or -1 for a unit with a data error
 *   out_score_ret  [L][H][N] float64 b_i(S0), or NULL
 *   out_twin_ret   [L][H][N] int32 argmax of b_i(S0), or NULL
 *   out_score_all  [L][H][N] float64 b_i(all), or NULL; when both this and
 *                  out_twin_all are NULL the evicted columns are skipped entirely
 *                  (O(N K d) instead of O(N^2 d), Sec. 3.5)
 *   out_twin_all   [L][H][N] int32, or NULL
 *   out_status     [L*H] int32 per-unit twinkv_status, or NULL
 */
twinkv_status twinkv_repair(const void* keys, twinkv_shape s, const uint8_t* retained_mask,
                            const int32_t* budget, float threshold,
                            const twinkv_params* params, uint8_t* out_mask,
                            int32_t* out_swaps, int32_t* out_nswaps, double* out_score_ret,
                            int32_t* out_twin_ret, double* out_score_all,
                            int32_t* out_twin_all, int32_t* out_status, void* workspace,
                            size_t workspace_bytes, void* stream);

/*
 * The classification, ranking and swap of twinkv_repair alone, on caller-supplied
 * b_i(S0) values (Sec. 3.4).  Same arguments and outputs as twinkv_repair; s.d and
 * s.dtype are ignored.  score_ret [L][H][N] float64 device.  Orphans compare
 * b < (double)threshold, donors b >= (double)threshold.
 */
twinkv_status twinkv_repair_select(const double* score_ret, twinkv_shape s,
                                   const uint8_t* retained_mask, const int32_t* budget,
                                   float threshold, const twinkv_params* params,
                                   uint8_t* out_mask, int32_t* out_swaps,
                                   int32_t* out_nswaps, int32_t* out_status,
                                   void* workspace, size_t workspace_bytes, void* stream);

/*
 * twinkv_repair_select for callers that may not allocate device memory: the same
 * classification, ranking and swap, with the same arguments and outputs, but without a
 * workspace argument.  The paper has no counterpart to this entry point; it exists for
 * callers that cannot call cudaMalloc: a plugin inside a serving engine or framework
 * that owns every device allocation through its own memory pool, or a latency-critical
 * loop that cannot afford the device-wide synchronization cudaMalloc and cudaFree may
 * imply.  The sort buffers live in a fixed array of device memory inside this library
 * (about 6 MiB per GPU that loads it, held until the process exits), so:
 *   - L*H*N may be at most TWINKV_NOALLOC_MAX_POSITIONS; larger requests return
 *     TWINKV_ERR_TOO_LARGE and enqueue nothing;
 *   - every call on a device shares that one array: two calls that may run at the
 *     same time on the GPU (for example on different streams without ordering between
 *     them) race and corrupt each other's results; order them on one stream;
 *   - the first call on each device looks up the array's device address (a host-side
 *     setup step, done once per device and kept until the process exits, so
 *     cudaDeviceReset after it is not supported); make that first call before any
 *     stream capture.
 * Nothing is allocated, by this call or on its behalf.
 */
#define TWINKV_NOALLOC_MAX_POSITIONS 262144
twinkv_status twinkv_repair_select_noalloc(const double* score_ret, twinkv_shape s,
                                           const uint8_t* retained_mask, const int32_t* budget,
                                           float threshold, const twinkv_params* params,
                                           uint8_t* out_mask, int32_t* out_swaps,
                                           int32_t* out_nswaps, int32_t* out_status,
                                           void* stream);

/*
 * twinkv_repair on a cache held in host memory (for example a KV cache offloaded to the
 * host): the same audit and swap (Sec. 3.4), with every tensor argument a HOST pointer
 * of the layout above (page-locked memory lets the copies run asynchronously).  The
 * units' keys go to the device in chunks of at most `chunk_units` units (0: the value
 * twinkv_host_default_chunk returns).  Nothing computes while the first chunk copies
 * in and each chunk's compute has to cover the next one's copy, so the chunks grow
 * from one unit by x2.5 (sizes of a whole wave of 128-row blocks or more rounded to
 * the nearest multiple of such a wave) up to `chunk_units`.
 * Per chunk, ordered by events:
 *   - its keys and mask are copied in on a copy stream the library keeps per device;
 *   - its prefix counts, retained-first layout and audit run on `stream`;
 *   - the exact values of its winners run on a second library stream, in blocks that
 *     fit on the SMs beside the next chunk's audit;
 *   - its scores and twins are copied back on a third.
 * Three chunk buffers let chunk c + 1's copy run while chunk c - 1 is still being
 * finished.  One selection over all units follows the last chunk, and S1,
 * the swap lists, counts and statuses are copied back after it.
 *   arena        caller-owned DEVICE memory of twinkv_host_arena_size(s, chunk_units)
 *                bytes, 256-byte aligned: three chunk buffers of keys and three chunk
 *                workspaces, the mask, b and twins of every unit, the outputs and the
 *                selection's workspace.  The library allocates nothing.
 *   out_*        host outputs as in twinkv_repair (out_score_ret .. out_twin_all may be
 *                NULL); valid once `stream` has completed.  Unlike twinkv_repair, the
 *                entries of out_swaps past out_nswaps[u] are overwritten with
 *                unspecified values (the whole swap array is copied back).
 * Calls on one device are ordered after each other's use of the arena.
 */
size_t twinkv_host_arena_size(twinkv_shape s, int32_t chunk_units);
/* The chunk size twinkv_repair_host and twinkv_host_arena_size use for chunk_units = 0
 * on the current device: about L*H / 8 units, rounded to the nearest multiple of
 * sms / gcd(sms, ceil(N / 128)), the number of units whose 128-row blocks fill every
 * SM an equal number of times (so no chunk's audit ends in a partial wave), clamped
 * to [1, L*H]; without a device, L*H / 8 unrounded.  Returns 0 for an invalid shape. */
int32_t twinkv_host_default_chunk(twinkv_shape s);
twinkv_status twinkv_repair_host(const void* keys, twinkv_shape s, const uint8_t* retained_mask,
                                 const int32_t* budget, float threshold,
                                 const twinkv_params* params, uint8_t* out_mask,
                                 int32_t* out_swaps, int32_t* out_nswaps, double* out_score_ret,
                                 int32_t* out_twin_ret, double* out_score_all,
                                 int32_t* out_twin_all, int32_t* out_status,
                                 int32_t chunk_units, void* arena, size_t arena_bytes,
                                 void* stream);

/*
 * twinkv_repair with a donor never evicted together with its twin (Sec. 3.4: a donor
 * is redundant because its twin, the argmax of b_i(S0), holds the same content; the
 * literal rule can still evict both members of a retained twin pair).  Donors are
 * walked in severity order (b descending, position ascending); a donor is skipped when
 * its twin is already being evicted, or when it is the twin of an evicted donor; the
 * walk stops after |O| evictions, so m = the number of evictions <= min(|O|, |D|).  The
 * m most severe orphans are admitted, the k-th evicted donor paired with the k-th
 * orphan.  Arguments, outputs and the workspace (TWINKV_OP_REPAIR) as for
 * twinkv_repair; N must not exceed 524288 (TWINKV_ERR_UNSUPPORTED otherwise: the walk
 * keeps two bits per donor in shared memory).  The walk is sequential per unit, so a
 * unit with many donors takes longer than in twinkv_repair.
 */
twinkv_status twinkv_repair_dedup(const void* keys, twinkv_shape s, const uint8_t* retained_mask,
                                  const int32_t* budget, float threshold,
                                  const twinkv_params* params, uint8_t* out_mask,
                                  int32_t* out_swaps, int32_t* out_nswaps, double* out_score_ret,
                                  int32_t* out_twin_ret, double* out_score_all,
                                  int32_t* out_twin_all, int32_t* out_status, void* workspace,
                                  size_t workspace_bytes, void* stream);

/*
 * The selection of twinkv_repair_dedup alone, on caller-supplied b_i(S0) and twins.
 *   score_ret   [L][H][N] float64 device, b_i(S0)
 *   twin_ret    [L][H][N] int32 device, the position of each b_i(S0)'s argmax (-1 none)
 *   other arguments as for twinkv_repair_select; workspace TWINKV_OP_REPAIR_SELECT_DEDUP
 */
twinkv_status twinkv_repair_select_dedup(const double* score_ret, const int32_t* twin_ret,
                                         twinkv_shape s, const uint8_t* retained_mask,
                                         const int32_t* budget, float threshold,
                                         const twinkv_params* params, uint8_t* out_mask,
                                         int32_t* out_swaps, int32_t* out_nswaps,
                                         int32_t* out_status, void* workspace,
                                         size_t workspace_bytes, void* stream);

/*
 * The standalone TwinKV policy (Sec. 3.2, Eq. 2-3): every key's redundancy count
 *     r_i = #{ j : |i-j| > w, j != i, sim(i,j) > tau }          (Eq. 2, strict)
 * and, per unit, the budget[u] positions with the highest score s_i = -r_i / N (Eq. 3),
 * the sink and recent regions first (they carry the maximum score and tie among
 * themselves), equal scores in position order (lower first).  All units in one pass;
 * the N x N similarities are never stored.
 *   keys        [L][H][N][d] device, dtype per s.dtype, 16-byte aligned
 *   budget      [L*H] int32 device: positions kept per unit, e.g. ceil((1 - rho) N)
 *               (Sec. 3.1); a budget below the protected count keeps the lowest
 *               protected positions
 *   threshold   tau (finite); overrides params->threshold
 *   params      host pointer or NULL (defaults); window, n_sink, n_recent are used
 *   out_mask    [L][H][N] uint8: 1 for a kept position
 *   out_count   [L][H][N] int32: r_i, or NULL (then kept in the workspace)
 *   out_status  [L*H] int32: 0, or TWINKV_ERR_INVALID_ARG where budget[u] is outside
 *               [0, N] (that unit's mask is all 0); or NULL
 * Precision: each pair is decided by one fp32 fused multiply-add on the unrounded
 * product, x_ij * (1/||k_j||) - tau * ||k_i||, x_ij the fp32 tensor-core dot product of
 * the bf16 keys: pairs whose similarity is within about 1e-6 of tau may count
 * differently than in exact arithmetic.
 * Workspace: twinkv_workspace_size(s, TWINKV_OP_POLICY) bytes, 256-byte aligned.
 */
twinkv_status twinkv_policy(const void* keys, twinkv_shape s, const int32_t* budget,
                            float threshold, const twinkv_params* params, uint8_t* out_mask,
                            int32_t* out_count, int32_t* out_status, void* workspace,
                            size_t workspace_bytes, void* stream);

/* Static description of a status code. */
const char* twinkv_status_string(twinkv_status st);

/*
 * Sticky asynchronous error of the current device: synchronizes the device, returns
 * TWINKV_ERR_TIMEOUT if a kernel's wait gave up, TWINKV_ERR_CUDA on a pending CUDA
 * error, else TWINKV_OK, and clears the sticky timeout.
 */
twinkv_status twinkv_get_last_error(void);

/*
 * Upper bound, in nanoseconds, on any single device-side wait of the kernels launched
 * afterwards (default 2e9; at least 1e7, smaller values return TWINKV_ERR_INVALID_ARG
 * and leave the limit unchanged).  A wait that exceeds it makes the kernel record
 * TWINKV_ERR_TIMEOUT, drain the copies and tensor-core operations it already started
 * (waiting at least 0.2 s for them, whatever this limit), release its resources and
 * return.
 */
twinkv_status twinkv_set_wait_timeout_ns(uint64_t ns);

/*
 * Exercises that give-up path: launches one block that takes tensor memory, waits on
 * a barrier nothing will ever complete (bounded by timeout_ns), frees the tensor
 * memory and returns.  Synchronizes the stream and writes the status the kernel
 * recorded (TWINKV_ERR_TIMEOUT expected) to *out (host pointer).
 */
twinkv_status twinkv_wait_probe(uint64_t timeout_ns, int32_t* out, void* stream);

/*
 * Profiling hooks.  Between twinkv_profile_begin() and twinkv_profile_end(), every
 * kernel launch of this library is bracketed by CUDA events on its stream.
 * twinkv_profile_end() synchronizes those events and returns, per twinkv_kernel, the
 * number of launches and their summed device time in milliseconds (arrays of
 * TWINKV_KERNEL_COUNT host elements).
 */
twinkv_status twinkv_profile_begin(void);
twinkv_status twinkv_profile_end(int32_t* launches, double* total_ms);

/* Library build info: ABI version. */
int32_t twinkv_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* TWINKV_H */
