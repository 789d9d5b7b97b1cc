// twk_api.cu -- the C ABI of libtwinkv (declared in include/twinkv.h): argument
// validation, workspace carving, TMA tensor maps and the launch sequence of the
// TwinKV audit and repair pass (arXiv 2608.27128, Sec. 3.2 and 3.4).
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <numeric>
#include <vector>

#include "twinkv.h"
#include "twk_internal.h"

namespace twk {
namespace {

__device__ int g_error_word[4];   // sticky device-side status (see twk_ptx.cuh)
__device__ int g_probe_word[4];   // status written by the wait probe

constexpr int kMaxDevices = 64;
constexpr int64_t kMaxN = 1 << 20;

std::mutex g_mu;
std::mutex g_host_mu;   // orders twinkv_repair_host calls' use of the per-device streams
unsigned long long g_timeout_ns = 2000000000ull;

struct DeviceInfo {
    bool ready = false;
    int sms = 0;
    int cc_major = 0, cc_minor = 0;
    int* err = nullptr;
    int* probe = nullptr;
};
DeviceInfo g_dev[kMaxDevices];

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn g_encode = nullptr;

// ---------------------------------------------------------------- profiling hooks
struct ProfRecord {
    int kernel;
    cudaEvent_t start, stop;
};
bool g_prof_on = false;
std::vector<ProfRecord> g_prof;

struct ProfScope {
    int kernel;
    cudaStream_t st;
    cudaEvent_t start = nullptr, stop = nullptr;
    ProfScope(int k, cudaStream_t s) : kernel(k), st(s)
    {
        if (!g_prof_on) return;
        cudaEventCreate(&start);
        cudaEventCreate(&stop);
        cudaEventRecord(start, st);
    }
    ~ProfScope()
    {
        if (!start) return;
        cudaEventRecord(stop, st);
        std::lock_guard<std::mutex> lk(g_mu);
        g_prof.push_back({kernel, start, stop});
    }
};

// A failed CUDA call maps to TWINKV_ERR_CUDA; with TWINKV_DEBUG set in the environment
// its message also goes to stderr.
twinkv_status cuda_status(cudaError_t e)
{
    if (e == cudaSuccess) return TWINKV_OK;
    if (std::getenv("TWINKV_DEBUG")) std::fprintf(stderr, "twinkv: %s\n", cudaGetErrorString(e));
    return TWINKV_ERR_CUDA;
}

// Current device's cached facts; sets them up on first use (outside stream capture).
twinkv_status device_info(DeviceInfo** out)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
        return TWINKV_ERR_CUDA;
    std::lock_guard<std::mutex> lk(g_mu);
    DeviceInfo& d = g_dev[dev];
    if (!d.ready) {
        if (cudaDeviceGetAttribute(&d.sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&d.cc_major, cudaDevAttrComputeCapabilityMajor, dev) !=
                cudaSuccess ||
            cudaDeviceGetAttribute(&d.cc_minor, cudaDevAttrComputeCapabilityMinor, dev) !=
                cudaSuccess)
            return TWINKV_ERR_CUDA;
        if (cudaGetSymbolAddress(reinterpret_cast<void**>(&d.err), g_error_word) != cudaSuccess ||
            cudaGetSymbolAddress(reinterpret_cast<void**>(&d.probe), g_probe_word) !=
                cudaSuccess)
            return TWINKV_ERR_CUDA;
        if (!g_encode) {
            cudaDriverEntryPointQueryResult q;
            void* fn = nullptr;
            if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000,
                                                 cudaEnableDefault, &q) != cudaSuccess ||
                q != cudaDriverEntryPointSuccess || !fn)
                return TWINKV_ERR_CUDA;
            g_encode = reinterpret_cast<EncodeTiledFn>(fn);
        }
        d.ready = true;
    }
    // The kernels are built for sm_103a only.
    if (d.cc_major != 10 || d.cc_minor != 3) return TWINKV_ERR_UNSUPPORTED;
    *out = &d;
    return TWINKV_OK;
}

// bf16 rows of length d: a 2-D tensor map [rows][d] with 128-byte swizzle and a box of
// 64 elements x box_rows rows.
twinkv_status make_map(CUtensorMap* map, const void* base, int64_t rows, int d, int box_rows)
{
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(rows)};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(d) * 2};
    cuuint32_t box[2] = {64, static_cast<cuuint32_t>(box_rows)};
    cuuint32_t estr[2] = {1, 1};
    const CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base),
                                dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                                CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? TWINKV_OK : TWINKV_ERR_CUDA;
}

// ---------------------------------------------------------------- shapes, workspace
bool shape_ok(const twinkv_shape& s, bool need_d)
{
    if (s.L < 1 || s.H < 1 || s.N < 1 || s.N > kMaxN) return false;
    const int64_t U = static_cast<int64_t>(s.L) * s.H;
    if (U > 65535) return false;                             // units run on grid.y
    if (!need_d) return U * s.N < (1LL << 31);
    if (s.d != 64 && s.d != 128) return false;
    if (s.dtype != TWINKV_BF16 && s.dtype != TWINKV_F32) return false;
    if (U * s.N * s.d >= (1LL << 31)) return false;          // element offsets
    if (U * column_stride(s.N) >= (1LL << 31)) return false; // TMA row coordinates
    return true;
}

size_t up256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

struct Layout {
    size_t keys16 = 0, colrinv = 0, colpos = 0, norm2 = 0, ukk = 0, kp = 0, cnt = 0, kb = 0,
           twin0 = 0, twin1 = 0, bret = 0, k0 = 0, i0 = 0, k1 = 0, i1 = 0, rcount = 0,
           rank = 0, slots = 0;
    size_t total = 0;
};

Layout layout(const twinkv_shape& s, int op)
{
    Layout L;
    size_t off = 0;
    auto take = [&](size_t bytes) {
        const size_t o = off;
        off += up256(bytes);
        return o;
    };
    const size_t U = static_cast<size_t>(s.L) * s.H;
    const size_t N = static_cast<size_t>(s.N);
    if (op == TWINKV_OP_REDUNDANCY || op == TWINKV_OP_REPAIR || op == TWINKV_OP_POLICY ||
        op == TWINKV_OP_REDUNDANCY_SYMMETRIC) {
        const size_t NP = static_cast<size_t>(column_stride(s.N));
        if (s.dtype == TWINKV_F32) L.keys16 = take(U * N * s.d * 2);
        L.colrinv = take(U * NP * 4);
        L.colpos = take(U * NP * 4);
        L.norm2 = take(U * N * 16);
        if (op != TWINKV_OP_POLICY) L.ukk = take(U * 4);   // largest k.k per unit
        if (op == TWINKV_OP_REPAIR) {
            L.kp = take(U * NP * s.d * 2);
            L.cnt = take(U * N * 4);
            L.kb = take(U * 4);
            L.twin0 = take(U * N * 4);
            L.twin1 = take(U * N * 4);
            L.bret = take(U * N * 8);
        }
    }
    if (op == TWINKV_OP_POLICY) L.rcount = take(U * N * 4);
    if (op == TWINKV_OP_REDUNDANCY_SYMMETRIC) L.slots = take(U * N * 8);
    if (op == TWINKV_OP_REPAIR || op == TWINKV_OP_REPAIR_SELECT ||
        op == TWINKV_OP_REPAIR_SELECT_DEDUP) {
        L.k0 = take(U * N * 8);
        L.i0 = take(U * N * 4);
        L.k1 = take(U * N * 8);
        L.i1 = take(U * N * 4);
        if (op != TWINKV_OP_REPAIR_SELECT) L.rank = take(U * N * 4);   // dedup's rank table
    }
    L.total = off;
    return L;
}

template <typename T>
T* at(void* ws, size_t off)
{
    return reinterpret_cast<T*>(static_cast<char*>(ws) + off);
}

twinkv_status check_ws(const twinkv_shape& s, int op, void* ws, size_t bytes, Layout* out)
{
    *out = layout(s, op);
    if (out->total == 0) return TWINKV_OK;
    if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255) != 0 || bytes < out->total)
        return TWINKV_ERR_WORKSPACE;
    return TWINKV_OK;
}

// bf16 view of the keys (rounding float32 keys into the workspace first).
twinkv_status keys_bf16(const void* keys, const twinkv_shape& s, void* ws, const Layout& L,
                        cudaStream_t st, const uint16_t** out)
{
    if (s.dtype == TWINKV_BF16) {
        *out = static_cast<const uint16_t*>(keys);
        return TWINKV_OK;
    }
    uint16_t* k16 = at<uint16_t>(ws, L.keys16);
    ProfScope p(TWINKV_KERNEL_PREP, st);
    const int64_t n = static_cast<int64_t>(s.L) * s.H * s.N * s.d;
    const cudaError_t e = launch_round_bf16(static_cast<const float*>(keys), k16, n, st);
    *out = k16;
    return cuda_status(e);
}

twinkv_status run_audit(const DeviceInfo& dev, const twinkv_shape& s, const uint16_t* keys16,
                        const void* bkeys, int64_t b_rows, AuditArgs a, cudaStream_t st,
                        AuditMode mode = AuditMode::kArgmax)
{
    CUtensorMap tmA, tmB;
    const int64_t U = static_cast<int64_t>(s.L) * s.H;
    twinkv_status r = make_map(&tmA, keys16, U * s.N, s.d, kBM);
    if (r != TWINKV_OK) return r;
    r = make_map(&tmB, bkeys, b_rows, s.d, kBN);
    if (r != TWINKV_OK) return r;
    const int64_t items = U * a.RB;
    const int grid = static_cast<int>(items < dev.sms ? items : dev.sms);
    ProfScope p(TWINKV_KERNEL_AUDIT, st);
    return cuda_status(launch_audit(s.d, mode, tmA, tmB, a, grid, st));
}

twinkv_status params_ok(const twinkv_params& p, float threshold)
{
    if (!std::isfinite(threshold)) return TWINKV_ERR_INVALID_ARG;
    if (p.window < 0 || p.n_sink < 0 || p.n_recent < 0) return TWINKV_ERR_INVALID_ARG;
    return TWINKV_OK;
}

twinkv_status launch_select(const twinkv_shape& s, const double* b, const uint8_t* mask,
                            const int32_t* budget, float threshold, const twinkv_params& p,
                            uint8_t* out_mask, int32_t* out_swaps, int32_t* out_nswaps,
                            int32_t* out_status, void* ws, const Layout& L, cudaStream_t st,
                            const DeviceInfo* dev, const int32_t* twin = nullptr)
{
    RepairArgs r;
    r.U = s.L * s.H;
    r.N = s.N;
    r.b = b;
    r.mask = mask;
    r.budget = budget;
    r.tau = static_cast<double>(threshold);
    r.n_sink = p.n_sink;
    r.n_recent = p.n_recent;
    r.out_mask = out_mask;
    r.out_swaps = out_swaps;
    r.out_nswaps = out_nswaps;
    r.out_status = out_status;
    r.keys0 = at<uint64_t>(ws, L.k0);
    r.idx0 = at<int>(ws, L.i0);
    r.keys1 = at<uint64_t>(ws, L.k1);
    r.idx1 = at<int>(ws, L.i1);
    r.twin = twin;
    r.rank_of = twin ? at<int>(ws, L.rank) : nullptr;
    r.cluster = select_cluster_size(r.U, r.N, dev ? dev->sms : 0);
    if (const char* f = std::getenv("TWINKV_SELECT_CLUSTER")) {
        // test hook: force the cluster size of the literal selection (1, 2, 4, 8, 16)
        const int c = std::atoi(f);
        if (c == 1 || c == 2 || c == 4 || c == 8 || c == 16) r.cluster = c;
    }
    if (twin && s.N > kDedupMaxN) return TWINKV_ERR_UNSUPPORTED;
    ProfScope prof(TWINKV_KERNEL_REPAIR, st);
    return cuda_status(launch_repair(r, st));
}

twinkv_status run_refine(const uint16_t* k16, const twinkv_shape& s, const float4* norm2,
                         const int* t0, int* t1, double* b0, double* b1, cudaStream_t st,
                         bool beside_audit = false)
{
    ProfScope p(TWINKV_KERNEL_REFINE, st);
    return cuda_status(
        launch_refine(k16, s.L * s.H, s.N, s.d, norm2, t0, t1, b0, b1, st, beside_audit));
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

// ---- host-buffer pipeline (twinkv_repair_host) ------------------------------------
// The number of units whose 128-row blocks fill `sms` SMs an equal number of times.
int wave_units(const twinkv_shape& s, int sms)
{
    const int rb = (s.N + kBM - 1) / kBM;
    return sms > 0 ? sms / std::gcd(sms, rb) : 0;
}

// Units per chunk of the host path when the caller passes 0: about an eighth of the
// units, so that later chunks' copies hide behind earlier chunks' compute, rounded to
// the nearest multiple of the unit count whose row blocks are a whole number of waves
// over the SMs (the persistent audit then ends no launch in a partial wave).
int default_chunk_units(const twinkv_shape& s)
{
    const int U = s.L * s.H;
    int uc = (U + 7) / 8;
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) == cudaSuccess &&
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess &&
        sms > 0) {
        const int step = wave_units(s, sms);
        if (step <= U) uc = std::max(step, (uc + step / 2) / step * step);
    }
    return std::max(1, std::min(uc, U));
}

// Chunk buffers of the host path: with three, chunk c + 1's copy waits only for chunk
// c - 2's exact values, so it runs well ahead of the audit that needs it.
constexpr int kChunkBufs = 3;

struct HostArena {
    // keys and audit-stage workspaces: kChunkBufs chunk buffers each; every other array
    // covers all units
    size_t keys = 0, mask = 0, budget = 0, bret = 0, tret = 0, sall = 0, tall = 0, omask = 0,
           oswaps = 0, onswaps = 0, ostatus = 0;
    size_t key_buf = 0;                // bytes of one keys chunk buffer
    size_t ws = 0, ws_bytes = 0;       // workspaces of one chunk, ws_bytes apart
    size_t sel = 0, sel_bytes = 0;     // selection workspace over all units
    size_t total = 0;
};

HostArena host_arena(const twinkv_shape& s, int uc)
{
    HostArena A;
    size_t off = 0;
    auto take = [&](size_t bytes) {
        const size_t o = off;
        off += up256(bytes);
        return o;
    };
    const size_t N = static_cast<size_t>(s.N), U = static_cast<size_t>(s.L) * s.H;
    const size_t esize = s.dtype == TWINKV_F32 ? 4 : 2;
    A.key_buf = up256(static_cast<size_t>(uc) * N * s.d * esize);
    A.keys = take(kChunkBufs * A.key_buf);
    A.mask = take(U * N);
    A.budget = take(U * 4);
    A.bret = take(U * N * 8);
    A.tret = take(U * N * 4);
    A.sall = take(U * N * 8);
    A.tall = take(U * N * 4);
    A.omask = take(U * N);
    A.oswaps = take(U * (N / 2) * 2 * 4);
    A.onswaps = take(U * 4);
    A.ostatus = take(U * 4);
    twinkv_shape sc = s;
    sc.L = 1;
    sc.H = uc;
    A.ws_bytes = up256(layout(sc, TWINKV_OP_REPAIR).total);
    A.ws = take(kChunkBufs * A.ws_bytes);
    A.sel_bytes = layout(s, TWINKV_OP_REPAIR_SELECT).total;
    A.sel = take(A.sel_bytes);
    A.total = off;
    return A;
}

struct HostStreams {
    bool ready = false;
    cudaStream_t h2d = nullptr, post = nullptr, d2h = nullptr;   // copies in; refine; copies out
    cudaEvent_t in[kChunkBufs], aud[kChunkBufs], done[kChunkBufs], sel, fin;
};
HostStreams g_hs[kMaxDevices];

twinkv_status host_streams(HostStreams** out)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
        return TWINKV_ERR_CUDA;
    HostStreams& h = g_hs[dev];
    if (!h.ready) {
        if (cudaStreamCreateWithFlags(&h.h2d, cudaStreamNonBlocking) != cudaSuccess ||
            cudaStreamCreateWithFlags(&h.d2h, cudaStreamNonBlocking) != cudaSuccess ||
            cudaStreamCreateWithFlags(&h.post, cudaStreamNonBlocking) != cudaSuccess)
            return TWINKV_ERR_CUDA;
        for (int b = 0; b < kChunkBufs; ++b)
            if (cudaEventCreateWithFlags(&h.in[b], cudaEventDisableTiming) != cudaSuccess ||
                cudaEventCreateWithFlags(&h.aud[b], cudaEventDisableTiming) != cudaSuccess ||
                cudaEventCreateWithFlags(&h.done[b], cudaEventDisableTiming) != cudaSuccess)
                return TWINKV_ERR_CUDA;
        if (cudaEventCreateWithFlags(&h.sel, cudaEventDisableTiming) != cudaSuccess ||
            cudaEventCreateWithFlags(&h.fin, cudaEventDisableTiming) != cudaSuccess)
            return TWINKV_ERR_CUDA;
        h.ready = true;
    }
    *out = &h;
    return TWINKV_OK;
}

// ---- fixed device scratch for twinkv_repair_select_noalloc ------------------------
// The selection's sort buffers (two 8-byte keys and two 4-byte positions per position,
// each buffer rounded up to 256 bytes) for up to TWINKV_NOALLOC_MAX_POSITIONS positions.
// On the host, g_noalloc_scratch only names the symbol; its device address is looked
// up per device with cudaGetSymbolAddress.
constexpr size_t kNoAllocBytes = 24u * TWINKV_NOALLOC_MAX_POSITIONS + 4u * 256u;
__device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocBytes];
void* g_noalloc_ptr[kMaxDevices];

// Device address of g_noalloc_scratch on the current device (looked up on first use).
twinkv_status noalloc_scratch(void** out)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
        return TWINKV_ERR_CUDA;
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_noalloc_ptr[dev]) {
        void* p = nullptr;
        const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess || !p) return cuda_status(e == cudaSuccess ? cudaErrorUnknown : e);
        g_noalloc_ptr[dev] = p;
    }
    *out = g_noalloc_ptr[dev];
    return TWINKV_OK;
}

}  // namespace
}  // namespace twk

using namespace twk;

extern "C" {

int32_t twinkv_abi_version(void) { return TWINKV_ABI_VERSION; }

twinkv_params twinkv_default_params(void)
{
    twinkv_params p;
    p.threshold = 0.85f;
    p.window = 32;
    p.n_sink = 4;
    p.n_recent = 64;
    return p;
}

size_t twinkv_swaps_capacity(twinkv_shape s)
{
    if (!shape_ok(s, false)) return 0;
    return static_cast<size_t>(s.L) * s.H * static_cast<size_t>(s.N / 2) * 2;
}

size_t twinkv_workspace_size(twinkv_shape s, int32_t op)
{
    if (op < TWINKV_OP_REDUNDANCY || op > TWINKV_OP_REDUNDANCY_SYMMETRIC) return 0;
    if (!shape_ok(s, op != TWINKV_OP_REPAIR_SELECT && op != TWINKV_OP_REPAIR_SELECT_DEDUP))
        return 0;
    return layout(s, op).total;
}

const char* twinkv_status_string(twinkv_status st)
{
    switch (st) {
    case TWINKV_OK: return "ok";
    case TWINKV_ERR_INVALID_ARG: return "invalid argument";
    case TWINKV_ERR_UNSUPPORTED: return "unsupported (needs an sm_103 GPU; d in {64, 128})";
    case TWINKV_ERR_BUDGET: return "retained count differs from the budget";
    case TWINKV_ERR_CUDA: return "CUDA error";
    case TWINKV_ERR_TIMEOUT: return "a device-side wait timed out";
    case TWINKV_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
    case TWINKV_ERR_TOO_LARGE:
        return "L*H*N exceeds TWINKV_NOALLOC_MAX_POSITIONS (the fixed scratch of "
               "twinkv_repair_select_noalloc)";
    }
    return "unknown status";
}

twinkv_status twinkv_set_wait_timeout_ns(uint64_t ns)
{
    if (ns < kMinWaitLimitNs) return TWINKV_ERR_INVALID_ARG;
    std::lock_guard<std::mutex> lk(g_mu);
    g_timeout_ns = ns;
    return TWINKV_OK;
}

twinkv_status twinkv_get_last_error(void)
{
    DeviceInfo* dev = nullptr;
    const twinkv_status r = device_info(&dev);
    if (r != TWINKV_OK) return r;
    const cudaError_t sync = cudaDeviceSynchronize();
    const cudaError_t last = cudaGetLastError();
    if (sync != cudaSuccess || last != cudaSuccess) return TWINKV_ERR_CUDA;
    int word[4];
    if (cudaMemcpyFromSymbol(word, g_error_word, sizeof word) != cudaSuccess)
        return TWINKV_ERR_CUDA;
    if (word[0] != 0) {
        const int zero[4] = {0, 0, 0, 0};
        cudaMemcpyToSymbol(g_error_word, zero, sizeof zero);
        return static_cast<twinkv_status>(word[0]);
    }
    return TWINKV_OK;
}

twinkv_status twinkv_wait_probe(uint64_t timeout_ns, int32_t* out, void* stream)
{
    if (!out || timeout_ns == 0) return TWINKV_ERR_INVALID_ARG;
    DeviceInfo* dev = nullptr;
    twinkv_status r = device_info(&dev);
    if (r != TWINKV_OK) return r;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (cudaMemsetAsync(dev->probe, 0, 4 * sizeof(int), st) != cudaSuccess) return TWINKV_ERR_CUDA;
    if (launch_wait_probe(dev->probe, timeout_ns, st) != cudaSuccess) return TWINKV_ERR_CUDA;
    int word[4];
    if (cudaMemcpyAsync(word, dev->probe, sizeof word, cudaMemcpyDeviceToHost, st) != cudaSuccess ||
        cudaStreamSynchronize(st) != cudaSuccess)
        return TWINKV_ERR_CUDA;
    *out = word[0];
    return TWINKV_OK;
}

twinkv_status twinkv_profile_begin(void)
{
    std::lock_guard<std::mutex> lk(g_mu);
    for (auto& r : g_prof) {
        cudaEventDestroy(r.start);
        cudaEventDestroy(r.stop);
    }
    g_prof.clear();
    g_prof_on = true;
    return TWINKV_OK;
}

twinkv_status twinkv_profile_end(int32_t* launches, double* total_ms)
{
    std::vector<ProfRecord> recs;
    {
        std::lock_guard<std::mutex> lk(g_mu);
        g_prof_on = false;
        recs.swap(g_prof);
    }
    twinkv_status st = TWINKV_OK;
    for (int k = 0; k < TWINKV_KERNEL_COUNT; ++k) {
        if (launches) launches[k] = 0;
        if (total_ms) total_ms[k] = 0.0;
    }
    for (auto& r : recs) {
        float ms = 0.f;
        if (cudaEventSynchronize(r.stop) != cudaSuccess ||
            cudaEventElapsedTime(&ms, r.start, r.stop) != cudaSuccess)
            st = TWINKV_ERR_CUDA;
        if (launches) launches[r.kernel] += 1;
        if (total_ms) total_ms[r.kernel] += ms;
        cudaEventDestroy(r.start);
        cudaEventDestroy(r.stop);
    }
    return st;
}

}  // extern "C"

namespace {
twinkv_status redundancy_impl(const void* keys, twinkv_shape s, int32_t window, double* out_score,
                              int32_t* out_twin, void* workspace, size_t workspace_bytes,
                              void* stream, bool symmetric)
{
    if (!keys || !aligned16(keys) || !out_score || !out_twin || window < 0 || !shape_ok(s, true))
        return TWINKV_ERR_INVALID_ARG;
    const int op = symmetric ? TWINKV_OP_REDUNDANCY_SYMMETRIC : TWINKV_OP_REDUNDANCY;
    Layout L;
    twinkv_status r = check_ws(s, op, workspace, workspace_bytes, &L);
    if (r != TWINKV_OK) return r;
    DeviceInfo* dev = nullptr;
    if ((r = device_info(&dev)) != TWINKV_OK) return r;
    cudaStream_t st = static_cast<cudaStream_t>(stream);

    const uint16_t* k16 = nullptr;
    if ((r = keys_bf16(keys, s, workspace, L, st, &k16)) != TWINKV_OK) return r;
    const int U = s.L * s.H;
    const int64_t NP = column_stride(s.N);
    float* colrinv = at<float>(workspace, L.colrinv);
    int* colpos = at<int>(workspace, L.colpos);
    float4* norm2 = at<float4>(workspace, L.norm2);
    unsigned long long* slots = symmetric ? at<unsigned long long>(workspace, L.slots) : nullptr;
    {
        ProfScope p(TWINKV_KERNEL_PREP, st);
        unsigned* ukk = at<unsigned>(workspace, L.ukk);
        if (cudaMemsetAsync(ukk, 0, static_cast<size_t>(U) * 4, st) != cudaSuccess ||
            launch_norms_identity(k16, U, s.N, s.d, NP, colrinv, colpos, norm2, st, 1.0f, ukk) !=
                cudaSuccess ||
            launch_scale_columns(colrinv, U, NP, ukk, st) != cudaSuccess ||
            (symmetric && cudaMemsetAsync(slots, 0, static_cast<size_t>(U) * s.N * 8, st) !=
                              cudaSuccess))
            return TWINKV_ERR_CUDA;
    }
    AuditArgs a;
    std::memset(&a, 0, sizeof a);
    a.U = U;
    a.N = s.N;
    a.NP = static_cast<int>(NP);
    a.RB = (s.N + kBM - 1) / kBM;
    a.window = window < s.N ? window : s.N;
    a.repair_mode = 0;
    a.need_all = 0;
    a.b_rows_per_unit = s.N;
    a.colrinv = colrinv;
    a.colpos = colpos;
    a.out_t0 = out_twin;
    a.slots = slots;
    a.err = dev->err;
    a.timeout_ns = g_timeout_ns;
    a.mant_mask = 0xFFFFFFE0u;
    if ((r = run_audit(*dev, s, k16, k16, static_cast<int64_t>(U) * s.N, a, st,
                       symmetric ? AuditMode::kSymmetric : AuditMode::kArgmax)) != TWINKV_OK)
        return r;
    if (symmetric) {
        ProfScope p(TWINKV_KERNEL_REFINE, st);   // post-processing of the audit's slots
        if (launch_slots_to_twins(slots, static_cast<int64_t>(U) * s.N, out_twin, st) !=
            cudaSuccess)
            return TWINKV_ERR_CUDA;
    }
    return run_refine(k16, s, norm2, out_twin, nullptr, out_score, nullptr, st);
}
}  // namespace

extern "C" {

twinkv_status twinkv_redundancy(const void* keys, twinkv_shape s, int32_t window,
                                double* out_score, int32_t* out_twin, void* workspace,
                                size_t workspace_bytes, void* stream)
{
    return redundancy_impl(keys, s, window, out_score, out_twin, workspace, workspace_bytes,
                           stream, false);
}

twinkv_status twinkv_redundancy_symmetric(const void* keys, twinkv_shape s, int32_t window,
                                          double* out_score, int32_t* out_twin, void* workspace,
                                          size_t workspace_bytes, void* stream)
{
    return redundancy_impl(keys, s, window, out_score, out_twin, workspace, workspace_bytes,
                           stream, true);
}

twinkv_status twinkv_policy(const void* keys, twinkv_shape s, const int32_t* budget,
                            float threshold, const twinkv_params* params, uint8_t* out_mask,
                            int32_t* out_count, int32_t* out_status, void* workspace,
                            size_t workspace_bytes, void* stream)
{
    const twinkv_params p = params ? *params : twinkv_default_params();
    if (!keys || !aligned16(keys) || !budget || !out_mask || !shape_ok(s, true))
        return TWINKV_ERR_INVALID_ARG;
    twinkv_status r = params_ok(p, threshold);
    if (r != TWINKV_OK) return r;
    Layout L;
    if ((r = check_ws(s, TWINKV_OP_POLICY, workspace, workspace_bytes, &L)) != TWINKV_OK) return r;
    DeviceInfo* dev = nullptr;
    if ((r = device_info(&dev)) != TWINKV_OK) return r;
    cudaStream_t st = static_cast<cudaStream_t>(stream);

    const uint16_t* k16 = nullptr;
    if ((r = keys_bf16(keys, s, workspace, L, st, &k16)) != TWINKV_OK) return r;
    const int U = s.L * s.H;
    const int64_t NP = column_stride(s.N);
    float* colrinv = at<float>(workspace, L.colrinv);
    int* colpos = at<int>(workspace, L.colpos);
    float4* norm2 = at<float4>(workspace, L.norm2);
    int* count = out_count ? out_count : at<int>(workspace, L.rcount);
    {
        ProfScope pr(TWINKV_KERNEL_PREP, st);
        if (launch_norms_identity(k16, U, s.N, s.d, NP, colrinv, colpos, norm2, st,
                                  kCountScale) !=
            cudaSuccess)
            return TWINKV_ERR_CUDA;
    }
    AuditArgs a;
    std::memset(&a, 0, sizeof a);
    a.U = U;
    a.N = s.N;
    a.NP = static_cast<int>(NP);
    a.RB = (s.N + kBM - 1) / kBM;
    a.window = p.window < s.N ? p.window : s.N;
    a.repair_mode = 0;
    a.need_all = 0;
    a.b_rows_per_unit = s.N;
    a.colrinv = colrinv;
    a.colpos = colpos;
    a.err = dev->err;
    a.timeout_ns = g_timeout_ns;
    a.mant_mask = 0xFFFFFFE0u;
    a.count_tau = threshold;
    a.out_count = count;
    if ((r = run_audit(*dev, s, k16, k16, static_cast<int64_t>(U) * s.N, a, st,
                       AuditMode::kCount)) != TWINKV_OK)
        return r;
    ProfScope pr(TWINKV_KERNEL_REPAIR, st);
    return cuda_status(launch_policy_select(count, U, s.N, budget, p.n_sink, p.n_recent,
                                            out_mask, out_status, st));
}

}  // extern "C"

namespace {
// The audit stages of the repair for one set of units: bf16 keys, retained-first
// gather, audit, exact values.  Writes b_i(S0) to bret and its twin's position to t0;
// b_i(all) and its twin to out_score_all / out_twin_all when either is given.
// The audit's inputs in `workspace`: bf16 keys (fp32 keys are rounded), the retained
// prefix counts, and the retained-first column layout with its metadata and the norm
// records.  *k16 receives the bf16 keys.
twinkv_status prep_stages(const void* keys, const twinkv_shape& s, const uint8_t* retained_mask,
                          void* workspace, const Layout& L, cudaStream_t st,
                          const uint16_t** k16)
{
    twinkv_status r;
    if ((r = keys_bf16(keys, s, workspace, L, st, k16)) != TWINKV_OK) return r;
    const int U = s.L * s.H;
    const int64_t NP = column_stride(s.N);
    {
        ProfScope pr(TWINKV_KERNEL_PREP, st);
        if (launch_scan(retained_mask, U, s.N, at<int>(workspace, L.cnt),
                        at<int>(workspace, L.kb), st) != cudaSuccess)
            return TWINKV_ERR_CUDA;
    }
    ProfScope pr(TWINKV_KERNEL_PREP, st);
    unsigned* ukk = at<unsigned>(workspace, L.ukk);
    if (cudaMemsetAsync(ukk, 0, static_cast<size_t>(U) * 4, st) != cudaSuccess ||
        launch_gather(*k16, retained_mask, at<int>(workspace, L.cnt), at<int>(workspace, L.kb),
                      U, s.N, s.d, NP, at<uint16_t>(workspace, L.kp),
                      at<float>(workspace, L.colrinv), at<int>(workspace, L.colpos),
                      at<float4>(workspace, L.norm2), ukk, st) != cudaSuccess ||
        launch_scale_columns(at<float>(workspace, L.colrinv), U, NP, ukk, st) != cudaSuccess)
        return TWINKV_ERR_CUDA;
    return TWINKV_OK;
}

// The audit (Eq. 4 and b_i(all)) and the exact value of each winner, on the inputs
// prep_stages left in `workspace`.  With refine_st given, the exact values run there
// after the audit (ordered by audit_done), in blocks that fit beside the next audit.
twinkv_status main_stages(const DeviceInfo* dev, const uint16_t* k16, const twinkv_shape& s,
                          const twinkv_params& p, double* bret, int* t0, double* out_score_all,
                          int32_t* out_twin_all, void* workspace, const Layout& L,
                          cudaStream_t st, cudaStream_t refine_st = nullptr,
                          cudaEvent_t audit_done = nullptr)
{
    twinkv_status r;
    const int U = s.L * s.H;
    const int64_t NP = column_stride(s.N);
    float* colrinv = at<float>(workspace, L.colrinv);
    int* colpos = at<int>(workspace, L.colpos);
    float4* norm2 = at<float4>(workspace, L.norm2);
    uint16_t* kp = at<uint16_t>(workspace, L.kp);
    int* cnt = at<int>(workspace, L.cnt);
    int* kb = at<int>(workspace, L.kb);
    const bool need_all = out_score_all || out_twin_all;
    int* t1 = need_all ? (out_twin_all ? out_twin_all : at<int>(workspace, L.twin1)) : nullptr;
    AuditArgs a;
    std::memset(&a, 0, sizeof a);
    a.U = U;
    a.N = s.N;
    a.NP = static_cast<int>(NP);
    a.RB = (s.N + kBM - 1) / kBM;
    a.window = p.window < s.N ? p.window : s.N;
    a.repair_mode = 1;
    a.need_all = need_all ? 1 : 0;
    a.b_rows_per_unit = NP;
    a.colrinv = colrinv;
    a.colpos = colpos;
    a.cnt = cnt;
    a.kb = kb;
    a.out_t0 = t0;
    a.out_t1 = t1;
    a.err = dev->err;
    a.timeout_ns = g_timeout_ns;
    a.mant_mask = 0xFFFFFFE0u;
    if ((r = run_audit(*dev, s, k16, kp, static_cast<int64_t>(U) * NP, a, st)) != TWINKV_OK)
        return r;
    if (!refine_st) return run_refine(k16, s, norm2, t0, t1, bret, out_score_all, st);
    if (cudaEventRecord(audit_done, st) != cudaSuccess ||
        cudaStreamWaitEvent(refine_st, audit_done, 0) != cudaSuccess)
        return TWINKV_ERR_CUDA;
    return run_refine(k16, s, norm2, t0, t1, bret, out_score_all, refine_st, true);
}

twinkv_status audit_stages(const DeviceInfo* dev, const void* keys, const twinkv_shape& s,
                           const uint8_t* retained_mask, const twinkv_params& p, double* bret,
                           int* t0, double* out_score_all, int32_t* out_twin_all,
                           void* workspace, const Layout& L, cudaStream_t st)
{
    const uint16_t* k16 = nullptr;
    const twinkv_status r = prep_stages(keys, s, retained_mask, workspace, L, st, &k16);
    if (r != TWINKV_OK) return r;
    return main_stages(dev, k16, s, p, bret, t0, out_score_all, out_twin_all, workspace, L, st);
}

twinkv_status repair_impl(const void* keys, twinkv_shape s, const uint8_t* retained_mask,
                          const int32_t* budget, float threshold, const twinkv_params* params,
                          uint8_t* out_mask, int32_t* out_swaps, int32_t* out_nswaps,
                          double* out_score_ret, int32_t* out_twin_ret, double* out_score_all,
                          int32_t* out_twin_all, int32_t* out_status, void* workspace,
                          size_t workspace_bytes, void* stream, bool dedup)
{
    const twinkv_params p = params ? *params : twinkv_default_params();
    if (!keys || !aligned16(keys) || !retained_mask || !out_mask || !out_nswaps ||
        !shape_ok(s, true) || (!out_swaps && s.N >= 2))   // with N < 2 no swap fits
        return TWINKV_ERR_INVALID_ARG;
    twinkv_status r = params_ok(p, threshold);
    if (r != TWINKV_OK) return r;
    Layout L;
    if ((r = check_ws(s, TWINKV_OP_REPAIR, workspace, workspace_bytes, &L)) != TWINKV_OK) return r;
    DeviceInfo* dev = nullptr;
    if ((r = device_info(&dev)) != TWINKV_OK) return r;
    cudaStream_t st = static_cast<cudaStream_t>(stream);

    int* t0 = out_twin_ret ? out_twin_ret : at<int>(workspace, L.twin0);
    double* bret = out_score_ret ? out_score_ret : at<double>(workspace, L.bret);
    if ((r = audit_stages(dev, keys, s, retained_mask, p, bret, t0, out_score_all,
                          out_twin_all, workspace, L, st)) != TWINKV_OK)
        return r;
    return launch_select(s, bret, retained_mask, budget, threshold, p, out_mask, out_swaps,
                         out_nswaps, out_status, workspace, L, st, dev, dedup ? t0 : nullptr);
}
}  // namespace

extern "C" {

twinkv_status twinkv_repair(const void* keys, twinkv_shape s, const uint8_t* retained_mask,
                            const int32_t* budget, float threshold, const twinkv_params* params,
                            uint8_t* out_mask, int32_t* out_swaps, int32_t* out_nswaps,
                            double* out_score_ret, int32_t* out_twin_ret, double* out_score_all,
                            int32_t* out_twin_all, int32_t* out_status, void* workspace,
                            size_t workspace_bytes, void* stream)
{
    return repair_impl(keys, s, retained_mask, budget, threshold, params, out_mask, out_swaps,
                       out_nswaps, out_score_ret, out_twin_ret, out_score_all, out_twin_all,
                       out_status, workspace, workspace_bytes, stream, false);
}

twinkv_status twinkv_repair_dedup(const void* keys, twinkv_shape s, const uint8_t* retained_mask,
                                  const int32_t* budget, float threshold,
                                  const twinkv_params* params, uint8_t* out_mask,
                                  int32_t* out_swaps, int32_t* out_nswaps, double* out_score_ret,
                                  int32_t* out_twin_ret, double* out_score_all,
                                  int32_t* out_twin_all, int32_t* out_status, void* workspace,
                                  size_t workspace_bytes, void* stream)
{
    return repair_impl(keys, s, retained_mask, budget, threshold, params, out_mask, out_swaps,
                       out_nswaps, out_score_ret, out_twin_ret, out_score_all, out_twin_all,
                       out_status, workspace, workspace_bytes, stream, true);
}

twinkv_status twinkv_repair_select_dedup(const double* score_ret, const int32_t* twin_ret,
                                         twinkv_shape s, const uint8_t* retained_mask,
                                         const int32_t* budget, float threshold,
                                         const twinkv_params* params, uint8_t* out_mask,
                                         int32_t* out_swaps, int32_t* out_nswaps,
                                         int32_t* out_status, void* workspace,
                                         size_t workspace_bytes, void* stream)
{
    const twinkv_params p = params ? *params : twinkv_default_params();
    if (!score_ret || !twin_ret || !retained_mask || !out_mask || !out_nswaps ||
        !shape_ok(s, false) || (!out_swaps && s.N >= 2))
        return TWINKV_ERR_INVALID_ARG;
    twinkv_status r = params_ok(p, threshold);
    if (r != TWINKV_OK) return r;
    Layout L;
    if ((r = check_ws(s, TWINKV_OP_REPAIR_SELECT_DEDUP, workspace, workspace_bytes, &L)) !=
        TWINKV_OK)
        return r;
    DeviceInfo* dev = nullptr;
    if ((r = device_info(&dev)) != TWINKV_OK) return r;
    return launch_select(s, score_ret, retained_mask, budget, threshold, p, out_mask, out_swaps,
                         out_nswaps, out_status, workspace, L, static_cast<cudaStream_t>(stream),
                         dev, twin_ret);
}

twinkv_status twinkv_repair_select(const double* score_ret, twinkv_shape s,
                                   const uint8_t* retained_mask, const int32_t* budget,
                                   float threshold, const twinkv_params* params,
                                   uint8_t* out_mask, int32_t* out_swaps, int32_t* out_nswaps,
                                   int32_t* out_status, void* workspace, size_t workspace_bytes,
                                   void* stream)
{
    const twinkv_params p = params ? *params : twinkv_default_params();
    if (!score_ret || !retained_mask || !out_mask || !out_nswaps || !shape_ok(s, false) ||
        (!out_swaps && s.N >= 2))
        return TWINKV_ERR_INVALID_ARG;
    twinkv_status r = params_ok(p, threshold);
    if (r != TWINKV_OK) return r;
    Layout L;
    if ((r = check_ws(s, TWINKV_OP_REPAIR_SELECT, workspace, workspace_bytes, &L)) != TWINKV_OK)
        return r;
    DeviceInfo* dev = nullptr;
    if ((r = device_info(&dev)) != TWINKV_OK) return r;
    return launch_select(s, score_ret, retained_mask, budget, threshold, p, out_mask, out_swaps,
                         out_nswaps, out_status, workspace, L, static_cast<cudaStream_t>(stream),
                         dev);
}

twinkv_status twinkv_repair_select_noalloc(const double* score_ret, twinkv_shape s,
                                           const uint8_t* retained_mask, const int32_t* budget,
                                           float threshold, const twinkv_params* params,
                                           uint8_t* out_mask, int32_t* out_swaps,
                                           int32_t* out_nswaps, int32_t* out_status,
                                           void* stream)
{
    const twinkv_params p = params ? *params : twinkv_default_params();
    if (!score_ret || !retained_mask || !out_mask || !out_nswaps || !shape_ok(s, false) ||
        (!out_swaps && s.N >= 2))
        return TWINKV_ERR_INVALID_ARG;
    twinkv_status r = params_ok(p, threshold);
    if (r != TWINKV_OK) return r;
    if (static_cast<int64_t>(s.L) * s.H * s.N > TWINKV_NOALLOC_MAX_POSITIONS)
        return TWINKV_ERR_TOO_LARGE;
    const Layout L = layout(s, TWINKV_OP_REPAIR_SELECT);
    if (L.total > kNoAllocBytes) return TWINKV_ERR_TOO_LARGE;
    DeviceInfo* dev = nullptr;
    if ((r = device_info(&dev)) != TWINKV_OK) return r;
    void* scratch = nullptr;
    if ((r = noalloc_scratch(&scratch)) != TWINKV_OK) return r;
    // The sort buffers are fully written before they are read: nothing needs clearing.
    return launch_select(s, score_ret, retained_mask, budget, threshold, p, out_mask, out_swaps,
                         out_nswaps, out_status, scratch, L, static_cast<cudaStream_t>(stream),
                         dev);
}

int32_t twinkv_host_default_chunk(twinkv_shape s)
{
    return shape_ok(s, true) ? default_chunk_units(s) : 0;
}

size_t twinkv_host_arena_size(twinkv_shape s, int32_t chunk_units)
{
    if (!shape_ok(s, true) || chunk_units < 0) return 0;
    const int U = s.L * s.H;
    const int uc = chunk_units == 0 ? default_chunk_units(s) : (chunk_units < U ? chunk_units : U);
    return host_arena(s, uc).total;
}

twinkv_status twinkv_repair_host(const void* keys, twinkv_shape s, const uint8_t* retained_mask,
                                 const int32_t* budget, float threshold,
                                 const twinkv_params* params, uint8_t* out_mask,
                                 int32_t* out_swaps, int32_t* out_nswaps, double* out_score_ret,
                                 int32_t* out_twin_ret, double* out_score_all,
                                 int32_t* out_twin_all, int32_t* out_status,
                                 int32_t chunk_units, void* arena, size_t arena_bytes,
                                 void* stream)
{
    const twinkv_params p = params ? *params : twinkv_default_params();
    if (!keys || !retained_mask || !out_mask || !out_nswaps || !shape_ok(s, true) ||
        (!out_swaps && s.N >= 2) || chunk_units < 0)
        return TWINKV_ERR_INVALID_ARG;
    twinkv_status r = params_ok(p, threshold);
    if (r != TWINKV_OK) return r;
    const int U = s.L * s.H;
    const int uc = chunk_units == 0 ? default_chunk_units(s) : (chunk_units < U ? chunk_units : U);
    const HostArena A = host_arena(s, uc);
    if (!arena || (reinterpret_cast<uintptr_t>(arena) & 255) != 0 || arena_bytes < A.total)
        return TWINKV_ERR_WORKSPACE;
    DeviceInfo* dev = nullptr;
    if ((r = device_info(&dev)) != TWINKV_OK) return r;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    std::lock_guard<std::mutex> call_lk(g_host_mu);
    HostStreams* hs = nullptr;
    if ((r = host_streams(&hs)) != TWINKV_OK) return r;

    char* base = static_cast<char*>(arena);
    const size_t N = static_cast<size_t>(s.N);
    const size_t esize = s.dtype == TWINKV_F32 ? 4 : 2;
    auto ck = [&](cudaError_t e) { return e == cudaSuccess; };
    // An error after work was enqueued: hs->fin is made to follow everything already
    // queued on the three library streams and on `stream`, so that the next call, which
    // waits on hs->fin before it reuses the arena, cannot overlap that work.  If even
    // that fails, the streams are synchronized.
    auto fail = [&](twinkv_status e) {
        cudaStream_t q[3] = {hs->h2d, hs->post, st};
        bool ok = true;
        for (cudaStream_t x : q)
            ok = ok && ck(cudaEventRecord(hs->sel, x)) && ck(cudaStreamWaitEvent(hs->d2h, hs->sel, 0));
        ok = ok && ck(cudaEventRecord(hs->fin, hs->d2h));
        if (!ok) {
            cudaStreamSynchronize(hs->h2d);
            cudaStreamSynchronize(hs->post);
            cudaStreamSynchronize(hs->d2h);
            cudaStreamSynchronize(st);
        }
        return e;
    };
    uint8_t* d_mask = reinterpret_cast<uint8_t*>(base + A.mask);
    int32_t* d_budget = budget ? reinterpret_cast<int32_t*>(base + A.budget) : nullptr;
    double* d_bret = reinterpret_cast<double*>(base + A.bret);
    int32_t* d_tret = reinterpret_cast<int32_t*>(base + A.tret);
    double* d_sall = reinterpret_cast<double*>(base + A.sall);
    int32_t* d_tall = reinterpret_cast<int32_t*>(base + A.tall);
    const bool need_all = out_score_all || out_twin_all;
    // A previous call's copies and selection finish before this call reuses the arena.
    if (!ck(cudaStreamWaitEvent(hs->h2d, hs->fin, 0)) || !ck(cudaStreamWaitEvent(st, hs->fin, 0)))
        return fail(TWINKV_ERR_CUDA);
    if (budget && !ck(cudaMemcpyAsync(d_budget, budget, U * 4, cudaMemcpyHostToDevice, hs->h2d)))
        return fail(TWINKV_ERR_CUDA);
    // Nothing computes while the first chunk copies in, and each chunk's compute has to
    // cover the next chunk's copy: the chunks grow from one unit by x2.5 (the audit of a
    // unit takes about three times the copy of its keys) up to uc.  A size of one wave
    // of units (wave_units) or more is rounded to the nearest whole number of waves.
    const int step = wave_units(s, dev->sms);
    auto next_size = [&](int prev) {
        int n = prev <= 0 ? 1 : std::max(prev + 1, (5 * prev + 1) / 2);
        if (n >= step && step > 0) n = std::max(step, (n + step / 2) / step * step);
        return std::min(n, uc);
    };
    int want = 0, last = 0;
    size_t u0 = 0;
    for (int c = 0; u0 < static_cast<size_t>(U); ++c) {
        const int b = c % kChunkBufs;
        want = next_size(want);
        const int un = static_cast<int>(U - u0 < static_cast<size_t>(want) ? U - u0 : want);
        char* kbuf = base + A.keys + b * A.key_buf;
        // inputs, once the audit and refine that last used this buffer pair are done
        if (c >= kChunkBufs && !ck(cudaStreamWaitEvent(hs->h2d, hs->done[b], 0)))
            return fail(TWINKV_ERR_CUDA);
        if (!ck(cudaMemcpyAsync(kbuf, static_cast<const char*>(keys) + u0 * N * s.d * esize,
                                un * N * s.d * esize, cudaMemcpyHostToDevice, hs->h2d)) ||
            !ck(cudaMemcpyAsync(d_mask + u0 * N, retained_mask + u0 * N, un * N,
                                cudaMemcpyHostToDevice, hs->h2d)) ||
            !ck(cudaEventRecord(hs->in[b], hs->h2d)) ||
            !ck(cudaStreamWaitEvent(st, hs->in[b], 0)))
            return fail(TWINKV_ERR_CUDA);
        // Prefix counts, retained-first layout and audit of this chunk on `stream`, into
        // this buffer's workspace and the all-unit arrays; the exact values on the
        // refine stream, beside the next chunk's audit.
        twinkv_shape sc = s;
        sc.L = 1;
        sc.H = un;
        const Layout Lc = layout(sc, TWINKV_OP_REPAIR);
        char* wsb = base + A.ws + b * A.ws_bytes;
        const uint16_t* k16 = nullptr;
        if ((r = prep_stages(kbuf, sc, d_mask + u0 * N, wsb, Lc, st, &k16)) != TWINKV_OK)
            return fail(r);
        r = main_stages(dev, k16, sc, p, d_bret + u0 * N, d_tret + u0 * N,
                        need_all ? d_sall + u0 * N : nullptr, need_all ? d_tall + u0 * N : nullptr,
                        wsb, Lc, st, hs->post, hs->aud[b]);
        if (r != TWINKV_OK) return fail(r);
        if (!ck(cudaEventRecord(hs->done[b], hs->post))) return fail(TWINKV_ERR_CUDA);
        last = b;
        // this chunk's scores and twins go back while later chunks run
        if (!ck(cudaStreamWaitEvent(hs->d2h, hs->done[b], 0))) return fail(TWINKV_ERR_CUDA);
        auto d2h = [&](void* dst, const void* src, size_t bytes) {
            return ck(cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDeviceToHost, hs->d2h));
        };
        if ((out_score_ret && !d2h(out_score_ret + u0 * N, d_bret + u0 * N, un * N * 8)) ||
            (out_twin_ret && !d2h(out_twin_ret + u0 * N, d_tret + u0 * N, un * N * 4)) ||
            (out_score_all && !d2h(out_score_all + u0 * N, d_sall + u0 * N, un * N * 8)) ||
            (out_twin_all && !d2h(out_twin_all + u0 * N, d_tall + u0 * N, un * N * 4)))
            return fail(TWINKV_ERR_CUDA);
        u0 += un;
    }
    // one selection over every unit (Sec. 3.4), after every chunk's exact values (the
    // refine stream runs them in order), then its results go back
    if (!ck(cudaStreamWaitEvent(st, hs->done[last], 0))) return fail(TWINKV_ERR_CUDA);
    const Layout Lsel = layout(s, TWINKV_OP_REPAIR_SELECT);
    uint8_t* d_omask = reinterpret_cast<uint8_t*>(base + A.omask);
    int32_t* d_oswaps = reinterpret_cast<int32_t*>(base + A.oswaps);
    int32_t* d_onswaps = reinterpret_cast<int32_t*>(base + A.onswaps);
    int32_t* d_ostatus = reinterpret_cast<int32_t*>(base + A.ostatus);
    if ((r = launch_select(s, d_bret, d_mask, d_budget, threshold, p, d_omask, d_oswaps,
                           d_onswaps, d_ostatus, base + A.sel, Lsel, st, dev)) != TWINKV_OK)
        return fail(r);
    if (!ck(cudaEventRecord(hs->sel, st)) || !ck(cudaStreamWaitEvent(hs->d2h, hs->sel, 0)))
        return fail(TWINKV_ERR_CUDA);
    const size_t swaps_bytes = static_cast<size_t>(U) * (N / 2) * 2 * 4;
    if (!ck(cudaMemcpyAsync(out_mask, d_omask, U * N, cudaMemcpyDeviceToHost, hs->d2h)) ||
        (out_swaps && swaps_bytes &&
         !ck(cudaMemcpyAsync(out_swaps, d_oswaps, swaps_bytes, cudaMemcpyDeviceToHost, hs->d2h))) ||
        !ck(cudaMemcpyAsync(out_nswaps, d_onswaps, U * 4, cudaMemcpyDeviceToHost, hs->d2h)) ||
        (out_status &&
         !ck(cudaMemcpyAsync(out_status, d_ostatus, U * 4, cudaMemcpyDeviceToHost, hs->d2h))) ||
        !ck(cudaEventRecord(hs->fin, hs->d2h)))
        return fail(TWINKV_ERR_CUDA);
    // The caller's stream completes only after the results reached the host.
    if (!ck(cudaStreamWaitEvent(st, hs->fin, 0))) return TWINKV_ERR_CUDA;
    return TWINKV_OK;
}

}  // extern "C"
