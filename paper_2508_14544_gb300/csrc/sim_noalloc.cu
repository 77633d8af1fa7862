// sim_run_noalloc: the whole simulation (staging + simulation kernels) for callers that cannot
// allocate device memory.
//
// Some callers cannot call cudaMalloc: a serving process that reserved all of the GPU's memory
// for its own pool at start-up (a cudaMalloc would fail or fragment that reservation), or a
// latency-sensitive loop that must not make the implicitly synchronising allocation calls
// (cudaFree waits for the whole device).  For them this entry point takes caller-owned inputs
// and outputs and keeps everything else -- the staged request records, the per-instance
// constants, the work counter, the queue buffers and the per-warp workspaces -- in one
// file-scope __device__ array of fixed size.  It calls no cudaMalloc, cudaFree or other
// allocating routine.
//
// The array is reserved on every GPU that loads the library, until the process exits.  All calls
// on a device share it and it keeps the last call's contents, so two calls whose work overlaps on
// the GPU (different streams, or different host threads) race on it; calls on one stream are
// ordered by the stream and are safe.  The work counter, the only part that must start at zero,
// is cleared by every call; everything else is fully rewritten before it is read.
#include <cuda_runtime.h>

#include <algorithm>
#include <mutex>

#include "sim.h"
#include "sim_internal.h"

namespace simgb {
void set_global_error(const char *msg);
}

namespace {

// Limits of the fixed scratch array (the entry point rejects larger inputs with SIM_E_INVAL).
constexpr int64_t kNaMaxInstances = 16384;        // instances per call
constexpr int64_t kNaMaxTotal = int64_t(1) << 18;  // requests per call (262,144)
constexpr int64_t kNaMaxPerInstance = 2048;       // requests per instance
constexpr int kNaWarpsPerBlock = 4;
constexpr int kNaBlocks = 32;
constexpr int64_t kNaSlots = int64_t(kNaBlocks) * kNaWarpsPerBlock;  // simulating warps
constexpr int kNaDeltaCap = simgb::kDcap;

constexpr size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

// Workspace bytes per warp for an active-set capacity of kNaMaxPerInstance (same formula as the
// simulation kernel's carve: 6 x ca + 2 x (ca + 4) int32, 16-byte aligned, then the delta queue
// and the main-queue head cache, and the int32 scratch of the window and the merge histogram).
// A run-time check compares it with the kernel's own size.
constexpr size_t ws_bytes_max() {
    size_t b = size_t(6) * kNaMaxPerInstance * 4 + size_t(2) * (kNaMaxPerInstance + 4) * 4;
    b = (b + 15) & ~size_t(15);
    b += size_t(kNaDeltaCap + 64) * sizeof(simgb::QEnt) + size_t(kNaDeltaCap + 4 + 68) * 4;
    return (b + 15) & ~size_t(15);
}

constexpr size_t kOffOff = 0;
constexpr size_t kOffRec = align256(kOffOff + size_t(kNaMaxInstances + 1) * sizeof(int64_t));
constexpr size_t kOffRecA = align256(kOffRec + size_t(kNaMaxTotal) * sizeof(simgb::QEnt));
constexpr size_t kOffInfo = align256(kOffRecA + size_t(kNaMaxTotal) * sizeof(int32_t));
constexpr size_t kOffCounter = align256(kOffInfo + size_t(kNaMaxInstances) * sizeof(simgb::InstInfo));
constexpr size_t kOffMain = align256(kOffCounter + 256);
constexpr size_t kOffWs = align256(kOffMain + size_t(kNaSlots) * 2 * kNaMaxPerInstance * sizeof(simgb::QEnt));
constexpr size_t kScratchBytes = align256(kOffWs + size_t(kNaSlots) * ws_bytes_max());  // about 23 MB

static __device__ __align__(256) unsigned char g_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
unsigned char *g_dev_ptr[kMaxDevices] = {};

int fail(int code, const char *msg) {
    simgb::set_global_error(msg);
    return code;
}

}  // namespace

extern "C" int sim_run_noalloc(int policy, int64_t M, int32_t n_instances, const int64_t *offsets,
                               const int32_t *arrival_t, const int32_t *prompt_s, const int32_t *lower_l,
                               const int32_t *upper_u, const int32_t *true_o, sim_result *results,
                               void *cuda_stream) {
    if (policy < SIM_AMAX || policy > SIM_HSF) return fail(SIM_E_INVAL, "sim_run_noalloc: bad policy");
    if (M < 1 || M > simgb::kMaxM) return fail(SIM_E_INVAL, "sim_run_noalloc: M outside [1, 2^26]");
    if (n_instances < 1 || n_instances > kNaMaxInstances)
        return fail(SIM_E_INVAL, "sim_run_noalloc: n_instances must be in [1, 16384]");
    if (!offsets || !results) return fail(SIM_E_INVAL, "sim_run_noalloc: NULL offsets or results");
    if (offsets[0] != 0) return fail(SIM_E_INVAL, "sim_run_noalloc: offsets[0] must be 0");
    int64_t n_max = 0;
    for (int32_t i = 0; i < n_instances; ++i) {
        const int64_t d = offsets[i + 1] - offsets[i];
        if (d < 0) return fail(SIM_E_INVAL, "sim_run_noalloc: offsets decrease");
        n_max = std::max(n_max, d);
    }
    const int64_t nt = offsets[n_instances];
    if (n_max > kNaMaxPerInstance)
        return fail(SIM_E_INVAL, "sim_run_noalloc: an instance has more than 2048 requests (the fixed scratch limit)");
    if (nt > kNaMaxTotal)
        return fail(SIM_E_INVAL, "sim_run_noalloc: more than 262144 requests in total (the fixed scratch limit)");
    if (nt > 0 && (!arrival_t || !prompt_s || !lower_l || !upper_u || !true_o))
        return fail(SIM_E_INVAL, "sim_run_noalloc: NULL input array");

    if (simgb::warp_ws_bytes(int(kNaMaxPerInstance)) > ws_bytes_max())
        return fail(SIM_E_STATE, "sim_run_noalloc: workspace layout mismatch");
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess || dev < 0 || dev >= kMaxDevices) return fail(SIM_E_CUDA, "sim_run_noalloc: cudaGetDevice failed");
    unsigned char *base = nullptr;
    {
        // One-time set-up per device, with that device current: the host-side name g_scratch is
        // not a device address, so its device address is looked up once and kept.
        std::lock_guard<std::mutex> lk(g_mu);
        if (!g_dev_ptr[dev]) {
            void *p = nullptr;
            e = cudaGetSymbolAddress(&p, g_scratch);
            if (e != cudaSuccess || !p) return fail(SIM_E_CUDA, "sim_run_noalloc: cudaGetSymbolAddress failed");
            g_dev_ptr[dev] = static_cast<unsigned char *>(p);
        }
        base = g_dev_ptr[dev];
    }
    cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
    int64_t *d_off = reinterpret_cast<int64_t *>(base + kOffOff);
    simgb::QEnt *d_rec = reinterpret_cast<simgb::QEnt *>(base + kOffRec);
    int32_t *d_rec_a = reinterpret_cast<int32_t *>(base + kOffRecA);
    simgb::InstInfo *d_info = reinterpret_cast<simgb::InstInfo *>(base + kOffInfo);
    int32_t *d_counter = reinterpret_cast<int32_t *>(base + kOffCounter);

    e = cudaMemcpyAsync(d_off, offsets, size_t(n_instances + 1) * sizeof(int64_t), cudaMemcpyHostToDevice, st);
    if (e != cudaSuccess) return fail(SIM_E_CUDA, "sim_run_noalloc: copy of the offsets failed");
    simgb::StageParams sp;
    sp.policy = policy;
    sp.M = M;
    sp.n_inst = n_instances;
    sp.n_max = int32_t(n_max);
    sp.max_total = kNaMaxTotal;     // checked again on the device, against the offsets it reads
    sp.max_n = int32_t(kNaMaxPerInstance);
    sp.step_cap = 0;
    sp.off = d_off;
    sp.a = arrival_t;
    sp.s = prompt_s;
    sp.l = lower_l;
    sp.u = upper_u;
    sp.o = true_o;
    sp.rank = nullptr;
    sp.lu = nullptr;
    sp.rec = d_rec;
    sp.rec_a = d_rec_a;
    sp.info = d_info;
    e = simgb::launch_stage(sp, st);
    if (e != cudaSuccess) return fail(SIM_E_CUDA, "sim_run_noalloc: staging kernel launch failed");

    e = cudaMemsetAsync(d_counter, 0, sizeof(int32_t), st);
    if (e != cudaSuccess) return fail(SIM_E_CUDA, "sim_run_noalloc: clearing the work counter failed");
    simgb::RunParams p;
    p.M = M;
    p.n_work = n_instances;
    p.work = nullptr;
    p.counter = d_counter;
    p.rec = d_rec;
    p.rec_a = d_rec_a;
    p.info = d_info;
    p.res = reinterpret_cast<simgb::DevResult *>(results);
    p.completion = nullptr;
    p.lu = nullptr;
    p.tie_seed = nullptr;  // seed 0 for every instance, as sim_run without sim_set_tie_seeds
    p.work_count = nullptr;
    p.batch_time = nullptr;
    p.ca = int32_t(((std::max<int64_t>(n_max, 128) + 127) / 128) * 128);  // >= any active set: no fallback
    p.use_smem = 0;
    p.debug = 0;
    p.evict_index = 0;
    p.gws = base + kOffWs;
    p.gws_stride = int64_t(ws_bytes_max());
    p.mainbuf = reinterpret_cast<simgb::QEnt *>(base + kOffMain);
    p.main_cap = kNaMaxPerInstance;
    const int blocks = int(std::min<int64_t>(kNaBlocks, (n_instances + kNaWarpsPerBlock - 1) / kNaWarpsPerBlock));
    e = simgb::launch_run(policy, p, blocks, kNaWarpsPerBlock, 0, false, st);
    if (e != cudaSuccess) return fail(SIM_E_CUDA, "sim_run_noalloc: simulation kernel launch failed");
    return SIM_OK;
}
