// C ABI of the batched scheduler simulator (declared in include/sim.h).
//
// Host side only: argument checks, device buffers owned by the context, launches of the staging
// and simulation kernels (sim_kernels.cu), and the capacity fallback (instances whose active set
// outgrows the shared-memory workspace are re-run with a global-memory workspace).
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <new>
#include <string>
#include <vector>

#include "sim.h"
#include "sim_internal.h"

using simgb::DevResult;
using simgb::InstInfo;
using simgb::QEnt;

struct sim_ctx {
    int policy = 0;
    int64_t M = 0;
    int32_t n_inst = 0;
    // options
    int64_t step_cap = 0;
    int record_completions = 0;
    int wpb = 4;
    bool wpb_set = false;  // SIM_OPT_WARPS_PER_BLOCK given by the caller
    int warps_per_sm = 0;
    int debug_checks = 0;
    int tune_residency = 0;
    int dense = 0;  // SIM_OPT_DENSE_RESIDENCY
    int evict_index = 0;
    int count_work = 0;
    int batch_time = 0;
    // residency chosen by SIM_OPT_TUNE_RESIDENCY for the load shape tuned_shape (n_inst, n_total,
    // n_max): warps per SM, or 0 for the default; tuned_shape[0] < 0 when not tuned
    int tuned_wps = 0;
    int tuned_dense = 0;
    int64_t tuned_shape[3] = {-1, -1, -1};
    int smem_ca = simgb::kSmemCaDefault;
    // state
    int device = -1;
    bool loaded = false;
    bool ran = false;
    bool comp_valid = false;
    int64_t n_total = 0;
    int32_t n_max = 0;
    // device buffers
    int64_t *d_off = nullptr;
    int32_t *d_raw = nullptr;  // 6 * cap_total: a, s, l, u, o, rank
    int2 *d_lu = nullptr;      // A_ell: (l, u) per request, cap_total
    int64_t cap_total = 0;
    QEnt *d_rec = nullptr;
    int32_t *d_rec_a = nullptr;
    InstInfo *d_info = nullptr;
    DevResult *d_res = nullptr;
    int64_t *d_comp = nullptr;
    int32_t *d_counter = nullptr;
    int32_t *d_work = nullptr;
    unsigned char *d_gws = nullptr;
    size_t gws_bytes = 0;
    QEnt *d_main = nullptr;
    size_t main_bytes = 0;
    double *d_cr = nullptr;
    uint64_t *d_seed = nullptr;          // A_min tie seeds (n_inst), null until sim_set_tie_seeds
    int64_t *d_wc = nullptr;             // work counters, 4 per instance (SIM_OPT_COUNT_WORK)
    bool wc_valid = false;
    int64_t *d_bt = nullptr;             // batch-time sums, 6 per instance (SIM_OPT_BATCH_TIME)
    double *d_btout = nullptr;           // 2 per instance
    bool bt_valid = false;
    cudaStream_t load_stream = nullptr;  // non-blocking stream of sim_load (independent of other threads' work)
    int64_t *h_off = nullptr;            // pinned copy of the offsets (n_inst + 1) for their upload
    int64_t launches = 0;
    std::vector<DevResult> h_res;
    std::string err;
};

static_assert(sizeof(sim_result) == 56, "sim_result must be 56 bytes");
static_assert(sizeof(DevResult) == sizeof(sim_result), "device result layout");

namespace {

thread_local std::string g_create_err;

int fail(sim_ctx *c, int code, const char *fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    if (c) c->err = buf; else g_create_err = buf;
    return code;
}

int cuda_fail(sim_ctx *c, cudaError_t e, const char *what) {
    return fail(c, SIM_E_CUDA, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

template <typename T>
void dfree(T *&p) {
    if (p) cudaFree(p);
    p = nullptr;
}

template <typename T>
cudaError_t dalloc(T *&p, size_t bytes) {
    dfree(p);
    if (bytes == 0) bytes = 16;
    void *q = nullptr;
    cudaError_t e = cudaMalloc(&q, bytes);
    if (e == cudaSuccess) p = static_cast<T *>(q);
    return e;
}

int check_device(sim_ctx *c) {
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(c, e, "cudaGetDevice");
    if (c->device >= 0 && dev != c->device)
        return fail(c, SIM_E_STATE, "current device %d differs from the device %d the data was loaded on", dev,
                    c->device);
    c->device = dev;
    return SIM_OK;
}

}  // namespace

namespace simgb {
// Message for sim_last_error(NULL) from entry points that have no context.
void set_global_error(const char *msg) { g_create_err = msg ? msg : ""; }
}  // namespace simgb

extern "C" {

int sim_create(int policy, int64_t M, int32_t n_instances, sim_ctx **out) {
    if (!out) return fail(nullptr, SIM_E_INVAL, "sim_create: out is NULL");
    *out = nullptr;
    if (policy < SIM_AMAX || policy > SIM_AELL) return fail(nullptr, SIM_E_INVAL, "sim_create: bad policy %d", policy);
    if (M < 1 || M > simgb::kMaxM)
        return fail(nullptr, SIM_E_INVAL, "sim_create: M=%lld outside [1, 2^26]", (long long)M);
    if (n_instances < 1) return fail(nullptr, SIM_E_INVAL, "sim_create: n_instances=%d < 1", n_instances);
    sim_ctx *c = new (std::nothrow) sim_ctx();
    if (!c) return fail(nullptr, SIM_E_NOMEM, "sim_create: out of host memory");
    c->policy = policy;
    c->M = M;
    c->n_inst = n_instances;
    g_create_err.clear();
    *out = c;
    return SIM_OK;
}

int sim_set_option(sim_ctx *c, int key, int64_t value) {
    if (!c) return SIM_E_INVAL;
    c->err.clear();
    switch (key) {
        case SIM_OPT_STEP_CAP:
            if (value < 0) return fail(c, SIM_E_INVAL, "STEP_CAP must be >= 0");
            c->step_cap = value;
            if (c->loaded) c->loaded = false;  // the cap is staged with the data: reload required
            return SIM_OK;
        case SIM_OPT_RECORD_COMPLETIONS:
            c->record_completions = value ? 1 : 0;
            return SIM_OK;
        case SIM_OPT_WARPS_PER_BLOCK:
            if (value < 1 || value > 8) return fail(c, SIM_E_INVAL, "WARPS_PER_BLOCK must be in [1, 8]");
            c->wpb = int(value);
            c->wpb_set = true;
            return SIM_OK;
        case SIM_OPT_WARPS_PER_SM:
            if (value < 0 || value > 64) return fail(c, SIM_E_INVAL, "WARPS_PER_SM must be in [0, 64]");
            c->warps_per_sm = int(value);
            return SIM_OK;
        case SIM_OPT_DEBUG_CHECKS:
            c->debug_checks = value ? 1 : 0;
            return SIM_OK;
        case SIM_OPT_TUNE_RESIDENCY:
            c->tune_residency = value ? 1 : 0;
            c->tuned_shape[0] = -1;
            return SIM_OK;
        case SIM_OPT_EVICT_TIES:
            if (value != 0 && value != 1) return fail(c, SIM_E_INVAL, "EVICT_TIES must be 0 (random) or 1 (index)");
            c->evict_index = int(value);
            return SIM_OK;
        case SIM_OPT_DENSE_RESIDENCY:
            c->dense = value ? 1 : 0;
            return SIM_OK;
        case SIM_OPT_COUNT_WORK:
            c->count_work = value ? 1 : 0;
            return SIM_OK;
        case SIM_OPT_BATCH_TIME:
            c->batch_time = value ? 1 : 0;
            return SIM_OK;
        case SIM_OPT_SMEM_ACTIVE_CAP:
            if (value < 128 || value > 4096 || value % 128)
                return fail(c, SIM_E_INVAL, "SMEM_ACTIVE_CAP must be a multiple of 128 in [128, 4096]");
            c->smem_ca = int(value);
            return SIM_OK;
        default:
            return fail(c, SIM_E_INVAL, "unknown option %d", key);
    }
}

static int load_impl(sim_ctx *c, const int64_t *offsets, const int32_t *a, const int32_t *s, const int32_t *l,
                     const int32_t *u, const int32_t *o, const int32_t *rank, int device_ptrs) {
    if (!c) return SIM_E_INVAL;
    c->err.clear();
    c->loaded = false;
    c->ran = false;
    c->comp_valid = false;
    if (!offsets) return fail(c, SIM_E_INVAL, "sim_load: offsets is NULL");
    if (offsets[0] != 0) return fail(c, SIM_E_INVAL, "sim_load: offsets[0] must be 0");
    int64_t n_max = 0;
    for (int32_t i = 0; i < c->n_inst; ++i) {
        const int64_t d = offsets[i + 1] - offsets[i];
        if (d < 0) return fail(c, SIM_E_INVAL, "sim_load: offsets decrease at instance %d", i);
        if (d > INT32_MAX / 2) return fail(c, SIM_E_INVAL, "sim_load: instance %d has too many requests", i);
        n_max = std::max(n_max, d);
    }
    const int64_t nt = offsets[c->n_inst];
    if (nt > 0 && (!a || !s || !l || !u || !o)) return fail(c, SIM_E_INVAL, "sim_load: NULL input array");
    if (c->policy == SIM_AR && nt > 0 && !rank)
        return fail(c, SIM_E_INVAL, "sim_load: A_r needs the permutation ranks (sim_load_ranked_csr)");
    int rc = check_device(c);
    if (rc) return rc;
    cudaError_t e;
    if (nt > c->cap_total || !c->d_raw) {
        const int64_t cap = std::max<int64_t>(nt, 1);
        if ((e = dalloc(c->d_raw, size_t(6) * cap * sizeof(int32_t))) != cudaSuccess ||
            (e = dalloc(c->d_rec, size_t(cap) * sizeof(QEnt))) != cudaSuccess ||
            (e = dalloc(c->d_rec_a, size_t(cap) * sizeof(int32_t))) != cudaSuccess ||
            (c->policy == SIM_AELL && (e = dalloc(c->d_lu, size_t(cap) * sizeof(int2))) != cudaSuccess)) {
            c->cap_total = 0;
            return e == cudaErrorMemoryAllocation ? fail(c, SIM_E_NOMEM, "sim_load: device allocation failed")
                                                  : cuda_fail(c, e, "cudaMalloc");
        }
        dfree(c->d_comp);
        c->cap_total = cap;
    }
    if (!c->d_off) {
        if ((e = dalloc(c->d_off, size_t(c->n_inst + 1) * sizeof(int64_t))) != cudaSuccess ||
            (e = dalloc(c->d_info, size_t(c->n_inst) * sizeof(InstInfo))) != cudaSuccess ||
            (e = dalloc(c->d_res, size_t(c->n_inst) * sizeof(DevResult))) != cudaSuccess ||
            (e = dalloc(c->d_counter, sizeof(int32_t) * 4)) != cudaSuccess ||
            (e = dalloc(c->d_work, size_t(c->n_inst) * sizeof(int32_t))) != cudaSuccess)
            return e == cudaErrorMemoryAllocation ? fail(c, SIM_E_NOMEM, "sim_load: device allocation failed")
                                                  : cuda_fail(c, e, "cudaMalloc");
    }
    if (!c->load_stream && (e = cudaStreamCreateWithFlags(&c->load_stream, cudaStreamNonBlocking)) != cudaSuccess)
        return cuda_fail(c, e, "sim_load: stream creation");
    const cudaStream_t ls = c->load_stream;
    // Device inputs are read in place by the staging kernel (sim_load returns only after it has
    // finished, so the caller may reuse them afterwards); host inputs are copied in first.
    const int32_t *src[6] = {a, s, l, u, o, rank};
    const int nsrc = (c->policy == SIM_AR) ? 6 : 5;
    const int32_t *in[6];
    for (int k = 0; k < 6; ++k) in[k] = c->d_raw + size_t(k) * c->cap_total;
    for (int k = 0; k < nsrc; ++k) {
        if (nt == 0) break;
        if (device_ptrs) {
            in[k] = src[k];
            continue;
        }
        e = cudaMemcpyAsync(c->d_raw + size_t(k) * c->cap_total, src[k], size_t(nt) * sizeof(int32_t),
                            cudaMemcpyHostToDevice, ls);
        if (e != cudaSuccess) return cuda_fail(c, e, "sim_load: copy of the input arrays");
    }
    if (!c->h_off && (e = cudaMallocHost(&c->h_off, size_t(c->n_inst + 1) * sizeof(int64_t))) != cudaSuccess) {
        c->h_off = nullptr;
        return cuda_fail(c, e, "sim_load: pinned offsets buffer");
    }
    std::memcpy(c->h_off, offsets, size_t(c->n_inst + 1) * sizeof(int64_t));
    e = cudaMemcpyAsync(c->d_off, c->h_off, size_t(c->n_inst + 1) * sizeof(int64_t), cudaMemcpyHostToDevice, ls);
    if (e != cudaSuccess) return cuda_fail(c, e, "sim_load: copy of the offsets");
    simgb::StageParams sp;
    sp.policy = c->policy;
    sp.M = c->M;
    sp.n_inst = c->n_inst;
    sp.n_max = int32_t(n_max);
    sp.max_total = c->cap_total;
    sp.max_n = INT32_MAX;
    sp.step_cap = c->step_cap;
    sp.off = c->d_off;
    sp.a = in[0];
    sp.s = in[1];
    sp.l = in[2];
    sp.u = in[3];
    sp.o = in[4];
    sp.rank = in[5];
    sp.lu = c->d_lu;
    sp.rec = c->d_rec;
    sp.rec_a = c->d_rec_a;
    sp.info = c->d_info;
    e = simgb::launch_stage(sp, ls);
    if (e != cudaSuccess) return cuda_fail(c, e, "sim_load: staging kernel launch");
    if (c->n_inst > 0) ++c->launches;
    e = cudaStreamSynchronize(ls);
    if (e != cudaSuccess) return cuda_fail(c, e, "sim_load: staging kernel");
    c->n_total = nt;
    c->n_max = int32_t(n_max);
    c->loaded = true;
    return SIM_OK;
}

int sim_load_csr(sim_ctx *c, const int64_t *offsets, const int32_t *a, const int32_t *s, const int32_t *l,
                 const int32_t *u, const int32_t *o, int device_ptrs) {
    return load_impl(c, offsets, a, s, l, u, o, nullptr, device_ptrs);
}

int sim_load_ranked_csr(sim_ctx *c, const int64_t *offsets, const int32_t *a, const int32_t *s,
                        const int32_t *l, const int32_t *u, const int32_t *o, const int32_t *rank,
                        int device_ptrs) {
    return load_impl(c, offsets, a, s, l, u, o, rank, device_ptrs);
}

int sim_load(sim_ctx *c, int32_t n, const int32_t *a, const int32_t *s, const int32_t *l, const int32_t *u,
             const int32_t *o, int device_ptrs) {
    if (!c) return SIM_E_INVAL;
    if (n < 0) return fail(c, SIM_E_INVAL, "sim_load: n_per_instance=%d < 0", n);
    std::vector<int64_t> off(size_t(c->n_inst) + 1);
    for (int32_t i = 0; i <= c->n_inst; ++i) off[i] = int64_t(i) * n;
    return sim_load_csr(c, off.data(), a, s, l, u, o, device_ptrs);
}

// One launch of the simulation kernel over n_work instances (all, or the device list work_dev).
// smem: the active sets in shared memory (else a global-memory workspace of n_max slots);
// dense: the 12-warps-per-SM configuration (blocks of 4 warps, 384 shared-memory slots); not with
// the instrumented kernel, which keeps its own register budget.
static int run_launch(sim_ctx *c, cudaStream_t st, const int32_t *work_dev, int32_t n_work, bool smem,
                      int warps_per_sm, bool dense = false) {
    cudaError_t e;
    int dev = c->device;
    int n_sm = 0, smem_optin = 0;
    cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev);
    cudaDeviceGetAttribute(&smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    dense = dense && smem && !c->count_work && !c->batch_time;
    int wpb = dense ? simgb::kDenseWarps : c->wpb;
    // no more instances than SMs: one warp per block, so that each instance gets an SM to itself
    // (64 instances of 10^5 requests: 1.5-3.7 % faster than four to a block on 16 SMs)
    if (!dense && !c->wpb_set && n_work <= n_sm) wpb = 1;
    int ca = smem ? (dense ? simgb::kDenseCa : c->smem_ca) : ((std::max(c->n_max, 128) + 127) / 128) * 128;
    size_t per_warp = simgb::warp_ws_bytes(ca);
    size_t smem_bytes = 0;
    if (smem) {
        while (wpb > 1 && per_warp * wpb > size_t(smem_optin)) --wpb;
        if (per_warp * wpb > size_t(smem_optin)) return fail(c, SIM_E_INVAL, "workspace does not fit shared memory");
        smem_bytes = per_warp * wpb;
        e = simgb::set_run_smem_limit(c->policy, smem_bytes);
        if (e != cudaSuccess) return cuda_fail(c, e, "cudaFuncSetAttribute");
    }
    int per_sm = 1;
    if (smem) {
        int smem_sm = 0;
        cudaDeviceGetAttribute(&smem_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev);
        per_sm = std::max(1, int(size_t(smem_sm) / (smem_bytes + 1024)));
        per_sm = std::min(per_sm, dense ? 3 : 64 / wpb);
    } else {
        per_sm = std::max(1, 16 / wpb);
    }
    if (warps_per_sm > 0 && !dense) per_sm = std::max(1, std::min(per_sm, warps_per_sm / wpb));
    int64_t blocks = int64_t(n_sm) * per_sm;
    blocks = std::min<int64_t>(blocks, (n_work + wpb - 1) / wpb);
    blocks = std::max<int64_t>(blocks, 1);
    const int64_t slots = blocks * wpb;
    const int64_t main_cap = std::max<int64_t>(c->n_max, 1);
    const size_t main_need = size_t(slots) * 2 * main_cap * sizeof(QEnt);
    if (main_need > c->main_bytes) {
        if ((e = dalloc(c->d_main, main_need)) != cudaSuccess) {
            c->main_bytes = 0;
            return e == cudaErrorMemoryAllocation ? fail(c, SIM_E_NOMEM, "sim_run: queue buffers") : cuda_fail(c, e, "cudaMalloc");
        }
        c->main_bytes = main_need;
    }
    if (!smem) {
        const size_t need = size_t(slots) * per_warp;
        if (need > c->gws_bytes) {
            if ((e = dalloc(c->d_gws, need)) != cudaSuccess) {
                c->gws_bytes = 0;
                return e == cudaErrorMemoryAllocation ? fail(c, SIM_E_NOMEM, "sim_run: workspace") : cuda_fail(c, e, "cudaMalloc");
            }
            c->gws_bytes = need;
        }
    }
    simgb::RunParams p;
    p.M = c->M;
    p.n_work = n_work;
    p.work = work_dev;
    p.counter = c->d_counter;
    p.rec = c->d_rec;
    p.rec_a = c->d_rec_a;
    p.info = c->d_info;
    p.res = c->d_res;
    p.completion = c->record_completions ? c->d_comp : nullptr;
    p.lu = c->d_lu;
    p.tie_seed = c->d_seed;
    p.work_count = c->count_work ? c->d_wc : nullptr;
    p.batch_time = c->batch_time ? c->d_bt : nullptr;
    p.ca = ca;
    p.use_smem = smem ? 1 : 0;
    p.debug = c->debug_checks;
    p.evict_index = c->evict_index;
    p.gws = c->d_gws;
    p.gws_stride = int64_t(per_warp);
    p.mainbuf = c->d_main;
    p.main_cap = main_cap;
    if ((e = cudaMemsetAsync(c->d_counter, 0, sizeof(int32_t), st)) != cudaSuccess)
        return cuda_fail(c, e, "cudaMemsetAsync");
    e = simgb::launch_run(c->policy, p, int(blocks), wpb, smem_bytes, dense, st);
    if (e != cudaSuccess) return cuda_fail(c, e, "sim_run: kernel launch");
    ++c->launches;
    return SIM_OK;
}

// Simulate every instance (shared-memory kernel, then a global-memory re-run of the instances whose
// active set outgrew it) and copy the results to c->h_res; ms (optional) receives the device time
// of the whole, measured by events on the stream.
static int simulate(sim_ctx *c, cudaStream_t st, int wps, bool dense, float *ms) {
    cudaError_t e;
    cudaEvent_t ev[2] = {nullptr, nullptr};
    if (ms) {
        for (auto &x : ev)
            if ((e = cudaEventCreate(&x)) != cudaSuccess) return cuda_fail(c, e, "cudaEventCreate");
        cudaEventRecord(ev[0], st);
    }
    int rc = run_launch(c, st, nullptr, c->n_inst, !c->debug_checks, wps, dense);
    if (rc == SIM_OK) {
        c->h_res.resize(size_t(c->n_inst));
        e = cudaMemcpyAsync(c->h_res.data(), c->d_res, sizeof(DevResult) * size_t(c->n_inst), cudaMemcpyDeviceToHost,
                            st);
        if (e == cudaSuccess) e = cudaStreamSynchronize(st);
        if (e != cudaSuccess) rc = cuda_fail(c, e, "sim_run: simulation kernel");
    }
    // instances whose active set outgrew the shared-memory workspace: re-run from global memory
    std::vector<int32_t> redo;
    if (rc == SIM_OK)
        for (int32_t i = 0; i < c->n_inst; ++i)
            if (c->h_res[i].status == simgb::kStatusCapacity) redo.push_back(i);
    if (rc == SIM_OK && !redo.empty()) {
        e = cudaMemcpyAsync(c->d_work, redo.data(), redo.size() * sizeof(int32_t), cudaMemcpyHostToDevice, st);
        if (e != cudaSuccess) rc = cuda_fail(c, e, "sim_run: work list");
        if (rc == SIM_OK) rc = run_launch(c, st, c->d_work, int32_t(redo.size()), false, c->warps_per_sm);
        if (rc == SIM_OK) {
            e = cudaMemcpyAsync(c->h_res.data(), c->d_res, sizeof(DevResult) * size_t(c->n_inst),
                                cudaMemcpyDeviceToHost, st);
            if (e == cudaSuccess) e = cudaStreamSynchronize(st);
            if (e != cudaSuccess) rc = cuda_fail(c, e, "sim_run: simulation kernel (global workspace)");
        }
    }
    if (ms) {
        if (rc == SIM_OK) {
            cudaEventRecord(ev[1], st);
            if ((e = cudaEventSynchronize(ev[1])) == cudaSuccess) cudaEventElapsedTime(ms, ev[0], ev[1]);
            else rc = cuda_fail(c, e, "sim_run: residency tuning");
        }
        for (auto &x : ev) cudaEventDestroy(x);
    }
    return rc;
}

int sim_run(sim_ctx *c, sim_result *out, void *stream) {
    if (!c) return SIM_E_INVAL;
    c->err.clear();
    if (!c->loaded) return fail(c, SIM_E_STATE, "sim_run: nothing loaded (call sim_load first)");
    if (!out) return fail(c, SIM_E_INVAL, "sim_run: out is NULL");
    int rc = check_device(c);
    if (rc) return rc;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    cudaError_t e;
    if (c->record_completions) {
        if (!c->d_comp && (e = dalloc(c->d_comp, size_t(c->cap_total) * sizeof(int64_t))) != cudaSuccess)
            return fail(c, SIM_E_NOMEM, "sim_run: completion buffer");
        if ((e = cudaMemsetAsync(c->d_comp, 0, size_t(std::max<int64_t>(c->n_total, 1)) * sizeof(int64_t), st)) !=
            cudaSuccess)
            return cuda_fail(c, e, "cudaMemsetAsync");
    }
    c->wc_valid = false;
    c->bt_valid = false;
    if (c->batch_time && !c->d_bt &&
        (e = dalloc(c->d_bt, size_t(c->n_inst) * 6 * sizeof(int64_t))) != cudaSuccess)
        return fail(c, SIM_E_NOMEM, "sim_run: batch-time buffer");
    if (c->count_work) {
        if (!c->d_wc && (e = dalloc(c->d_wc, size_t(c->n_inst) * 4 * sizeof(int64_t))) != cudaSuccess)
            return fail(c, SIM_E_NOMEM, "sim_run: work-counter buffer");
        if ((e = cudaMemsetAsync(c->d_wc, 0, size_t(c->n_inst) * 4 * sizeof(int64_t), st)) != cudaSuccess)
            return cuda_fail(c, e, "cudaMemsetAsync");
    }
    // with SIM_OPT_DEBUG_CHECKS every instance runs in the checking global-memory kernel
    int wps = c->warps_per_sm;
    bool dense = c->dense != 0;
    bool simulated = false;  // a tuning run already wrote the results (they do not depend on residency)
    if (c->tune_residency && !c->debug_checks) {
        const int64_t shape[3] = {c->n_inst, c->n_total, c->n_max};
        if (!std::equal(shape, shape + 3, c->tuned_shape)) {
            // one warp per scheduler (4 schedulers per SM), the default (two), and the dense copy
            // (three), each timed on the stream with its capacity re-runs
            const int cand_wps[3] = {4, 0, 0};
            const bool cand_dense[3] = {false, false, true};
            float best = 0.f;
            int pick = 1;
            for (int k = 0; k < 3; ++k) {
                float ms = 0.f;
                rc = simulate(c, st, cand_wps[k], cand_dense[k], &ms);
                if (rc) return rc;
                if (k == 0 || ms < best) {
                    best = ms;
                    pick = k;
                }
            }
            c->tuned_wps = cand_wps[pick];
            c->tuned_dense = cand_dense[pick] ? 1 : 0;
            std::copy(shape, shape + 3, c->tuned_shape);
            simulated = true;
        }
        wps = c->tuned_wps;
        dense = c->tuned_dense != 0;
    }
    if (!simulated) {
        rc = simulate(c, st, wps, dense && !c->debug_checks, nullptr);
        if (rc) return rc;
    }
    int worst = SIM_OK;
    for (int32_t i = 0; i < c->n_inst; ++i) {
        const DevResult &d = c->h_res[i];
        sim_result &r = out[i];
        r.total_latency = d.total_latency;
        r.makespan = d.makespan;
        r.peak_memory = d.peak_memory;
        r.evictions = d.evictions;
        r.steps = d.steps;
        r.request_steps = d.request_steps;
        r.status = d.status;
        r._pad = 0;
        if (d.status == simgb::kStatusCapacity) r.status = SIM_E_STATE;
        worst = std::min(worst, int(r.status));
    }
    c->ran = true;
    c->comp_valid = c->record_completions != 0;
    c->wc_valid = c->count_work != 0;
    c->bt_valid = c->batch_time != 0;
    if (worst == SIM_E_STATE) fail(c, SIM_E_STATE, "sim_run: an internal consistency check failed");
    else if (worst == SIM_E_STEPCAP) fail(c, SIM_E_STEPCAP, "sim_run: an instance hit the step cap");
    else if (worst == SIM_E_INFEASIBLE)
        fail(c, SIM_E_INFEASIBLE, "sim_run: an instance has a request with s+o > M (or s+u > M under A_max, A_ell)");
    else if (worst == SIM_E_INVAL)
        fail(c, SIM_E_INVAL, "sim_run: an instance violates 1 <= l <= o <= u, s >= 1, a >= 0 (rank >= 0 under A_r, "
                             "a < 2^30 under A_ell)");
    return worst;
}

int sim_set_tie_seeds(sim_ctx *c, const uint64_t *seeds) {
    if (!c) return SIM_E_INVAL;
    c->err.clear();
    int rc = check_device(c);
    if (rc) return rc;
    if (!seeds) {
        dfree(c->d_seed);
        return SIM_OK;
    }
    cudaError_t e;
    if (!c->d_seed && (e = dalloc(c->d_seed, size_t(c->n_inst) * sizeof(uint64_t))) != cudaSuccess)
        return e == cudaErrorMemoryAllocation ? fail(c, SIM_E_NOMEM, "sim_set_tie_seeds: device allocation failed")
                                              : cuda_fail(c, e, "cudaMalloc");
    e = cudaMemcpy(c->d_seed, seeds, size_t(c->n_inst) * sizeof(uint64_t), cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return cuda_fail(c, e, "sim_set_tie_seeds: copy");
    return SIM_OK;
}

int sim_get_work_counts(sim_ctx *c, int64_t *counts) {
    if (!c) return SIM_E_INVAL;
    c->err.clear();
    if (!counts) return fail(c, SIM_E_INVAL, "sim_get_work_counts: NULL output");
    if (!c->wc_valid || !c->d_wc)
        return fail(c, SIM_E_STATE, "sim_get_work_counts: set SIM_OPT_COUNT_WORK=1 and call sim_run first");
    cudaError_t e = cudaMemcpy(counts, c->d_wc, size_t(c->n_inst) * 4 * sizeof(int64_t), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(c, e, "sim_get_work_counts: copy");
    return SIM_OK;
}

int sim_get_batch_time_sums(sim_ctx *c, int64_t *sums) {
    if (!c) return SIM_E_INVAL;
    c->err.clear();
    if (!sums) return fail(c, SIM_E_INVAL, "sim_get_batch_time_sums: NULL output");
    if (!c->bt_valid || !c->d_bt)
        return fail(c, SIM_E_STATE, "sim_get_batch_time_sums: set SIM_OPT_BATCH_TIME=1 and call sim_run first");
    cudaError_t e = cudaMemcpy(sums, c->d_bt, size_t(c->n_inst) * 6 * sizeof(int64_t), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(c, e, "sim_get_batch_time_sums: copy");
    return SIM_OK;
}

int sim_batch_time(sim_ctx *c, const double *coef, double *out, void *stream) {
    if (!c) return SIM_E_INVAL;
    c->err.clear();
    if (!coef || !out) return fail(c, SIM_E_INVAL, "sim_batch_time: NULL coefficients or output");
    for (int k = 0; k < 5; ++k)
        if (!(coef[k] == coef[k]) || coef[k] - coef[k] != 0.0)
            return fail(c, SIM_E_INVAL, "sim_batch_time: coefficient %d is not finite", k);
    if (!c->bt_valid || !c->d_bt)
        return fail(c, SIM_E_STATE, "sim_batch_time: set SIM_OPT_BATCH_TIME=1 and call sim_run first");
    int rc = check_device(c);
    if (rc) return rc;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    cudaError_t e;
    if (!c->d_btout && (e = dalloc(c->d_btout, size_t(c->n_inst) * 2 * sizeof(double))) != cudaSuccess)
        return fail(c, SIM_E_NOMEM, "sim_batch_time: buffer");
    e = simgb::launch_batch_time(c->d_bt, c->d_res, coef, c->d_btout, c->n_inst, st);
    if (e != cudaSuccess) return cuda_fail(c, e, "sim_batch_time: launch");
    ++c->launches;
    e = cudaMemcpyAsync(out, c->d_btout, size_t(c->n_inst) * 2 * sizeof(double), cudaMemcpyDeviceToHost, st);
    if (e != cudaSuccess) return cuda_fail(c, e, "sim_batch_time: copy");
    e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return cuda_fail(c, e, "sim_batch_time: sync");
    return SIM_OK;
}

int sim_get_completions(sim_ctx *c, int64_t *completion_t) {
    if (!c) return SIM_E_INVAL;
    c->err.clear();
    if (!completion_t) return fail(c, SIM_E_INVAL, "sim_get_completions: NULL output");
    if (!c->comp_valid || !c->d_comp)
        return fail(c, SIM_E_STATE, "sim_get_completions: set SIM_OPT_RECORD_COMPLETIONS=1 and call sim_run first");
    if (c->n_total == 0) return SIM_OK;
    cudaError_t e =
        cudaMemcpy(completion_t, c->d_comp, size_t(c->n_total) * sizeof(int64_t), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(c, e, "sim_get_completions: copy");
    return SIM_OK;
}

int sim_competitive_ratio(const sim_ctx *cp, const sim_ctx *ch, double *cr_out, void *stream) {
    sim_ctx *c = const_cast<sim_ctx *>(cp);
    if (!cp || !ch || !cr_out) return SIM_E_INVAL;
    c->err.clear();
    if (cp->n_inst != ch->n_inst) return fail(c, SIM_E_INVAL, "sim_competitive_ratio: instance counts differ");
    if (ch->policy != SIM_HSF) return fail(c, SIM_E_INVAL, "sim_competitive_ratio: reference context is not H-SF");
    if (!cp->ran || !ch->ran) return fail(c, SIM_E_STATE, "sim_competitive_ratio: run both contexts first");
    if (cp->device != ch->device) return fail(c, SIM_E_INVAL, "sim_competitive_ratio: contexts on different devices");
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    cudaError_t e;
    if (!c->d_cr && (e = dalloc(c->d_cr, size_t(c->n_inst) * sizeof(double))) != cudaSuccess)
        return fail(c, SIM_E_NOMEM, "sim_competitive_ratio: buffer");
    e = simgb::launch_ratio(cp->d_res, ch->d_res, c->d_cr, c->n_inst, st);
    if (e != cudaSuccess) return cuda_fail(c, e, "sim_competitive_ratio: launch");
    ++c->launches;
    e = cudaMemcpyAsync(cr_out, c->d_cr, size_t(c->n_inst) * sizeof(double), cudaMemcpyDeviceToHost, st);
    if (e != cudaSuccess) return cuda_fail(c, e, "sim_competitive_ratio: copy");
    e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return cuda_fail(c, e, "sim_competitive_ratio: sync");
    return SIM_OK;
}

int64_t sim_kernel_launches(const sim_ctx *c) { return c ? c->launches : -1; }

const char *sim_last_error(const sim_ctx *c) { return c ? c->err.c_str() : g_create_err.c_str(); }

void sim_destroy(sim_ctx *c) {
    if (!c) return;
    dfree(c->d_off);
    dfree(c->d_raw);
    dfree(c->d_lu);
    dfree(c->d_rec);
    dfree(c->d_rec_a);
    dfree(c->d_info);
    dfree(c->d_res);
    dfree(c->d_comp);
    dfree(c->d_counter);
    dfree(c->d_work);
    dfree(c->d_gws);
    dfree(c->d_main);
    dfree(c->d_cr);
    dfree(c->d_seed);
    dfree(c->d_wc);
    dfree(c->d_bt);
    dfree(c->d_btout);
    if (c->load_stream) cudaStreamDestroy(c->load_stream);
    if (c->h_off) cudaFreeHost(c->h_off);
    delete c;
}

/* ---- analytic competitive ratios (Lemma thm:Amin, Corollary A/B) --------------------------- */

int sim_cr_amin_lemma(int32_t n_hist, int32_t len, int32_t l, double s, const double *x, double *cr_out,
                      int device_ptrs, void *cuda_stream) {
    if (n_hist < 0 || len < 1 || len > 8192 || l < 1 || !(s >= 0.0) || int64_t(l) + len - 1 > INT32_MAX)
        return fail(nullptr, SIM_E_INVAL, "sim_cr_amin_lemma: need n_hist >= 0, 1 <= len <= 8192, l >= 1, s >= 0");
    if (n_hist == 0) return SIM_OK;
    if (!x || !cr_out) return fail(nullptr, SIM_E_INVAL, "sim_cr_amin_lemma: NULL x or cr_out");
    cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
    cudaError_t e;
    if (device_ptrs) {
        e = simgb::launch_lemma(n_hist, len, l, s, x, cr_out, st);
        if (e != cudaSuccess) return cuda_fail(nullptr, e, "sim_cr_amin_lemma: kernel launch");
        return SIM_OK;
    }
    double *dx = nullptr, *dout = nullptr;
    const size_t nx = size_t(n_hist) * size_t(len);
    if ((e = cudaMalloc(&dx, nx * sizeof(double))) != cudaSuccess ||
        (e = cudaMalloc(&dout, size_t(n_hist) * sizeof(double))) != cudaSuccess) {
        cudaFree(dx);
        return e == cudaErrorMemoryAllocation ? fail(nullptr, SIM_E_NOMEM, "sim_cr_amin_lemma: device allocation")
                                              : cuda_fail(nullptr, e, "sim_cr_amin_lemma: cudaMalloc");
    }
    int rc = SIM_OK;
    if ((e = cudaMemcpyAsync(dx, x, nx * sizeof(double), cudaMemcpyHostToDevice, st)) != cudaSuccess ||
        (e = simgb::launch_lemma(n_hist, len, l, s, dx, dout, st)) != cudaSuccess ||
        (e = cudaMemcpyAsync(cr_out, dout, size_t(n_hist) * sizeof(double), cudaMemcpyDeviceToHost, st)) !=
            cudaSuccess ||
        (e = cudaStreamSynchronize(st)) != cudaSuccess)
        rc = cuda_fail(nullptr, e, "sim_cr_amin_lemma");
    cudaFree(dx);
    cudaFree(dout);
    return rc;
}

int sim_cr_amin_rho(int32_t n_u, const int32_t *u_values, double *rho_out) {
    if (n_u < 0) return fail(nullptr, SIM_E_INVAL, "sim_cr_amin_rho: n_u < 0");
    if (n_u == 0) return SIM_OK;
    if (!u_values || !rho_out) return fail(nullptr, SIM_E_INVAL, "sim_cr_amin_rho: NULL argument");
    int32_t umax = 0;
    for (int32_t k = 0; k < n_u; ++k) {
        if (u_values[k] < 1 || u_values[k] > (1 << 20))
            return fail(nullptr, SIM_E_INVAL, "sim_cr_amin_rho: u_values[%d]=%d outside [1, 2^20]", k, u_values[k]);
        umax = std::max(umax, u_values[k]);
    }
    // batches of at most 256 MB of vectors (3 u doubles per value)
    const int64_t stride = 3 * int64_t(umax);
    const int64_t per_batch = std::max<int64_t>(1, (int64_t(256) << 20) / (stride * int64_t(sizeof(double))));
    const int32_t nb = int32_t(std::min<int64_t>(per_batch, n_u));
    double *scratch = nullptr, *dout = nullptr;
    int32_t *dus = nullptr;
    cudaError_t e;
    if ((e = cudaMalloc(&scratch, size_t(nb) * size_t(stride) * sizeof(double))) != cudaSuccess ||
        (e = cudaMalloc(&dout, size_t(nb) * sizeof(double))) != cudaSuccess ||
        (e = cudaMalloc(&dus, size_t(nb) * sizeof(int32_t))) != cudaSuccess) {
        cudaFree(scratch);
        cudaFree(dout);
        return e == cudaErrorMemoryAllocation ? fail(nullptr, SIM_E_NOMEM, "sim_cr_amin_rho: device allocation")
                                              : cuda_fail(nullptr, e, "sim_cr_amin_rho: cudaMalloc");
    }
    int rc = SIM_OK;
    for (int32_t b = 0; b < n_u && rc == SIM_OK; b += nb) {
        const int32_t m = std::min(nb, n_u - b);
        if ((e = cudaMemcpy(dus, u_values + b, size_t(m) * sizeof(int32_t), cudaMemcpyHostToDevice)) != cudaSuccess ||
            (e = simgb::launch_rho(m, dus, dout, scratch, stride, 200, nullptr)) != cudaSuccess ||
            (e = cudaMemcpy(rho_out + b, dout, size_t(m) * sizeof(double), cudaMemcpyDeviceToHost)) != cudaSuccess)
            rc = cuda_fail(nullptr, e, "sim_cr_amin_rho");
    }
    cudaFree(scratch);
    cudaFree(dout);
    cudaFree(dus);
    return rc;
}

}  // extern "C"
