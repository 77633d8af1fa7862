// Internal declarations shared by the C ABI (sim_api.cpp) and the CUDA kernels (sim_kernels.cu).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <climits>

namespace simgb {

// Internal per-instance status: the active set outgrew the per-instance capacity of the launch;
// the host re-runs such instances with a larger, global-memory workspace.
constexpr int32_t kStatusCapacity = -100;
constexpr int64_t kMaxM = int64_t(1) << 26;
// Steps are int32: an instance stops with SIM_E_STEPCAP before a step passes kMaxStep, which leaves
// room for a projected length (<= M <= 2^26) on top of any step.
constexpr int32_t kMaxStep = INT32_MAX - (int32_t(1) << 27);
// A_ell queue keys are 2 a (arrival) and 2 t + 1 (promotion at step t): steps stay below 2^30.
constexpr int32_t kAellMaxStep = (int32_t(1) << 30) - 1;

// One waiting request as the queue stores it; queues are ordered by (key, idx).
struct QEnt {
    int32_t key;  // sort key: u (A_max), o (H-SF), current lower bound (A_min), permutation rank
                  // (A_r), queue position 2 a / 2 t + 1 (A_ell)
    int32_t idx;  // request index within its instance
    int32_t s;    // prompt size
    int32_t o;    // true output length
};

// Per-instance constants produced by the staging kernel.
struct InstInfo {
    int64_t base;     // offset of the instance's first request
    int64_t sum_a;    // sum of arrival steps (TEL = sum of completions - sum_a)
    int64_t cap;      // step cap
    int32_t n;        // number of requests
    int32_t status;   // 0 or a sim_status from validation
    int32_t lmax;     // largest u_i or o_i of the instance (bounds every projected length)
    int32_t pad;
};

struct DevResult {
    int64_t total_latency, makespan, peak_memory, evictions, steps, request_steps;
    int32_t status, pad;
};

struct StageParams {
    int policy;
    int64_t M;
    int32_t n_inst;
    int32_t n_max;             // largest instance (sizes the staging kernel's shared memory; 0: unknown)
    int64_t max_total;         // capacity of rec / rec_a: an instance reaching past it is rejected (INVAL)
    int32_t max_n;             // requests per instance above this are rejected (INVAL)
    int64_t step_cap;          // 0: default 64 * (n + sum o)
    const int64_t *off;        // n_inst + 1
    const int32_t *a, *s, *l, *u, *o;  // raw copies, n_total each
    const int32_t *rank;       // A_r: permutation rank per request (n_total), else unused
    QEnt *rec;                 // out: per instance, sorted by (a, key, idx)
    int2 *lu;                  // out (A_ell only, else null): (l, u) of request idx at base + idx
    int32_t *rec_a;            // out: arrival step of rec[i]
    InstInfo *info;            // out: n_inst
};

struct RunParams {
    int64_t M;
    int32_t n_work;            // instances to run in this launch
    const int32_t *work;       // instance ids (n_work)
    int32_t *counter;          // work-queue cursor (zeroed before launch)
    const QEnt *rec;
    const int32_t *rec_a;
    const InstInfo *info;
    DevResult *res;
    int64_t *completion;       // optional, n_total
    const int2 *lu;            // A_ell: (l, u) per request (staged), else null
    const uint64_t *tie_seed;  // A_min: seed of the random eviction ties per instance, or null (0 for all)
    int64_t *work_count;       // optional, 4 per instance: S2 adds, S3 compare-exchanges, S5 endpoint
                               // evaluations of the per-step method, global bytes moved by the queue
    int64_t *batch_time;       // optional, 6 per instance: the batch-time sums X0..X3, F2, F3
    // workspace
    int32_t ca;                // active-set capacity per instance (multiple of 32)
    int32_t use_smem;          // 1: active set + delta queue in shared memory; 0: global workspace
    int32_t debug;             // 1: check the simulation state's invariants every iteration (global kernel)
    int32_t evict_index;       // 1: A_min eviction ties by request index instead of the random tie key
    unsigned char *gws;        // global workspace base (use_smem == 0)
    int64_t gws_stride;        // bytes per warp slot
    QEnt *mainbuf;             // ping-pong main-queue buffers, 2 * main_cap per warp slot
    int64_t main_cap;
};

size_t warp_ws_bytes(int ca);  // workspace bytes per warp slot for ca active-set slots

cudaError_t launch_stage(const StageParams &p, cudaStream_t st);
// dense: the 12-warps-per-SM copy of the plain shared-memory kernel (blocks of 4 warps, kDenseCa slots)
cudaError_t launch_run(int policy, const RunParams &p, int blocks, int warps_per_block, size_t smem_bytes, bool dense,
                       cudaStream_t st);
constexpr int kDenseCa = 384;      // active-set slots per warp of the dense configuration
constexpr int kDenseWarps = 4;     // warps per block of the dense configuration
constexpr int kSmemCaDefault = 512;  // active-set slots per warp in shared memory by default
constexpr int kDcap = 256;         // delta-queue capacity per warp slot (multiple of 32)
cudaError_t launch_ratio(const DevResult *pol, const DevResult *ref, double *out, int32_t n, cudaStream_t st);
cudaError_t launch_batch_time(const int64_t *sums, const DevResult *res, const double *coef, double *out, int32_t n,
                              cudaStream_t st);
cudaError_t set_run_smem_limit(int policy, size_t bytes);
cudaError_t launch_lemma(int32_t n_hist, int32_t len, int32_t l, double s, const double *x, double *out,
                         cudaStream_t st);
cudaError_t launch_rho(int32_t n_u, const int32_t *us, double *out, double *scratch, int64_t stride,
                       int32_t max_iter, cudaStream_t st);

}  // namespace simgb
