/*
 * sim.h - C ABI of the batched scheduler simulator (libsim.so, CUDA, sm_103a).
 *
 * The library simulates many independent instances of the single-worker LLM-inference
 * scheduling problem of arXiv 2508.14544 ("Adaptively Robust LLM Inference Optimization under
 * Prediction Uncertainty") on one GPU, under one of five policies:
 *
 *   SIM_AMAX - A_max, Algorithm malb (Section 3.2): every output length is taken to be its
 *              predicted upper bound u_i; each step admits the largest prefix of the waiting set,
 *              sorted by (u_i, request index), that keeps the projected memory within M at every
 *              future step (eq. Constraint).  Never cancels a job.
 *   SIM_AMIN - A_min, Algorithms milb and milbrevise (Section 4, 4.2): each request starts with the
 *              lower bound l_i as its length estimate; when the next step would exceed M, active
 *              jobs are cancelled in ascending estimate order until the rest fits, ties broken
 *              uniformly at random (a fresh draw at every step, see sim_set_tie_seeds), and each
 *              cancelled job's estimate becomes max(estimate, tokens generated); the waiting set is
 *              then admitted as for A_max, using the estimates.
 *   SIM_HSF  - the hindsight shortest-first benchmark H-SF, Algorithm off (Section 3.1, Appendix
 *              B): like A_max with the true output lengths.
 *   SIM_AR   - the auxiliary policy A_r, Algorithm random (Appendix B): a fixed random permutation
 *              of the requests (given by the caller as ranks, see sim_load_ranked_csr) and the true
 *              output lengths; each step admits the largest feasible prefix in permutation order.
 *   SIM_AELL - the promote-l policy A_ell, Algorithm promote_l (Section 5, two-point output
 *              distributions; here with each request's own l_i and u_i): a FIFO waiting queue,
 *              length estimate l_i; at the start of a step a job that has generated l_i tokens
 *              without finishing is cancelled, takes u_i as its estimate and joins the end of the
 *              queue (after the requests that arrived in that step; several in index order).
 *              Each such promotion counts as a cancellation.  Steps must stay below 2^30.
 *
 * Model (Section 2): a worker with a KV cache of M tokens runs one batch per unit of time; every
 * member generates one token; a job's memory is its prompt size s_i plus the tokens generated so
 * far, and the memory of each step (counted after the step's tokens) must not exceed M
 * (eq. constraintM).  Request i becomes eligible at step a_i (the paper has a_i = 0; arrivals are
 * an extension); its completion step C_i is one past the step that generated its last token.
 *
 * Ties in the waiting set's order, which the paper breaks "uniformly at random", are broken by the
 * smaller request index (0-based position within the instance): with requests drawn i.i.d. the
 * index order of requests that have not run yet is itself a uniformly random order.  A_min's
 * cancellation ties are drawn afresh at every step from a counter-based generator: the tie key of
 * request i at step t is the high 32 bits of SplitMix64 output number t * 2^32 + i + 1 for the
 * instance's seed (sim_set_tie_seeds), and the cancellation order is (estimate, tie key, index).
 * Outputs are deterministic given the seeds and bit-identical to the CPU reference of the same
 * rules.
 *
 * Threading: a context must not be used from two threads at once.  Different contexts are
 * independent.  All calls act on the CUDA device that is current on the calling thread.
 */
#ifndef SIM_H_
#define SIM_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum { SIM_AMAX = 0, SIM_AMIN = 1, SIM_HSF = 2, SIM_AR = 3, SIM_AELL = 4 } sim_policy;

typedef enum {
    SIM_OK = 0,
    SIM_E_INVAL = -1,      /* bad argument, or an instance with l > o, o > u, l < 1, s < 1, a < 0 */
    SIM_E_INFEASIBLE = -2, /* an instance has a request with s + o > M (or s + u > M under A_max, A_ell) */
    SIM_E_STEPCAP = -3,    /* an instance processed step_cap batches without finishing, or its step
                              counter reached 2^31 - 2^27 (2^30 under A_ell) */
    SIM_E_CUDA = -4,       /* a CUDA runtime call failed; see sim_last_error */
    SIM_E_STATE = -5,      /* call out of order (e.g. sim_run before sim_load), or an internal check failed */
    SIM_E_NOMEM = -6       /* host or device allocation failed */
} sim_status;

/* Per-instance result of sim_run (56 bytes). */
typedef struct {
    int64_t total_latency; /* TEL = sum_i (C_i - a_i)  (eq. latency) */
    int64_t makespan;      /* max_i C_i */
    int64_t peak_memory;   /* max over steps of the step's memory, sum over the batch of (s + tokens) */
    int64_t evictions;     /* number of cancellations (always 0 for A_max and H-SF) */
    int64_t steps;         /* batches processed (steps skipped while idle are not counted) */
    int64_t request_steps; /* sum over steps of the batch size (tokens generated, wasted ones included) */
    int32_t status;        /* sim_status of this instance */
    int32_t _pad;
} sim_result;

typedef struct sim_ctx sim_ctx;

/* Options for sim_set_option. */
enum {
    SIM_OPT_STEP_CAP = 1,           /* int64 > 0: stop an instance after this many batches
                                       (status SIM_E_STEPCAP).  0 (default): 64 * (n + sum_i o_i). */
    SIM_OPT_RECORD_COMPLETIONS = 2, /* 0/1: keep each request's completion step for
                                       sim_get_completions (default 0). */
    SIM_OPT_WARPS_PER_BLOCK = 3,    /* 1..8: simulation warps per thread block (default 4; unset,
                                       a launch with no more instances than SMs uses 1, so that
                                       each instance has an SM to itself).  Results do not depend
                                       on it. */
    SIM_OPT_SMEM_ACTIVE_CAP = 4,    /* 128..4096, multiple of 128: active-set slots kept in shared
                                       memory per instance (default 512).  Instances that need more
                                       are re-run automatically with the active set in global
                                       memory; results are identical. */
    SIM_OPT_WARPS_PER_SM = 5,       /* 0..64: at most this many simulation warps resident per SM
                                       (0, the default: as many as shared memory allows).  Results
                                       do not depend on it. */
    SIM_OPT_DEBUG_CHECKS = 6,       /* 0/1: run every instance in the global-memory kernel and check
                                       the simulation state's invariants between events (active set
                                       sorted by projected end, suffix sums and prefix maxima of the
                                       set, queue order; no job past its projected end under A_max,
                                       H-SF and A_r).  A violation gives that instance SIM_E_STATE.
                                       Slower; results are otherwise identical. */
    SIM_OPT_TUNE_RESIDENCY = 7,     /* 0/1: on the first sim_run of a load shape (n_instances, total
                                       and largest instance size), time three residencies -- one
                                       simulation warp per scheduler (4 per SM), the default (two),
                                       and the dense configuration of SIM_OPT_DENSE_RESIDENCY
                                       (three) -- each with its global-memory re-runs, and use the
                                       fastest for every later sim_run of that shape, across
                                       sim_load calls (default 0).  A launch is as long as its
                                       slowest instance: one warp per scheduler wins when a few
                                       instances dominate, more when there are many even ones.  The
                                       tuning run simulates three times; results do not depend on
                                       it.  Overrides SIM_OPT_WARPS_PER_SM and
                                       SIM_OPT_DENSE_RESIDENCY while set. */
    SIM_OPT_EVICT_TIES = 8,         /* 0 (default): A_min's cancellation ties are broken at random
                                       as Algorithm milb states (see sim_set_tie_seeds); 1: by the
                                       request index instead, a fixed order that always cancels the
                                       earliest-started of the tied jobs (for sensitivity studies). */
    SIM_OPT_COUNT_WORK = 9,         /* 0/1: record per instance the work that the paper's per-step
                                       method does (sim_get_work_counts; default 0).  Results are
                                       identical; the counting costs a few instructions per event. */
    SIM_OPT_BATCH_TIME = 10,        /* 0/1: record per instance the integer sums that give total
                                       latency and makespan in time units under a linear batch-time
                                       model (sim_batch_time, sim_get_batch_time_sums; default 0). */
    SIM_OPT_DENSE_RESIDENCY = 11    /* 0/1: simulate with three blocks of four warps per SM (12
                                       warps; a kernel copy limited to 170 registers a thread) and
                                       384 active-set slots in shared memory per instance, instead
                                       of two blocks and SIM_OPT_SMEM_ACTIVE_CAP slots (default 0).
                                       Faster when there are many instances whose active sets stay
                                       below 384 jobs; instances that need more are re-run in global
                                       memory.  Not used with SIM_OPT_COUNT_WORK or
                                       SIM_OPT_BATCH_TIME.  Results do not depend on it. */
};

/*
 * sim_create: set up a context for `n_instances` independent instances simulated under `policy`
 * with KV-cache limit M tokens (Section 2).
 *   policy      SIM_AMAX, SIM_AMIN, SIM_HSF, SIM_AR or SIM_AELL.
 *   M           1 <= M <= 2^26.
 *   n_instances >= 1.
 *   out         receives the new context (owned by the caller; free with sim_destroy).
 * Touches no GPU memory.  Returns SIM_OK, SIM_E_INVAL or SIM_E_NOMEM.
 */
int sim_create(int policy, int64_t M, int32_t n_instances, sim_ctx **out);

/*
 * sim_load: load n_per_instance requests for every instance (uniform sizes).  Each array holds
 * n_instances * n_per_instance int32 values, instance-major: request j of instance i is at
 * [i * n_per_instance + j].
 *   arrival_t  a_i >= 0: first step at which the request may be scheduled.
 *   prompt_s   s_i >= 1: prompt size in tokens (Section 2; per-request as in Section 6).
 *   lower_l    l_i: predicted lower bound of the output length, 1 <= l_i <= o_i.
 *   upper_u    u_i: predicted upper bound, o_i <= u_i.
 *   true_o     o_i >= 1: true output length (hidden from A_max and A_min; used by H-SF and by the
 *              simulation itself to know when a job finishes).
 *   device_ptrs 0: the arrays are host memory; 1: device memory on the current device, already
 *               written (the call does not order itself after the caller's streams).
 * The library stages the data into device buffers it owns (host arrays are copied in first; device
 * arrays are read in place by the staging kernel), on a stream of its own, so the call does not
 * wait for other work on the device, and returns when staging has finished: the caller may free
 * or reuse its arrays as soon as the call returns.  Per-instance input problems (INVAL, INFEASIBLE) do not fail
 * the call: they are reported in that instance's sim_result.status by sim_run.
 * Returns SIM_OK, SIM_E_INVAL (n_per_instance < 0, null pointer; under SIM_AR, which needs
 * sim_load_ranked_csr), SIM_E_NOMEM or SIM_E_CUDA.
 */
int sim_load(sim_ctx *ctx, int32_t n_per_instance, const int32_t *arrival_t, const int32_t *prompt_s,
             const int32_t *lower_l, const int32_t *upper_u, const int32_t *true_o, int device_ptrs);

/*
 * sim_load_csr: like sim_load with per-instance sizes.  `offsets` is HOST memory with
 * n_instances + 1 non-decreasing int64 values, offsets[0] = 0; instance i owns requests
 * [offsets[i], offsets[i+1]) of each array.  Empty instances are allowed (their result is all
 * zeros with status SIM_OK).
 */
int sim_load_csr(sim_ctx *ctx, const int64_t *offsets, const int32_t *arrival_t, const int32_t *prompt_s,
                 const int32_t *lower_l, const int32_t *upper_u, const int32_t *true_o, int device_ptrs);

/*
 * sim_load_ranked_csr: sim_load_csr plus the random permutation that Algorithm random (A_r,
 * Appendix B) draws before it starts; the draw is the caller's, so runs are reproducible.
 *   rank   int32 per request, same layout and memory kind as the other arrays: rank_i >= 0 is the
 *          position of request i in its instance's permutation (a permutation of 0..n-1 is the
 *          intended use; equal ranks are ordered by request index).  Required (non-NULL) under
 *          SIM_AR; ignored under the other policies.
 * A negative rank makes that instance SIM_E_INVAL.  Returns as sim_load_csr.
 */
int sim_load_ranked_csr(sim_ctx *ctx, const int64_t *offsets, const int32_t *arrival_t, const int32_t *prompt_s,
                        const int32_t *lower_l, const int32_t *upper_u, const int32_t *true_o,
                        const int32_t *rank, int device_ptrs);

/*
 * sim_run: simulate every loaded instance and write n_instances results to `out` (HOST memory).
 *   cuda_stream  a cudaStream_t of the current device, or NULL for the default stream.
 * Synchronous: returns after the results are in `out`.  Re-running without reloading gives
 * identical results.  Returns the most negative per-instance status (SIM_OK if all succeeded),
 * or SIM_E_STATE (nothing loaded), SIM_E_CUDA, SIM_E_NOMEM.
 */
int sim_run(sim_ctx *ctx, sim_result *out, void *cuda_stream);

/*
 * sim_set_tie_seeds: seeds of A_min's random cancellation ties (Algorithm milb / milbrevise,
 * Section 4: "sort S_t in ascending order of the lower bound; break ties uniformly at random").
 *   seeds  HOST, n_instances uint64 values, one per instance; NULL resets every seed to 0 (the
 *          default).  Copied before the call returns.
 * At a step t with an overflow, the active jobs are cancelled in ascending (estimate, r, index)
 * order, r = the high 32 bits of output number t * 2^32 + i + 1 of the SplitMix64 generator
 * (Steele, Lea and Flood 2014) seeded with the instance's seed, i the request index: a fresh,
 * reproducible random order of the tied jobs at every step.  Takes effect at the next sim_run (no
 * reload needed); ignored under the other policies and under SIM_OPT_EVICT_TIES = 1.
 * Returns SIM_OK, SIM_E_INVAL, SIM_E_STATE (another device is current), SIM_E_NOMEM or SIM_E_CUDA.
 */
int sim_set_tie_seeds(sim_ctx *ctx, const uint64_t *seeds);

/*
 * sim_get_work_counts: the work counters of the last sim_run (SIM_OPT_COUNT_WORK = 1), four int64
 * per instance, instance-major, into `counts` (HOST, 4 * n_instances).  They count the work of
 * the per-step method that Theorem complexity (Section 4) bounds, summed over the instance's
 * processed steps, with A_t the active set at the start of step t, A'_t + k_t the batch after
 * cancellations and admission (k_t admitted) and Q_t the waiting set at admission:
 *   [0] sum_t A_t                                    (memory accounting of S_t: one add per job)
 *   [1] sum over steps with an overflow (A_min) of A_t * ceil(log2 A_t)^2
 *                                                    (compare-exchanges of a sort of S_t)
 *   [2] sum_t (A'_t + k_t) * ceil(log2(Q_t + 1))     (endpoint evaluations of an admission that
 *                                                     binary-searches the largest feasible prefix)
 *   [3] bytes of global memory the waiting queue moved (arrival runs, head reloads, merges).
 * The simulator itself skips most of this work (quiet steps in closed form, incremental order);
 * the counters measure the method, not the kernel.  Returns SIM_OK, SIM_E_INVAL, SIM_E_STATE
 * (counting was off for the last sim_run) or SIM_E_CUDA.
 */
int sim_get_work_counts(sim_ctx *ctx, int64_t *counts);

/*
 * sim_batch_time: total latency and makespan of every instance of the last sim_run in time units,
 * under a linear batch-time model (Section 6 times each batch with a linear regression predictor;
 * the paper prints no coefficients, so they are the caller's).  A processed step t with batch B_t
 * takes
 *     f(B_t) = c0 + c1 |B_t| + c2 mem(t) + c3 prefill(t),
 * mem(t) = sum over B_t of (s_i + tokens), the step's KV tokens; prefill(t) = the prompt tokens of
 * the requests started (or restarted) at t; a step with nothing to run takes c_idle.  Request i's
 * latency in time units is the total time of steps a_i .. C_i - 1.
 *   coef  HOST, 5 doubles: c0, c1, c2, c3, c_idle (finite).
 *   out   HOST, 2 * n_instances doubles: [2i] = total latency in time units = c0 X0 + c1 X1 +
 *         c2 X2 + c3 X3, [2i+1] = makespan in time units = c0 F0 + c1 F1 + c2 F2 + c3 F3 +
 *         c_idle F4, each evaluated left to right in IEEE double without fused multiply-adds, with
 *         the integer sums of sim_get_batch_time_sums (F0 = steps, F1 = request steps, F4 =
 *         makespan - steps); NaN for an instance whose status is not SIM_OK.
 * Requires SIM_OPT_BATCH_TIME = 1 before sim_run; coefficients can then change without
 * re-simulating.  Synchronous on cuda_stream.  Returns SIM_OK, SIM_E_INVAL, SIM_E_STATE,
 * SIM_E_NOMEM or SIM_E_CUDA.
 */
int sim_batch_time(sim_ctx *ctx, const double *coef, double *out, void *cuda_stream);

/*
 * sim_get_batch_time_sums: the integer sums behind sim_batch_time, six int64 per instance
 * (HOST, 6 * n_instances): X0..X3 = sum over requests i of the number of processed steps, batch
 * sizes |B_t|, step memories mem(t) and prefill tokens prefill(t) of the steps a_i .. C_i - 1 (no
 * step inside a request's interval is idle); F2, F3 = the totals of mem(t) and prefill(t) over
 * all processed steps.  Zeros for an instance whose status is not SIM_OK.  X2 stays exact while
 * M * total latency < 2^63.  Returns SIM_OK, SIM_E_INVAL, SIM_E_STATE or SIM_E_CUDA.
 */
int sim_get_batch_time_sums(sim_ctx *ctx, int64_t *sums);

/*
 * sim_get_completions: copy every request's completion step C_i of the last sim_run into
 * `completion_t` (HOST, n_total int64, same layout as the loaded arrays; 0 for instances that did
 * not run).  Requires SIM_OPT_RECORD_COMPLETIONS = 1 before sim_run; otherwise SIM_E_STATE.
 */
int sim_get_completions(sim_ctx *ctx, int64_t *completion_t);

/*
 * sim_competitive_ratio: per-instance ratio TEL(policy) / TEL(H-SF) (Definition cr, Section 3.1)
 * of two contexts that ran the same instances, computed on the device in IEEE double.
 *   ctx_policy, ctx_hsf  contexts after sim_run with equal n_instances (ctx_hsf under SIM_HSF).
 *   cr_out               HOST, n_instances doubles; NaN where either instance failed or TEL(H-SF)=0.
 * Returns SIM_OK, SIM_E_INVAL or SIM_E_STATE.
 */
int sim_competitive_ratio(const sim_ctx *ctx_policy, const sim_ctx *ctx_hsf, double *cr_out, void *cuda_stream);

/* sim_kernel_launches: number of CUDA kernels this context has launched since sim_create
 * (staging, simulation, fallback and ratio kernels).  ctx NULL -> -1. */
int64_t sim_kernel_launches(const sim_ctx *ctx);

/*
 * sim_run_noalloc: stage and simulate in one call WITHOUT allocating any device memory.  The
 * paper has no counterpart: this is a library convenience for callers that cannot call cudaMalloc
 * -- a process whose GPU memory is all reserved up front by its own pool allocator (a cudaMalloc
 * would fail or fragment that reservation), or a latency-sensitive loop that must avoid the
 * implicitly synchronising allocation calls (cudaFree waits for the whole device).
 * Semantics and results are those of sim_load_csr + sim_run with default options.
 *   policy, M, n_instances  as for sim_create, policy SIM_AMAX, SIM_AMIN or SIM_HSF
 *               (1 <= n_instances <= 16384).
 *   offsets     HOST, n_instances + 1 int64, as for sim_load_csr.
 *   arrival_t .. true_o     DEVICE int32 arrays (current device), layout as for sim_load_csr.
 *   results     DEVICE, n_instances sim_result, written by the kernels.
 *   cuda_stream a cudaStream_t or NULL.  The call only enqueues work: read `results` after
 *               synchronising the stream.  Per-instance statuses are in results[i].status.
 * Everything except the inputs and outputs lives in one fixed array of about 23 MB that every GPU
 * loading the library holds until the process exits.  Limits: at most 2048 requests per instance
 * and 262,144 requests per call; larger inputs are rejected with SIM_E_INVAL and a message in
 * sim_last_error(NULL).  The staging kernel checks the offsets it reads against the same limits
 * again: an instance that reaches past them gets status SIM_E_INVAL in its result and nothing of
 * it is staged.  The fixed array holds the workspaces of 128 simulating warps (32 blocks of 4),
 * so on a 152-SM GPU most SMs stay idle: with many instances expect several times the time of
 * sim_run, which sizes its launch to the whole GPU.  All calls share that array and it keeps the last call's contents: calls
 * that overlap on the GPU (different streams or threads) race; calls on one stream are safe.
 * The first call on each device looks up the array's device address (cudaGetSymbolAddress) with
 * that device current.  Allocates nothing.
 * Returns SIM_OK, SIM_E_INVAL, SIM_E_CUDA or SIM_E_STATE.
 */
int sim_run_noalloc(int policy, int64_t M, int32_t n_instances, const int64_t *offsets, const int32_t *arrival_t,
                    const int32_t *prompt_s, const int32_t *lower_l, const int32_t *upper_u, const int32_t *true_o,
                    sim_result *results, void *cuda_stream);

/*
 * sim_cr_amin_lemma: the large-M competitive ratio of A_min given by Lemma thm:Amin (Section 4.1)
 * for a batch of output-length histograms, in IEEE double.  Every request has prompt size s and
 * an output length in [l, u], u = l + len - 1; histogram h gives x_k, the fraction (or count) of
 * requests of length k, at x[h * len + (k - l)].
 *   CR = sum_k d(k) S1(k) (d(k) S2(k) + 2 G(k)) / sum_k k (s+k) x_k (x_k + 2 sum_{i>k} x_i),
 *   d(l) = s + l, d(k) = 1 otherwise, S1(k) = sum_{i>=k} i x_i, S2(k) = sum_{i>=k} x_i / (s+i),
 *   G(k) = sum_{i>k} (i-k) x_i / (s+i).
 *   n_hist     >= 0 histograms; 1 <= len <= 8192; l >= 1; s >= 0.
 *   x, cr_out  n_hist * len and n_hist doubles; HOST memory (device_ptrs = 0: the call copies,
 *              computes and returns with the results in cr_out) or DEVICE memory of the current
 *              device (device_ptrs = 1: the call only enqueues the kernel on cuda_stream).
 * Entries must be >= 0 with a positive denominator (at least one x_k > 0); otherwise the ratio is
 * not a number.  Returns SIM_OK, SIM_E_INVAL (message in sim_last_error(NULL)), SIM_E_NOMEM,
 * SIM_E_CUDA.  No counterpart needs a context.
 */
int sim_cr_amin_lemma(int32_t n_hist, int32_t len, int32_t l, double s, const double *x, double *cr_out,
                      int device_ptrs, void *cuda_stream);

/*
 * sim_cr_amin_rho: for each u, the spectral radius of B_u^{-1} A_u (Corollary A/B, s = 0, l = 1:
 * a_ij = min(i,j)^2/(ij) ((i+j)^2/2 - min(i,j)^2), b_ij = min(i,j)^2), the largest value of the
 * Rayleigh quotient x'A_u x / x'B_u x and thus the bound on CR(A_min) of Section 4.1 (<= H_u).
 *   u_values  HOST, n_u values in [1, 2^20];  rho_out  HOST, n_u doubles.
 * Power iteration in double on the current device, synchronous; converges to the relative
 * precision of double in well under 200 iterations (the second eigenvalue is below a third of the
 * first for every u tried).  Returns SIM_OK, SIM_E_INVAL, SIM_E_NOMEM or SIM_E_CUDA.
 */
int sim_cr_amin_rho(int32_t n_u, const int32_t *u_values, double *rho_out);

/* sim_set_option: set one of the SIM_OPT_* options.  Returns SIM_OK or SIM_E_INVAL. */
int sim_set_option(sim_ctx *ctx, int key, int64_t value);

/* sim_last_error: NUL-terminated message of the last failing call on ctx ("" if none).  The
 * pointer stays valid until the next call on ctx.  ctx may be NULL (message of the last sim_create). */
const char *sim_last_error(const sim_ctx *ctx);

/* sim_destroy: free the context and every device buffer it owns.  NULL is allowed. */
void sim_destroy(sim_ctx *ctx);

#ifdef __cplusplus
}
#endif

#endif /* SIM_H_ */
