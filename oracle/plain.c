/*
 * Plain CPU oracle of the batched schedulers A_max, A_min, H-SF, A_r and A_ell (endpoint
 * evaluation).
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the CPU-baseline leg of
 * bench.py may load this library.  It shares no code, header, table or helper with the CUDA path.
 *
 * Same semantics as oracle/literal.py (see the readings listed there): the W memory-timing
 * reading of eq. constraintM (Section 2), the future-feasibility check of eq. Constraint
 * (Section 3.1) with the policy's length estimate (o for H-SF, Algorithm off; u for A_max,
 * Algorithm malb; the running lower bound for A_min, Algorithms milb / milbrevise), admission of
 * the largest feasible prefix of the waiting set sorted by (key, index), and A_min's
 * overflow eviction in ascending lower-bound order, ties broken by a random key drawn afresh at
 * every step (SplitMix64 of the instance's seed and the counter step * 2^32 + index; the index
 * order instead when evict_index is set), with the refinement
 * lower_bound <- max(lower_bound, tokens generated).  A_r (Algorithm random): true lengths and a
 * given permutation rank as the queue key.  A_ell (Algorithm promote_l): FIFO queue (key 2 a_i on
 * arrival, 2 t + 1 on re-entry at step t), estimate l_i, and at the start of a step a request that
 * has used up its estimate unfinished is removed, takes u_i and re-enters at the end.
 *
 * The only difference from the literal oracle is how the constraint is checked: instead of
 * every future step t', it is checked at the projected last steps ("endpoints") of the jobs.
 * With every start <= t, the set of jobs still projected to run shrinks as t' grows and the sum
 * grows linearly between two endpoints, so the maximum over t' >= t is reached at an endpoint;
 * at endpoint x the value is  sum_{e_j >= x} (s_j - p_j + 1 + x).
 *
 * Batch time (Section 6, a linear batch-time predictor with caller-supplied coefficients): the
 * optional time_sums output holds, per instance, X0..X3 = sum over requests of the number of
 * processed steps, batch sizes, step memories and prefill (prompt tokens started) of the steps
 * a_i .. C_i - 1, and F2, F3 = the totals of step memory and prefill over all processed steps.
 * They are kept as prefix sums: an arrival at t subtracts the prefix up to t, a completion at C
 * adds the prefix up to C.
 *
 * Data structures are the textbook ones: a binary min-heap keyed by (key, index) for the waiting
 * set, an unsorted array for the active set, qsort for the endpoint sweep and the eviction order.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

enum { O_AMAX = 0, O_AMIN = 1, O_HSF = 2, O_AR = 3, O_AELL = 4 };
enum { O_OK = 0, O_E_INVAL = -1, O_E_INFEASIBLE = -2, O_E_STEPCAP = -3, O_E_NOMEM = -6 };

typedef struct {
    int64_t total_latency, makespan, peak_memory, evictions, steps, request_steps;
    int32_t status, pad;
} oracle_result;

/* ---- waiting set: binary min-heap of (key << 32 | index) ------------------------------------ */
typedef struct {
    uint64_t *v;
    int32_t n;
} heap_t;

static void heap_push(heap_t *h, uint64_t x) {
    int32_t i = h->n++;
    while (i > 0) {
        int32_t par = (i - 1) / 2;
        if (h->v[par] <= x) break;
        h->v[i] = h->v[par];
        i = par;
    }
    h->v[i] = x;
}

static uint64_t heap_pop(heap_t *h) {
    uint64_t top = h->v[0];
    uint64_t last = h->v[--h->n];
    int32_t i = 0;
    for (;;) {
        int32_t c = 2 * i + 1;
        if (c >= h->n) break;
        if (c + 1 < h->n && h->v[c + 1] < h->v[c]) c++;
        if (last <= h->v[c]) break;
        h->v[i] = h->v[c];
        i = c;
    }
    if (h->n > 0) h->v[i] = last;
    return top;
}

/* ---- endpoint sweep -------------------------------------------------------------------------- */
typedef struct {
    int64_t e; /* last projected step */
    int64_t c; /* s - p + 1: the job's memory at step x is c + x */
} ep_t;

static int cmp_ep_desc(const void *pa, const void *pb) {
    const ep_t *a = (const ep_t *)pa, *b = (const ep_t *)pb;
    return (a->e < b->e) - (a->e > b->e);
}

/* max over endpoints x of sum_{e_j >= x} (c_j + x) <= M ?  (sorts buf) */
static int endpoints_fit(ep_t *buf, int32_t m, int64_t M) {
    qsort(buf, (size_t)m, sizeof(ep_t), cmp_ep_desc);
    int64_t cnt = 0, sumc = 0;
    int32_t i = 0;
    while (i < m) {
        int64_t x = buf[i].e;
        while (i < m && buf[i].e == x) {
            cnt++;
            sumc += buf[i].c;
            i++;
        }
        if (sumc + cnt * x > M) return 0;
    }
    return 1;
}

/* ---- per-instance validation (Section 2 model; interface requirements) ------------------------ */
static int validate(int policy, int64_t M, int32_t n, const int32_t *a, const int32_t *s,
                    const int32_t *l, const int32_t *u, const int32_t *o, const int32_t *rank) {
    if (policy == O_AR && !rank) return O_E_INVAL;
    for (int32_t i = 0; i < n; i++) {
        if (s[i] < 1 || a[i] < 0 || l[i] < 1 || l[i] > o[i] || o[i] > u[i]) return O_E_INVAL;
        if (policy == O_AR && rank[i] < 0) return O_E_INVAL;
    }
    for (int32_t i = 0; i < n; i++) {
        if ((int64_t)s[i] + o[i] > M) return O_E_INFEASIBLE;
        if ((policy == O_AMAX || policy == O_AELL) && (int64_t)s[i] + u[i] > M) return O_E_INFEASIBLE;
    }
    return O_OK;
}

/* ---- A_min's random eviction ties ---------------------------------------------------------------
 * SplitMix64 (Steele, Lea and Flood, OOPSLA 2014; finalizer of Vigna's public-domain splitmix64.c):
 * output number k >= 1 for a seed is the state seed + k * 0x9E3779B97F4A7C15 (mod 2^64) passed
 * through two xor-shift-multiply rounds and a final xor-shift.  The tie key of request i at step t
 * is the high half of output number (t * 2^32 + i) + 1. */
static uint64_t splitmix64_at(uint64_t seed, uint64_t k) {
    uint64_t z = seed + k * 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

uint32_t oracle_tie_key(uint64_t seed, int64_t t, int32_t i) {
    const uint64_t k = (((uint64_t)t << 32) | (uint32_t)i) + 1u;
    return (uint32_t)(splitmix64_at(seed, k) >> 32);
}

typedef struct {
    int32_t key, idx;
    uint32_t tie; /* random tie key (0 for every job under the index rule) */
    int64_t w;
} evk_t;

static int cmp_evk(const void *pa, const void *pb) {
    const evk_t *a = (const evk_t *)pa, *b = (const evk_t *)pb;
    if (a->key != b->key) return (a->key > b->key) - (a->key < b->key);
    if (a->tie != b->tie) return (a->tie > b->tie) - (a->tie < b->tie);
    return (a->idx > b->idx) - (a->idx < b->idx);
}

typedef struct {
    int64_t a, i;
} arr_t;

static int cmp_arr(const void *pa, const void *pb) {
    const arr_t *x = (const arr_t *)pa, *y = (const arr_t *)pb;
    if (x->a != y->a) return (x->a > y->a) - (x->a < y->a);
    return (x->i > y->i) - (x->i < y->i);
}

int64_t oracle_default_step_cap(int32_t n, const int32_t *o) {
    int64_t so = 0;
    for (int32_t i = 0; i < n; i++) so += o[i];
    return 64 * ((int64_t)n + so);
}

/*
 * Simulate one instance.  step_cap <= 0 selects the default cap 64 * (n + sum o).
 * completion (optional, n entries) receives each request's completion step C_i.
 * rank (A_r only; may be NULL otherwise) is the permutation position of each request.
 * tie_seed seeds A_min's random eviction ties; evict_index != 0 breaks them by index instead.
 */
int oracle_run_full(int policy, int64_t M, int32_t n, const int32_t *a, const int32_t *s,
                    const int32_t *l, const int32_t *u, const int32_t *o, const int32_t *rank,
                    uint64_t tie_seed, int evict_index, int64_t step_cap, oracle_result *res,
                    int64_t *completion, int64_t *time_sums) {
    if (time_sums)
        for (int k = 0; k < 6; k++) time_sums[k] = 0;
    memset(res, 0, sizeof(*res));
    if (completion)
        for (int32_t i = 0; i < n; i++) completion[i] = 0;
    if (policy < 0 || policy > 4 || n < 0) {
        res->status = O_E_INVAL;
        return O_E_INVAL;
    }
    int st = validate(policy, M, n, a, s, l, u, o, rank);
    if (st != O_OK || n == 0) {
        res->status = st;
        return st;
    }
    int64_t cap = step_cap > 0 ? step_cap : oracle_default_step_cap(n, o);

    /* per-request state */
    int64_t *start = (int64_t *)malloc(sizeof(int64_t) * n);
    int32_t *otil = (int32_t *)malloc(sizeof(int32_t) * n);
    int64_t *qkey = (int64_t *)malloc(sizeof(int64_t) * n);
    int32_t *act = (int32_t *)malloc(sizeof(int32_t) * n);
    int32_t *nxt = (int32_t *)malloc(sizeof(int32_t) * n);
    arr_t *arr = (arr_t *)malloc(sizeof(arr_t) * n);
    ep_t *ep = (ep_t *)malloc(sizeof(ep_t) * (size_t)n);
    ep_t *tmp = (ep_t *)malloc(sizeof(ep_t) * (size_t)n);
    evk_t *ev = (evk_t *)malloc(sizeof(evk_t) * n);
    heap_t q;
    q.v = (uint64_t *)malloc(sizeof(uint64_t) * n);
    q.n = 0;
    if (!start || !otil || !qkey || !act || !nxt || !arr || !ep || !tmp || !ev || !q.v) {
        free(start); free(otil); free(qkey); free(act); free(nxt); free(arr); free(ep); free(tmp);
        free(ev); free(q.v);
        res->status = O_E_NOMEM;
        return O_E_NOMEM;
    }
    for (int32_t i = 0; i < n; i++) {
        otil[i] = l[i];
        qkey[i] = 2 * (int64_t)a[i];
        arr[i].a = a[i];
        arr[i].i = i;
    }
    qsort(arr, (size_t)n, sizeof(arr_t), cmp_arr);

    int64_t tel = 0, makespan = 0, peak = 0, evictions = 0, steps = 0, rsteps = 0;
    int64_t memsum = 0, pfsum = 0, xs[4] = {0, 0, 0, 0}; /* batch-time prefix sums and X0..X3 */
    int32_t an = 0, n_done = 0, ap = 0;
    int64_t t = arr[0].a;
    int status = O_OK;

#define EST(i) (policy == O_HSF || policy == O_AR ? o[i] : policy == O_AMAX ? u[i] : otil[i])
#define QKEY(i) (policy == O_AR ? (uint32_t)rank[i] : policy == O_AELL ? (uint32_t)qkey[i] : (uint32_t)EST(i))

    while (n_done < n) {
        if (steps >= cap) {
            status = O_E_STEPCAP;
            break;
        }
        /* arrivals: requests with a_i <= t join the waiting set */
        while (ap < n && arr[ap].a <= t) {
            int32_t i = (int32_t)arr[ap].i;
            xs[0] -= steps;
            xs[1] -= rsteps;
            xs[2] -= memsum;
            xs[3] -= pfsum;
            heap_push(&q, ((uint64_t)QKEY(i) << 32) | (uint32_t)i);
            ap++;
        }
        if (an == 0 && q.n == 0) { /* idle: jump to the next arrival */
            t = arr[ap].a;
            continue;
        }

        /* A_min: overflow of the next step -> evict in ascending (lower bound, tie key, index) */
        if (policy == O_AMIN) {
            int64_t need = 0;
            for (int32_t k = 0; k < an; k++) need += s[act[k]] + (t - start[act[k]]) + 1;
            if (need > M) {
                for (int32_t k = 0; k < an; k++) {
                    int32_t i = act[k];
                    ev[k].key = otil[i];
                    ev[k].idx = i;
                    ev[k].tie = evict_index ? 0u : oracle_tie_key(tie_seed, t, i);
                    ev[k].w = s[i] + (t - start[i]) + 1;
                }
                qsort(ev, (size_t)an, sizeof(evk_t), cmp_evk);
                for (int32_t k = 0; k < an && need > M; k++) {
                    int32_t i = ev[k].idx;
                    int64_t g = t - start[i];
                    need -= ev[k].w;
                    if (g > otil[i]) otil[i] = (int32_t)g;
                    start[i] = -1;
                    evictions++;
                    heap_push(&q, ((uint64_t)(uint32_t)otil[i] << 32) | (uint32_t)i);
                }
                int32_t m = 0;
                for (int32_t k = 0; k < an; k++)
                    if (start[act[k]] >= 0) act[m++] = act[k];
                an = m;
            }
        }

        /* A_ell: a request that used up its estimate unfinished goes to the end of the queue */
        if (policy == O_AELL) {
            int32_t m = 0;
            for (int32_t k = 0; k < an; k++) {
                int32_t i = act[k];
                if (t - start[i] == otil[i]) {
                    otil[i] = u[i];
                    start[i] = -1;
                    qkey[i] = 2 * t + 1;
                    evictions++;
                    heap_push(&q, ((uint64_t)QKEY(i) << 32) | (uint32_t)i);
                } else {
                    act[m++] = i;
                }
            }
            an = m;
        }

        /* admission: largest feasible prefix of the waiting set in (key, index) order */
        int32_t base = 0;
        for (int32_t k = 0; k < an; k++) {
            int32_t i = act[k];
            int64_t e = start[i] + EST(i) - 1;
            if (policy == O_AMIN && e < t) e = t;
            ep[base].e = e;
            ep[base].c = s[i] - start[i] + 1;
            base++;
        }
        int32_t nadm = 0;
        while (q.n > 0) {
            uint64_t top = heap_pop(&q);
            int32_t i = (int32_t)(top & 0xffffffffu);
            ep[base + nadm].e = t + EST(i) - 1;
            ep[base + nadm].c = s[i] - t + 1;
            memcpy(tmp, ep, sizeof(ep_t) * (size_t)(base + nadm + 1));
            if (!endpoints_fit(tmp, base + nadm + 1, M)) {
                heap_push(&q, top);
                break;
            }
            nxt[nadm++] = i;
        }
        for (int32_t k = 0; k < nadm; k++) {
            start[nxt[k]] = t;
            act[an++] = nxt[k];
            pfsum += s[nxt[k]];
        }

        /* process the batch: every member generates one token */
        int64_t mem = 0;
        int32_t m = 0, ncomp = 0;
        for (int32_t k = 0; k < an; k++) {
            int32_t i = act[k];
            int64_t g = t - start[i] + 1;
            mem += s[i] + g;
            if (g == o[i]) {
                int64_t C = t + 1;
                if (completion) completion[i] = C;
                tel += C - a[i];
                if (C > makespan) makespan = C;
                n_done++;
                ncomp++;
            } else {
                act[m++] = i;
            }
        }
        rsteps += an;
        an = m;
        if (mem > peak) peak = mem;
        steps++;
        memsum += mem;
        xs[0] += ncomp * steps; /* prefixes up to C = t + 1 */
        xs[1] += ncomp * rsteps;
        xs[2] += ncomp * memsum;
        xs[3] += ncomp * pfsum;
        t++;
    }
#undef QKEY
#undef EST

    res->total_latency = tel;
    res->makespan = makespan;
    res->peak_memory = peak;
    res->evictions = evictions;
    res->steps = steps;
    res->request_steps = rsteps;
    res->status = status;
    if (time_sums && status == O_OK) {
        for (int k = 0; k < 4; k++) time_sums[k] = xs[k];
        time_sums[4] = memsum;
        time_sums[5] = pfsum;
    }
    free(start); free(otil); free(qkey); free(act); free(nxt); free(arr); free(ep); free(tmp);
    free(ev); free(q.v);
    return status;
}

int oracle_run_seeded(int policy, int64_t M, int32_t n, const int32_t *a, const int32_t *s,
                      const int32_t *l, const int32_t *u, const int32_t *o, const int32_t *rank,
                      uint64_t tie_seed, int evict_index, int64_t step_cap, oracle_result *res,
                      int64_t *completion) {
    return oracle_run_full(policy, M, n, a, s, l, u, o, rank, tie_seed, evict_index, step_cap, res,
                           completion, NULL);
}

int oracle_run_ex(int policy, int64_t M, int32_t n, const int32_t *a, const int32_t *s,
                  const int32_t *l, const int32_t *u, const int32_t *o, const int32_t *rank,
                  int64_t step_cap, oracle_result *res, int64_t *completion) {
    return oracle_run_seeded(policy, M, n, a, s, l, u, o, rank, 0, 0, step_cap, res, completion);
}

int oracle_run(int policy, int64_t M, int32_t n, const int32_t *a, const int32_t *s,
               const int32_t *l, const int32_t *u, const int32_t *o, int64_t step_cap,
               oracle_result *res, int64_t *completion) {
    return oracle_run_ex(policy, M, n, a, s, l, u, o, NULL, step_cap, res, completion);
}

/* ---- many instances (CSR), spread over threads ------------------------------------------------ */
typedef struct {
    int policy;
    int64_t M;
    int32_t n_inst;
    const int64_t *off;
    const int32_t *a, *s, *l, *u, *o, *rank;
    const uint64_t *tie_seed;
    int evict_index;
    int64_t step_cap;
    oracle_result *res;
    int64_t *completion;
    int64_t *time_sums;
    int32_t next;
    pthread_mutex_t mu;
} batch_t;

static void *batch_worker(void *arg) {
    batch_t *b = (batch_t *)arg;
    for (;;) {
        pthread_mutex_lock(&b->mu);
        int32_t i = b->next++;
        pthread_mutex_unlock(&b->mu);
        if (i >= b->n_inst) break;
        int64_t lo = b->off[i], hi = b->off[i + 1];
        oracle_run_full(b->policy, b->M, (int32_t)(hi - lo), b->a + lo, b->s + lo, b->l + lo,
                        b->u + lo, b->o + lo, b->rank ? b->rank + lo : NULL,
                        b->tie_seed ? b->tie_seed[i] : 0, b->evict_index, b->step_cap, &b->res[i],
                        b->completion ? b->completion + lo : NULL,
                        b->time_sums ? b->time_sums + 6 * (int64_t)i : NULL);
    }
    return NULL;
}

/* Many instances (CSR offsets); tie_seed (optional, one per instance, else 0 for all);
 * time_sums (optional, 6 per instance). */
int oracle_run_batch_full(int policy, int64_t M, int32_t n_inst, const int64_t *offsets,
                          const int32_t *a, const int32_t *s, const int32_t *l, const int32_t *u,
                          const int32_t *o, const int32_t *rank, const uint64_t *tie_seed,
                          int evict_index, int64_t step_cap, oracle_result *res,
                          int64_t *completion, int64_t *time_sums, int32_t n_threads) {
    batch_t b;
    b.time_sums = time_sums;
    b.policy = policy;
    b.M = M;
    b.n_inst = n_inst;
    b.off = offsets;
    b.a = a; b.s = s; b.l = l; b.u = u; b.o = o; b.rank = rank;
    b.tie_seed = tie_seed;
    b.evict_index = evict_index;
    b.step_cap = step_cap;
    b.res = res;
    b.completion = completion;
    b.next = 0;
    pthread_mutex_init(&b.mu, NULL);
    if (n_threads < 1) n_threads = 1;
    if (n_threads > 1024) n_threads = 1024;
    pthread_t th[1024];
    int32_t started = 0;
    for (int32_t k = 1; k < n_threads; k++)
        if (pthread_create(&th[started], NULL, batch_worker, &b) == 0) started++;
    batch_worker(&b);
    for (int32_t k = 0; k < started; k++) pthread_join(th[k], NULL);
    pthread_mutex_destroy(&b.mu);
    int worst = O_OK;
    for (int32_t i = 0; i < n_inst; i++)
        if (res[i].status < worst) worst = res[i].status;
    return worst;
}

int oracle_run_batch_seeded(int policy, int64_t M, int32_t n_inst, const int64_t *offsets,
                            const int32_t *a, const int32_t *s, const int32_t *l, const int32_t *u,
                            const int32_t *o, const int32_t *rank, const uint64_t *tie_seed,
                            int evict_index, int64_t step_cap, oracle_result *res,
                            int64_t *completion, int32_t n_threads) {
    return oracle_run_batch_full(policy, M, n_inst, offsets, a, s, l, u, o, rank, tie_seed,
                                 evict_index, step_cap, res, completion, NULL, n_threads);
}

int oracle_run_batch_ex(int policy, int64_t M, int32_t n_inst, const int64_t *offsets,
                        const int32_t *a, const int32_t *s, const int32_t *l, const int32_t *u,
                        const int32_t *o, const int32_t *rank, int64_t step_cap, oracle_result *res,
                        int64_t *completion, int32_t n_threads) {
    return oracle_run_batch_seeded(policy, M, n_inst, offsets, a, s, l, u, o, rank, NULL, 0,
                                   step_cap, res, completion, n_threads);
}

int oracle_run_batch(int policy, int64_t M, int32_t n_inst, const int64_t *offsets,
                     const int32_t *a, const int32_t *s, const int32_t *l, const int32_t *u,
                     const int32_t *o, int64_t step_cap, oracle_result *res, int64_t *completion,
                     int32_t n_threads) {
    return oracle_run_batch_ex(policy, M, n_inst, offsets, a, s, l, u, o, NULL, step_cap, res,
                               completion, n_threads);
}

/*
 * Total latency and makespan in time units under the linear batch-time model
 * coef = (c0, c1, c2, c3, c_idle) (Section 6): from time_sums = [X0, X1, X2, X3, F2, F3] and the
 * result's steps (F0), request steps (F1) and makespan (F4 = makespan - steps),
 *   out[0] = c0 X0 + c1 X1 + c2 X2 + c3 X3,
 *   out[1] = c0 F0 + c1 F1 + c2 F2 + c3 F3 + c_idle F4,
 * each evaluated left to right in IEEE double (built without contraction into fused multiply-adds);
 * NaN for an instance that did not finish.
 */
void oracle_batch_time(const int64_t *time_sums, const oracle_result *res, const double *coef, double *out) {
    if (res->status != O_OK) {
        out[0] = out[1] = NAN;
        return;
    }
    const double x0 = (double)time_sums[0], x1 = (double)time_sums[1], x2 = (double)time_sums[2];
    const double x3 = (double)time_sums[3], f2 = (double)time_sums[4], f3 = (double)time_sums[5];
    out[0] = coef[0] * x0 + coef[1] * x1 + coef[2] * x2 + coef[3] * x3;
    out[1] = coef[0] * (double)res->steps + coef[1] * (double)res->request_steps + coef[2] * f2 +
             coef[3] * f3 + coef[4] * (double)(res->makespan - res->steps);
}

