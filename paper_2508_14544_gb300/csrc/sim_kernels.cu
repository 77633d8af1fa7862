// CUDA kernels of the batched scheduler simulator (sm_103a).
//
//   k_stage  - per instance: validate the requests (Section 2 model), compute TEL/step-cap
//              constants, and sort the requests by (arrival step, policy key, index) so that every
//              arrival batch is already ordered the way the waiting set R_t is sorted
//              (Algorithm malb: key u; Algorithm milb/milbrevise: key l; Algorithm off: key o).
//   k_run    - one warp simulates one instance at a time, step by step (persistent warps pulling
//              instance ids from a work queue).  Per step: arrivals join R_t; A_min resolves an
//              overflow of the next step by cancelling in ascending (estimate, index) order
//              (Algorithm milb); the head of R_t is admitted while the future-memory check of
//              eq. Constraint holds (largest feasible prefix); the batch is processed (one token per
//              member, eq. constraintM accounting, completions, TEL of eq. latency).
//   k_ratio  - per-instance competitive ratio TEL(pi) / TEL(H-SF) (Definition cr).
//
// Active set layout (per warp, shared memory when it fits): structure-of-arrays sorted by the
// projected last step E (ascending):
//   E = p + Lhat - 1   projected last step (Lhat = u, o or the A_min estimate)
//   F = p + o - 1      true last step (completion at step F, C = F + 1)
//   B = s - p + 1      so the job's memory at step x is B + x
//   P = p, I = request index, K = the estimate (A_min sort key)
// Derived arrays, rebuilt whenever the set changes, relative to a time base tb:
//   SB[i] = sum_{j >= i} (B_j + tb)                      (suffix sums; SB[A] = 0)
//   PM[h] = max_{i < h} (SB[i] + (A - i)(E_i - tb) + E_i - tb)   (prefix maxima; PM[0] = -inf)
// With these, the future memory of the active set at its endpoint E_i is
// V(E_i) = SB[i] + (A - i)(E_i - tb) (exact for the first entry of each group of equal E, and a
// lower bound for the others, so maxima are exact), and the check "the head of R_t, started now,
// keeps every future step within M" costs O(1) per step (see head_fits).
#include <climits>
#include <cstdint>

#include "sim_internal.h"

namespace simgb {

namespace {

constexpr unsigned FULL = 0xffffffffu;
enum { P_AMAX = 0, P_AMIN = 1, P_HSF = 2 };
enum { ST_OK = 0, ST_INVAL = -1, ST_INFEASIBLE = -2, ST_STEPCAP = -3, ST_STATE = -5 };

__device__ __forceinline__ bool qless(const QEnt &a, const QEnt &b) {
    return a.key < b.key || (a.key == b.key && a.idx < b.idx);
}

__device__ __forceinline__ int lane_id() { return threadIdx.x & 31; }

__device__ __forceinline__ int64_t warp_sum64(int64_t v) {
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1) v += __shfl_xor_sync(FULL, v, d);
    return v;
}

__device__ __forceinline__ int warp_min32(int v) {
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1) v = min(v, __shfl_xor_sync(FULL, v, d));
    return v;
}

__device__ __forceinline__ int sat32(int64_t v) {
    const int64_t hi = int64_t(1) << 30;
    if (v > hi) return int(hi);
    if (v < -hi) return int(-hi);
    return int(v);
}

__device__ __forceinline__ QEnt shfl_q(const QEnt &q, int src) {
    QEnt r;
    r.key = __shfl_sync(FULL, q.key, src);
    r.idx = __shfl_sync(FULL, q.idx, src);
    r.s = __shfl_sync(FULL, q.s, src);
    r.o = __shfl_sync(FULL, q.o, src);
    return r;
}

// Number of leading positions i in [0, len) with pred(i) true, for a predicate that is true on a
// prefix.  Two ballots over 32 samples: O(1) dependent loads for len <= 1024.
template <class Pred>
__device__ __forceinline__ int warp_prefix_count(int len, Pred pred) {
    if (len <= 0) return 0;
    const int lane = lane_id();
    const int c = (len + 31) >> 5;
    const int pos = min((lane + 1) * c - 1, len - 1);
    const int full = __popc(__ballot_sync(FULL, pred(pos)));
    int cnt = full * c;
    if (cnt >= len) return len;
    const int end = min(cnt + c, len);
    for (int off = cnt; off < end; off += 32) {
        const int i = off + lane;
        const unsigned b = __ballot_sync(FULL, i < end && pred(i));
        const int k = __popc(b);
        cnt += k;
        if (k < 32) break;
    }
    return cnt;
}

// ---------------------------------------------------------------------------------------------
// Per-warp workspace
// ---------------------------------------------------------------------------------------------
struct Ws {
    int32_t *E, *F, *B, *P, *I, *K;  // active set, capacity ca
    int32_t *SB, *PM;                // ca + 1
    QEnt *dq;                        // delta queue, capacity dcap, sorted DESCENDING (head at the end)
    int32_t *cnt;                    // dcap + 1 (merge histogram)
    QEnt *mb0, *mb1;                 // global ping-pong main-queue buffers
    int32_t ca, dcap;
};

__host__ __device__ inline size_t ws_bytes_impl(int ca, int dcap) {
    size_t b = 0;
    b += size_t(6) * ca * sizeof(int32_t);
    b += size_t(2) * (ca + 1) * sizeof(int32_t);
    b = (b + 15) & ~size_t(15);
    b += size_t(dcap) * sizeof(QEnt);
    b += size_t(dcap + 1) * sizeof(int32_t);
    b = (b + 15) & ~size_t(15);
    return b;
}

__device__ inline Ws carve_ws(unsigned char *base, int ca, int dcap) {
    Ws w;
    int32_t *p = reinterpret_cast<int32_t *>(base);
    w.E = p; p += ca;
    w.F = p; p += ca;
    w.B = p; p += ca;
    w.P = p; p += ca;
    w.I = p; p += ca;
    w.K = p; p += ca;
    w.SB = p; p += ca + 1;
    w.PM = p; p += ca + 1;
    size_t off = (reinterpret_cast<unsigned char *>(p) - base);
    off = (off + 15) & ~size_t(15);
    w.dq = reinterpret_cast<QEnt *>(base + off);
    w.cnt = reinterpret_cast<int32_t *>(w.dq + dcap);
    w.ca = ca;
    w.dcap = dcap;
    return w;
}

// ---------------------------------------------------------------------------------------------
// Waiting set R_t: a sorted main array in global memory [mh, me) plus a small sorted delta array
// (the workspace, descending so that its head is the last element).  Together they hold R_t in
// (key, idx) order.  Inserts go to the delta; a full delta is merged into the main array.
// ---------------------------------------------------------------------------------------------
struct Queue {
    const QEnt *mq;  // main array (global, ascending); may point into the staged records
    int mh, me;      // head / end
    int mbuf;        // -1: mq is read-only staged data; 0/1: ping-pong buffer in use
    int dn;          // delta size
    int mcb;         // main head cache base (lane l caches mq[mcb + l]), -1 invalid
    QEnt mc;         // this lane's cached main entry
};

__device__ __forceinline__ bool queue_empty(const Queue &q) { return q.mh >= q.me && q.dn == 0; }

// Merge the delta into the main array (into the other ping-pong buffer).
__device__ void merge_delta(const Ws &w, Queue &q) {
    const int lane = lane_id();
    const int dn = q.dn;
    const int nx = q.me - q.mh;
    QEnt *out = (q.mbuf == 0) ? w.mb1 : w.mb0;
    const QEnt *X = q.mq + q.mh;
    // delta ascending view: Yasc(j) = dq[dn - 1 - j]
    for (int j = lane; j <= dn; j += 32) w.cnt[j] = 0;
    __syncwarp();
    const int c = (nx + 31) >> 5;
    const int s0 = lane * c;
    const int s1 = min(s0 + c, nx);
    if (s0 < s1) {
        // r = #Y < X[s0]  (binary search over the ascending view)
        const QEnt x0 = X[s0];
        int lo = 0, hi = dn;
        while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (qless(w.dq[dn - 1 - mid], x0)) lo = mid + 1; else hi = mid;
        }
        int r = lo, run_r = lo, run_len = 0;
        for (int i = s0; i < s1; ++i) {
            const QEnt x = X[i];
            while (r < dn && qless(w.dq[dn - 1 - r], x)) ++r;
            out[i + r] = x;
            if (r != run_r) {
                if (run_len) atomicAdd(&w.cnt[run_r], run_len);
                run_r = r;
                run_len = 0;
            }
            ++run_len;
        }
        if (run_len) atomicAdd(&w.cnt[run_r], run_len);
    }
    __syncwarp();
    // delta element j (ascending) goes to j + sum_{r <= j} cnt[r]
    int carry = 0;
    for (int c0 = 0; c0 < dn; c0 += 32) {
        const int j = c0 + lane;
        int v = (j < dn) ? w.cnt[j] : 0;
#pragma unroll
        for (int d = 1; d < 32; d <<= 1) {
            const int y = __shfl_up_sync(FULL, v, d);
            if (lane >= d) v += y;
        }
        v += carry;
        if (j < dn) out[j + v] = w.dq[dn - 1 - j];
        carry = __shfl_sync(FULL, v, 31);
    }
    __syncwarp();
    __threadfence_block();
    q.mq = out;
    q.mbuf = (q.mbuf == 0) ? 1 : 0;
    q.mh = 0;
    q.me = nx + dn;
    q.dn = 0;
    q.mcb = -1;
}

// Insert one entry into the delta (merging the delta into main first if it is full).
__device__ void delta_insert(const Ws &w, Queue &q, const QEnt &e) {
    const int lane = lane_id();
    if (q.dn == w.dcap) merge_delta(w, q);
    const int dn = q.dn;
    // descending order: pos = #entries greater than e
    const int pos = warp_prefix_count(dn, [&](int i) { return qless(e, w.dq[i]); });
    for (int hi = dn; hi > pos; hi -= 32) {
        const int lo = max(pos, hi - 32);
        const int i = lo + lane;
        QEnt v;
        const bool act = i < hi;
        if (act) v = w.dq[i];
        __syncwarp();
        if (act) w.dq[i + 1] = v;
        __syncwarp();
    }
    if (lane == 0) w.dq[pos] = e;
    __syncwarp();
    q.dn = dn + 1;
}

// Head of R_t (smallest (key, idx)); the queue must not be empty.  src: 0 main, 1 delta.
__device__ __forceinline__ QEnt queue_head(const Ws &w, Queue &q, int &src) {
    const int lane = lane_id();
    bool have_m = q.mh < q.me;
    QEnt hm, hd;
    if (have_m) {
        if (q.mcb < 0 || q.mh < q.mcb || q.mh >= q.mcb + 32) {
            q.mcb = q.mh;
            const int i = q.mcb + lane;
            if (i < q.me) q.mc = q.mq[i];
        }
        hm = shfl_q(q.mc, q.mh - q.mcb);
    }
    if (q.dn > 0) hd = w.dq[q.dn - 1];
    if (have_m && (q.dn == 0 || qless(hm, hd))) {
        src = 0;
        return hm;
    }
    src = 1;
    return hd;
}

__device__ __forceinline__ void queue_pop(Queue &q, int src) {
    if (src == 0) ++q.mh; else --q.dn;
}

// Arrival batch (ascending, global): becomes the main array if R_t is empty; a few entries go
// into the delta one by one; a long batch is copied into the (emptied) delta in chunks, each
// chunk merged into the main array.
__device__ void insert_run(const Ws &w, Queue &q, const QEnt *run, int len) {
    const int lane = lane_id();
    if (len <= 0) return;
    if (queue_empty(q)) {
        q.mq = run;
        q.mh = 0;
        q.me = len;
        q.mbuf = -1;
        q.mcb = -1;
        return;
    }
    int done = 0;
    while (done < len) {
        const int rem = len - done;
        if (rem <= 8) {
            for (int j = 0; j < rem; ++j) delta_insert(w, q, run[done + j]);
            break;
        }
        if (q.dn > 0) merge_delta(w, q);
        const int k = min(rem, w.dcap);
        for (int j = lane; j < k; j += 32) w.dq[j] = run[done + k - 1 - j];  // descending
        __syncwarp();
        q.dn = k;
        done += k;
    }
}

// ---------------------------------------------------------------------------------------------
// Active set maintenance
// ---------------------------------------------------------------------------------------------
// Rebuild SB / PM for the current A entries relative to time base tb; also returns min F.
__device__ void rebuild(const Ws &w, int A, int tb, int &SB0, int &nextF) {
    const int lane = lane_id();
    int carry = 0;
    if (A > 0) {
        for (int c0 = ((A - 1) >> 5) << 5; c0 >= 0; c0 -= 32) {
            const int i = c0 + lane;
            int x = (i < A) ? w.B[i] + tb : 0;
#pragma unroll
            for (int d = 1; d < 32; d <<= 1) {
                const int y = __shfl_down_sync(FULL, x, d);
                if (lane + d < 32) x += y;
            }
            x += carry;
            if (i < A) w.SB[i] = x;
            carry = __shfl_sync(FULL, x, 0);
        }
    }
    if (lane == 0) {
        w.SB[A] = 0;
        w.PM[0] = INT_MIN;
    }
    SB0 = carry;
    __syncwarp();
    int run = INT_MIN;
    int fmin = INT_MAX;
    for (int c0 = 0; c0 < A; c0 += 32) {
        const int i = c0 + lane;
        int h = INT_MIN;
        if (i < A) {
            const int64_t e = int64_t(w.E[i]) - tb;
            h = sat32(int64_t(w.SB[i]) + int64_t(A - i) * e + e);
            fmin = min(fmin, w.F[i]);
        }
#pragma unroll
        for (int d = 1; d < 32; d <<= 1) {
            const int y = __shfl_up_sync(FULL, h, d);
            if (lane >= d) h = max(h, y);
        }
        h = max(h, run);
        if (i < A) w.PM[i + 1] = h;
        run = __shfl_sync(FULL, h, 31);
    }
    nextF = warp_min32(fmin);
    __syncwarp();
}

// Remove entries marked dead (F < 0), keeping the order.  Returns the new size.
__device__ int compact(const Ws &w, int A) {
    const int lane = lane_id();
    int wpos = 0;
    for (int c0 = 0; c0 < A; c0 += 32) {
        const int i = c0 + lane;
        const bool in = i < A;
        int e = 0, f = -1, b = 0, p = 0, id = 0, k = 0;
        if (in) {
            f = w.F[i];
            e = w.E[i];
            b = w.B[i];
            p = w.P[i];
            id = w.I[i];
            k = w.K[i];
        }
        const bool live = in && f >= 0;
        const unsigned bal = __ballot_sync(FULL, live);
        const int dst = wpos + __popc(bal & ((1u << lane) - 1u));
        __syncwarp();
        if (live) {
            w.E[dst] = e;
            w.F[dst] = f;
            w.B[dst] = b;
            w.P[dst] = p;
            w.I[dst] = id;
            w.K[dst] = k;
        }
        __syncwarp();
        wpos += __popc(bal);
    }
    return wpos;
}

// Insert one active job keeping E ascending (after equal E).  Returns false if full.
__device__ bool insert_active(const Ws &w, int &A, int e, int f, int b, int p, int id, int k) {
    const int lane = lane_id();
    if (A >= w.ca) return false;
    const int pos = warp_prefix_count(A, [&](int i) { return w.E[i] <= e; });
    for (int hi = A; hi > pos; hi -= 32) {
        const int lo = max(pos, hi - 32);
        const int i = lo + lane;
        const bool act = i < hi;
        int ve = 0, vf = 0, vb = 0, vp = 0, vi = 0, vk = 0;
        if (act) {
            ve = w.E[i];
            vf = w.F[i];
            vb = w.B[i];
            vp = w.P[i];
            vi = w.I[i];
            vk = w.K[i];
        }
        __syncwarp();
        if (act) {
            w.E[i + 1] = ve;
            w.F[i + 1] = vf;
            w.B[i + 1] = vb;
            w.P[i + 1] = vp;
            w.I[i + 1] = vi;
            w.K[i + 1] = vk;
        }
        __syncwarp();
    }
    if (lane == 0) {
        w.E[pos] = e;
        w.F[pos] = f;
        w.B[pos] = b;
        w.P[pos] = p;
        w.I[pos] = id;
        w.K[pos] = k;
    }
    __syncwarp();
    ++A;
    return true;
}

// ---------------------------------------------------------------------------------------------
// One instance, simulated by one warp.  All lanes hold identical copies of the scalar state.
// ---------------------------------------------------------------------------------------------
template <int POL>
__device__ void sim_instance(const RunParams &P, const Ws &w, int inst) {
    const int lane = lane_id();
    const InstInfo info = P.info[inst];
    DevResult r;
    r.total_latency = r.makespan = r.peak_memory = r.evictions = r.steps = r.request_steps = 0;
    r.status = info.status;
    r.pad = 0;
    if (info.status != ST_OK || info.n == 0) {
        if (lane == 0) P.res[inst] = r;
        return;
    }
    const int n = info.n;
    const QEnt *rec = P.rec + info.base;
    const int32_t *ra = P.rec_a + info.base;
    const int64_t M = P.M;
    const int64_t cap = info.cap;

    Queue q;
    q.mq = rec;
    q.mh = q.me = 0;
    q.mbuf = -1;
    q.dn = 0;
    q.mcb = -1;

    int A = 0, tb = 0, SB0 = 0, nextF = INT_MAX;
    int t = ra[0];
    int ap = 0;
    int next_a = t;
    int64_t sumC = 0, peak = 0, steps = 0, rsteps = 0, nev = 0;
    int64_t makespan = 0;
    int ndone = 0;
    int status = ST_OK;

    bool hvalid = false;
    QEnt h;
    int hsrc = 0;
    bool pdirty = true;
    int64_t y_prev = 0;
    int hi = 0, lb = 0;

    for (;;) {
        if (steps >= cap) {
            status = ST_STEPCAP;
            break;
        }
        // ---- S1: arrivals with a <= t join R_t (a sorted run of the staged records)
        if (ap < n && next_a <= t) {
            int ae = ap;
            for (;;) {
                const int i = ae + lane;
                const bool ok = i < n && ra[i] <= t;
                const unsigned b = __ballot_sync(FULL, ok);
                const int k = __popc(b);
                ae += k;
                if (k < 32) break;
            }
            insert_run(w, q, rec + ap, ae - ap);
            ap = ae;
            next_a = (ap < n) ? ra[ap] : INT_MAX;
            hvalid = false;
        }
        if (A == 0 && queue_empty(q)) {
            if (ap >= n) {
                status = ST_STATE;
                break;
            }
            t = next_a;  // idle: jump to the next arrival
            continue;
        }
        // ---- S2/S3: A_min overflow of the next step -> cancel in ascending (estimate, index)
        if (POL == P_AMIN) {
            int64_t need = int64_t(SB0) + int64_t(A) * (t - tb);
            if (need > M) {
                while (need > M) {
                    unsigned long long best = ~0ull;
                    int bi = -1;
                    for (int i = lane; i < A; i += 32) {
                        if (w.F[i] >= 0) {
                            const unsigned long long kk =
                                (static_cast<unsigned long long>(static_cast<unsigned>(w.K[i])) << 32) |
                                static_cast<unsigned>(w.I[i]);
                            if (kk < best) {
                                best = kk;
                                bi = i;
                            }
                        }
                    }
#pragma unroll
                    for (int d = 16; d >= 1; d >>= 1) {
                        const unsigned long long ob = __shfl_xor_sync(FULL, best, d);
                        const int oi = __shfl_xor_sync(FULL, bi, d);
                        if (ob < best) {
                            best = ob;
                            bi = oi;
                        }
                    }
                    if (bi < 0) {
                        status = ST_STATE;
                        break;
                    }
                    const int b = w.B[bi], p = w.P[bi], f = w.F[bi], k = w.K[bi], id = w.I[bi];
                    __syncwarp();
                    if (lane == 0) w.F[bi] = -1;
                    __syncwarp();
                    QEnt e;
                    e.key = max(k, t - p);  // refined lower bound: max(estimate, tokens generated)
                    e.idx = id;
                    e.s = b + p - 1;
                    e.o = f - p + 1;
                    need -= int64_t(b) + t;
                    ++nev;
                    delta_insert(w, q, e);
                }
                if (status != ST_OK) break;
                A = compact(w, A);
                tb = t;
                rebuild(w, A, tb, SB0, nextF);
                hvalid = false;
                pdirty = true;
            }
        }
        // ---- S4/S5: admit the head of R_t while it fits (largest feasible prefix)
        for (;;) {
            if (!hvalid) {
                if (queue_empty(q)) break;
                h = queue_head(w, q, hsrc);
                hvalid = true;
                pdirty = true;
            }
            const int64_t dt = int64_t(t) - tb;
            const int64_t need = int64_t(SB0) + int64_t(A) * dt;
            bool fits = need + h.s + 1 <= M;
            if (fits && A > 0) {
                const int64_t y = int64_t(t) + h.key - 1;
                if (pdirty || y != y_prev + 1) {
                    hi = warp_prefix_count(A, [&](int i) { return w.E[i] <= y; });
                    lb = warp_prefix_count(hi, [&](int i) { return w.E[i] < y; });
                } else {
                    lb = hi;
                    while (hi < A && w.E[hi] <= y) ++hi;
                }
                pdirty = false;
                y_prev = y;
                const int pm = w.PM[hi];
                if (int64_t(pm) + h.s + 1 - dt > M) fits = false;
                const int64_t v = int64_t(w.SB[lb]) + int64_t(A - lb) * (y - tb);
                if (v + h.s + h.key > M) fits = false;
            } else if (fits) {
                fits = int64_t(h.s) + h.key <= M;
            }
            if (!fits) break;
            queue_pop(q, hsrc);
            const int e = t + h.key - 1;
            const int f = t + h.o - 1;
            if (!insert_active(w, A, e, f, h.s - t + 1, t, h.idx, h.key)) {
                status = kStatusCapacity;
                break;
            }
            tb = t;
            rebuild(w, A, tb, SB0, nextF);
            hvalid = false;
            pdirty = true;
        }
        if (status != ST_OK) break;
        // ---- S6: process the batch
        const int64_t mem = int64_t(SB0) + int64_t(A) * (int64_t(t) - tb);
        if (mem > M) {
            status = ST_STATE;
            break;
        }
        if (mem > peak) peak = mem;
        rsteps += A;
        ++steps;
        if (t == nextF) {
            int c = 0;
            for (int i = lane; i < A; i += 32) {
                if (w.F[i] == t) {
                    ++c;
                    if (P.completion) P.completion[info.base + w.I[i]] = int64_t(t) + 1;
                    w.F[i] = -1;
                }
            }
            c = int(warp_sum64(c));
            __syncwarp();
            sumC += int64_t(c) * (int64_t(t) + 1);
            makespan = int64_t(t) + 1;
            ndone += c;
            A = compact(w, A);
            tb = t + 1;
            rebuild(w, A, tb, SB0, nextF);
            pdirty = true;
            if (ndone >= n) break;
        }
        ++t;
    }
    if (lane == 0) {
        r.status = status;
        r.total_latency = sumC - info.sum_a;
        r.makespan = makespan;
        r.peak_memory = peak;
        r.evictions = nev;
        r.steps = steps;
        r.request_steps = rsteps;
        P.res[inst] = r;
    }
    __syncwarp();
}

template <int POL>
__global__ void __launch_bounds__(256) k_run(RunParams P) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int lane = lane_id();
    const int wib = threadIdx.x >> 5;
    const int64_t slot = int64_t(blockIdx.x) * (blockDim.x >> 5) + wib;
    unsigned char *base = P.use_smem ? smem_raw + size_t(wib) * ws_bytes_impl(P.ca, P.dcap)
                                     : P.gws + slot * P.gws_stride;
    Ws w = carve_ws(base, P.ca, P.dcap);
    w.mb0 = P.mainbuf + slot * 2 * P.main_cap;
    w.mb1 = w.mb0 + P.main_cap;
    for (;;) {
        int k = 0;
        if (lane == 0) k = atomicAdd(P.counter, 1);
        k = __shfl_sync(FULL, k, 0);
        if (k >= P.n_work) break;
        const int inst = P.work ? P.work[k] : k;
        sim_instance<POL>(P, w, inst);
    }
}

// ---------------------------------------------------------------------------------------------
// Staging: validate, constants, sort by (a, key, idx)
// ---------------------------------------------------------------------------------------------
__device__ __forceinline__ bool stage_less(int aa, const QEnt &x, int ab, const QEnt &y) {
    if (aa != ab) return aa < ab;
    if (x.key != y.key) return x.key < y.key;
    return x.idx < y.idx;
}

template <typename T>
__device__ T block_reduce(T v, T *sh, bool is_max) {
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = blockDim.x >> 5;
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1) {
        const T o = __shfl_xor_sync(FULL, v, d);
        v = is_max ? (o > v ? o : v) : v + o;
    }
    __syncthreads();
    if (lane == 0) sh[wid] = v;
    __syncthreads();
    T acc = sh[0];
    for (int i = 1; i < nw; ++i) acc = is_max ? (sh[i] > acc ? sh[i] : acc) : acc + sh[i];
    return acc;
}

__global__ void __launch_bounds__(256) k_stage(StageParams S) {
    __shared__ int64_t sh64[32];
    const int inst = blockIdx.x;
    const int64_t base = S.off[inst];
    const int n = int(S.off[inst + 1] - base);
    int64_t bad_inval = 0, bad_inf = 0, sum_a = 0, sum_o = 0, work = 0;
    for (int j = threadIdx.x; j < n; j += blockDim.x) {
        const int64_t g = base + j;
        const int a = S.a[g], s = S.s[g], l = S.l[g], u = S.u[g], o = S.o[g];
        if (s < 1 || a < 0 || l < 1 || l > o || o > u) bad_inval = 1;
        if (int64_t(s) + o > S.M) bad_inf = 1;
        if (S.policy == P_AMAX && int64_t(s) + u > S.M) bad_inf = 1;
        const int key = (S.policy == P_AMAX) ? u : (S.policy == P_HSF ? o : l);
        QEnt e;
        e.key = key;
        e.idx = j;
        e.s = s;
        e.o = o;
        S.rec[g] = e;
        S.rec_a[g] = a;
        sum_a += a;
        sum_o += o;
        work += int64_t(s) * o + int64_t(o) * o / 2;
    }
    bad_inval = block_reduce<int64_t>(bad_inval, sh64, true);
    bad_inf = block_reduce<int64_t>(bad_inf, sh64, true);
    sum_a = block_reduce<int64_t>(sum_a, sh64, false);
    sum_o = block_reduce<int64_t>(sum_o, sh64, false);
    work = block_reduce<int64_t>(work, sh64, false);
    int status = ST_OK;
    if (bad_inval) status = ST_INVAL;
    else if (bad_inf) status = ST_INFEASIBLE;
    if (threadIdx.x == 0) {
        InstInfo in;
        in.base = base;
        in.n = n;
        in.status = status;
        in.sum_a = sum_a;
        in.cap = S.step_cap > 0 ? S.step_cap : 64 * (int64_t(n) + sum_o);
        in.work = work;
        S.info[inst] = in;
    }
    if (status != ST_OK || n <= 1) return;
    __syncthreads();
    // bitonic sort of [base, base + n) by (a, key, idx), padded virtually to a power of two
    int N = 1;
    while (N < n) N <<= 1;
    QEnt *R = S.rec + base;
    int32_t *RA = S.rec_a + base;
    for (int k = 2; k <= N; k <<= 1) {
        for (int p = threadIdx.x; p < N / 2; p += blockDim.x) {
            const int half = k >> 1;
            const int i = (p / half) * k + (p % half);
            const int j = i ^ (k - 1);
            if (j < n) {
                const QEnt x = R[i], y = R[j];
                const int ax = RA[i], ay = RA[j];
                if (stage_less(ay, y, ax, x)) {
                    R[i] = y;
                    R[j] = x;
                    RA[i] = ay;
                    RA[j] = ax;
                }
            }
        }
        __syncthreads();
        for (int d = k >> 2; d >= 1; d >>= 1) {
            for (int p = threadIdx.x; p < N / 2; p += blockDim.x) {
                const int i = (p / d) * 2 * d + (p % d);
                const int j = i + d;
                if (j < n) {
                    const QEnt x = R[i], y = R[j];
                    const int ax = RA[i], ay = RA[j];
                    if (stage_less(ay, y, ax, x)) {
                        R[i] = y;
                        R[j] = x;
                        RA[i] = ay;
                        RA[j] = ax;
                    }
                }
            }
            __syncthreads();
        }
    }
}

__global__ void k_ratio(const DevResult *pol, const DevResult *ref, double *out, int32_t n) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= n) return;
    const DevResult a = pol[i], b = ref[i];
    double v = __longlong_as_double(0x7ff8000000000000ll);  // NaN
    if (a.status == ST_OK && b.status == ST_OK && b.total_latency > 0)
        v = double(a.total_latency) / double(b.total_latency);
    out[i] = v;
}

}  // namespace

size_t warp_ws_bytes(int ca, int dcap) { return ws_bytes_impl(ca, dcap); }

cudaError_t launch_stage(const StageParams &p, cudaStream_t st) {
    if (p.n_inst <= 0) return cudaSuccess;
    k_stage<<<p.n_inst, 256, 0, st>>>(p);
    return cudaGetLastError();
}

cudaError_t set_run_smem_limit(int policy, size_t bytes) {
    const void *fn = policy == P_AMAX ? (const void *)k_run<P_AMAX>
                   : policy == P_AMIN ? (const void *)k_run<P_AMIN>
                                      : (const void *)k_run<P_HSF>;
    return cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, int(bytes));
}

cudaError_t launch_run(int policy, const RunParams &p, int blocks, int warps_per_block, size_t smem_bytes,
                       cudaStream_t st) {
    const dim3 grid(blocks), block(32 * warps_per_block);
    switch (policy) {
        case P_AMAX: k_run<P_AMAX><<<grid, block, smem_bytes, st>>>(p); break;
        case P_AMIN: k_run<P_AMIN><<<grid, block, smem_bytes, st>>>(p); break;
        default: k_run<P_HSF><<<grid, block, smem_bytes, st>>>(p); break;
    }
    return cudaGetLastError();
}

cudaError_t launch_ratio(const DevResult *pol, const DevResult *ref, double *out, int32_t n, cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    k_ratio<<<(n + 255) / 256, 256, 0, st>>>(pol, ref, out, n);
    return cudaGetLastError();
}

}  // namespace simgb
