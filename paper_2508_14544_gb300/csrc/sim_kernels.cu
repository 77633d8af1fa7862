// Simulation kernel of the batched scheduler simulator (sm_103a): k_run<policy, shared, instrumented, layout>.
//
// One warp simulates one instance at a time (persistent warps pull instance ids from a work
// queue).  Each step follows the paper's algorithms:
//   S1  arrivals with a_i <= t join the waiting set R_t (extension: the paper has a_i = 0);
//   S3  A_min only (Algorithm milb): if the next step of the active set would exceed M, cancel
//       jobs in ascending estimate order, ties broken uniformly at random by a key drawn afresh
//       at every step (SplitMix64 of the instance's seed and the counter t * 2^32 + index, then
//       the index), until it fits; each cancelled job's estimate becomes max(estimate, tokens
//       generated) and it re-enters R_t in the same step (the cancelled jobs stay in the
//       active-set arrays, marked, until something reads those arrays: see the S2/S3 block);
//   S5  admit the largest prefix of R_t (sorted by (key, index)) for which eq. Constraint holds at
//       every future step (Algorithms malb / milb / off);
//   S6  process the batch: one token per member, the step's memory sum(s + tokens) (eq.
//       constraintM), completions, TEL (eq. latency).
// Two more policies share the loop: A_r (Algorithm random: the queue key is a given permutation
// rank, the projected length the true o) and A_ell (Algorithm promote_l: FIFO queue, estimate l;
// at the start of a step a job that used up its estimate unfinished is removed, takes u and
// re-enters the queue at its end; the queue key is 2 a on arrival and 2 t + 1 on re-entry).
//
// Active set (per warp, shared memory; a global-memory workspace of the same layout serves
// instances that outgrow it), structure of arrays sorted by the projected last step E:
//   E = p + Lhat - 1   projected last step (Lhat = u, o or the A_min estimate)
//   F = p + o - 1      true last step (completion at step F, C = F + 1); F = -1 marks a cancelled
//                      (A_min) or promoted (A_ell) job
//   B = s - p + 1      the job's memory at step x is B + x
//   P = p, I = request index, K = the estimate (A_min key)
// Derived arrays, recomputed in one warp pass whenever the set changes (after A_min
// cancellations: when they are next read), relative to a time base tb:
//   SB[i] = sum_{j >= i} (B_j + tb),  SB[A] = 0                    (suffix sums)
//   PM[h] = max_{i < h} H_i,  H_i = SB[i] + (A - i)(E_i - tb) + (E_i - tb),  PM[0] = -inf
// V(x) = SB[lb] + (A - lb)(x - tb), lb = #{E < x}, is the projected memory of the active set at
// step x (eq. Constraint restricted to S'); H_i is V(E_i) + E_i - tb for the first entry of each
// group of equal E and a lower bound for the others, so prefix maxima are exact.  The head
// candidate (prompt s, estimate L) started at step t fits iff
//   (1) SB[0] + A (t - tb) + s + 1 <= M                 (the coming step),
//   (2) PM[#{E <= y}] + s + 1 - (t - tb) <= M            (every active endpoint it covers),
//   (3) V(y) + s + L <= M,  y = t + L - 1                (its own last step),
// so a step in which nothing changes costs O(1), and a run of such steps is processed in closed
// form up to the next event (completion, arrival, A_min overflow, or the first step at which
// the head fits, found by scanning the segments between active endpoints).  When the head fits,
// the whole admitted prefix is found at once on a window of the first 32 entries of R_t: with
// CS[k] = sum_{m<k} (s_m + 1), prefix k adds CS[k] - CS[r] + (k - r)(x - t) to the projected
// memory at step x, where r counts the window entries that end before x; each point (x = t,
// every active endpoint, every window entry's endpoint) yields the first k at which it exceeds
// M, and the admitted count is the minimum of those, less one.
#include <climits>
#include <cstdint>
#include <type_traits>

#include "sim_internal.h"

namespace simgb {

namespace {

constexpr unsigned FULL = 0xffffffffu;
enum { P_AMAX = 0, P_AMIN = 1, P_HSF = 2, P_AR = 3, P_AELL = 4 };
enum { ST_OK = 0, ST_INVAL = -1, ST_STEPCAP = -3, ST_STATE = -5 };
// Loops whose trip count is known only at run time carry `#pragma unroll 1`: their unrolled copies
// added 15-20 % to the code of the simulation loop, which two warps on one scheduler share through
// its instruction cache.
constexpr int kChunk = 128;  // active-set entries per warp pass (4 per lane)
constexpr int kWin = 32;     // admission window (one candidate per lane)
constexpr int kMc = 64;      // cached entries of the main queue (two per lane)
constexpr int64_t kBig = int64_t(1) << 60;

__device__ __forceinline__ int lane_id() { return threadIdx.x & 31; }

// Random tie key of request i at step t for A_min's cancellation order: the high 32 bits of
// output number t * 2^32 + i + 1 of the SplitMix64 generator seeded with `seed` (Steele, Lea and
// Flood, OOPSLA 2014, with the finalizer of Vigna's splitmix64.c): the state after k steps is
// seed + k * 0x9E3779B97F4A7C15, mixed by two xor-shift-multiply rounds and a final xor-shift.
// `base` = seed + t * 2^32 * 0x9E3779B97F4A7C15 (mod 2^64) is computed once per step.
__device__ __forceinline__ uint64_t tie_base(uint64_t seed, int t) {
    return seed + (uint64_t(uint32_t(t) * 0x7F4A7C15u) << 32);  // t * 2^32 * gamma mod 2^64
}

__device__ __forceinline__ unsigned tie_key(uint64_t base, int i) {
    uint64_t z = base + uint64_t(uint32_t(i) + 1u) * 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    z ^= z >> 31;
    return unsigned(z >> 32);
}


__device__ __forceinline__ bool qless(const QEnt &a, const QEnt &b) {
    return a.key < b.key || (a.key == b.key && a.idx < b.idx);
}

// The admission code reads an entry's key as its projected length.  For A_max, A_min and H-SF the
// sort key is that length; A_r projects the true length o and A_ell the current estimate (l before
// a promotion, u after: promotions have odd keys).
template <int POL>
__device__ __forceinline__ QEnt proj(const RunParams &P, int64_t base, QEnt e) {
    if (POL == P_AR) e.key = e.o;
    if (POL == P_AELL) {
        const int2 lu = P.lu[base + e.idx];
        e.key = (e.key & 1) ? lu.y : lu.x;
    }
    return e;
}

// Memory sums of the active set (projected memory at an endpoint, the next step's memory) are
// compared with M <= 2^26.  The shared-memory kernel computes them in 32 bits: every instance it
// runs has capacity x (2 lmax + 2) + 2^27 < 2^31 (lmax = the longest u or o of the instance), and
// then every offset from the time base (E - tb, y - tb, t - tb) is at most lmax + 1 in size, every
// product (count x offset) at most capacity x (lmax + 1), and every sum of B + tb at most the
// memory of a step, so nothing overflows.  Instances outside that bound, and instances whose set
// outgrows shared memory, run in the global-memory kernel, which keeps 64 bits and saturates at
// 2^30 (enough for every comparison with M).
template <bool N>
using wint = typename std::conditional<N, int32_t, int64_t>::type;

template <bool N>
__device__ __forceinline__ int satw(wint<N> v) {
    if (N) return int(v);
    const int64_t hi = int64_t(1) << 30;
    return int(v > hi ? hi : (v < -hi ? -hi : v));
}

// floor(a / b) for b > 0 in 32-bit arithmetic.  The numerators here are M minus memory sums that
// are >= 0, so they are <= M <= 2^26; a numerator below -2^30 is raised to -2^30, which keeps the
// quotient negative enough for every use (each one only asks whether a step lies before t).
__device__ __forceinline__ int floor_div32(int64_t a, int b) {
    const int ai = int(max(min(a, int64_t(INT_MAX)), -(int64_t(1) << 30)));
    int q = ai / b;
    if ((ai % b != 0) && (ai < 0)) --q;
    return q;
}

// Exclusive prefix sum over lanes; total = sum over all lanes.
__device__ __forceinline__ int excl_scan_add(int v, int &total) {
    const int lane = lane_id();
    int x = v;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
        const int y = __shfl_up_sync(FULL, x, d);
        if (lane >= d) x += y;
    }
    total = __shfl_sync(FULL, x, 31);
    return x - v;
}

// Exclusive count over lanes of the entries marked in lv (four per lane, entry 4 lane + j), by one
// ballot per slot; total = all marked entries.
__device__ __forceinline__ int excl_count4(const bool (&lv)[4], int &total) {
    const unsigned lt = (1u << lane_id()) - 1u;
    int off = 0, tot = 0;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const unsigned b = __ballot_sync(FULL, lv[j]);
        off += __popc(b & lt);
        tot += __popc(b);
    }
    total = tot;
    return off;
}

// Sum over lanes above this one; total = sum over all lanes.
__device__ __forceinline__ int excl_suffix_add(int v, int &total) {
    const int lane = lane_id();
    int x = v;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
        const int y = __shfl_down_sync(FULL, x, d);
        if (lane + d < 32) x += y;
    }
    total = __shfl_sync(FULL, x, 0);
    return x - v;
}

// Max over lanes below this one (INT_MIN for lane 0).
__device__ __forceinline__ int excl_scan_max(int v) {
    const int lane = lane_id();
    int x = v;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
        const int y = __shfl_up_sync(FULL, x, d);
        if (lane >= d) x = max(x, y);
    }
    const int ex = __shfl_up_sync(FULL, x, 1);
    return lane == 0 ? INT_MIN : ex;
}

// Number of leading positions i in [0, len) with pred(i) true (pred true on a prefix); warp-wide.
template <class Pred>
__device__ __forceinline__ int warp_prefix_count(int len, Pred pred) {
    if (len <= 0) return 0;
    const int lane = lane_id();
    if (len <= 64) {  // two entries per lane: one round
        const bool p0 = lane < len && pred(lane);
        const bool p1 = lane + 32 < len && pred(lane + 32);
        return __popc(__ballot_sync(FULL, p0)) + __popc(__ballot_sync(FULL, p1));
    }
    const int c = (len + 31) >> 5;
    const int pos = min((lane + 1) * c - 1, len - 1);
    const int full = __popc(__ballot_sync(FULL, pred(pos)));
    int cnt = full * c;
    if (cnt >= len) return len;
    const int end = min(cnt + c, len);
    #pragma unroll 1
    for (int off = cnt; off < end; off += 32) {
        const int i = off + lane;
        const unsigned b = __ballot_sync(FULL, i < end && pred(i));
        const int k = __popc(b);
        cnt += k;
        if (k < 32) break;
    }
    return cnt;
}

// #{i < len : E[i] <= y} and #{i < len : E[i] < y} for E ascending, searched in step (a
// coarse round over 32 splitters, then one fine round each).
__device__ __forceinline__ void prefix_le_lt(const int32_t *E, int len, int64_t y, int &hi, int &lb) {
    hi = lb = 0;
    if (len <= 0) return;
    const int lane = lane_id();
    const int c = (len + 31) >> 5;
    const int e = E[min((lane + 1) * c - 1, len - 1)];
    int h = min(__popc(__ballot_sync(FULL, e <= y)) * c, len);
    int l = min(__popc(__ballot_sync(FULL, e < y)) * c, len);
    const int eh = min(h + c, len), el = min(l + c, len);
    bool dh = h >= len, dl = l >= len;
    int oh = h, ol = l;
    #pragma unroll 1
    while (!(dh && dl)) {
        const int ih = oh + lane, il = ol + lane;
        const bool ph = !dh && ih < eh && E[ih] <= y;
        const bool pl = !dl && il < el && E[il] < y;
        const int kh = __popc(__ballot_sync(FULL, ph)), kl = __popc(__ballot_sync(FULL, pl));
        if (!dh) {
            h += kh;
            oh += 32;
            dh = kh < 32 || oh >= eh;
        }
        if (!dl) {
            l += kl;
            ol += 32;
            dl = kl < 32 || ol >= el;
        }
    }
    hi = h;
    lb = l;
}

// The same, computed by one lane alone (binary search).
template <class Pred>
__device__ __forceinline__ int lane_prefix_count(int len, Pred pred) {
    int lo = 0, hi = len;
    #pragma unroll 1
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (pred(mid)) lo = mid + 1; else hi = mid;
    }
    return lo;
}

// Position of the job A_min cancels when several live jobs (F >= 0) of the active set share the
// smallest estimate mk: the smallest (tie key, index) among them, the tie key drawn from `base`
// (tie_base of the step) or, under the index rule, the index itself.  Warp-wide; every lane gets
// the position.  Out of line: ties are a small share of the cancellation rounds, and keeping the
// hashing out of the simulation loop keeps that loop's code small (the loop is sensitive to the
// instruction cache).
__device__ __noinline__ int tie_position(const int32_t *F, const int32_t *K, const int32_t *I, int A, unsigned mk,
                                         uint64_t base, int rnd) {
    const int lane = lane_id();
    unsigned br = UINT_MAX, bi = UINT_MAX;
    int bp = -1;
    #pragma unroll 1
    for (int i = lane; i < A; i += 32) {
        if (F[i] >= 0 && unsigned(K[i]) == mk) {
            const unsigned id = unsigned(I[i]);
            const unsigned r = rnd ? tie_key(base, int(id)) : id;
            if (r < br || (r == br && id < bi)) {
                br = r;
                bi = id;
                bp = i;
            }
        }
    }
    const unsigned mr = __reduce_min_sync(FULL, br);
    const unsigned mi = __reduce_min_sync(FULL, br == mr ? bi : UINT_MAX);
    const unsigned b = __ballot_sync(FULL, bp >= 0 && br == mr && bi == mi);
    return b ? __shfl_sync(FULL, bp, __ffs(b) - 1) : -1;
}

// ---------------------------------------------------------------------------------------------
// Per-warp workspace
// ---------------------------------------------------------------------------------------------
struct Ws {
    int32_t *E, *F, *B, *P, *I, *K;  // active set, capacity ca (multiple of kChunk), 16-byte aligned
    int32_t *SB, *PM;                // ca + 4
    QEnt *dq;                        // delta queue, dcap entries, sorted DESCENDING (head = dq[dn-1])
    QEnt *mc;                        // cached head of the main queue, kMc entries
    int32_t *cnt;                    // dcap + 4 (merge histogram)
    int32_t *wkey, *wcs;             // window keys and prefix sums CS[0..kWin] (wide-set prefix search)
    QEnt *mb0, *mb1;                 // global ping-pong main-queue buffers
    int32_t ca, dcap;
};

__host__ __device__ inline size_t ws_bytes_impl(int ca, int dcap) {
    size_t b = size_t(6) * ca * sizeof(int32_t) + size_t(2) * (ca + 4) * sizeof(int32_t);
    b = (b + 15) & ~size_t(15);
    b += size_t(dcap + kMc) * sizeof(QEnt);
    b += size_t(dcap + 4) * sizeof(int32_t) + size_t(kWin + kWin + 4) * sizeof(int32_t);
    return (b + 15) & ~size_t(15);
}

__device__ __forceinline__ Ws carve_ws(unsigned char *base, int ca, int dcap) {
    Ws w;
    int32_t *p = reinterpret_cast<int32_t *>(base);
    w.E = p; p += ca;
    w.F = p; p += ca;
    w.B = p; p += ca;
    w.P = p; p += ca;
    w.I = p; p += ca;
    w.K = p; p += ca;
    w.SB = p; p += ca + 4;
    w.PM = p; p += ca + 4;
    size_t off = size_t(reinterpret_cast<unsigned char *>(p) - base);
    off = (off + 15) & ~size_t(15);
    w.dq = reinterpret_cast<QEnt *>(base + off);
    w.mc = w.dq + dcap;
    w.cnt = reinterpret_cast<int32_t *>(w.mc + kMc);
    w.wkey = w.cnt + dcap + 4;
    w.wcs = w.wkey + kWin;
    w.ca = ca;
    w.dcap = dcap;
    return w;
}

__device__ __forceinline__ int4 ld4(const int32_t *a, int i) { return *reinterpret_cast<const int4 *>(a + i); }

// ---------------------------------------------------------------------------------------------
// Waiting set R_t: a sorted main array in global memory [mh, me) (its first kWin entries cached
// in the workspace) plus a small sorted delta array (descending, so the head is the last
// entry).  Together they hold R_t in (key, idx) order.  Inserts go to the delta; a full delta is
// merged into the main array.
// ---------------------------------------------------------------------------------------------
struct Queue {
    const QEnt *mq;  // main array (global, ascending); may point into the staged records
    int mh, me;      // head / end
    int mbuf;        // -1: mq is read-only staged data; 0/1: ping-pong buffer in use
    int dn;          // delta size
    int mcb;         // main cache base: w.mc[i] = mq[mcb + i] for i < kMc; -1 invalid
};

__device__ __forceinline__ bool queue_empty(const Queue &q) { return q.mh >= q.me && q.dn == 0; }

// Make w.mc cover mq[mh .. mh + kWin): keep the cached run while the head is within its first
// kMc - kWin entries, otherwise reload kMc entries from the head.  gb counts the global-memory bytes
// the queue moves (a work counter of the instrumented kernel; a dead variable otherwise).
__device__ __forceinline__ void main_cache_at_head(const Ws &w, Queue &q, int64_t &gb) {
    if (q.mcb >= 0 && q.mh >= q.mcb && q.mh - q.mcb <= kMc - kWin) return;
    const int lane = lane_id();
    gb += int64_t(min(kMc, q.me - q.mh)) * int64_t(sizeof(QEnt));
    const int i0 = q.mh + lane, i1 = q.mh + 32 + lane;
    QEnt a, b;
    if (i0 < q.me) a = q.mq[i0];
    if (i1 < q.me) b = q.mq[i1];
    if (i0 < q.me) w.mc[lane] = a;
    if (i1 < q.me) w.mc[32 + lane] = b;
    __syncwarp();
    q.mcb = q.mh;
}

// Merge the delta into the main array (into the other ping-pong buffer).  Rare (a full delta, or
// a long arrival run), so it is kept out of line: the simulation loop stays small enough for the
// instruction cache when two warps share a scheduler.  Takes the few workspace pointers it needs
// by value and the queue by pointer; gb (null in the plain kernel) counts the global bytes moved.
__device__ __noinline__ void merge_delta(int32_t *cnt, const QEnt *dq, QEnt *mb0, QEnt *mb1, Queue *qp, int64_t *gb) {
    const int lane = lane_id();
    Queue q = *qp;
    const int dn = q.dn;
    const int nx = q.me - q.mh;
    QEnt *out = (q.mbuf == 0) ? mb1 : mb0;
    const QEnt *X = q.mq + q.mh;
    #pragma unroll 1
    for (int j = lane; j <= dn; j += 32) cnt[j] = 0;
    __syncwarp();
    const int c = (nx + 31) >> 5;
    const int s0 = lane * c;
    const int s1 = min(s0 + c, nx);
    if (s0 < s1) {
        const QEnt x0 = X[s0];
        int r = lane_prefix_count(dn, [&](int m) { return qless(dq[dn - 1 - m], x0); });
        int run_r = r, run_len = 0;
        #pragma unroll 1
        for (int i = s0; i < s1; ++i) {
            const QEnt x = X[i];
            #pragma unroll 1
            while (r < dn && qless(dq[dn - 1 - r], x)) ++r;
            out[i + r] = x;
            if (r != run_r) {
                if (run_len) atomicAdd(&cnt[run_r], run_len);
                run_r = r;
                run_len = 0;
            }
            ++run_len;
        }
        if (run_len) atomicAdd(&cnt[run_r], run_len);
    }
    __syncwarp();
    // delta element j (ascending) goes to j + #{main entries smaller} = j + sum_{r <= j} cnt[r]
    int carry = 0;
    #pragma unroll 1
    for (int c0 = 0; c0 < dn; c0 += 32) {
        const int j = c0 + lane;
        int v = (j < dn) ? cnt[j] : 0;
#pragma unroll
        for (int d = 1; d < 32; d <<= 1) {
            const int y = __shfl_up_sync(FULL, v, d);
            if (lane >= d) v += y;
        }
        v += carry;
        if (j < dn) out[j + v] = dq[dn - 1 - j];
        carry = __shfl_sync(FULL, v, 31);
    }
    __syncwarp();
    __threadfence_block();
    if (gb && lane == 0) *gb += int64_t(2 * nx + dn) * int64_t(sizeof(QEnt));  // main read once, merged written
    q.mq = out;
    q.mbuf = (q.mbuf == 0) ? 1 : 0;
    q.mh = 0;
    q.me = nx + dn;
    q.dn = 0;
    q.mcb = -1;
    *qp = q;
}

__device__ __forceinline__ void merge_delta(const Ws &w, Queue &q, int64_t *gb) {
    Queue qq = q;
    merge_delta(w.cnt, w.dq, w.mb0, w.mb1, &qq, gb);
    q = qq;
}

// Insert one entry into the delta (merging the delta into main first if it is full).
__device__ __forceinline__ void delta_insert(const Ws &w, Queue &q, const QEnt &e, int64_t *gb) {
    const int lane = lane_id();
    if (q.dn == w.dcap) merge_delta(w, q, gb);
    const int dn = q.dn;
    if (dn < 64) {
        // two entries per lane: count the entries greater than e (they lead the descending delta),
        // then the smaller ones move one place right straight from registers
        QEnt d0, d1;
        const bool h0 = lane < dn, h1 = lane + 32 < dn;
        if (h0) d0 = w.dq[lane];
        if (h1) d1 = w.dq[lane + 32];
        const int pos = __popc(__ballot_sync(FULL, h0 && qless(e, d0))) + __popc(__ballot_sync(FULL, h1 && qless(e, d1)));
        __syncwarp();
        if (h0 && lane >= pos) w.dq[lane + 1] = d0;
        if (h1 && lane + 32 >= pos) w.dq[lane + 33] = d1;
        if (lane == 0) w.dq[pos] = e;
        __syncwarp();
        q.dn = dn + 1;
        return;
    }
    const int pos = warp_prefix_count(dn, [&](int i) { return qless(e, w.dq[i]); });  // #entries > e
    #pragma unroll 1
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

// Head of R_t (smallest (key, idx)); the queue must not be empty.
__device__ __forceinline__ QEnt queue_head(const Ws &w, Queue &q, int64_t &gb) {
    const bool have_m = q.mh < q.me;
    QEnt hm;
    if (have_m) {
        main_cache_at_head(w, q, gb);
        hm = w.mc[q.mh - q.mcb];
    }
    if (q.dn > 0) {
        const QEnt hd = w.dq[q.dn - 1];
        if (!have_m || qless(hd, hm)) return hd;
    }
    return hm;
}

// Arrival batch (ascending run in global memory): becomes the main array if R_t is empty; a few
// entries go into the delta one by one; a long batch is copied into the emptied delta in chunks.
__device__ __forceinline__ void insert_run(const Ws &w, Queue &q, const QEnt *run, int len, int64_t &gb,
                                           int64_t *gbp) {
    const int lane = lane_id();
    if (len <= 0) return;
    gb += int64_t(len) * int64_t(sizeof(QEnt));
    if (queue_empty(q)) {
        q.mq = run;
        q.mh = 0;
        q.me = len;
        q.mbuf = -1;
        q.mcb = -1;
        return;
    }
    int done = 0;
    #pragma unroll 1
    while (done < len) {
        const int rem = len - done;
        if (rem <= 8) {
            #pragma unroll 1
            for (int j = 0; j < rem; ++j) delta_insert(w, q, run[done + j], gbp);
            break;
        }
        if (q.dn > 0) merge_delta(w, q, gbp);
        const int k = min(rem, w.dcap);
        #pragma unroll 1
        for (int j = lane; j < k; j += 32) w.dq[j] = run[done + k - 1 - j];  // descending
        __syncwarp();
        q.dn = k;
        done += k;
    }
}

// First kWin entries of R_t in (key, idx) order from the cached head of the main array (ascending)
// and the delta (descending): lane m returns entry m in `mine` (src 0 main, 1 delta).  Returns how
// many there are.
__device__ __forceinline__ int build_window(const Ws &w, Queue &q, QEnt &mine, int &msrc, int64_t &gb) {
    const int lane = lane_id();
    const int nmain = max(q.me - q.mh, 0);
    if (nmain > 0) main_cache_at_head(w, q, gb);
    const int na = min(kWin, nmain);
    const int dn = q.dn;
    const int nb = min(kWin, dn);
    // The main head A (ascending, lane i holds A[i]) followed by the delta head B in descending
    // order (lane i holds B[31 - i]) is a bitonic sequence of 64; the lane-wise minimum of the two
    // halves holds the 32 smallest entries of both as a bitonic sequence, which five shuffle stages
    // sort.  Missing entries are +infinity (key and index INT_MAX, above every real entry).  With one
    // source empty the other's head, read in ascending order, is the window as it stands.
    QEnt x;
    x.key = x.idx = INT_MAX;
    x.s = x.o = 0;
    int src = 0;
    if (lane < na) x = w.mc[q.mh - q.mcb + lane];
    const int jb = (na > 0) ? kWin - 1 - lane : lane;  // one source only: its head is the window
    if (jb < nb) {
        const QEnt y = w.dq[dn - 1 - jb];
        if (qless(y, x)) {
            x = y;
            src = 1;
        }
    }
#pragma unroll
    for (int d = 16; na > 0 && nb > 0 && d >= 1; d >>= 1) {
        QEnt y;
        y.key = __shfl_xor_sync(FULL, x.key, d);
        y.idx = __shfl_xor_sync(FULL, x.idx, d);
        y.s = __shfl_xor_sync(FULL, x.s, d);
        y.o = __shfl_xor_sync(FULL, x.o, d);
        const int ysrc = __shfl_xor_sync(FULL, src, d);
        const bool lower = (lane & d) == 0;
        if (lower == qless(y, x)) {  // the lower lane keeps the smaller entry
            x = y;
            src = ysrc;
        }
    }
    const int W = min(kWin, na + nb);
    msrc = 0;
    if (lane < W) {
        mine = x;
        msrc = src;
    }
    return W;
}

// ---------------------------------------------------------------------------------------------
// Active set maintenance
// ---------------------------------------------------------------------------------------------
__device__ __forceinline__ void store_job(const Ws &w, int i, int e, int f, int b, int p, int id, int k) {
    w.E[i] = e;
    w.F[i] = f;
    w.B[i] = b;
    w.P[i] = p;
    w.I[i] = id;
    w.K[i] = k;
}

// SB, PM, SB0 and min F for the A entries (no dead entries), time base tb.
template <bool N>
__device__ __forceinline__ void derive(const Ws &w, int A, int tb, int &SB0, int &nextF) {
    const int lane = lane_id();
    int carry = 0;
    const int last = ((A - 1) / kChunk) * kChunk;
    #pragma unroll 1
    for (int cb = last; A > 0 && cb >= 0; cb -= kChunk) {
        const int base = cb + 4 * lane;
        const int4 b4 = ld4(w.B, base);
        const int bb[4] = {b4.x, b4.y, b4.z, b4.w};
        int s[4];
        int acc = 0;
#pragma unroll
        for (int j = 3; j >= 0; --j) {
            acc += (base + j < A) ? bb[j] + tb : 0;
            s[j] = acc;
        }
        int tot;
        const int after = excl_suffix_add(acc, tot) + carry;
#pragma unroll
        for (int j = 0; j < 4; ++j)
            if (base + j < A) w.SB[base + j] = s[j] + after;
        carry += tot;
    }
    __syncwarp();
    if (lane == 0) {
        w.SB[A] = 0;
        w.PM[0] = INT_MIN;
    }
    SB0 = carry;
    int run = INT_MIN;
    int fmin = INT_MAX;
    #pragma unroll 1
    for (int cb = 0; cb < A; cb += kChunk) {
        const int base = cb + 4 * lane;
        const int4 e4 = ld4(w.E, base), s4 = ld4(w.SB, base), f4 = ld4(w.F, base);
        const int ee[4] = {e4.x, e4.y, e4.z, e4.w};
        const int ss[4] = {s4.x, s4.y, s4.z, s4.w};
        const int ff[4] = {f4.x, f4.y, f4.z, f4.w};
        int m[4];
        int mx = INT_MIN;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            int h = INT_MIN;
            if (base + j < A) {
                const wint<N> e = wint<N>(ee[j]) - tb;
                h = satw<N>(wint<N>(ss[j]) + wint<N>(A - base - j) * e + e);
                fmin = min(fmin, ff[j]);
            }
            mx = max(mx, h);
            m[j] = mx;
        }
        const int before = max(excl_scan_max(mx), run);
#pragma unroll
        for (int j = 0; j < 4; ++j)
            if (base + j < A) w.PM[base + j + 1] = max(before, m[j]);
        run = max(run, __reduce_max_sync(FULL, mx));
    }
    nextF = __reduce_min_sync(FULL, fmin);
    __syncwarp();
}

// One-chunk sets (0 < A <= kChunk) after an insertion: derive() in one pass, the suffix sums kept
// in registers for the prefix maxima.
template <bool N>
__device__ __forceinline__ void derive_one(const Ws &w, int A, int tb, int &SB0, int &nextF) {
    const int lane = lane_id();
    {
        const int base = 4 * lane;
        const int4 b4 = ld4(w.B, base), e4 = ld4(w.E, base), f4 = ld4(w.F, base);
        const int bb[4] = {b4.x, b4.y, b4.z, b4.w}, ee[4] = {e4.x, e4.y, e4.z, e4.w};
        const int ff[4] = {f4.x, f4.y, f4.z, f4.w};
        int s[4];
        int acc = 0;
#pragma unroll
        for (int j = 3; j >= 0; --j) {
            acc += (base + j < A) ? bb[j] + tb : 0;
            s[j] = acc;
        }
        int tot;
        const int after = excl_suffix_add(acc, tot);
        int m[4];
        int mx = INT_MIN, fmin = INT_MAX;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            int h = INT_MIN;
            if (base + j < A) {
                const wint<N> e = wint<N>(ee[j]) - tb;
                h = satw<N>(wint<N>(s[j] + after) + wint<N>(A - base - j) * e + e);
                fmin = min(fmin, ff[j]);
            }
            mx = max(mx, h);
            m[j] = mx;
        }
        const int before = excl_scan_max(mx);
        nextF = __reduce_min_sync(FULL, fmin);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            if (base + j < A) {
                w.SB[base + j] = s[j] + after;
                w.PM[base + j + 1] = max(before, m[j]);
            }
        }
        if (lane == 0) {
            w.SB[A] = 0;
            w.PM[0] = INT_MIN;
        }
        SB0 = tot;
        __syncwarp();
        return;
    }
}

// Remove the entries that ended before the new time base tb (completed at tb - 1, or marked with
// F = -1), keeping the order; entries only move left.
__device__ __forceinline__ void compact(const Ws &w, int &A, int tb) {
    const int lane = lane_id();
    int wpos = 0;
    #pragma unroll 1
    for (int cb = 0; cb < A; cb += kChunk) {
        const int base = cb + 4 * lane;
        const int4 e4 = ld4(w.E, base), f4 = ld4(w.F, base), b4 = ld4(w.B, base);
        const int4 p4 = ld4(w.P, base), i4 = ld4(w.I, base), k4 = ld4(w.K, base);
        const int ee[4] = {e4.x, e4.y, e4.z, e4.w}, ff[4] = {f4.x, f4.y, f4.z, f4.w};
        const int bb[4] = {b4.x, b4.y, b4.z, b4.w}, pp[4] = {p4.x, p4.y, p4.z, p4.w};
        const int ii[4] = {i4.x, i4.y, i4.z, i4.w}, kk[4] = {k4.x, k4.y, k4.z, k4.w};
        bool lv[4];
        int lc = 0;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            lv[j] = (base + j < A) && ff[j] >= tb;
            lc += lv[j] ? 1 : 0;
        }
        int L;
        const int off = excl_count4(lv, L);
        __syncwarp();
        int qd = wpos + off;
#pragma unroll
        for (int j = 0; j < 4; ++j)
            if (lv[j]) store_job(w, qd++, ee[j], ff[j], bb[j], pp[j], ii[j], kk[j]);
        __syncwarp();
        wpos += L;
    }
    A = wpos;
}

// Remove the entries with F < tb (see compact) and recompute the derived arrays, in one pass when the
// set fits one chunk (positions, suffix sums and prefix maxima of the compacted order are known
// from the live counts before anything is stored).
template <bool N>
__device__ __forceinline__ void compact_derive(const Ws &w, int &A, int tb, int &SB0, int &nextF) {
    if (A > kChunk) {
        compact(w, A, tb);
        derive<N>(w, A, tb, SB0, nextF);
        return;
    }
    const int lane = lane_id();
    const int base = 4 * lane;
    const int4 e4 = ld4(w.E, base), f4 = ld4(w.F, base), b4 = ld4(w.B, base);
    const int4 p4 = ld4(w.P, base), i4 = ld4(w.I, base), k4 = ld4(w.K, base);
    const int ee[4] = {e4.x, e4.y, e4.z, e4.w}, ff[4] = {f4.x, f4.y, f4.z, f4.w};
    const int bb[4] = {b4.x, b4.y, b4.z, b4.w}, pp[4] = {p4.x, p4.y, p4.z, p4.w};
    const int ii[4] = {i4.x, i4.y, i4.z, i4.w}, kk[4] = {k4.x, k4.y, k4.z, k4.w};
    bool lv[4];
    int lc = 0;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        lv[j] = (base + j < A) && ff[j] >= tb;
        lc += lv[j] ? 1 : 0;
    }
    int L;
    const int off = excl_count4(lv, L);
    int sfx[4];
    int acc = 0;
#pragma unroll
    for (int j = 3; j >= 0; --j) {
        acc += lv[j] ? bb[j] + tb : 0;
        sfx[j] = acc;
    }
    int tot;
    const int after = excl_suffix_add(acc, tot);
    int q = off, mx = INT_MIN, fmin = INT_MAX;
    int qp[4], mm[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        qp[j] = q;
        if (lv[j]) {
            const wint<N> e = wint<N>(ee[j]) - tb;
            mx = max(mx, satw<N>(wint<N>(sfx[j] + after) + wint<N>(L - q) * e + e));
            fmin = min(fmin, ff[j]);
            ++q;
        }
        mm[j] = mx;
    }
    const int before = excl_scan_max(mx);
    nextF = __reduce_min_sync(FULL, fmin);
    __syncwarp();
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        if (lv[j]) {
            store_job(w, qp[j], ee[j], ff[j], bb[j], pp[j], ii[j], kk[j]);
            w.SB[qp[j]] = sfx[j] + after;
            w.PM[qp[j] + 1] = max(before, mm[j]);
        }
    }
    if (lane == 0) {
        w.SB[L] = 0;
        w.PM[0] = INT_MIN;
    }
    A = L;
    SB0 = tot;
    __syncwarp();
}

// Insert the K window entries admitted at step t (lane m < K holds entry m, ascending E) into the
// compact active set, keeping E ascending (new entries after equal old ones): with
// cnt_m = #{old E <= E_m}, new entry m goes to m + cnt_m and old entry p moves right by
// #{m : cnt_m <= p}.  Entries only move right, so chunks are processed from the back.
// Returns false if the capacity is exceeded.
__device__ __forceinline__ bool insert_window(const Ws &w, int &A, int K, int t, const QEnt &mine, int le) {
    const int lane = lane_id();
    if (A + K > w.ca) return false;
    const int ne = t + mine.key - 1;
    // le >= 0: #{old E <= E_m} already found by the admission test
    const int cnt = (lane < K) ? (le >= 0 ? le : lane_prefix_count(A, [&](int i) { return w.E[i] <= ne; })) : INT_MAX;
    const int last = ((A - 1) / kChunk) * kChunk;
    #pragma unroll 1
    for (int cb = last; A > 0 && cb >= 0; cb -= kChunk) {
        const int base = cb + 4 * lane;
        const int4 e4 = ld4(w.E, base), f4 = ld4(w.F, base), b4 = ld4(w.B, base);
        const int4 p4 = ld4(w.P, base), i4 = ld4(w.I, base), k4 = ld4(w.K, base);
        const int ee[4] = {e4.x, e4.y, e4.z, e4.w}, ff[4] = {f4.x, f4.y, f4.z, f4.w};
        const int bb[4] = {b4.x, b4.y, b4.z, b4.w}, pp[4] = {p4.x, p4.y, p4.z, p4.w};
        const int ii[4] = {i4.x, i4.y, i4.z, i4.w}, kk[4] = {k4.x, k4.y, k4.z, k4.w};
        int sh[4] = {0, 0, 0, 0};
        #pragma unroll 1
        for (int m = 0; m < K; ++m) {
            const int c = __shfl_sync(FULL, cnt, m);
#pragma unroll
            for (int j = 0; j < 4; ++j) sh[j] += (base + j >= c) ? 1 : 0;
        }
        __syncwarp();
#pragma unroll
        for (int j = 0; j < 4; ++j)
            if (base + j < A) store_job(w, base + j + sh[j], ee[j], ff[j], bb[j], pp[j], ii[j], kk[j]);
        __syncwarp();
    }
    if (lane < K) store_job(w, lane + cnt, ne, t + mine.o - 1, mine.s - t + 1, t, mine.idx, mine.key);
    __syncwarp();
    A += K;
    return true;
}

// Largest admissible prefix of the window at step t (see the file comment), for any active-set
// size: per point a binary search for the first failing prefix length.  Lane m holds window entry
// m (m < W); the active set is compact with derived arrays for time base tb.
template <bool N>
__device__ __forceinline__ int admissible_prefix_search(const Ws &w, int A, int tb, int SB0, int64_t M, int t,
                                                        int W, const QEnt &mine) {
    const int lane = lane_id();
    // prefix sums CS[k] = sum_{m<k} (s_m + 1)
    int tot;
    const int add = lane < W ? mine.s + 1 : 0;
    const int ex = excl_scan_add(add, tot);
    const int incl = ex + add;
    if (lane < W) {
        w.wkey[lane] = mine.key;
        w.wcs[lane + 1] = incl;
    }
    if (lane == 0) w.wcs[0] = 0;
    __syncwarp();
    const wint<N> dt = wint<N>(t) - tb;
    const wint<N> need = wint<N>(SB0) + wint<N>(A) * dt;
    const wint<N> csW = tot;
    // the coming step (x = t): every window entry adds s + 1
    const unsigned ball = __ballot_sync(FULL, lane < W && need + incl > wint<N>(M));
    int phi = ball ? __ffs(ball) : W + 1;
    // active endpoints x = E_j >= t
    #pragma unroll 1
    for (int j = lane; j < A; j += 32) {
        const int ej = w.E[j];
        if (ej < t) continue;
        const wint<N> d = wint<N>(ej) - t;
        const wint<N> v0 = wint<N>(w.SB[j]) + wint<N>(A - j) * (wint<N>(ej) - tb);
        if (v0 + csW + wint<N>(W) * d <= wint<N>(M)) continue;
        if (v0 > wint<N>(M)) {
            phi = 0;
            continue;
        }
        const int r = lane_prefix_count(W, [&](int m) { return wint<N>(w.wkey[m]) <= d; });
        if (r >= W) continue;
        const wint<N> base = v0 - w.wcs[r] - wint<N>(r) * d;
        if (base + csW + wint<N>(W) * d <= wint<N>(M)) continue;
        int lo = r + 1, hi = W;
        #pragma unroll 1
        while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (base + w.wcs[mid] + wint<N>(mid) * d > wint<N>(M)) hi = mid; else lo = mid + 1;
        }
        phi = min(phi, lo);
    }
    // the window entries' own last steps x = t + key_m - 1
    if (lane < W) {
        const wint<N> d = wint<N>(mine.key) - 1;
        const wint<N> y = wint<N>(t) + d;
        const int lb = lane_prefix_count(A, [&](int i) { return wint<N>(w.E[i]) < y; });
        const wint<N> av = wint<N>(w.SB[lb]) + wint<N>(A - lb) * (y - tb);
        const wint<N> base = av - ex - wint<N>(lane) * d;  // ex = CS[lane]
        if (base + csW + wint<N>(W) * d > wint<N>(M)) {
            int lo = lane + 1, hi = W;
            #pragma unroll 1
            while (lo < hi) {
                const int mid = (lo + hi) >> 1;
                if (base + w.wcs[mid] + wint<N>(mid) * d > wint<N>(M)) hi = mid; else lo = mid + 1;
            }
            phi = min(phi, lo);
        }
    }
    phi = __reduce_min_sync(FULL, phi);
    return min(max(phi - 1, 0), W);
}

// Largest admissible prefix of the window at step t when the active set fits one chunk: every
// point keeps its projected memory in a register and the window entries are added one at a time
// (candidate k-1 adds s + 1 + (x - t) at every point x it reaches: the coming step x = t, the
// active endpoints E_j with key > E_j - t, and the endpoints of window entries 0..k-1); the first
// k at which any point exceeds M ends the prefix.  Falls back to the binary-search form otherwise.
template <bool N>
__device__ __forceinline__ int admissible_prefix(const Ws &w, int A, int tb, int SB0, int64_t M, int t, int W,
                                                 const QEnt &mine, int &le) {
    le = -1;
    if (A > kChunk) return admissible_prefix_search<N>(w, A, tb, SB0, M, t, W, mine);
    const int lane = lane_id();
    const int Mi = int(M);
    // active endpoints at or after t: V(E_j) and d_j = E_j - t
    const int base = 4 * lane;
    const int4 e4 = ld4(w.E, base), s4 = ld4(w.SB, base);
    const int ee[4] = {e4.x, e4.y, e4.z, e4.w};
    const int ss[4] = {s4.x, s4.y, s4.z, s4.w};
    int va[4], da[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const bool ok = base + j < A && ee[j] >= t;
        da[j] = ok ? ee[j] - t : INT_MAX;
        va[j] = ok ? satw<N>(wint<N>(ss[j]) + wint<N>(A - base - j) * (wint<N>(ee[j]) - tb)) : INT_MIN;
    }
    // this lane's window entry: V(y) of the active set at its last step y = t + key - 1
    const int dm = mine.key - 1;
    int vc = INT_MIN;
    int av = 0;
    if (lane < W) {
        // #{E < y} for V(y), and #{E <= y}, where the entry goes if it is admitted (insert_window),
        // by two binary searches in step
        const int y = t + dm;
        int lo1 = 0, hi1 = A, lo2 = 0, hi2 = A;
        #pragma unroll 1
        while (lo1 < hi1 || lo2 < hi2) {
            const int m1 = (lo1 + hi1) >> 1, m2 = (lo2 + hi2) >> 1;
            const int e1 = w.E[min(m1, A - 1)], e2 = w.E[min(m2, A - 1)];
            if (lo1 < hi1) {
                if (e1 < y) lo1 = m1 + 1; else hi1 = m1;
            }
            if (lo2 < hi2) {
                if (e2 <= y) lo2 = m2 + 1; else hi2 = m2;
            }
        }
        const int lb = lo1;
        le = lo2;
        av = satw<N>(wint<N>(w.SB[lb]) + wint<N>(A - lb) * wint<N>(y - tb));
    }
    wint<N> need = wint<N>(SB0) + wint<N>(A) * (wint<N>(t) - tb);
    // two candidates per round: the state after both is used only if neither fails
    #pragma unroll 1
    for (int k = 1; k <= W; k += 2) {
        const bool two = k < W;
        const int s1 = __shfl_sync(FULL, mine.s, k - 1) + 1;
        const int k1 = __shfl_sync(FULL, mine.key, k - 1);
        const int s2 = __shfl_sync(FULL, mine.s, k) + 1;
        const int k2 = __shfl_sync(FULL, mine.key, k);
        const wint<N> need1 = need + s1;
        const wint<N> need2 = need1 + s2;
        bool f1 = false, f2 = false;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            if (k1 > da[j]) va[j] += s1 + da[j];
            f1 = f1 || va[j] > Mi;
            if (k2 > da[j]) va[j] += s2 + da[j];
            f2 = f2 || va[j] > Mi;
        }
        if (lane == k - 1) vc = av + s1 + dm;
        else if (lane < k - 1) vc += s1 + dm;
        f1 = f1 || vc > Mi;
        if (lane == k) vc = av + s2 + dm;
        else if (lane < k) vc += s2 + dm;
        f2 = f2 || vc > Mi;
        const unsigned b1 = __ballot_sync(FULL, f1);
        const unsigned b2 = __ballot_sync(FULL, f2);
        if (b1 != 0 || need1 > wint<N>(M)) return k - 1;
        if (!two) break;
        if (b2 != 0 || need2 > wint<N>(M)) return k;
        need = need2;
    }
    return W;
}

// Largest admissible prefix when the window is in queue order but not in length order (A_r: the
// permutation, A_ell: the FIFO queue).  Candidate c reaches a point x iff its last step
// t + L_c - 1 >= x, so every point keeps its own sum: the active endpoints' projected memory is kept
// in the K array (these policies do not use it) and each window entry m accumulates, in a register,
// the candidates so far whose length is >= L_m (itself included); entry m's point counts once m is
// admitted.  Any active-set size.
template <bool N>
__device__ __forceinline__ int admissible_prefix_general(const Ws &w, int A, int tb, int SB0, int64_t M, int t,
                                                         int W, const QEnt &mine) {
    const int lane = lane_id();
    const int Mi = int(M);
    #pragma unroll 1
    for (int j = lane; j < A; j += 32) {
        const int ej = w.E[j];
        w.K[j] = (ej >= t) ? satw<N>(wint<N>(w.SB[j]) + wint<N>(A - j) * (wint<N>(ej) - tb)) : INT_MIN;
    }
    const int Lm = mine.key, dm = Lm - 1;
    int av = 0, acc = 0;
    if (lane < W) {
        const int64_t y = int64_t(t) + dm;
        const int lb = lane_prefix_count(A, [&](int i) { return int64_t(w.E[i]) < y; });
        av = satw<N>(wint<N>(w.SB[lb]) + wint<N>(A - lb) * wint<N>(y - tb));
    }
    wint<N> need = wint<N>(SB0) + wint<N>(A) * (wint<N>(t) - tb);
    #pragma unroll 1
    for (int k = 1; k <= W; ++k) {
        const int c = k - 1;
        const int sc = __shfl_sync(FULL, mine.s, c) + 1;
        const int Lc = __shfl_sync(FULL, mine.key, c);
        need += sc;
        bool fail = false;
        #pragma unroll 1
        for (int j = lane; j < A; j += 32) {  // each lane updates only its own points
            const int v = w.K[j];
            const int dj = w.E[j] - t;
            if (v != INT_MIN && Lc > dj) {
                const int nv = v + sc + dj;
                w.K[j] = nv;
                fail = fail || nv > Mi;
            }
        }
        if (lane < W && Lc >= Lm) acc += sc + dm;
        if (lane <= c) fail = fail || wint<N>(av) + acc > wint<N>(M);
        if (__ballot_sync(FULL, fail) != 0 || need > wint<N>(M)) return k - 1;
    }
    return W;
}

// Order the K admitted window entries by projected length (the active set is sorted by the last
// step E = t + L - 1); equal lengths keep their queue order.
__device__ __forceinline__ void sort_admitted(const Ws &w, int K, QEnt &mine) {
    const int lane = lane_id();
    int rk = 0;
    #pragma unroll 1
    for (int m = 0; m < K; ++m) {
        const int Lo = __shfl_sync(FULL, mine.key, m);
        rk += (Lo < mine.key || (Lo == mine.key && m < lane)) ? 1 : 0;
    }
    __syncwarp();
    if (lane < K) w.cnt[rk] = lane;  // the merge histogram is free here
    __syncwarp();
    const int src = lane < K ? w.cnt[lane] : lane;
    __syncwarp();
    QEnt o;
    o.key = __shfl_sync(FULL, mine.key, src);
    o.idx = __shfl_sync(FULL, mine.idx, src);
    o.s = __shfl_sync(FULL, mine.s, src);
    o.o = __shfl_sync(FULL, mine.o, src);
    if (lane < K) mine = o;
}

// First step tau in (t, tau_lim) at which the head candidate (prompt s, estimate L) fits, with the
// active set unchanged; kBig if none; -1 if the answer needs the arrays and arrays_ok is false
// (they hold cancelled jobs whose compaction was deferred).  In terms of y = tau + L - 1, the interval between active
// endpoints (E[j-1], E[j]] has #{E < y} = j, and #{E <= y} = j below E[j] and the end of E[j]'s
// group at y = E[j] (whose prefix maximum is PM[j+1]: within a group of equal E that lies at or
// after tb the first entry has the largest H).  Conditions (1)-(3) give, per interval, a lower
// bound on y from (2) and upper bounds from (1) and (3).
// All quantities are taken relative to the time base tb (they stay within the 32-bit bound of the
// shared-memory kernel); PM[0] is the -infinity sentinel and takes no arithmetic.
template <bool N>
__device__ __forceinline__ int64_t first_fit_step(const Ws &w, int A, int tb, int SB0, int64_t M, int t, int s,
                                                  int L, int64_t tau_lim, bool arrays_ok) {
    using W = wint<N>;
    const int lane = lane_id();
    const W BIG = N ? W(1 << 29) : W(int64_t(1) << 60);
    const W y0 = W(t - tb) + L - 1;
    const W ylim = W(min(tau_lim - tb, int64_t(BIG))) - 1 + L - 1;
    // (1) already fails at step t + 1 (the usual case, tested without the division below)
    if (int64_t(SB0) + int64_t(A) * (int64_t(t) + 1 - tb) + s + 1 > M) return kBig;
    const W tau1 = floor_div32(M - s - 1 - SB0, A);  // (1)
    const W yup = min(ylim, tau1 + L - 1);
    if (yup <= y0) return kBig;
    if (!arrays_ok) return -1;  // the arrays hold cancelled jobs: the caller compacts them first
    const W C = W(M) - s - L;  // (2): PM - C <= y;  (3): y <= floor((C - SB[j]) / (A - j))
    W best = BIG;
    #pragma unroll 1
    for (int j = lane; j <= A; j += 32) {
        const W prev = (j == 0) ? -BIG : W(w.E[j - 1] - tb);
        const W cur = (j == A) ? BIG : W(w.E[j] - tb);
        if (cur <= y0 || prev >= yup) continue;
        const W y3 = (A - j > 0) ? W(floor_div32(int64_t(C) - w.SB[j], A - j)) : BIG;
        const W up = min(yup, y3);
        const W lo = max(prev + 1, y0 + 1);
        const W cand = (j == 0) ? lo : max(lo, W(w.PM[j]) - C);
        if (cand <= min(cur - 1, up)) best = min(best, cand);
        if (j < A && cur > prev && cur >= y0 + 1 && cur <= up && W(w.PM[j + 1]) - C <= cur)
            best = min(best, cur);
    }
    // warp minimum: candidates lie in (y0, yup], so y - y0 fits 32 bits
    const unsigned off = (best == BIG) ? UINT_MAX : unsigned(best - y0);
    const unsigned m = __reduce_min_sync(FULL, off);
    if (m == UINT_MAX) return kBig;
    return int64_t(tb) + int64_t(y0) + m - L + 1;
}

// Invariants of the simulation state between events (SIM_OPT_DEBUG_CHECKS; global-memory kernel
// only): the active set is sorted by E; SB and PM are the suffix sums and prefix maxima of the
// current set and time base; SB0 and nextF match them; under A_max, H-SF and A_r no job runs past
// its projected last step; the delta queue is strictly descending and the cached head of the main
// array ascending.  Returns false on the first violation.
template <int POL, bool N>
__device__ bool state_ok(const Ws &w, const Queue &q, int A, int tb, int SB0, int nextF) {
    const int lane = lane_id();
    bool bad = false;
    int fmin = INT_MAX;
    #pragma unroll 1
    for (int i = lane; i < A; i += 32) {
        const int e = w.E[i];
        if (i + 1 < A && e > w.E[i + 1]) bad = true;
        if (w.SB[i] != w.SB[i + 1] + w.B[i] + tb) bad = true;
        const wint<N> d = wint<N>(e) - tb;
        const int h = satw<N>(wint<N>(w.SB[i]) + wint<N>(A - i) * d + d);
        if (w.PM[i + 1] != max(w.PM[i], h)) bad = true;
        fmin = min(fmin, w.F[i]);
        if ((POL == P_AMAX || POL == P_HSF || POL == P_AR) && w.F[i] > e) bad = true;
    }
    if (lane == 0 && (w.SB[A] != 0 || w.PM[0] != INT_MIN || (A > 0 && w.SB[0] != SB0))) bad = true;
    #pragma unroll 1
    for (int i = lane; i + 1 < q.dn; i += 32)
        if (!qless(w.dq[i + 1], w.dq[i])) bad = true;
    if (q.mcb >= 0)
        #pragma unroll 1
        for (int i = q.mh + lane; i + 1 < min(q.me, q.mcb + kMc); i += 32)
            if (i >= q.mcb && !qless(w.mc[i - q.mcb], w.mc[i + 1 - q.mcb])) bad = true;
    fmin = __reduce_min_sync(FULL, fmin);
    if (A > 0 && fmin != nextF) bad = true;
    return __ballot_sync(FULL, bad) == 0;
}

// ---------------------------------------------------------------------------------------------
// One instance, simulated by one warp.  All lanes hold identical copies of the scalar state.
// INS: the instrumented copy, which also keeps the work counters of the per-step method and the
// batch-time sums; the plain copy has neither.
// ---------------------------------------------------------------------------------------------
template <int POL, bool N, bool INS>
__device__ __forceinline__ void sim_instance(const RunParams &P, const Ws &w0, int inst) {
    const int lane = lane_id();
    const InstInfo info = P.info[inst];
    // delta capacity for this instance: shifts in the delta cost O(capacity) per insertion, merges
    // into the main array O(n) per capacity insertions; a small delta suits a short queue
    Ws w = w0;
    w.dcap = info.n <= 1024 ? min(w0.dcap, 64) : (info.n <= 4096 ? min(w0.dcap, 128) : w0.dcap);
    DevResult r;
    r.total_latency = r.makespan = r.peak_memory = r.evictions = r.steps = r.request_steps = 0;
    r.status = info.status;
    r.pad = 0;
    if (info.status == ST_OK && int64_t(info.n) > P.main_cap) r.status = ST_INVAL;  // larger than the queue buffers
    if (r.status != ST_OK || info.n == 0) {
        if (lane == 0) P.res[inst] = r;
        return;
    }
    if (N && int64_t(P.ca) * (2 * int64_t(info.lmax) + 2) + (int64_t(1) << 27) >= (int64_t(1) << 31)) {
        r.status = kStatusCapacity;  // too long for 32-bit sums: the global-memory kernel runs it
        if (lane == 0) P.res[inst] = r;
        return;
    }
    const int n = info.n;
    const QEnt *rec = P.rec + info.base;
    const int32_t *ra = P.rec_a + info.base;
    const uint64_t tie_seed = (POL == P_AMIN && P.tie_seed) ? P.tie_seed[inst] : 0ull;
    const int64_t M = P.M;
    const int64_t cap = info.cap;

    Queue q;
    q.mq = rec;
    q.mh = q.me = 0;
    q.mbuf = -1;
    q.dn = 0;
    q.mcb = -1;
    // global-memory bytes moved by the queue (instrumented kernel); the merge adds through gbp
    int64_t gbq = 0;
    int64_t *const gbp = INS ? &gbq : nullptr;
    // work counters of the paper's per-step method (Theorem complexity), accumulated per step in
    // closed form: S2 adds (the active set), S3 compare-exchanges of the overflow sort
    // (A ceil(log2 A)^2), S5 endpoint evaluations of a binary-search admission
    // ((A' + k) ceil(log2(Q + 1))); k_step / ev_step: admitted / removed at the current step
    int64_t cS2 = 0, cS3 = 0, cS5 = 0;
    int k_step = 0, ev_step = 0;

    // Batch time (Section 6's linear batch-time model, coefficients given later): bx0..bx3 =
    // X0..X3, the sums over requests of the processed steps, batch sizes, step memories and
    // prefill tokens of the steps a_i .. C_i - 1 (an arrival at t subtracts the prefixes up to t,
    // a completion at C adds those up to C); bmem, bpf the prefixes of step memory and prefill
    // (steps and request steps have their own counters).
    const bool bt = INS && P.batch_time != nullptr;
    int64_t bx0 = 0, bx1 = 0, bx2 = 0, bx3 = 0, bmem = 0, bpf = 0;
    // A: live jobs; Ad: entries of the active-set arrays, which after an A_min cancellation whose
    // compaction is deferred also hold the cancelled jobs (F = -1).  SB0 and A are exact either way;
    // SB and PM describe the arrays only when Ad == A.
    int A = 0, Ad = 0, tb = 0, SB0 = 0, nextF = INT_MAX;
    if (lane == 0) {  // derived arrays of the empty active set (the workspace is reused)
        w.SB[0] = 0;
        w.PM[0] = INT_MIN;
    }
    __syncwarp();
    int t = ra[0];
    int ap = 0;
    int next_a = t;
    int64_t sumC = 0, rsteps = 0, nev = 0;
    // 32 bits suffice (fewer live registers): steps <= t + 1 and makespan <= t + 1 with
    // t <= kMaxStep + 1, and the peak is a step's memory, <= M <= 2^26
    int steps = 0, makespan = 0, peak = 0;
    int ndone = 0;
    int status = ST_OK;

    bool hvalid = false;
    QEnt h;
    bool pdirty = true;
    int y_prev = 0;  // t + key - 1 <= kMaxStep + 2^26 < 2^31
    int hi = 0, lb = 0;

    bool pend_compact = false, done_step = false;
    int tb_next = 0;
    for (;;) {
        if (pend_compact) {
            // cancelled jobs (F = -1) and jobs completed at the previous step (F = tb - 1) leave
            // the active set.  Both kinds of removal share this one site: the loop body stays
            // small, which matters when two warps at different points of it share a scheduler's
            // instruction cache.
            tb = tb_next;
            const int A0 = A;
            compact_derive<N>(w, Ad, tb, SB0, nextF);
            A = Ad;
            pend_compact = false;
            pdirty = true;
            if (done_step) {  // the jobs completed at step tb - 1 (C = tb) have left the set
                const int c = A0 - A;
                sumC += int64_t(c) * tb;
                if (bt) {
                    bx0 += int64_t(c) * steps;
                    bx1 += int64_t(c) * rsteps;
                    bx2 += int64_t(c) * bmem;
                    bx3 += int64_t(c) * bpf;
                }
                ndone += c;
                done_step = false;
                if (ndone >= n) break;
            }
        }
        if (!N && P.debug && !state_ok<POL, N>(w, q, A, tb, SB0, nextF)) {
            status = ST_STATE;  // a consistency check of SIM_OPT_DEBUG_CHECKS failed
            break;
        }
        if (steps >= cap || t > kMaxStep) {
            status = ST_STEPCAP;
            break;
        }
        // ---- S1: arrivals with a <= t join R_t (a sorted run of the staged records)
        if (ap < n && next_a <= t) {
            int ae = ap;
            for (;;) {
                const int i = ae + lane;
                const unsigned b = __ballot_sync(FULL, i < n && ra[i] <= t);
                const int k = __popc(b);
                ae += k;
                if (k < 32) break;
            }
            insert_run(w, q, rec + ap, ae - ap, gbq, gbp);
            if (INS) gbq += int64_t(ae - ap) * 4;  // their arrival steps
            if (bt) {
                const int64_t m = ae - ap;
                bx0 -= m * steps;
                bx1 -= m * rsteps;
                bx2 -= m * bmem;
                bx3 -= m * bpf;
            }
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
        // ---- S2/S3: A_min overflow of the next step -> cancel in ascending (estimate, tie key, index)
        if (POL == P_AMIN) {
            wint<N> need = wint<N>(SB0) + wint<N>(A) * (t - tb);
            if (need > wint<N>(M)) {
                if (INS) {
                    const int lg = A > 1 ? 32 - __clz(A - 1) : 0;
                    cS3 += int64_t(A) * lg * lg;
                }
                // Cancellation order (estimate, r, index), r the step's tie key (SplitMix64 of the seed
                // and t * 2^32 + index; under the index rule r = index, the same order).  A round
                // finds the smallest estimate by one warp minimum; only when several live jobs share
                // it does tie_position draw and compare their keys.  (On the 40960 x 2000 workload
                // 1.3 % of the overflow steps have a tie at the smallest estimate.)
                // One-chunk sets keep the lane's four estimates in registers for all of the step's
                // cancellations, `live` marking those still in the set (the array itself is never
                // written by a run-time position, which would put it in local memory).
                const bool reg = Ad <= kChunk;
                unsigned rk[4] = {0u, 0u, 0u, 0u};
                unsigned live = 0;
                if (reg) {
                    const int base = 4 * lane;
                    const int4 k4 = ld4(w.K, base), f4 = ld4(w.F, base);
                    const int kk[4] = {k4.x, k4.y, k4.z, k4.w}, ff[4] = {f4.x, f4.y, f4.z, f4.w};
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        rk[j] = unsigned(kk[j]);
                        if (base + j < Ad && ff[j] >= 0) live |= 1u << j;
                    }
                }
                bool defer = !P.debug;  // no cancelled job is the next to complete
                #pragma unroll 1
                while (need > wint<N>(M)) {
                    int pos = -1;
                    unsigned mk;
                    int tot = 0;
                    if (reg) {
                        const unsigned q0 = (live & 1u) ? rk[0] : UINT_MAX, q1 = (live & 2u) ? rk[1] : UINT_MAX;
                        const unsigned q2 = (live & 4u) ? rk[2] : UINT_MAX, q3 = (live & 8u) ? rk[3] : UINT_MAX;
                        mk = __reduce_min_sync(FULL, min(min(q0, q1), min(q2, q3)));
#pragma unroll
                        for (int j = 0; j < 4; ++j) {
                            const unsigned b = __ballot_sync(FULL, ((live >> j) & 1u) && rk[j] == mk);
                            tot += __popc(b);
                            if (b) pos = 4 * (__ffs(b) - 1) + j;
                        }
                    } else {
                        // one pass: the smallest estimate, how many live jobs share it, and where
                        unsigned bk = UINT_MAX;
                        int bc = 0, bp = -1;
                        #pragma unroll 1
                        for (int cb = 0; cb < Ad; cb += kChunk) {
                            const int base = cb + 4 * lane;
                            const int4 f4 = ld4(w.F, base), k4 = ld4(w.K, base);
                            const int ff[4] = {f4.x, f4.y, f4.z, f4.w}, kk[4] = {k4.x, k4.y, k4.z, k4.w};
#pragma unroll
                            for (int j = 0; j < 4; ++j) {
                                if (base + j < Ad && ff[j] >= 0) {
                                    const unsigned k = unsigned(kk[j]);
                                    if (k < bk) {
                                        bk = k;
                                        bc = 1;
                                        bp = base + j;
                                    } else if (k == bk) {
                                        ++bc;
                                    }
                                }
                            }
                        }
                        mk = __reduce_min_sync(FULL, bk);
                        tot = int(__reduce_add_sync(FULL, bk == mk ? unsigned(bc) : 0u));
                        const unsigned b = __ballot_sync(FULL, bk == mk && bc > 0);
                        if (b) pos = __shfl_sync(FULL, bp, __ffs(b) - 1);
                    }
                    if (mk == UINT_MAX) pos = -1;
                    else if (tot > 1) pos = tie_position(w.F, w.K, w.I, Ad, mk, tie_base(tie_seed, t), P.evict_index == 0);
                    if (reg && pos >= 0 && (pos >> 2) == lane) live &= ~(1u << (pos & 3));
                    if (pos < 0) {  // UINT_MAX: no live entry
                        status = ST_STATE;
                        break;
                    }
                    const int b = w.B[pos], p = w.P[pos], f = w.F[pos], k = w.K[pos], id = w.I[pos];
                    QEnt e;
                    e.key = max(k, t - p);  // refined lower bound: max(estimate, tokens generated)
                    e.idx = id;
                    e.s = b + p - 1;
                    e.o = f - p + 1;
                    __syncwarp();
                    if (lane == 0) w.F[pos] = -1;
                    __syncwarp();
                    need -= wint<N>(b) + t;
                    SB0 -= b + tb;
                    --A;
                    if (f == nextF) defer = false;
                    ++nev;
                    if (INS) ++ev_step;
                    delta_insert(w, q, e, gbp);
                    if (hvalid && qless(e, h)) h = e;  // the head of R_t is the smaller of the two
                }
                if (status != ST_OK) break;
                // The cancelled jobs stay in the arrays (F = -1) until the next compaction, which
                // happens when something reads SB, PM or the order of the arrays (an admission
                // test past its O(1) part, a first-fit search, an insertion) or after the next
                // completion step; until then SB0, A and nextF describe the live jobs.  On the
                // 40960 x 2000 workload 62 % of the steps with cancellations need no compaction
                // of their own.
                if (!defer) {
                    tb_next = t;
                    pend_compact = true;
                }
                continue;
            }
        }
        // ---- A_ell: jobs that used up their estimate unfinished (E < t; the set is sorted by E, so
        // they lead it) leave the batch and re-enter the queue at its end with the estimate u
        if (POL == P_AELL && A > 0 && w.E[0] < t) {
            if (t > kAellMaxStep) {
                status = ST_STEPCAP;
                break;
            }
            const int c = warp_prefix_count(A, [&](int i) { return w.E[i] < t; });
            #pragma unroll 1
            for (int j = 0; j < c; ++j) {  // in position order; the delta orders equal keys by index
                const int b = w.B[j], p = w.P[j], f = w.F[j], id = w.I[j];
                QEnt e;
                e.key = 2 * t + 1;
                e.idx = id;
                e.s = b + p - 1;
                e.o = f - p + 1;
                __syncwarp();
                if (lane == 0) w.F[j] = -1;
                __syncwarp();
                delta_insert(w, q, e, gbp);
            }
            nev += c;
            if (INS) ev_step += c;
            tb_next = t;
            pend_compact = true;
            hvalid = false;
            continue;
        }
        // ---- S4/S5: admit the largest feasible prefix of R_t
        for (;;) {
            if (!hvalid) {
                if (queue_empty(q)) break;
                h = proj<POL>(P, info.base, queue_head(w, q, gbq));
                hvalid = true;
                pdirty = true;
            }
            // quick test of the head alone (the prefix of length one)
            const wint<N> dt = wint<N>(t) - tb;
            const wint<N> need = wint<N>(SB0) + wint<N>(A) * dt;
            bool fits = need + h.s + 1 <= wint<N>(M);
            if (fits && Ad > A) {  // the rest of the test reads the arrays: compact them first
                tb_next = tb;
                pend_compact = true;
                break;
            }
            if (fits && A > 0) {
                const int64_t y = int64_t(t) + h.key - 1;
                if (pdirty || y != int64_t(y_prev) + 1) {
                    prefix_le_lt(w.E, A, y, hi, lb);
                } else {
                    lb = hi;
                    #pragma unroll 1
                    while (hi < A && w.E[hi] <= y) ++hi;
                }
                pdirty = false;
                y_prev = int(y);
                // PM[0] is the INT_MIN sentinel: compare without adding to it
                if (wint<N>(w.PM[hi]) > wint<N>(M) - h.s - 1 + dt) fits = false;
                const wint<N> v = wint<N>(w.SB[lb]) + wint<N>(A - lb) * wint<N>(y - tb);
                if (v + h.s + h.key > wint<N>(M)) fits = false;
            } else if (fits) {
                fits = int64_t(h.s) + h.key <= M;
            }
            if (!fits) break;
            // the head fits: find the whole admissible prefix on the window
            QEnt mine;
            mine.key = mine.idx = mine.s = mine.o = 0;
            int msrc = 0;
            const int W = build_window(w, q, mine, msrc, gbq);
            if (POL == P_AR || POL == P_AELL) {
                if (lane < W) mine = proj<POL>(P, info.base, mine);
            }
            int le = -1;
            const int Kadm = (POL == P_AR || POL == P_AELL)
                                 ? admissible_prefix_general<N>(w, A, tb, SB0, M, t, W, mine)
                                 : admissible_prefix<N>(w, A, tb, SB0, M, t, W, mine, le);
            if (Kadm <= 0) {
                status = ST_STATE;  // the head test and the window disagree: internal error
                break;
            }
            if (INS) k_step += Kadm;
            if (bt)  // prefill: the prompts of the admitted requests
                bpf += int64_t(__reduce_add_sync(FULL, lane < Kadm ? unsigned(mine.s) : 0u));
            const int cm = __popc(__ballot_sync(FULL, lane < Kadm && msrc == 0));
            q.mh += cm;
            q.dn -= Kadm - cm;
            // entries >= Kadm stay in their lanes, so the new head below is unaffected
            if ((POL == P_AR || POL == P_AELL) && Kadm > 1) sort_admitted(w, Kadm, mine);
            if (!insert_window(w, A, Kadm, t, mine, le)) {
                status = kStatusCapacity;
                break;
            }
            Ad = A;
            tb = t;
            if (A <= kChunk) derive_one<N>(w, A, tb, SB0, nextF);
            else derive<N>(w, A, tb, SB0, nextF);
            pdirty = true;
            if (Kadm < W) {
                // window entry Kadm is the new head, and it does not fit at step t
                h.key = __shfl_sync(FULL, mine.key, Kadm);
                h.idx = __shfl_sync(FULL, mine.idx, Kadm);
                h.s = __shfl_sync(FULL, mine.s, Kadm);
                h.o = __shfl_sync(FULL, mine.o, Kadm);
                hvalid = true;
                break;
            }
            hvalid = false;
        }
        if (status != ST_OK) break;
        if (pend_compact) continue;  // the admission test asked for the deferred compaction
        // ---- S6: process the batch
        if (t == nextF) {
            const wint<N> mem = wint<N>(SB0) + wint<N>(A) * (wint<N>(t) - tb);
            if (mem > wint<N>(M)) {
                status = ST_STATE;
                break;
            }
            if (mem > peak) peak = int(mem);
            rsteps += A;
            ++steps;
            if (bt) bmem += int64_t(mem);
            if (INS) {
                const int Qa = (q.me - q.mh) + q.dn;  // R_t after admission
                cS2 += A - k_step + ev_step;
                cS5 += int64_t(A) * (32 - __clz(Qa + k_step));
                k_step = ev_step = 0;
            }
            // the jobs with F = t complete (C = t + 1): the compaction at the top of the next
            // iteration removes them (F < the new time base) and counts them
            if (P.completion) {
#pragma unroll 1
                for (int i = lane; i < Ad; i += 32)
                    if (w.F[i] == t) P.completion[info.base + w.I[i]] = int64_t(t) + 1;
            }
            makespan = t + 1;
            tb_next = t + 1;
            pend_compact = true;
            done_step = true;
            ++t;
        } else {
            // steps t .. tau-1 change nothing: no completion before nextF, no arrival before
            // next_a, (A_min) no overflow before tau_ov, and the head does not fit before tau_fit
            int64_t tau = nextF;
            if (ap < n) tau = min(tau, int64_t(next_a));
            if (POL == P_AMIN && A > 0) tau = min(tau, int64_t(tb) + floor_div32(M - SB0, A) + 1);
            if (POL == P_AELL && A > 0) tau = min(tau, int64_t(w.E[0]) + 1);
            tau = min(tau, int64_t(t) + (cap - steps));
            tau = min(tau, int64_t(kMaxStep) + 1);
            if (tau > int64_t(t) + 1 && hvalid && A > 0) {
                const int64_t ff = first_fit_step<N>(w, A, tb, SB0, M, t, h.s, h.key, tau, Ad == A);
                if (ff < 0) {  // the search reads the arrays: compact them first
                    tb_next = tb;
                    pend_compact = true;
                    continue;
                }
                tau = min(tau, ff);
            }
            const int64_t c = max(tau - int64_t(t), int64_t(1));
            const int64_t mem = int64_t(SB0) + int64_t(A) * (int64_t(t) + c - 1 - tb);
            if (mem > M) {
                status = ST_STATE;
                break;
            }
            if (mem > peak) peak = int(mem);
            rsteps += int64_t(A) * c;
            steps += int(c);
            if (bt)  // steps t .. t+c-1 have memory SB0 + A (x - tb)
                bmem += c * int64_t(SB0) + int64_t(A) * (c * (int64_t(t) - tb) + c * (c - 1) / 2);
            if (INS) {
                const int Qa = (q.me - q.mh) + q.dn;
                cS2 += int64_t(A) * c - k_step + ev_step;
                cS5 += int64_t(A) * (32 - __clz(Qa + k_step)) + int64_t(A) * (c - 1) * (32 - __clz(Qa));
                k_step = ev_step = 0;
            }
            t += int(c);
        }
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
        if (bt) {
            int64_t *o = P.batch_time + 6 * int64_t(inst);
            const bool ok = status == ST_OK;
            o[0] = ok ? bx0 : 0;
            o[1] = ok ? bx1 : 0;
            o[2] = ok ? bx2 : 0;
            o[3] = ok ? bx3 : 0;
            o[4] = ok ? bmem : 0;
            o[5] = ok ? bpf : 0;
        }
        if (INS && P.work_count) {
            int64_t *wc = P.work_count + 4 * int64_t(inst);
            wc[0] = cS2;
            wc[1] = cS3;
            wc[2] = cS5;
            wc[3] = gbq;
        }
    }
    __syncwarp();
}

// LAY: the workspace layout.  1 (dense): three blocks of four warps per SM (12 simulating warps,
// at most 170 registers a thread) and kDenseCa active-set slots; 2: the default kSmemCaDefault
// slots; 0: P.ca slots (the global-memory kernel, other shared-memory capacities and the
// instrumented copy).  With 1 and 2 the layout is fixed at compile time, so the workspace arrays
// are constant offsets from one shared-memory base instead of pointers held in registers.  Other
// than dense: blocks of up to 256 threads and as many registers as the code wants.
template <int POL, bool SMEM, bool INS, int LAY>
__global__ void __launch_bounds__(LAY == 1 ? 128 : 256, LAY == 1 ? 3 : 1) k_run(RunParams P) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int lane = lane_id();
    const int wib = threadIdx.x >> 5;
    const int64_t slot = int64_t(blockIdx.x) * (blockDim.x >> 5) + wib;
    const int ca = LAY == 1 ? kDenseCa : (LAY == 2 ? kSmemCaDefault : P.ca);
    unsigned char *base;
    if (SMEM) base = smem_raw + size_t(wib) * ws_bytes_impl(ca, kDcap);
    else base = P.gws + slot * P.gws_stride;
    Ws w = carve_ws(base, ca, kDcap);
    w.mb0 = P.mainbuf + slot * 2 * P.main_cap;
    w.mb1 = w.mb0 + P.main_cap;
    for (;;) {
        int k = 0;
        if (lane == 0) k = atomicAdd(P.counter, 1);
        k = __shfl_sync(FULL, k, 0);
        if (k >= P.n_work) break;
        const int inst = P.work ? P.work[k] : k;
        sim_instance<POL, SMEM, INS>(P, w, inst);
    }
}

// The shared-memory copies: v = 0 plain with P.ca slots, 1 instrumented, 2 dense, 3 plain with
// the default slots.
template <int POL>
const void *smem_fn(int v) {
    switch (v) {
        case 0: return (const void *)k_run<POL, true, false, 0>;
        case 1: return (const void *)k_run<POL, true, true, 0>;
        case 2: return (const void *)k_run<POL, true, false, 1>;
        default: return (const void *)k_run<POL, true, false, 2>;
    }
}

template <int POL>
void launch_pol(const RunParams &p, dim3 grid, dim3 block, size_t smem_bytes, bool dense, cudaStream_t st) {
    const bool sm = p.use_smem != 0;
    const bool ins = p.work_count != nullptr || p.batch_time != nullptr;
    if (ins) {
        if (sm) k_run<POL, true, true, 0><<<grid, block, smem_bytes, st>>>(p);
        else k_run<POL, false, true, 0><<<grid, block, smem_bytes, st>>>(p);
    } else if (sm && dense) {
        k_run<POL, true, false, 1><<<grid, block, smem_bytes, st>>>(p);
    } else if (sm && p.ca == kSmemCaDefault) {
        k_run<POL, true, false, 2><<<grid, block, smem_bytes, st>>>(p);
    } else {
        if (sm) k_run<POL, true, false, 0><<<grid, block, smem_bytes, st>>>(p);
        else k_run<POL, false, false, 0><<<grid, block, smem_bytes, st>>>(p);
    }
}

}  // namespace

size_t warp_ws_bytes(int ca) { return ws_bytes_impl(ca, kDcap); }

cudaError_t set_run_smem_limit(int policy, size_t bytes) {
    for (int v = 0; v < 4; ++v) {
        const void *fn = policy == P_AMAX ? smem_fn<P_AMAX>(v)
                         : policy == P_AMIN ? smem_fn<P_AMIN>(v)
                         : policy == P_HSF  ? smem_fn<P_HSF>(v)
                         : policy == P_AR   ? smem_fn<P_AR>(v)
                                            : smem_fn<P_AELL>(v);
        const cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, int(bytes));
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

cudaError_t launch_run(int policy, const RunParams &p, int blocks, int warps_per_block, size_t smem_bytes, bool dense,
                       cudaStream_t st) {
    const dim3 grid(blocks), block(32 * warps_per_block);
    switch (policy) {
        case P_AMAX: launch_pol<P_AMAX>(p, grid, block, smem_bytes, dense, st); break;
        case P_AMIN: launch_pol<P_AMIN>(p, grid, block, smem_bytes, dense, st); break;
        case P_HSF: launch_pol<P_HSF>(p, grid, block, smem_bytes, dense, st); break;
        case P_AR: launch_pol<P_AR>(p, grid, block, smem_bytes, dense, st); break;
        default: launch_pol<P_AELL>(p, grid, block, smem_bytes, dense, st); break;
    }
    return cudaGetLastError();
}

}  // namespace simgb
