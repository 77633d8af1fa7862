// Staging and result kernels of the batched scheduler simulator (sm_103a).
//
//   k_stage  - per instance (one CTA): validate the requests against the Section 2 model
//              (1 <= l <= o <= u, s >= 1, a >= 0, s + o <= M; s + u <= M under A_max), compute the
//              constants the simulation needs (sum of arrivals for TEL, the step cap), and sort
//              the requests by (arrival step, policy key, index) so that every arrival batch is
//              already in the order of the waiting set R_t (key u for Algorithm malb, l for
//              Algorithms milb / milbrevise, o for Algorithm off, the given permutation rank for
//              Algorithm random, and the FIFO position 2 a for Algorithm promote_l, which also
//              gets its (l, u) table).
//   k_ratio  - per instance TEL(pi) / TEL(H-SF) in IEEE double (Definition cr).
//   k_batch_time - per instance total latency and makespan in time units under a linear
//              batch-time model (Section 6), from the integer sums the simulation recorded.
#include <climits>
#include <cstdint>

#include "sim_internal.h"

namespace simgb {

namespace {

constexpr unsigned FULL = 0xffffffffu;
enum { P_AMAX = 0, P_AMIN = 1, P_HSF = 2, P_AR = 3, P_AELL = 4 };
enum { ST_OK = 0, ST_INVAL = -1, ST_INFEASIBLE = -2 };

struct BtCoef {
    double k[5];
};

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

// Bitonic sort of n records by (a, key, idx) in place in global memory, padded virtually to a
// power of two (positions >= n take no part): instances too large for shared memory.
__device__ void bitonic_sort(QEnt *R, int32_t *RA, int n) {
    int N = 1;
    while (N < n) N <<= 1;
    for (int k = 2; k <= N; k <<= 1) {
        for (int d = k >> 1, ld = __ffs(d) - 1; d >= 1; d >>= 1, --ld) {
            for (int p = threadIdx.x; p < N / 2; p += blockDim.x) {
                const int i = ((p >> ld) << (ld + 1)) | (p & (d - 1));  // d is a power of two
                const int j = (d == (k >> 1)) ? (i | (k - 1)) - (i & (k - 1)) : i + d;  // first pass: mirror
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

// Instances of up to this many requests are sorted in shared memory: per request its key, arrival,
// prompt and true length and two index buffers (24 bytes), plus the radix counters.
constexpr int kStageSmemN = 2048;
constexpr int kStageSmemBytesPerReq = 24;
constexpr int kStageSmemIpt = kStageSmemN / 256;  // elements per thread of a radix pass
constexpr size_t kStageCntBytes = size_t(16) * kStageSmemIpt * 8 * sizeof(uint16_t);

// Instances held in shared memory are sorted by an LSD radix sort of request indices, 4-bit digits
// of the policy key and then of the arrival step, each pass stable, so the order is (a, key, idx)
// (both are >= 0 in a valid instance).  A pass ranks element e = r * 256 + thread (iteration r):
// within a warp and iteration, __match_any_sync groups the lanes with equal digits and a lane's
// rank in its group is the number of group lanes below it; the groups' sizes go to counters in
// (digit, iteration, warp) order, whose exclusive prefix sums are the groups' first output
// positions.  Elements are thereby placed in (digit, e) order: stable.
constexpr int kRadixBits = 4;
constexpr int kRadixBins = 1 << kRadixBits;
constexpr int kStageThreads = 256;
constexpr int kStageWarps = kStageThreads / 32;

template <int IPT>
__device__ __forceinline__ void radix_pass(const int32_t *keyof, const int32_t *in, int32_t *out, uint16_t *cnt,
                                           int *wsum, int n, int shift) {
    constexpr int kCnt = kRadixBins * IPT * kStageWarps;  // a multiple of 4 * kStageThreads / 4
    const int t = threadIdx.x, lane = t & 31, w = t >> 5;
    const unsigned lt = (1u << lane) - 1u;
    for (int f = t; f < kCnt; f += kStageThreads) cnt[f] = 0;
    __syncthreads();
    int dg[IPT], rk[IPT], ix[IPT];
#pragma unroll
    for (int r = 0; r < IPT; ++r) {
        const int e = r * kStageThreads + t;
        const bool v = e < n;
        ix[r] = v ? in[e] : 0;
        dg[r] = v ? ((keyof[ix[r]] >> shift) & (kRadixBins - 1)) : kRadixBins;  // past the end: a group of its own
        const unsigned peers = __match_any_sync(FULL, dg[r]);
        rk[r] = __popc(peers & lt);
        if (v && rk[r] == 0) cnt[(dg[r] * IPT + r) * kStageWarps + w] = uint16_t(__popc(peers));
    }
    __syncthreads();
    // exclusive prefix sums of the counters, kCnt / kStageThreads consecutive ones per thread
    constexpr int kPer = kCnt / kStageThreads;
    int c[kPer], sum = 0;
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
        c[i] = cnt[kPer * t + i];
        sum += c[i];
    }
    int x = sum;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
        const int y = __shfl_up_sync(FULL, x, d);
        if (lane >= d) x += y;
    }
    if (lane == 31) wsum[w] = x;
    __syncthreads();
    int run = x - sum;
    for (int i = 0; i < w; ++i) run += wsum[i];
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
        cnt[kPer * t + i] = uint16_t(run);
        run += c[i];
    }
    __syncthreads();
#pragma unroll
    for (int r = 0; r < IPT; ++r) {
        const int e = r * kStageThreads + t;
        if (e < n) out[cnt[(dg[r] * IPT + r) * kStageWarps + w] + rk[r]] = ix[r];
    }
    __syncthreads();
}

// Sorts the indices 0..n-1 held in i0 (scratch i1) by (ka, kk, index); returns the buffer that
// holds the result.  kmax, amax: the largest key and arrival step (>= 0).
__device__ int32_t *radix_sort_idx(const int32_t *kk, const int32_t *ka, int32_t *i0, int32_t *i1, uint16_t *cnt,
                                   int *wsum, int n, int kmax, int amax) {
    int32_t *in = i0, *out = i1;
    const int kbits = kmax > 0 ? 32 - __clz(kmax) : 0;
    const int abits = amax > 0 ? 32 - __clz(amax) : 0;
    for (int sh = 0; sh < kbits; sh += kRadixBits) {
        radix_pass<kStageSmemIpt>(kk, in, out, cnt, wsum, n, sh);
        int32_t *tmp = in;
        in = out;
        out = tmp;
    }
    for (int sh = 0; sh < abits; sh += kRadixBits) {
        radix_pass<kStageSmemIpt>(ka, in, out, cnt, wsum, n, sh);
        int32_t *tmp = in;
        in = out;
        out = tmp;
    }
    return in;
}


__global__ void __launch_bounds__(kStageThreads) k_stage(StageParams S, int np) {
    __shared__ int64_t sh64[32];
    __shared__ int wsum[kStageWarps];
    extern __shared__ __align__(16) unsigned char stage_smem[];
    const int inst = blockIdx.x;
    const int64_t base = S.off[inst];
    const int64_t n64 = S.off[inst + 1] - base;
    // offsets that reach outside the staged buffers (or above the per-instance limit) reject the
    // instance before anything is written: it is staged as empty with status INVAL
    const bool oob = base < 0 || n64 < 0 || n64 > S.max_n || base + n64 > S.max_total;
    const int n = oob ? 0 : int(n64);
    int64_t bad_inval = oob ? 1 : 0, bad_inf = 0, sum_a = 0, sum_o = 0, lmax = 0, kmax = 0, amax = 0;
    const bool in_smem = n <= np;
    int32_t *kk = reinterpret_cast<int32_t *>(stage_smem);
    int32_t *ka = kk + np;
    int32_t *ss = ka + np;
    int32_t *so = ss + np;
    int32_t *i0 = so + np;
    int32_t *i1 = i0 + np;
    uint16_t *cnt = reinterpret_cast<uint16_t *>(i1 + np);
    for (int j = threadIdx.x; j < n; j += blockDim.x) {
        const int64_t g = base + j;
        const int a = S.a[g], s = S.s[g], l = S.l[g], u = S.u[g], o = S.o[g];
        if (s < 1 || a < 0 || l < 1 || l > o || o > u) bad_inval = 1;
        if (int64_t(s) + o > S.M) bad_inf = 1;
        if ((S.policy == P_AMAX || S.policy == P_AELL) && int64_t(s) + u > S.M) bad_inf = 1;
        int key;
        switch (S.policy) {
            case P_AMAX: key = u; break;
            case P_HSF: key = o; break;
            case P_AR: key = S.rank[g]; break;
            case P_AELL: key = 2 * min(a, kAellMaxStep); break;
            default: key = l; break;
        }
        if (S.policy == P_AR && key < 0) bad_inval = 1;
        if (S.policy == P_AELL) {
            if (a > kAellMaxStep) bad_inval = 1;
            S.lu[g] = make_int2(l, u);  // indexed by request: j == idx below
        }
        if (in_smem) {
            kk[j] = key;
            ka[j] = a;
            ss[j] = s;
            so[j] = o;
            i0[j] = j;
        } else {
            QEnt e;
            e.key = key;
            e.idx = j;
            e.s = s;
            e.o = o;
            S.rec[g] = e;
            S.rec_a[g] = a;
        }
        sum_a += a;
        sum_o += o;
        lmax = max(lmax, int64_t(max(u, o)));
        kmax = max(kmax, int64_t(key));
        amax = max(amax, int64_t(a));
    }
    bad_inval = block_reduce<int64_t>(bad_inval, sh64, true);
    bad_inf = block_reduce<int64_t>(bad_inf, sh64, true);
    sum_a = block_reduce<int64_t>(sum_a, sh64, false);
    sum_o = block_reduce<int64_t>(sum_o, sh64, false);
    lmax = block_reduce<int64_t>(lmax, sh64, true);
    if (in_smem) {
        kmax = block_reduce<int64_t>(kmax, sh64, true);
        amax = block_reduce<int64_t>(amax, sh64, true);
    }
    int status = ST_OK;
    if (bad_inval) status = ST_INVAL;
    else if (bad_inf) status = ST_INFEASIBLE;
    if (threadIdx.x == 0) {
        InstInfo in;
        in.base = oob ? 0 : base;
        in.n = n;
        in.status = status;
        in.sum_a = sum_a;
        in.cap = S.step_cap > 0 ? S.step_cap : 64 * (int64_t(n) + sum_o);
        in.lmax = int32_t(lmax);
        in.pad = 0;
        S.info[inst] = in;
    }
    __syncthreads();
    if (!in_smem) {
        if (status == ST_OK && n > 1) bitonic_sort(S.rec + base, S.rec_a + base, n);
        return;
    }
    const int32_t *ord = i0;
    if (status == ST_OK && n > 1) ord = radix_sort_idx(kk, ka, i0, i1, cnt, wsum, n, int(kmax), int(amax));
    // write the (sorted, or for a rejected instance unsorted) records out
    for (int j = threadIdx.x; j < n; j += blockDim.x) {
        const int idx = ord[j];
        QEnt e;
        e.key = kk[idx];
        e.idx = idx;
        e.s = ss[idx];
        e.o = so[idx];
        S.rec[base + j] = e;
        S.rec_a[base + j] = ka[idx];
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

// Total latency and makespan in time units under the linear batch-time model (Section 6: each
// batch's time from a linear predictor; coef = c0, c1, c2, c3, c_idle):
//   out[2i]     = c0 X0 + c1 X1 + c2 X2 + c3 X3,
//   out[2i + 1] = c0 steps + c1 request_steps + c2 F2 + c3 F3 + c_idle (makespan - steps),
// from sums = X0..X3, F2, F3 of instance i, evaluated left to right with round-to-nearest products
// and sums (no fused multiply-add), so the result is the IEEE value of that expression.  NaN for an
// instance that did not finish.
__global__ void k_batch_time(const int64_t *sums, const DevResult *res, BtCoef c, double *out, int32_t n) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= n) return;
    const DevResult r = res[i];
    const int64_t *x = sums + 6 * int64_t(i);
    double tel = __longlong_as_double(0x7ff8000000000000ll), span = tel;
    if (r.status == ST_OK) {
        tel = __dadd_rn(__dadd_rn(__dadd_rn(__dmul_rn(c.k[0], __ll2double_rn(x[0])), __dmul_rn(c.k[1], __ll2double_rn(x[1]))),
                                  __dmul_rn(c.k[2], __ll2double_rn(x[2]))),
                        __dmul_rn(c.k[3], __ll2double_rn(x[3])));
        span = __dadd_rn(__dadd_rn(__dadd_rn(__dadd_rn(__dmul_rn(c.k[0], __ll2double_rn(r.steps)),
                                                       __dmul_rn(c.k[1], __ll2double_rn(r.request_steps))),
                                             __dmul_rn(c.k[2], __ll2double_rn(x[4]))),
                                   __dmul_rn(c.k[3], __ll2double_rn(x[5]))),
                         __dmul_rn(c.k[4], __ll2double_rn(r.makespan - r.steps)));
    }
    out[2 * int64_t(i)] = tel;
    out[2 * int64_t(i) + 1] = span;
}

}  // namespace

cudaError_t launch_batch_time(const int64_t *sums, const DevResult *res, const double *coef, double *out, int32_t n,
                              cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    BtCoef c;
    for (int k = 0; k < 5; ++k) c.k[k] = coef[k];
    k_batch_time<<<(n + 255) / 256, 256, 0, st>>>(sums, res, c, out, n);
    return cudaGetLastError();
}

cudaError_t launch_stage(const StageParams &p, cudaStream_t st) {
    if (p.n_inst <= 0) return cudaSuccess;
    // shared memory for the largest instance up to kStageSmemN, rounded up to a power of two
    int np = 1;
    const int want = (p.n_max > 0 && p.n_max < kStageSmemN) ? p.n_max : kStageSmemN;
    while (np < want) np <<= 1;
    const size_t smem = size_t(np) * kStageSmemBytesPerReq + kStageCntBytes;
    if (smem > 48 * 1024) {
        const cudaError_t e = cudaFuncSetAttribute(k_stage, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
        if (e != cudaSuccess) return e;
    }
    k_stage<<<p.n_inst, kStageThreads, smem, st>>>(p, np);
    return cudaGetLastError();
}

cudaError_t launch_ratio(const DevResult *pol, const DevResult *ref, double *out, int32_t n, cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    k_ratio<<<(n + 255) / 256, 256, 0, st>>>(pol, ref, out, n);
    return cudaGetLastError();
}

}  // namespace simgb
