// Analytic competitive-ratio evaluators of A_min (double precision, sm_103a).
//
//   k_lemma   - Lemma thm:Amin for a batch of length histograms: one thread per histogram walks it
//               from the longest length down with the four running sums the lemma needs
//               (sum i x_i, sum x_i/(s+i), sum i x_i/(s+i), sum x_i over i >= k), about ten FP64
//               operations per length, with 1/(s+k) and k(s+k) from a shared-memory table.  The
//               histogram is read once; GB300's FP64 rate, not HBM, bounds the kernel.
//   k_rho     - spectral radius of B_u^{-1} A_u (Corollary A/B; s = 0, l = 1), the bound on the
//               Rayleigh quotient of Section 4.1, by power iteration.  A_u v is O(u) from prefix
//               and suffix sums (for j <= i, a_ij = ij/2 + j^2 - j^3/(2i); symmetric), B_u^{-1} is
//               the tridiagonal matrix printed in Section 4.1, and the estimate is the Rayleigh
//               quotient v'Av / v'Bv with (Bv)_i = sum_{j<=i} j^2 v_j + i^2 sum_{j>i} v_j.  One
//               warp per u; the vectors live in a global scratch of 3 u doubles per warp.
#include <algorithm>
#include <cmath>
#include <cstdint>

#include "sim_internal.h"

namespace simgb {

namespace {

constexpr unsigned FULL = 0xffffffffu;

__device__ __forceinline__ double warp_sum(double v) {
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1) v += __shfl_xor_sync(FULL, v, d);
    return v;
}

// Inclusive prefix sum over lanes.
__device__ __forceinline__ double prefix_incl(double v) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
        const double y = __shfl_up_sync(FULL, v, d);
        if (lane >= d) v += y;
    }
    return v;
}

__global__ void __launch_bounds__(256) k_lemma(int32_t n_hist, int32_t len, int32_t l, double s,
                                                const double *__restrict__ x, double *__restrict__ out) {
    // per-length constants shared by every histogram: 1/(s+k) and k(s+k)
    extern __shared__ double tab[];
    double *rinv = tab, *ck = tab + len;
    for (int j = threadIdx.x; j < len; j += blockDim.x) {
        const double k = double(l + j);
        rinv[j] = 1.0 / (s + k);
        ck[j] = k * (s + k);
    }
    __syncthreads();
    const int64_t h = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
    if (h >= n_hist) return;
    const double *xh = x + h * int64_t(len);
    // running sums over lengths > k (before the update) and >= k (after it)
    double S1 = 0.0, S2 = 0.0, T = 0.0, X = 0.0;
    double num = 0.0, den = 0.0;
    for (int j = len - 1; j >= 0; --j) {
        const double k = double(l + j);
        const double xk = __ldg(xh + j);
        // values over i > k
        const double gap = fma(-k, S2, T);      // sum_{i>k} (i-k) x_i/(s+i)
        const double twoXn = 2.0 * X;           // 2 sum_{i>k} x_i
        const double fr = xk * rinv[j];
        S1 = fma(k, xk, S1);                    // sum_{i>=k} i x_i
        S2 += fr;                               // sum_{i>=k} x_i/(s+i)
        T = fma(k, fr, T);                      // sum_{i>=k} i x_i/(s+i)
        X += xk;
        const double delta = (j == 0) ? (s + double(l)) : 1.0;
        num = fma(delta * S1, fma(2.0, gap, delta * S2), num);
        den = fma(ck[j] * xk, xk + twoXn, den);
    }
    out[h] = num / den;
}

// (A v)_i and (B v)_i for i = 1..u from prefix/suffix sums; v, av, bv in global scratch.
__device__ void rho_products(int u, const double *v, double *av, double *bv, double &vav, double &vbv) {
    const int lane = threadIdx.x & 31;
    // totals first: P1 = sum j v_j
    double p1 = 0.0;
    for (int b = 0; b < u; b += 32) {
        const int j = b + lane + 1;
        if (j <= u) p1 += double(j) * v[j - 1];
    }
    p1 = warp_sum(p1);
    // prefix sums Q2 = sum_{j<=i} j^2 v_j, Q3 = sum_{j<=i} j^3 v_j; suffix sums R0 = sum_{j>i} v_j,
    // R1 = sum_{j>i} v_j / j, obtained as totals minus prefixes
    double t0 = 0.0, t1 = 0.0;
    for (int b = 0; b < u; b += 32) {
        const int j = b + lane + 1;
        if (j <= u) {
            t0 += v[j - 1];
            t1 += v[j - 1] / double(j);
        }
    }
    t0 = warp_sum(t0);
    t1 = warp_sum(t1);
    double q2c = 0.0, q3c = 0.0, r0c = 0.0, r1c = 0.0;  // running prefixes of the four sums
    double sa = 0.0, sb = 0.0;
    for (int b = 0; b < u; b += 32) {
        const int i = b + lane + 1;
        const double di = double(i);
        const double vi = (i <= u) ? v[i - 1] : 0.0;
        const double q2 = prefix_incl(di * di * vi) + q2c;
        const double q3 = prefix_incl(di * di * di * vi) + q3c;
        const double p0 = prefix_incl(vi) + r0c;         // sum_{j<=i} v_j
        const double p1i = prefix_incl(vi / di) + r1c;   // sum_{j<=i} v_j / j
        if (i <= u) {
            const double R0 = t0 - p0, R1 = t1 - p1i;
            const double a = 0.5 * di * p1 + q2 - q3 / (2.0 * di) + di * di * R0 - 0.5 * di * di * di * R1;
            const double bb = q2 + di * di * R0;
            av[i - 1] = a;
            bv[i - 1] = bb;
            sa += vi * a;
            sb += vi * bb;
        }
        q2c = __shfl_sync(FULL, q2, 31);
        q3c = __shfl_sync(FULL, q3, 31);
        r0c = __shfl_sync(FULL, p0, 31);
        r1c = __shfl_sync(FULL, p1i, 31);
    }
    vav = warp_sum(sa);
    vbv = warp_sum(sb);
    __syncwarp();
}

__global__ void k_rho(int32_t n_u, const int32_t *__restrict__ us, double *__restrict__ out, double *scratch,
                      int64_t stride, int32_t max_iter) {
    const int lane = threadIdx.x & 31;
    const int64_t warp = (int64_t(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    if (warp >= n_u) return;
    const int u = us[warp];
    double *v = scratch + warp * stride;
    double *av = v + u;
    double *bv = av + u;
    for (int i = lane; i < u; i += 32) v[i] = 1.0;
    __syncwarp();
    double lam = 0.0;
    for (int it = 0; it < max_iter; ++it) {
        double vav, vbv;
        rho_products(u, v, av, bv, vav, vbv);
        const double nl = vav / vbv;  // generalized Rayleigh quotient of the current vector
        // next vector: B^{-1} (A v), tridiagonal, then scale by its largest entry
        double mx = 0.0;
        for (int b = 0; b < u; b += 32) {
            const int i = b + lane + 1;
            double z = 0.0;
            if (i <= u) {
                const double di = double(i);
                const double d = (i < u) ? 4.0 * di / (4.0 * di * di - 1.0) : 1.0 / (2.0 * di - 1.0);
                z = d * av[i - 1];
                if (i > 1) z -= av[i - 2] / (2.0 * (di - 1.0) + 1.0);
                if (i < u) z -= av[i] / (2.0 * di + 1.0);
            }
            __syncwarp();
            if (i <= u) bv[i - 1] = z;  // bv is free until the next products
            mx = fmax(mx, fabs(z));
        }
#pragma unroll
        for (int d = 16; d >= 1; d >>= 1) mx = fmax(mx, __shfl_xor_sync(FULL, mx, d));
        __syncwarp();
        for (int i = lane; i < u; i += 32) v[i] = bv[i] / mx;
        __syncwarp();
        const bool done = it > 0 && fabs(nl - lam) <= 1e-15 * nl;
        lam = nl;
        if (done) break;
    }
    if (lane == 0) out[warp] = lam;
}

}  // namespace

cudaError_t launch_lemma(int32_t n_hist, int32_t len, int32_t l, double s, const double *x, double *out,
                         cudaStream_t st) {
    if (n_hist <= 0) return cudaSuccess;
    const size_t smem = size_t(2) * len * sizeof(double);
    if (smem > 48 * 1024) {
        const cudaError_t e = cudaFuncSetAttribute(k_lemma, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
        if (e != cudaSuccess) return e;
    }
    k_lemma<<<(n_hist + 255) / 256, 256, smem, st>>>(n_hist, len, l, s, x, out);
    return cudaGetLastError();
}

cudaError_t launch_rho(int32_t n_u, const int32_t *us, double *out, double *scratch, int64_t stride,
                       int32_t max_iter, cudaStream_t st) {
    if (n_u <= 0) return cudaSuccess;
    k_rho<<<(n_u + 3) / 4, 128, 0, st>>>(n_u, us, out, scratch, stride, max_iter);
    return cudaGetLastError();
}

}  // namespace simgb
