// svd.cu -- the singular values of every matrix (Alg. 2 takes the SVD of each 2-D
// pseudo-gradient; Sec. 4.5's spectrum maps need the individual sigma_i).
//
// With the polar factor Q of Delta (Delta = U S V^T, Q = U V^T), H = Q^T Delta = V S V^T
// (Delta Q^T = U S U^T for a wide matrix) is symmetric positive semidefinite and its
// eigenvalues are the singular values of Delta.  A rotation error K in Q (Q U^T V = I + K,
// K skew) changes H's eigenvalues only at second order (v_i^T K H v_i = 0), so sigma_i
// comes out much more accurate than Q itself.  Per matrix:
//   k_svd_tridiag : Householder reduction of H (fp32, full symmetric storage, in place) to
//                   a symmetric tridiagonal T = (d, e), one CTA per matrix.  Step k takes
//                   the reflector I - tau v v^T of row k's part right of the diagonal, forms
//                   p = B v over the trailing block B, w = tau p - (tau^2 / 2)(p^T v) v and
//                   B -= v w^T + w v^T.  The update of step k and the product B' v' of step
//                   k + 1 share one pass over the block: row k + 1 is updated first, gives
//                   v', and every later row is updated and dotted with v' in the same sweep.
//   k_svd_bisect  : every eigenvalue of T by bisection on the Sturm count (the number of
//                   negative pivots of T - x I), one thread per eigenvalue: the j-th smallest
//                   is the j-th one found, so the result comes sorted.
// The reduction is BLAS-2 bound: about n^3 / 3 elements read and written per matrix.
#include "common.cuh"
#include "types.h"

namespace isoloco {

constexpr int kUnroll = 8;  // row elements per lane in flight in the sweeps over H

__device__ __forceinline__ float svd_warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Block-wide sum (kSvdThreads threads); `red` holds 32 floats; every thread gets the sum.
__device__ __forceinline__ float svd_block_sum(float v, float* red) {
    v = svd_warp_sum(v);
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    __syncthreads();
    if (l == 0) red[w] = v;
    __syncthreads();
    float s = (l < (kSvdThreads >> 5)) ? red[l] : 0.f;
    s = svd_warp_sum(s);
    return s;
}

// Householder vector of x = a[0 .. m-1] (row r0 - 1, the columns r0 ..), written to v with
// v[0] = 1; returns tau (0 when x is already a multiple of e_1) and beta (the new
// off-diagonal entry).
__device__ __forceinline__ float svd_householder(const float* a, int m, float* v, float* red, float* beta_out) {
    float s2 = 0.f;
    for (int i = 1 + static_cast<int>(threadIdx.x); i < m; i += kSvdThreads) {
        const float x = a[i];
        v[i] = x;
        s2 = fmaf(x, x, s2);
    }
    s2 = svd_block_sum(s2, red);
    const float alpha = a[0];
    if (!(s2 > 0.f)) {
        *beta_out = alpha;
        if (threadIdx.x == 0) v[0] = 1.f;
        for (int i = 1 + static_cast<int>(threadIdx.x); i < m; i += kSvdThreads) v[i] = 0.f;
        __syncthreads();
        return 0.f;
    }
    const float beta = -copysignf(sqrtf(alpha * alpha + s2), alpha);
    const float tau = (beta - alpha) / beta;
    const float scale = 1.f / (alpha - beta);
    for (int i = 1 + static_cast<int>(threadIdx.x); i < m; i += kSvdThreads) v[i] *= scale;
    if (threadIdx.x == 0) v[0] = 1.f;
    __syncthreads();
    *beta_out = beta;
    return tau;
}

// One CTA per matrix listed (grid.x = matrices).  h: the matrix's n x n fp32 H (leading
// dimension ld), overwritten; d[n], e[n - 1] at tri + tri_off[mi] (d) and + n (e).  A matrix
// whose Q is zero (final_buf == 2) gets T = 0.  Dynamic shared memory: 4 n floats + 32.
__global__ void __launch_bounds__(kSvdThreads) k_svd_tridiag(const MatDesc* __restrict__ mats,
                                                            const MatState* __restrict__ state,
                                                            float* __restrict__ hbuf,
                                                            const int64_t* __restrict__ hoff,
                                                            const int64_t* __restrict__ hss,
                                                            const int* __restrict__ nsplit,
                                                            float* __restrict__ tri,
                                                            const int64_t* __restrict__ tri_off) {
    extern __shared__ float sm[];
    const int mi = blockIdx.x;
    const MatDesc md = mats[mi];
    const int n = md.n, ld = md.ld_n;
    float* d = tri + tri_off[mi];
    float* e = d + n;
    if (state[mi].final_buf == 2) {
        for (int i = threadIdx.x; i < 2 * n - 1; i += kSvdThreads) d[i] = 0.f;
        return;
    }
    float* h = hbuf + hoff[mi];
    // split-K partials of H (the embedding's and head's long reductions): summed into split 0
    const int splits = nsplit[mi];
    if (splits > 1) {
        const int64_t ss = hss[mi];
        for (int64_t idx = threadIdx.x; idx < static_cast<int64_t>(n) * n; idx += kSvdThreads) {
            const int64_t o = (idx / n) * ld + idx % n;
            float s = h[o];
            for (int sp = 1; sp < splits; ++sp) s += h[o + sp * ss];
            h[o] = s;
        }
        __syncthreads();
    }
    float* v = sm;            // reflector of the current step (v[0] = 1)
    float* pv = sm + n;       // B v of the current step
    float* w = sm + 2 * n;    // w of the current step
    float* vn = sm + 3 * n;   // reflector of the next step
    float* red = sm + 4 * n;  // 32 floats
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    constexpr int kWarps = kSvdThreads / 32;
    if (n == 1) {
        if (threadIdx.x == 0) d[0] = h[0];
        return;
    }
    // step 0: reflector of row 0 and the product with the trailing block
    float beta;
    float tau = svd_householder(h + 1, n - 1, v, red, &beta);
    if (threadIdx.x == 0) {
        d[0] = h[0];
        e[0] = beta;
        if (n == 2) d[1] = h[ld + 1];  // a 2 x 2 matrix is already tridiagonal
    }
    {
        const int m = n - 1;
        for (int i = warp; i < m; i += kWarps) {
            const float* row = h + static_cast<int64_t>(1 + i) * ld + 1;
            float acc = 0.f;
            for (int j0 = 0; j0 < m; j0 += 32 * kUnroll) {
                float a[kUnroll];
#pragma unroll
                for (int u = 0; u < kUnroll; ++u) {
                    const int j = j0 + lane + 32 * u;
                    a[u] = j < m ? row[j] : 0.f;
                }
#pragma unroll
                for (int u = 0; u < kUnroll; ++u) {
                    const int j = j0 + lane + 32 * u;
                    if (j < m) acc = fmaf(a[u], v[j], acc);
                }
            }
            acc = svd_warp_sum(acc);
            if (lane == 0) pv[i] = acc;
        }
    }
    __syncthreads();
    for (int k = 0; k + 2 < n; ++k) {
        const int r0 = k + 1;     // first row / column of the trailing block B
        const int m = n - r0;     // its size
        // w = tau p - (tau^2 / 2)(p^T v) v, p = B v
        float pt = 0.f;
        for (int i = threadIdx.x; i < m; i += kSvdThreads) pt = fmaf(pv[i], v[i], pt);
        pt = svd_block_sum(pt, red);
        const float kk = -0.5f * tau * tau * pt;
        for (int i = threadIdx.x; i < m; i += kSvdThreads) w[i] = fmaf(kk, v[i], tau * pv[i]);
        __syncthreads();
        // row 0 of B (row r0 of H) first: it is the next step's x
        float* row0 = h + static_cast<int64_t>(r0) * ld + r0;
        const float v0 = v[0], w0 = w[0];
        for (int j = threadIdx.x; j < m; j += kSvdThreads) row0[j] -= v0 * w[j] + w0 * v[j];
        __syncthreads();
        if (threadIdx.x == 0) d[r0] = row0[0];
        if (m == 2) {
            // last 2 x 2 block: T's final entries
            if (threadIdx.x == 0) {
                e[r0] = row0[1];
                float* row1 = row0 + ld;
                d[r0 + 1] = row1[1] - (v[1] * w[1] + w[1] * v[1]);
            }
            break;
        }
        float beta_n;
        const float tau_n = svd_householder(row0 + 1, m - 1, vn, red, &beta_n);
        if (threadIdx.x == 0) e[r0] = beta_n;
        // rows 1 .. m - 1 of B: update columns 1 .. m - 1 and dot them with the next
        // reflector; each lane keeps kUnroll loads in flight (the sweep is latency bound)
        for (int i = 1 + warp; i < m; i += kWarps) {
            float* row = h + static_cast<int64_t>(r0 + i) * ld + r0;
            const float vi = v[i], wi = w[i];
            float acc = 0.f;
            for (int j0 = 1; j0 < m; j0 += 32 * kUnroll) {
                float a[kUnroll];
#pragma unroll
                for (int u = 0; u < kUnroll; ++u) {
                    const int j = j0 + lane + 32 * u;
                    a[u] = j < m ? row[j] : 0.f;
                }
#pragma unroll
                for (int u = 0; u < kUnroll; ++u) {
                    const int j = j0 + lane + 32 * u;
                    if (j < m) {
                        const float x = a[u] - (vi * w[j] + wi * v[j]);
                        row[j] = x;
                        acc = fmaf(x, vn[j - 1], acc);
                    }
                }
            }
            acc = svd_warp_sum(acc);
            if (lane == 0) pv[i - 1] = acc;
        }
        __syncthreads();
        for (int i = threadIdx.x; i < m - 1; i += kSvdThreads) v[i] = vn[i];
        tau = tau_n;
        __syncthreads();
    }
}

// Eigenvalues of the tridiagonal T (d, e) of matrix blockIdx.y by bisection; thread j finds
// the j-th smallest and stores it at sv + sv_off[mi] + (n - 1 - j) (descending order).
__global__ void __launch_bounds__(256) k_svd_bisect(const MatDesc* __restrict__ mats,
                                                    const float* __restrict__ tri,
                                                    const int64_t* __restrict__ tri_off,
                                                    float* __restrict__ sv, const int64_t* __restrict__ sv_off) {
    const int mi = blockIdx.y;
    const int n = mats[mi].n;
    const float* d = tri + tri_off[mi];
    const float* e = d + n;
    // Gershgorin interval of T (every thread computes it; n reads, cached)
    float gl = 3.4e38f, gu = -3.4e38f, emax2 = 0.f, tnorm = 0.f;
    for (int i = 0; i < n; ++i) {
        const float el = i > 0 ? fabsf(e[i - 1]) : 0.f;
        const float er = i + 1 < n ? fabsf(e[i]) : 0.f;
        gl = fminf(gl, d[i] - el - er);
        gu = fmaxf(gu, d[i] + el + er);
        emax2 = fmaxf(emax2, er * er);
        tnorm = fmaxf(tnorm, fabsf(d[i]) + el + er);
    }
    const float pivmin = fmaxf(1.17549435e-38f, 1.17549435e-38f * emax2);
    const int j = blockIdx.x * blockDim.x + threadIdx.x;
    if (j >= n) return;
    const float slack = 2.f * 1.1920929e-7f * tnorm * n + pivmin;
    float lo = gl - slack, hi = gu + slack;
    for (int it = 0; it < 64; ++it) {
        const float mid = 0.5f * (lo + hi);
        if (!(mid > lo && mid < hi)) break;
        // Sturm count: negative pivots of T - mid I
        int cnt = 0;
        float q = d[0] - mid;
        if (fabsf(q) < pivmin) q = -pivmin;
        cnt += q < 0.f;
        for (int i = 1; i < n; ++i) {
            q = d[i] - mid - e[i - 1] * e[i - 1] / q;
            if (fabsf(q) < pivmin) q = -pivmin;
            cnt += q < 0.f;
        }
        if (cnt > j)
            hi = mid;  // at least j + 1 eigenvalues below mid: the j-th smallest is below it
        else
            lo = mid;
    }
    sv[sv_off[mi] + (n - 1 - j)] = 0.5f * (lo + hi);
}

// One warp per matrix: sigma_bar = (sum of the singular values) / n (Alg. 2's mean).
__global__ void k_svd_sigma_bar(const MatDesc* __restrict__ mats, int nmat, MatState* __restrict__ state,
                                const float* __restrict__ sv, const int64_t* __restrict__ sv_off) {
    const int mi = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (mi >= nmat) return;
    const int n = mats[mi].n;
    double s = 0.0;
    for (int i = lane; i < n; i += 32) s += static_cast<double>(sv[sv_off[mi] + i]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (lane == 0 && state[mi].final_buf != 2) state[mi].sigma_bar = static_cast<float>(s / n);
}

}  // namespace isoloco
