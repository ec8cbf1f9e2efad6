/*
 * isoloco_oracle.c -- plain fp64 CPU oracle for the IsoLoCo / DiLoCo outer step.
 *
 * TEST INFRASTRUCTURE ONLY.  This is the slow, obviously correct restatement of
 * what the outer step computes.  It exists to check the CUDA library; only the
 * test suite, the smoke check and the benchmark's CPU-baseline leg load it.  It
 * shares no code, header or table with the CUDA path.
 *
 * Paper: "Can Model Merging Improve Aggregation in DiLoCo?" (arXiv 2607.03011).
 *   Alg. 1 (DiLoCo):  Delta = (1/R) sum_i (theta^{t-1} - theta_i), then OuterOpt.
 *   Alg. 2 (IsoLoCo): mean pseudo-gradient; for every tensor with dim == 2 take
 *       the SVD  Delta = U S V^T,  sigma_bar = (1/r) sum_k sigma_k,
 *       Delta <- sigma_bar U V^T;  then Nesterov momentum
 *       B <- mu B + Delta,  P <- Delta + mu B,  theta <- theta - eta_out P.
 *   Sec. 2.2 / Eq. 1: task arithmetic  theta_0 + lambda sum_t tau_t with
 *       tau_t = theta_t - theta_0; Iso-C sums the task matrices, takes the SVD
 *       and replaces every singular value by their mean.
 *
 * Everything here is double precision.  The SVD is a hand-written one-sided
 * (Hestenes) Jacobi iteration; tall matrices are first reduced by a Householder
 * QR so that only the n x n factor R is rotated.  No BLAS/LAPACK is used.
 *
 * Readings of points the paper leaves open (each one is listed in the design
 * notes of the repository):
 *   - sign: Delta_k = theta_global - theta_k and theta <- theta - eta P (Alg. 1/2);
 *   - r = min(m, n); singular values below r * eps * sigma_max count as zero and
 *     the polar factor is the partial isometry U_rho V_rho^T;
 *   - alpha (Iso-C's merging scale) multiplies only the 2-D Iso-C output;
 *   - non-matrix parameters use the plain mean pseudo-gradient (Sec. 4 text).
 *
 * Parity status: pinned.  The unit tests check these routines against closed
 * forms (2x2 polar), invariants (all output singular values equal alpha*sigma_bar,
 * nuclear norm preserved, Q^T Delta symmetric PSD), special cases (c * orthogonal,
 * diagonal, 1 x n), an independent scaled-Newton polar, a library SVD, and a
 * hand-worked Nesterov example.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#include <float.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORC_OK 0
#define ORC_ERR_INVALID (-1)
#define ORC_ERR_NOMEM (-2)
#define ORC_ERR_NOCONV (-3)

/* ------------------------------------------------------------------------- */
/* Element access for the worker replicas: fp32 or bf16 (upcast exactly).     */
/* ------------------------------------------------------------------------- */

static double bf16_bits_to_double(uint16_t h) {
    uint32_t u = ((uint32_t)h) << 16; /* bf16 is the top half of an fp32 */
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

static double replica_at(const void* rep, int dtype, int64_t i) {
    if (dtype == 0) return (double)((const float*)rep)[i];
    return bf16_bits_to_double(((const uint16_t*)rep)[i]);
}

int orc_num_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* ------------------------------------------------------------------------- */
/* Pseudo-gradient reduction (Alg. 1 "Average pseudo-gradients"; Alg. 2 mean)  */
/*   mode 0: (1/K) sum_k (theta - theta_k)       -- DiLoCo / IsoLoCo           */
/*   mode 1:       sum_k (theta - theta_k)                                     */
/*   mode 2:       sum_k (theta_k - theta)       -- task vectors, Eq. 1        */
/* Each difference is taken first and then summed, in fp64.                   */
/* ------------------------------------------------------------------------- */
void orc_pseudo_gradient(int64_t n, const float* theta, const void* const* reps,
                         int K, int dtype, int mode, double* out) {
    int64_t i;
#pragma omp parallel for schedule(static)
    for (i = 0; i < n; ++i) {
        double s = 0.0;
        for (int k = 0; k < K; ++k) {
            double d = (double)theta[i] - replica_at(reps[k], dtype, i);
            s += (mode == 2) ? -d : d;
        }
        out[i] = (mode == 0) ? s / (double)K : s;
    }
}

/* ------------------------------------------------------------------------- */
/* Nesterov outer optimiser, Alg. 2:                                          */
/*   B' = mu B + U;   P = U + mu B';   theta' = theta - eta P                  */
/* ------------------------------------------------------------------------- */
void orc_nesterov(int64_t n, const double* U, double mu, double eta,
                  const double* theta_in, const double* B_in,
                  double* theta_out, double* B_out) {
    int64_t i;
#pragma omp parallel for schedule(static)
    for (i = 0; i < n; ++i) {
        double b = mu * B_in[i] + U[i];
        double p = U[i] + mu * b;
        theta_out[i] = theta_in[i] - eta * p;
        B_out[i] = b;
    }
}

/* ------------------------------------------------------------------------- */
/* One-sided (Hestenes) Jacobi on the columns of W (column-major, m x n).      */
/* Rotates pairs of columns until every pair is numerically orthogonal:        */
/*   |w_p . w_q| <= tol * ||w_p|| ||w_q||.                                    */
/* V (column-major n x n) accumulates the rotations, so that on exit           */
/*   W_in V = W_out  with orthogonal columns,  sigma_i = ||w_i||.              */
/* Pairs are visited in round-robin (tournament) order, so the n/2 pairs of a  */
/* round touch disjoint columns and may be rotated concurrently.               */
/* A column whose squared norm is at most `neg2` = n (eps ||W||_F)^2 is below  */
/* Iso-C's zero cut r eps sigma_max (||W||_F <= sqrt(n) sigma_max, r = n): it  */
/* is not rotated.  Without this the rounding-level columns of an exactly      */
/* rank-deficient W keep rotating among themselves and the sweeps never end.   */
/* ------------------------------------------------------------------------- */
static int rotate_pair(int m, int n, double* wp, double* wq, double* vp, double* vq,
                       double tol, double neg2) {
    double a = 0.0, b = 0.0, c = 0.0;
    for (int i = 0; i < m; ++i) {
        a += wp[i] * wp[i];
        b += wq[i] * wq[i];
        c += wp[i] * wq[i];
    }
    if (a <= neg2 || b <= neg2) return 0;
    if (fabs(c) <= tol * sqrt(a) * sqrt(b)) return 0;
    /* Choose the rotation angle that zeroes the off-diagonal entry of the 2x2
     * Gram [[a, c], [c, b]]: t = tan(angle) is the smaller root of
     * t^2 + 2 zeta t - 1 = 0 with zeta = (b - a) / (2c). */
    double zeta = (b - a) / (2.0 * c);
    double t = (zeta >= 0.0 ? 1.0 : -1.0) / (fabs(zeta) + sqrt(1.0 + zeta * zeta));
    double cs = 1.0 / sqrt(1.0 + t * t);
    double sn = cs * t;
    for (int i = 0; i < m; ++i) {
        double x = wp[i], y = wq[i];
        wp[i] = cs * x - sn * y;
        wq[i] = sn * x + cs * y;
    }
    for (int i = 0; i < n; ++i) {
        double x = vp[i], y = vq[i];
        vp[i] = cs * x - sn * y;
        vq[i] = sn * x + cs * y;
    }
    return 1;
}

static int jacobi_svd_cols(int m, int n, double* W, double* V, int max_sweeps,
                           int* sweeps_out) {
    int n2 = n + (n & 1);
    int* order = (int*)malloc(sizeof(int) * (size_t)(n2 > 0 ? n2 : 1));
    if (!order) return ORC_ERR_NOMEM;
    for (int i = 0; i < n2; ++i) order[i] = i; /* index n is a bye when n is odd */
    for (int j = 0; j < n; ++j)
        for (int i = 0; i < n; ++i) V[(size_t)j * n + i] = (i == j) ? 1.0 : 0.0;
    double tol = (double)(m > 1 ? m : 1) * DBL_EPSILON;
    double fro2 = 0.0;
    for (size_t i = 0; i < (size_t)m * n; ++i) fro2 += W[i] * W[i];
    double neg2 = (double)n * DBL_EPSILON * DBL_EPSILON * fro2;
    int sweep = 0, converged = (n < 2);
    while (!converged && sweep < max_sweeps) {
        long rotated = 0;
        for (int round = 0; round < n2 - 1; ++round) {
            int k;
#pragma omp parallel for reduction(+ : rotated) schedule(dynamic, 4)
            for (k = 0; k < n2 / 2; ++k) {
                int p = order[k], q = order[n2 - 1 - k];
                if (p >= n || q >= n) continue;
                if (p > q) { int tmp = p; p = q; q = tmp; }
                rotated += rotate_pair(m, n, W + (size_t)p * m, W + (size_t)q * m,
                                       V + (size_t)p * n, V + (size_t)q * n, tol, neg2);
            }
            /* tournament schedule: keep order[0], cycle the rest by one seat */
            int last = order[n2 - 1];
            memmove(order + 2, order + 1, sizeof(int) * (size_t)(n2 - 2));
            order[1] = last;
        }
        ++sweep;
        converged = (rotated == 0);
    }
    free(order);
    if (sweeps_out) *sweeps_out = sweep;
    return converged ? ORC_OK : ORC_ERR_NOCONV;
}

/* ------------------------------------------------------------------------- */
/* Householder QR of a column-major m x n matrix (m >= n), in place.           */
/* On exit the upper triangle holds R; below the diagonal of column j sit the  */
/* trailing entries of v_j (whose leading entry is 1), and tau[j] its factor:  */
/*   H_j = I - tau_j v_j v_j^T,   Q = H_0 H_1 ... H_{n-1}.                     */
/* ------------------------------------------------------------------------- */
static void householder_qr(int m, int n, double* A, double* tau) {
    for (int j = 0; j < n; ++j) {
        double* x = A + (size_t)j * m + j; /* x = A[j:m, j] */
        int len = m - j;
        double alpha = x[0], s2 = 0.0;
        for (int i = 1; i < len; ++i) s2 += x[i] * x[i];
        if (s2 == 0.0) { tau[j] = 0.0; continue; } /* already upper triangular */
        double beta = -copysign(sqrt(alpha * alpha + s2), alpha);
        tau[j] = (beta - alpha) / beta;
        double inv = 1.0 / (alpha - beta);
        for (int i = 1; i < len; ++i) x[i] *= inv;
        x[0] = beta;
        int k;
#pragma omp parallel for schedule(static)
        for (k = j + 1; k < n; ++k) {
            double* c = A + (size_t)k * m + j;
            double w = c[0];
            for (int i = 1; i < len; ++i) w += x[i] * c[i];
            w *= tau[j];
            c[0] -= w;
            for (int i = 1; i < len; ++i) c[i] -= w * x[i];
        }
    }
}

/* Y (column-major m x n) <- Q Y with Q from householder_qr's reflectors. */
static void apply_q(int m, int n, const double* A, const double* tau, int ncols, double* Y) {
    for (int j = n - 1; j >= 0; --j) {
        if (tau[j] == 0.0) continue;
        const double* v = A + (size_t)j * m + j;
        int len = m - j;
        int k;
#pragma omp parallel for schedule(static)
        for (k = 0; k < ncols; ++k) {
            double* c = Y + (size_t)k * m + j;
            double w = c[0];
            for (int i = 1; i < len; ++i) w += v[i] * c[i];
            w *= tau[j];
            c[0] -= w;
            for (int i = 1; i < len; ++i) c[i] -= w * v[i];
        }
    }
}

/* ------------------------------------------------------------------------- */
/* Thin SVD of a tall column-major m x n matrix (m >= n):  A = U diag(S) V^T.  */
/* U: column-major m x n, S: n, V: column-major n x n.  A is destroyed.        */
/* ------------------------------------------------------------------------- */
static int svd_tall_colmajor(int m, int n, double* A, double* U, double* S, double* V,
                             int* sweeps) {
    int rc;
    if (m == n) {
        memcpy(U, A, sizeof(double) * (size_t)m * n);
        rc = jacobi_svd_cols(m, n, U, V, 80, sweeps);
    } else {
        double* tau = (double*)malloc(sizeof(double) * (size_t)n);
        double* R = (double*)calloc((size_t)n * n, sizeof(double));
        if (!tau || !R) { free(tau); free(R); return ORC_ERR_NOMEM; }
        householder_qr(m, n, A, tau);
        for (int j = 0; j < n; ++j)
            for (int i = 0; i <= j; ++i) R[(size_t)j * n + i] = A[(size_t)j * m + i];
        rc = jacobi_svd_cols(n, n, R, V, 80, sweeps);
        /* U = Q [W_R ; 0]; the columns are normalised below */
        memset(U, 0, sizeof(double) * (size_t)m * n);
        for (int j = 0; j < n; ++j)
            memcpy(U + (size_t)j * m, R + (size_t)j * n, sizeof(double) * (size_t)n);
        apply_q(m, n, A, tau, n, U);
        free(tau);
        free(R);
    }
    /* sigma_j = ||w_j||, u_j = w_j / sigma_j (zero columns stay zero) */
    for (int j = 0; j < n; ++j) {
        double s = 0.0;
        double* u = U + (size_t)j * m;
        for (int i = 0; i < m; ++i) s += u[i] * u[i];
        s = sqrt(s);
        S[j] = s;
        if (s > 0.0)
            for (int i = 0; i < m; ++i) u[i] /= s;
    }
    return rc;
}

/* ------------------------------------------------------------------------- */
/* Public: thin SVD of a row-major m x n matrix, any orientation.              */
/*   U: row-major m x r, S: r, V: row-major n x r, r = min(m, n);               */
/*   A = U diag(S) V^T.  Singular values are in no particular order.            */
/* ------------------------------------------------------------------------- */
int orc_svd(int m, int n, const double* A, double* U, double* S, double* V, int* sweeps) {
    if (m <= 0 || n <= 0) return ORC_ERR_INVALID;
    int tall = (m >= n);
    int M = tall ? m : n, N = tall ? n : m; /* work on the tall orientation */
    double* W = (double*)malloc(sizeof(double) * (size_t)M * N);
    double* Uc = (double*)malloc(sizeof(double) * (size_t)M * N);
    double* Vc = (double*)malloc(sizeof(double) * (size_t)N * N);
    if (!W || !Uc || !Vc) { free(W); free(Uc); free(Vc); return ORC_ERR_NOMEM; }
    /* column-major copy of T = A (tall) or A^T (wide):  T[i][j] at W[j*M + i] */
    for (int i = 0; i < M; ++i)
        for (int j = 0; j < N; ++j)
            W[(size_t)j * M + i] = tall ? A[(size_t)i * n + j] : A[(size_t)j * n + i];
    int rc = svd_tall_colmajor(M, N, W, Uc, S, Vc, sweeps);
    /* T = Uc S Vc^T.  If A = T^T then A = Vc S Uc^T: swap the roles. */
    const double* left = tall ? Uc : Vc;
    const double* right = tall ? Vc : Uc;
    int ldl = tall ? M : N, ldr = tall ? N : M;
    for (int i = 0; i < m; ++i)
        for (int k = 0; k < N; ++k) U[(size_t)i * N + k] = left[(size_t)k * ldl + i];
    for (int j = 0; j < n; ++j)
        for (int k = 0; k < N; ++k) V[(size_t)j * N + k] = right[(size_t)k * ldr + j];
    free(W);
    free(Uc);
    free(Vc);
    return rc;
}

/* ------------------------------------------------------------------------- */
/* Iso-C on one matrix (Sec. 2.2; Alg. 2 lines under "dim == 2"):               */
/*   U S V^T = SVD(D);  sigma_bar = (1/r) sum_k sigma_k;  out = alpha sigma_bar  */
/*   U_rho V_rho^T, where rho counts the singular values above r*eps*sigma_max.  */
/* Returns sigma_bar in *sigma_bar_out and the sweep count in *sweeps.          */
/* ------------------------------------------------------------------------- */
int orc_iso_c(int m, int n, const double* D, double alpha, double* out,
              double* sigma_bar_out, int* sweeps) {
    if (m <= 0 || n <= 0) return ORC_ERR_INVALID;
    int r = m < n ? m : n;
    double* U = (double*)malloc(sizeof(double) * (size_t)m * r);
    double* S = (double*)malloc(sizeof(double) * (size_t)r);
    double* V = (double*)malloc(sizeof(double) * (size_t)n * r);
    if (!U || !S || !V) { free(U); free(S); free(V); return ORC_ERR_NOMEM; }
    int rc = orc_svd(m, n, D, U, S, V, sweeps);
    double smax = 0.0, ssum = 0.0;
    for (int k = 0; k < r; ++k) {
        ssum += S[k];
        if (S[k] > smax) smax = S[k];
    }
    double sigma_bar = ssum / (double)r;
    double cut = (double)r * DBL_EPSILON * smax;
    for (int k = 0; k < r; ++k)
        if (!(S[k] > cut)) /* rank-deficient direction: drop from U V^T */
            for (int i = 0; i < m; ++i) U[(size_t)i * r + k] = 0.0;
    double scale = alpha * sigma_bar;
    int i;
#pragma omp parallel for schedule(static)
    for (i = 0; i < m; ++i) {
        const double* ui = U + (size_t)i * r;
        for (int j = 0; j < n; ++j) {
            const double* vj = V + (size_t)j * r;
            double acc = 0.0;
            for (int k = 0; k < r; ++k) acc += ui[k] * vj[k];
            out[(size_t)i * n + j] = scale * acc;
        }
    }
    if (sigma_bar_out) *sigma_bar_out = sigma_bar;
    free(U);
    free(S);
    free(V);
    return rc;
}

/* ------------------------------------------------------------------------- */
/* Whole outer steps over a parameter table.                                   */
/* Parameter p occupies [offs[p], offs[p] + rows[p]*max(cols[p],1)) of every    */
/* flat buffer; cols[p] == 0 marks a 1-D tensor of rows[p] elements.            */
/* ------------------------------------------------------------------------- */
static int check_table(const int64_t* offs, const int* rows, const int* cols, int np,
                       int64_t N) {
    for (int p = 0; p < np; ++p) {
        int64_t len = (int64_t)rows[p] * (cols[p] > 0 ? cols[p] : 1);
        if (rows[p] <= 0 || cols[p] < 0 || offs[p] < 0 || offs[p] + len > N)
            return ORC_ERR_INVALID;
    }
    return ORC_OK;
}

/* IsoLoCo outer step, Alg. 2.  reduce_mean = 1 follows Alg. 2 (mean); 0 sums.
 * theta_out / B_out: fp64 results of the step.  U_out (nullable): the update
 * direction U (alpha*sigma_bar*Q for 2-D, Delta for 1-D).  sigma_bar_out
 * (nullable): one entry per parameter (0 for 1-D).  Parameters with
 * do_param[p] == 0 are skipped entirely (their outputs are left untouched);
 * do_param may be NULL (all parameters).  */
int orc_isoloco_outer_step(const int64_t* offs, const int* rows, const int* cols, int np,
                           int64_t N, const float* theta, const float* B,
                           const void* const* reps, int K, int dtype, double alpha,
                           double eta, double mu, int reduce_mean, const int* do_param,
                           double* theta_out, double* B_out, double* U_out,
                           double* sigma_bar_out, int* sweeps_out) {
    if (K <= 0 || check_table(offs, rows, cols, np, N) != ORC_OK) return ORC_ERR_INVALID;
    int rc_all = ORC_OK;
    for (int p = 0; p < np; ++p) {
        if (do_param && !do_param[p]) continue;
        int64_t o = offs[p];
        int m = rows[p], n = cols[p];
        int64_t len = (int64_t)m * (n > 0 ? n : 1);
        double* D = (double*)malloc(sizeof(double) * (size_t)len);
        double* Uu = (double*)malloc(sizeof(double) * (size_t)len);
        double* th = (double*)malloc(sizeof(double) * (size_t)len);
        double* bb = (double*)malloc(sizeof(double) * (size_t)len);
        const void* rp[1024];
        if (!D || !Uu || !th || !bb || K > 1024) {
            free(D); free(Uu); free(th); free(bb);
            return ORC_ERR_NOMEM;
        }
        for (int k = 0; k < K; ++k)
            rp[k] = (const char*)reps[k] + (size_t)o * (dtype == 0 ? 4 : 2);
        orc_pseudo_gradient(len, theta + o, rp, K, dtype, reduce_mean ? 0 : 1, D);
        double sb = 0.0;
        int sw = 0;
        if (n > 0) {
            int rc = orc_iso_c(m, n, D, alpha, Uu, &sb, &sw);
            if (rc != ORC_OK) rc_all = rc;
        } else {
            memcpy(Uu, D, sizeof(double) * (size_t)len); /* 1-D: plain mean */
        }
        for (int64_t i = 0; i < len; ++i) {
            th[i] = (double)theta[o + i];
            bb[i] = (double)B[o + i];
        }
        orc_nesterov(len, Uu, mu, eta, th, bb, theta_out + o, B_out + o);
        if (U_out) memcpy(U_out + o, Uu, sizeof(double) * (size_t)len);
        if (sigma_bar_out) sigma_bar_out[p] = sb;
        if (sweeps_out) sweeps_out[p] = sw;
        free(D); free(Uu); free(th); free(bb);
    }
    return rc_all;
}

/* DiLoCo outer step, Alg. 1 with Nesterov SGD as OuterOpt (same update as
 * Alg. 2 without the Iso-C correction). */
int orc_diloco_outer_step(int64_t N, const float* theta, const float* B,
                          const void* const* reps, int K, int dtype, double eta, double mu,
                          int reduce_mean, double* theta_out, double* B_out) {
    if (K <= 0 || N < 0) return ORC_ERR_INVALID;
    double* D = (double*)malloc(sizeof(double) * (size_t)(N > 0 ? N : 1));
    double* th = (double*)malloc(sizeof(double) * (size_t)(N > 0 ? N : 1));
    double* bb = (double*)malloc(sizeof(double) * (size_t)(N > 0 ? N : 1));
    if (!D || !th || !bb) { free(D); free(th); free(bb); return ORC_ERR_NOMEM; }
    orc_pseudo_gradient(N, theta, reps, K, dtype, reduce_mean ? 0 : 1, D);
    for (int64_t i = 0; i < N; ++i) {
        th[i] = (double)theta[i];
        bb[i] = (double)B[i];
    }
    orc_nesterov(N, D, mu, eta, th, bb, theta_out, B_out);
    free(D); free(th); free(bb);
    return ORC_OK;
}

/* Iso-C model merge (Sec. 2.2 with Eq. 1's form): tau_k = theta_k - theta_base,
 * T = sum_k tau_k;  out = base + alpha * IsoC(T) for 2-D tensors and
 * out = base + alpha * T for the others. */
int orc_iso_c_merge(const int64_t* offs, const int* rows, const int* cols, int np, int64_t N,
                    const float* base, const void* const* experts, int K, int dtype,
                    double alpha, const int* do_param, double* out, double* sigma_bar_out) {
    if (K <= 0 || check_table(offs, rows, cols, np, N) != ORC_OK) return ORC_ERR_INVALID;
    int rc_all = ORC_OK;
    for (int p = 0; p < np; ++p) {
        if (do_param && !do_param[p]) continue;
        int64_t o = offs[p];
        int m = rows[p], n = cols[p];
        int64_t len = (int64_t)m * (n > 0 ? n : 1);
        double* T = (double*)malloc(sizeof(double) * (size_t)len);
        double* Uu = (double*)malloc(sizeof(double) * (size_t)len);
        const void* rp[1024];
        if (!T || !Uu || K > 1024) { free(T); free(Uu); return ORC_ERR_NOMEM; }
        for (int k = 0; k < K; ++k)
            rp[k] = (const char*)experts[k] + (size_t)o * (dtype == 0 ? 4 : 2);
        orc_pseudo_gradient(len, base + o, rp, K, dtype, 2, T);
        double sb = 0.0;
        if (n > 0) {
            int sw = 0;
            int rc = orc_iso_c(m, n, T, alpha, Uu, &sb, &sw);
            if (rc != ORC_OK) rc_all = rc;
        } else {
            for (int64_t i = 0; i < len; ++i) Uu[i] = alpha * T[i];
        }
        for (int64_t i = 0; i < len; ++i) out[o + i] = (double)base[o + i] + Uu[i];
        if (sigma_bar_out) sigma_bar_out[p] = sb;
        free(T); free(Uu);
    }
    return rc_all;
}
