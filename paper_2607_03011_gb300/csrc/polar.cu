// polar.cu -- per-iteration bookkeeping of the batched polar iteration, and sigma_bar.
//
//  k_gram_finalize : split-K buckets only: G = sum of the Gram partials as bf16 hi/lo
//                    planes, and per-tile sums of G^2, diag(G) and (G - I)^2 for the
//                    convergence test (the Gram GEMM's epilogue does this otherwise).
//  k_control       : one warp per matrix; sums the partials in a fixed order,
//                    normalises at t = 0 (s^2 = ||Delta^T Delta||_F >= sigma_max^2),
//                    tests ||X^T X - I||_F / sqrt(n) < tol (or, for an exactly
//                    rank-deficient Delta, the partial-isometry test below) and picks
//                    this iteration's polynomial: the next quintic of the schedule, the
//                    final cubic polish, or stop.
//  k_trace_partial / k_trace_final : sigma_bar = tr(Q^T Delta) / n (Alg. 2's mean
//                    singular value: for the polar factor Q, Q^T Delta = V S V^T).  The
//                    GEMM that writes a matrix's final Q sums its share in the epilogue
//                    (trace_fused); the partial pass covers the other matrices, reading Q's
//                    fp16 hi/lo planes and Delta's bf16 hi/lo planes.
//
// All reductions use fixed assignments and fixed shuffle trees: two runs on the same
// inputs give bitwise-identical results.
#include "common.cuh"
#include "ns_schedule.h"
#include "types.h"

namespace isoloco {

__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ double warp_sum_d(double v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Split-K buckets only: grid = one block (256 threads) per (matrix, kFinRows x 256 tile
// of the n x n Gram) listed in `ftiles`.  Sums the split partials, writes G as bf16 hi/lo
// and the tile's sums of G^2, diag(G) and (G - I)^2 (unsplit buckets do all of this
// in the Gram GEMM's epilogue).
__global__ void __launch_bounds__(256) k_gram_finalize(const MatDesc* __restrict__ mats,
                                                       const int2* __restrict__ ftiles,
                                                       const MatState* __restrict__ state,
                                                       const float* __restrict__ gpart,
                                                       const int64_t* __restrict__ gpart_off,
                                                       const int64_t* __restrict__ gpart_split_stride,
                                                       const int* __restrict__ nsplit,
                                                       __nv_bfloat16* __restrict__ ghi,
                                                       __nv_bfloat16* __restrict__ glo,
                                                       float* __restrict__ fin_part, int out_f16,
                                                       __nv_bfloat16* __restrict__ ypl, int skip_gs) {
    const int2 ft = ftiles[blockIdx.x];
    const int mi = ft.x;
    if (state[mi].done) return;
    if (skip_gs && mats[mi].gs) return;  // Gram-side matrices: their later Grams are n x n products
    // ypl != null: also write Y = yb I + yc G (hi plane) for the quintic step that may follow
    const float yb = state[mi].yb, yc = state[mi].yc;
    const MatDesc md = mats[mi];
    const int n = md.n, ld = md.ld_n;
    const int tiles_c = (n + BN - 1) / BN;
    const int r0 = (ft.y / tiles_c) * kFinRows, c0 = (ft.y % tiles_c) * BN;
    const int64_t poff = gpart_off[mi];
    const int64_t sstride = gpart_split_stride[mi];
    const int splits = nsplit[mi];

    // each thread owns 4-column groups (float4) of the tile; 8 independent loads per split
    // are in flight per thread.  Columns beyond n (row padding) are neither read as data
    // nor written.
    static_assert((kFinRows * BN / 4) % (8 * 256) == 0, "tile = 8 column groups per thread");
    constexpr int kGroups = kFinRows * BN / 4 / 256;  // column groups per thread (blockDim 256)
    float sq = 0.f, tr = 0.f, dev = 0.f;
    float4 acc[kGroups];
    int64_t idx[kGroups];
    bool any[kGroups];
#pragma unroll
    for (int i = 0; i < kGroups; ++i) {
        const int e = (threadIdx.x + i * 256) * 4;
        const int r = r0 + e / BN, c = c0 + e % BN;
        any[i] = r < n && c < n;
        idx[i] = static_cast<int64_t>(r) * ld + c;
        acc[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
    for (int sp = 0; sp < splits; ++sp) {
        const float* base = gpart + poff + sp * sstride;
        float4 t[kGroups];
#pragma unroll
        for (int i = 0; i < kGroups; ++i)
            t[i] = any[i] ? __ldg(reinterpret_cast<const float4*>(base + idx[i])) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int i = 0; i < kGroups; ++i) {
            acc[i].x += t[i].x;
            acc[i].y += t[i].y;
            acc[i].z += t[i].z;
            acc[i].w += t[i].w;
        }
    }
    const bool of16 = out_f16 != 0;
#pragma unroll
    for (int i = 0; i < kGroups; ++i) {
        if (!any[i]) continue;
        const int e = (threadIdx.x + i * 256) * 4;
        const int r = r0 + e / BN, c = c0 + e % BN;
        const float v[4] = {acc[i].x, acc[i].y, acc[i].z, acc[i].w};
        uint32_t hw[2], lw[2], yw[2];
        split16x2(v[0], v[1], of16, hw[0], lw[0]);
        split16x2(v[2], v[3], of16, hw[1], lw[1]);
        if (ypl) {
            yw[0] = round16x2(yc * v[0] + (r == c ? yb : 0.f), yc * v[1] + (r == c + 1 ? yb : 0.f), of16);
            yw[1] = round16x2(yc * v[2] + (r == c + 2 ? yb : 0.f), yc * v[3] + (r == c + 3 ? yb : 0.f), of16);
        }
        const int64_t o = md.gslot + idx[i];
        if (c + 3 < n) {
            *reinterpret_cast<uint2*>(reinterpret_cast<uint16_t*>(ghi) + o) = make_uint2(hw[0], hw[1]);
            *reinterpret_cast<uint2*>(reinterpret_cast<uint16_t*>(glo) + o) = make_uint2(lw[0], lw[1]);
            if (ypl) *reinterpret_cast<uint2*>(reinterpret_cast<uint16_t*>(ypl) + o) = make_uint2(yw[0], yw[1]);
        } else {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                if (c + q >= n) break;
                const int sh = (q & 1) * 16;
                reinterpret_cast<uint16_t*>(ghi)[o + q] = static_cast<uint16_t>(hw[q >> 1] >> sh);
                reinterpret_cast<uint16_t*>(glo)[o + q] = static_cast<uint16_t>(lw[q >> 1] >> sh);
                if (ypl) reinterpret_cast<uint16_t*>(ypl)[o + q] = static_cast<uint16_t>(yw[q >> 1] >> sh);
            }
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            if (c + q >= n) break;
            const float x = v[q];
            const bool dg = (r == c + q);
            sq += x * x;
            tr += dg ? x : 0.f;
            dev += dg ? (x - 1.f) * (x - 1.f) : x * x;
        }
    }
    __shared__ float red[3][8];
    sq = warp_sum_f(sq);
    tr = warp_sum_f(tr);
    dev = warp_sum_f(dev);
    const int w = threadIdx.x >> 5;
    if ((threadIdx.x & 31) == 0) {
        red[0][w] = sq;
        red[1][w] = tr;
        red[2][w] = dev;
    }
    __syncthreads();
    if (threadIdx.x < 3) {
        float s = 0.f;
        for (int i = 0; i < (int)(blockDim.x >> 5); ++i) s += red[threadIdx.x][i];
        // one slot of 3 per finalize tile, packed after the matrix's first slot
        fin_part[(static_cast<int64_t>(md.gpart_slot) * kPartSlots + ft.y) * 3 + threadIdx.x] = s;
    }
}

// Coefficients (a, b, c) of quintic step `step` of a matrix.  Near-square matrices (deep)
// start with one round of the deep schedule, which reaches singular values down to 1e-6
// of the normalisation.  Whatever was below that has grown by the product of its linear
// coefficients (~4e6): from 1e-8 up it is above 0.038, inside the design interval of the
// standard schedule's third step, so the next round starts there (5 steps instead of 7);
// any later round, and every round of the other matrices, is the full standard schedule.
// (Singular values under 1e-8 of s are below what the split arithmetic resolves.)
constexpr int kDeepRestart = 2;  // first standard step after the deep round

// Partial isometries (Alg. 2's Iso-C of a rank-deficient Delta: Q = U_rho V_rho^T).  A
// direction whose singular value is exactly 0 stays at 0 under every odd polynomial step,
// so ||X^T X - I||_F^2 keeps one unit per such direction and the full-rank test never
// passes.  The iteration cannot tell such a direction from a tiny nonzero one still being
// lifted, so singular values below kZeroFloor of the normalisation (under what the
// split-precision arithmetic resolves) are the ones taken as zero, and the test waits for
// the end of a round that started with every value at or above kZeroFloor inside the
// round's design interval (lift_round * kZeroFloor >= the round's first lower bound): the
// schedule then guarantees all of them in [0.998, 1.002], and what is left near 0 is zero.
// With rho = round(tr X^T X) < n directions at 1, the residual of the converged part,
// (||X^T X - I||_F^2 - (n - rho)) / rho (each zero direction adds ~1 to the first term),
// must be below tol^2; the matrix then takes the cubic polish, which keeps zeros at zero.
constexpr float kZeroFloor = 1e-8f;

// Rounds of the schedule (sched_row): a near-square matrix takes the deep round (steps
// 0 .. kSchedDeepSteps - 1), the restart round (kSchedSteps - kDeepRestart steps from the
// standard schedule's step kDeepRestart) and then standard rounds; any other matrix takes
// standard rounds.  True when `steps` quintic steps end a round; *lo is then the lower end
// of the design interval that round started from.
__device__ __forceinline__ bool round_end(bool deep, int steps, float* lo) {
    if (steps <= 0) return false;
    if (!deep) {
        *lo = kSchedLo[0];
        return steps % kSchedSteps == 0;
    }
    const int restart_end = kSchedDeepSteps + kSchedSteps - kDeepRestart;
    if (steps == kSchedDeepSteps) {
        *lo = kSchedDeepLo[0];
        return true;
    }
    if (steps == restart_end) {
        *lo = kSchedLo[kDeepRestart];
        return true;
    }
    *lo = kSchedLo[0];
    return steps > restart_end && (steps - restart_end) % kSchedSteps == 0;
}
__device__ __forceinline__ const float* sched_row(bool deep, int step) {
    if (!deep) return kSched[step % kSchedSteps];
    if (step < kSchedDeepSteps) return kSchedDeep[step];
    const int kk = step - kSchedDeepSteps;
    if (kk < kSchedSteps - kDeepRestart) return kSched[kDeepRestart + kk];
    return kSched[(kk - (kSchedSteps - kDeepRestart)) % kSchedSteps];
}

// Decision for matrix mi, taken by one warp.  t: iteration index (0 = first Gram of Delta).
__device__ void control_matrix(const MatDesc* __restrict__ mats, int mi, MatState* __restrict__ state,
                               const float* __restrict__ fin_part, int t, int max_iter, float tol,
                               uint32_t* __restrict__ err, int lane, int fast_steps, int4 gram_one,
                               int4 upd_one, int gs_on) {
    MatState& st = state[mi];
    if (st.done) {
        if (lane == 0) st.mode = 0;
        return;
    }
    const MatDesc md = mats[mi];
    // fp32 lane sums and a fixed shuffle tree: each lane adds at most a few dozen
    // non-negative terms (relative error ~1e-6, far below the tolerance this sum is
    // tested against), and fp32 keeps one SM off GB300's narrow fp64 pipe.
    // four independent accumulators per lane keep four slots' loads in flight
    const int nslots = kPartSlots * md.n_gtiles;
    const float* pp = fin_part + static_cast<int64_t>(md.gpart_slot) * kPartSlots * 3;
    float a_sq[4] = {0.f, 0.f, 0.f, 0.f}, a_tr[4] = {0.f, 0.f, 0.f, 0.f}, a_dev[4] = {0.f, 0.f, 0.f, 0.f};
    for (int i0 = lane; i0 < nslots; i0 += 128) {
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int i = i0 + 32 * u;
            if (i < nslots) {
                a_sq[u] += pp[3 * i];
                a_tr[u] += pp[3 * i + 1];
                a_dev[u] += pp[3 * i + 2];
            }
        }
    }
    float sqf = (a_sq[0] + a_sq[1]) + (a_sq[2] + a_sq[3]);
    float trf = (a_tr[0] + a_tr[1]) + (a_tr[2] + a_tr[3]);
    float devf = (a_dev[0] + a_dev[1]) + (a_dev[2] + a_dev[3]);
    sqf = warp_sum_f(sqf);
    trf = warp_sum_f(trf);
    devf = warp_sum_f(devf);
    if (lane != 0) return;
    const double sq = sqf, tr = trf;

    const double n = static_cast<double>(md.n);
    double d, gscale = 1.0, xscale = 1.0;
    const int st_step = st.step, st_iters = st.iters;  // one read each; st is global memory
    // this Gram ran a single pass (precision schedule: the step range of the matrix's kind,
    // gram_one = (standard from, to, deep from, to), and a large previous residual)
    const int g_from = md.deep ? gram_one.z : gram_one.x, g_to = md.deep ? gram_one.w : gram_one.y;
    const bool gram_single =
        !md.gs && t > 0 && st_step >= g_from && st_step < g_to && st.resid >= kOnePassGramResid;
    if (t == 0) {
        const double s2 = sqrt(sq);  // ||Delta^T Delta||_F >= sigma_max(Delta)^2
        if (!(s2 > 0.0) || !isfinite(s2)) {
            // Delta = 0 (or unusable): Q = 0, sigma_bar = 0, zero update.
            if (!isfinite(s2)) atomicOr(err, kErrNonFinite);
            st.mode = 0;
            st.done = 1;
            st.final_buf = 2;
            st.resid = 0.f;
            return;
        }
        gscale = 1.0 / s2;
        xscale = 1.0 / sqrt(s2);
        // fast variant (Sec. 4.3): sigma_bar = RMS of the singular values = ||Delta||_F / sqrt(r),
        // with ||Delta||_F^2 = tr(Delta^T Delta), the trace of this Gram
        if (fast_steps) st.sigma_bar = static_cast<float>(sqrt(fmax(0.0, tr) / n));
        // ||G/s2 - I||_F^2 = ||G||^2/s2^2 - 2 tr(G)/s2 + n, with ||G||^2/s2^2 = 1
        d = sqrt(fmax(0.0, 1.0 - 2.0 * tr * gscale + n) / n);
    } else {
        d = sqrtf(fmaxf(0.f, devf) / static_cast<float>(md.n));  // fp32: the narrow fp64 pipe is slow
    }
    st.resid = static_cast<float>(d);
    st.xscale = static_cast<float>(xscale);
    if (!isfinite(d)) {
        atomicOr(err, kErrNonFinite);
        st.mode = 0;
        st.done = 1;
        st.final_buf = 2;
        return;
    }
    // partial-isometry test at the end of a round (see kZeroFloor)
    const float lift = st.lift, lift_round = st.lift_round;
    float round_lo = 1.f;
    const bool at_round_end = round_end(md.deep != 0, st_step, &round_lo);
    bool partial = false;
    if (t > 0 && !fast_steps && at_round_end && lift_round * kZeroFloor >= round_lo) {
        const float rho = rintf(trf);
        const float ext = static_cast<float>(md.n) - rho;  // directions taken as zero
        if (rho >= 1.f && ext >= 1.f) partial = (devf - ext) / rho < tol * tol;
    }
    if (fast_steps) {
        // fast variant: a fixed number of standard quintic steps, no test, no polish (steps
        // after the schedule's last repeat it); the last one leaves Q in the buffer its
        // update writes
        const float* q = kSched[st_step < kSchedSteps ? st_step : kSchedSteps - 1];
        st.mode = 1;
        st.a = q[0];
        st.b = static_cast<float>(q[1] * gscale);
        st.c = static_cast<float>(q[2] * gscale * gscale);
        st.step = st_step + 1;
        st.iters = st_iters + 1;
        if (st_iters + 1 >= fast_steps) {
            st.done = 1;
            st.final_buf = (t + 1) & 1;
        }
    } else if ((d < tol || partial) && !gram_single) {
        // Cubic polish p(x) = 1.5 x - 0.5 x^3 on singular values already near 1 (or 0).
        // (Not from a single-pass Gram: the matrix then takes one more quintic step, and the
        // Gram after it, with a small residual, keeps its passes.)
        st.mode = 2;
        // the polish update's epilogue sums tr(Q^T Delta) (a Gram-side matrix's polish writes
        // Z, and its Q = Delta Z launch sums it instead)
        st.trace_fused = (gs_on && md.gs) ? 0 : 1;
        st.a = 1.5f;
        st.b = static_cast<float>(-0.5 * gscale);
        st.c = 0.f;
        st.iters = st_iters + 1;
        st.done = 1;
        st.final_buf = (t + 1) & 1;
    } else if (st_iters >= max_iter) {
        st.mode = 0;
        st.done = 1;
        st.final_buf = t & 1;
        st.status = kErrNotConverged;
        atomicOr(err, kErrNotConverged);
    } else {
        const float* q = sched_row(md.deep != 0, st_step);
        st.mode = 1;
        // the X this step writes needs no lo plane when the next Gram and update run single-pass
        // (next step in both ranges, this residual large: the next test cannot pass, no
        // polish) and the next iteration cannot hit max_iter (Q = X would be final)
        const int kn = st_step + 1;
        const int u_from = md.deep ? upd_one.z : upd_one.x, u_to = md.deep ? upd_one.w : upd_one.y;
        st.x_hi_only = (!md.gs && kn >= g_from && kn < g_to && kn >= u_from && kn < u_to &&
                        d >= kOnePassGramResid && st_iters + 2 <= max_iter) ? 1 : 0;
        if (st_step == 0 || at_round_end) st.lift_round = lift;  // this step starts a round
        st.lift = lift * q[0];
        st.a = q[0];
        st.b = static_cast<float>(q[1] * gscale);
        st.c = static_cast<float>(q[2] * gscale * gscale);
        st.step = st_step + 1;
        st.iters = st_iters + 1;
        // the next Gram writes Y = b I + c G of the step after this one (X normalised by then)
        const float* qn = sched_row(md.deep != 0, st_step + 1);
        st.yb = qn[1];
        st.yc = qn[2];
    }
}


// kControlThreads-thread blocks, one warp per matrix (grid = ceil(nmat / warps per block)).
// The last block to finish (a ticket counter; no block waits for another) compacts, per
// shape bucket, the matrices that still need a Gram (not done) and those that take a step
// this iteration (mode != 0), in matrix order; GEMM launches only enumerate the listed
// matrices.  As the last kernel of the polar graph's loop body (set_cond), it also sets the
// loop's condition: run the body again while some matrix is not done, at most until the
// iteration count passes max_iter (loopc[0] counts body runs in this call, reset at t = 0;
// loopc[1] counts them over the plan's life).  The ticket returns to 0 at the end.
__global__ void __launch_bounds__(kControlThreads) k_control(const MatDesc* __restrict__ mats, int nmat,
                                                             MatState* __restrict__ state,
                                                             const float* __restrict__ fin_part, int t,
                                                             int max_iter, float tol, uint32_t* __restrict__ err,
                                                             const int* __restrict__ bucket_first,
                                                             const int* __restrict__ bucket_count, int nbuckets,
                                                             int* __restrict__ list_gram, int* __restrict__ cnt_gram,
                                                             int* __restrict__ list_step, int* __restrict__ cnt_step,
                                                             cudaGraphConditionalHandle cond, int set_cond,
                                                             long long* __restrict__ loopc, int fast_steps,
                                                             int* __restrict__ ticket, int4 gram_one,
                                                             int4 upd_one, int gs_on) {
    constexpr int kWarps = kControlThreads / 32;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int mi = blockIdx.x * kWarps + warp; mi < nmat; mi += gridDim.x * kWarps) {
        control_matrix(mats, mi, state, fin_part, t, max_iter, tol, err, lane, fast_steps, gram_one, upd_one,
                       gs_on);
        __syncwarp();
    }
    __threadfence();
    __syncthreads();
    __shared__ int last;
    if (threadIdx.x == 0) last = (atomicAdd(ticket, 1) == static_cast<int>(gridDim.x) - 1);
    __syncthreads();
    if (!last) return;
    __threadfence();
    // other blocks' decisions: read past L1
    for (int bk = warp; bk < nbuckets; bk += kWarps) {
        const int first = bucket_first[bk], count = bucket_count[bk];
        int ng = 0, ns = 0;
        for (int j0 = 0; j0 < count; j0 += 32) {
            const int j = j0 + lane;
            bool g_on = false, s_on = false;
            if (j < count) {
                g_on = (__ldcg(&state[first + j].done) == 0);
                s_on = (__ldcg(&state[first + j].mode) != 0);
            }
            const unsigned bg = __ballot_sync(0xffffffffu, g_on), bs = __ballot_sync(0xffffffffu, s_on);
            const unsigned below = (1u << lane) - 1u;
            if (g_on) list_gram[first + ng + __popc(bg & below)] = j;
            if (s_on) list_step[first + ns + __popc(bs & below)] = j;
            ng += __popc(bg);
            ns += __popc(bs);
        }
        if (lane == 0) {
            cnt_gram[bk] = ng;
            cnt_step[bk] = ns;
        }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        *ticket = 0;
        if (t == 0) loopc[0] = 0;
        if (set_cond) {
            int active = 0;
            for (int bk = 0; bk < nbuckets; ++bk) active += cnt_gram[bk];
            const long long runs = ++loopc[0];
            ++loopc[1];
            const bool more = active > 0 && 2 * runs < static_cast<long long>(max_iter) + 2;
            cudaGraphSetConditional(cond, more ? 1u : 0u);
        }
    }
}

// Blocks of 256 threads take windows of 32 (matrix, row chunk) entries of `tchunks` (x =
// matrix, y = first row, z = rows, w = chunk index within the matrix), window w holding the
// entries w, w + W, w + 2W, ... (W windows; so one large matrix's chunks spread over many
// blocks): the first warp checks one entry per lane, and the block then sums the window's
// chunks whose matrix still needs its trace (no GEMM epilogue summed it: trace_fused), one
// chunk at a time.  Q comes from the final ping-pong
// buffer.
__global__ void __launch_bounds__(256) k_trace_partial(const MatDesc* __restrict__ mats,
                                                       const int4* __restrict__ tchunks, int ntchunks,
                                                       const MatState* __restrict__ state,
                                                       const __nv_bfloat16* __restrict__ dhi,
                                                       const __nv_bfloat16* __restrict__ dlo,
                                                       const __nv_bfloat16* __restrict__ x0hi,
                                                       const __nv_bfloat16* __restrict__ x0lo,
                                                       const __nv_bfloat16* __restrict__ x1hi,
                                                       const __nv_bfloat16* __restrict__ x1lo,
                                                       double* __restrict__ tpart) {
    __shared__ double red[8];
    __shared__ int todo[32];
    __shared__ int ntodo;
    const int nwin = (ntchunks + 31) / 32;
    for (int win = blockIdx.x; win < nwin; win += gridDim.x) {
        if (threadIdx.x < 32) {
            const int mine = win + static_cast<int>(threadIdx.x) * nwin;
            const bool need = mine < ntchunks && !state[tchunks[mine].x].trace_fused;
            const uint32_t m = __ballot_sync(0xffffffffu, need);
            if (need) todo[__popc(m & ((1u << threadIdx.x) - 1u))] = mine;
            if (threadIdx.x == 0) ntodo = __popc(m);
        }
        __syncthreads();
        const int cnt = ntodo;
        for (int k = 0; k < cnt; ++k) {
            const int4 tc = tchunks[todo[k]];
            const MatDesc md = mats[tc.x];
            const int fb = state[tc.x].final_buf;
            double acc = 0.0;
            if (fb == 0 || fb == 1) {
                const __nv_bfloat16* qh = (fb == 0 ? x0hi : x1hi) + md.slot;
                const __nv_bfloat16* ql = (fb == 0 ? x0lo : x1lo) + md.slot;
                const __nv_bfloat16* dh = dhi + md.slot;
                const __nv_bfloat16* dl = dlo + md.slot;
                float part = 0.f;
                if (md.ld == md.cols && (md.cols & 7) == 0) {
                    // contiguous rows: 8 elements per 16-byte load of each plane
                    const int64_t base = static_cast<int64_t>(tc.y) * md.cols;
                    const int nv = tc.z * md.cols / 8;
                    const uint4* a4 = reinterpret_cast<const uint4*>(qh + base);
                    const uint4* b4 = reinterpret_cast<const uint4*>(ql + base);
                    const uint4* c4 = reinterpret_cast<const uint4*>(dh + base);
                    const uint4* d4 = reinterpret_cast<const uint4*>(dl + base);
                    for (int v = threadIdx.x; v < nv; v += blockDim.x) {
                        const uint4 a = a4[v], bq = b4[v], c = c4[v], d = d4[v];
                        const uint32_t aw[4] = {a.x, a.y, a.z, a.w}, bw[4] = {bq.x, bq.y, bq.z, bq.w};
                        const uint32_t cw[4] = {c.x, c.y, c.z, c.w}, dw[4] = {d.x, d.y, d.z, d.w};
    #pragma unroll
                        for (int w = 0; w < 4; ++w) {
                            const float q0 = dec16(aw[w] & 0xFFFFu, true) + dec16(bw[w] & 0xFFFFu, true);
                            const float q1 = dec16(aw[w] >> 16, true) + dec16(bw[w] >> 16, true);
                            const float d0 = __uint_as_float(cw[w] << 16) + __uint_as_float(dw[w] << 16);
                            const float d1 = __uint_as_float(cw[w] & 0xFFFF0000u) + __uint_as_float(dw[w] & 0xFFFF0000u);
                            part = fmaf(q0, d0, part);
                            part = fmaf(q1, d1, part);
                        }
                    }
                } else {
                    for (int r = tc.y; r < tc.y + tc.z; ++r) {
                        for (int c = threadIdx.x; c < md.cols; c += blockDim.x) {
                            const int64_t idx = static_cast<int64_t>(r) * md.ld + c;
                            const float q = dec16(__bfloat16_as_ushort(qh[idx]), true) +
                                            dec16(__bfloat16_as_ushort(ql[idx]), true);
                            const float dv = __bfloat162float(dh[idx]) + __bfloat162float(dl[idx]);
                            part = fmaf(q, dv, part);
                        }
                    }
                }
                acc = static_cast<double>(part);
            }
            acc = warp_sum_d(acc);
            if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
            __syncthreads();
            if (threadIdx.x == 0) {
                double s = 0.0;
                for (int i = 0; i < (int)(blockDim.x >> 5); ++i) s += red[i];
                tpart[md.trace_part + tc.w] = s;
            }
            __syncthreads();  // red is reused by the next chunk
        }
        __syncthreads();  // todo and ntodo are rewritten by the next window
    }
}

// One block of 256 threads per matrix: sigma_bar = (sum of the trace partials) / n, the
// partials from k_trace_partial's row chunks or, for a matrix whose Q-writing GEMM summed them,
// from that GEMM's tile slots.  Fixed order: four strided accumulators per thread, then a fixed
// tree over the threads.
__global__ void __launch_bounds__(256) k_trace_final(const MatDesc* __restrict__ mats, int nmat,
                                                     MatState* __restrict__ state,
                                                     const double* __restrict__ tpart,
                                                     const double* __restrict__ tfpart) {
    const int mi = blockIdx.x;
    if (mi >= nmat) return;
    const MatDesc md = mats[mi];
    const bool fused = state[mi].trace_fused != 0;
    const double* src = fused ? tfpart + md.tf_part : tpart + md.trace_part;
    const int cnt = fused ? md.tf_slots : md.n_tchunks;
    double a[4] = {0.0, 0.0, 0.0, 0.0};
    for (int i0 = threadIdx.x; i0 < cnt; i0 += 4 * 256) {
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int i = i0 + 256 * u;
            if (i < cnt) a[u] += src[i];
        }
    }
    double s = (a[0] + a[1]) + (a[2] + a[3]);
    __shared__ double red[8];
    s = warp_sum_d(s);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
    __syncthreads();
    if (threadIdx.x == 0) {
        double t = 0.0;
        for (int w = 0; w < 8; ++w) t += red[w];
        MatState& st = state[mi];
        st.trace = t;
        st.sigma_bar = (st.final_buf == 2) ? 0.f : static_cast<float>(t / md.n);
    }
}

// Resets the per-matrix state before a step: every matrix is active for the first Gram,
// and the GEMM launches' tile counters restart at zero.
__global__ void k_reset_state(MatState* state, int nmat, uint32_t* err, const MatDesc* __restrict__ mats,
                              const int* __restrict__ bucket_first, const int* __restrict__ bucket_count,
                              int nbuckets, int* __restrict__ list_gram, int* __restrict__ cnt_gram,
                              int* __restrict__ counters, int ncounters) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i == 0) *err = 0u;
    for (int c = i; c < ncounters; c += gridDim.x * blockDim.x) counters[c] = 0;
    if (i < nbuckets) cnt_gram[i] = bucket_count[i];
    if (i < nmat) list_gram[i] = i - bucket_first[mats[i].bucket];
    if (i >= nmat) return;
    MatState s;
    s.a = s.b = s.c = 0.f;
    s.xscale = 1.f;
    s.resid = 0.f;
    s.sigma_bar = 0.f;
    s.mode = 0;
    s.step = 0;
    s.iters = 0;
    s.done = 0;
    s.final_buf = 2;
    s.yb = s.yc = 0.f;
    s.status = 0;
    s.lift = 1.f;
    s.lift_round = 1.f;
    s.xs0 = 1.f;
    s.x_hi_only = 0;
    s.trace = 0.0;
    s.trace_fused = 0;
    state[i] = s;
}

}  // namespace isoloco
