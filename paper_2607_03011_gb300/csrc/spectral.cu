// spectral.cu -- the clip_high / clip_low variants of Sec. 4.5: the singular values of
// Delta above (clip_high) or below (clip_low) their mean sigma_bar are set to sigma_bar,
// the others kept.
//
// For a tall matrix with polar factor Q (Delta = U S V^T, Q = U V^T), H = Q^T Delta =
// V S V^T and A' = H / sigma_bar - I = V (S / sigma_bar - I) V^T.  Q_A = sign(A') (the
// polar factor of that symmetric matrix) splits the right singular directions: P_lo =
// (I - Q_A) / 2 projects on those with s < sigma_bar, P_hi = (I + Q_A) / 2 on the others.
// Then, with P = P_lo (clip_high) or P_hi (clip_low),
//   S' = I + P A' P = V f(S) V^T / sigma_bar,   U_clip = sigma_bar Q S',
// f(s) = min(s, sigma_bar) or max(s, sigma_bar).  P appears on both sides so that its error
// in a direction with a large s (where A' is large) enters only at second order.  A wide
// matrix uses H = Delta Q^T and multiplies from the left.  The GEMMs (H; P A'; (P A') P;
// Q S') run on the split-precision tcgen05 kernel, sign(A') is the polar iteration of an
// auxiliary plan of the n x n matrices, and Q S' replaces Q in the other ping-pong buffer
// so that the apply pass forms U = alpha sigma_bar (Q S') as for Iso-C.  The kernels here
// move data between those stages, one CTA row per matrix (grid.y).
#include "common.cuh"
#include "types.h"

namespace isoloco {

// Eight 16-bit values of a hi/lo plane pair as floats (16-byte loads).
__device__ __forceinline__ void ld16x8(const __nv_bfloat16* hi, const __nv_bfloat16* lo, int64_t o, bool f16,
                                       float (&v)[8]) {
    const uint4 h = *reinterpret_cast<const uint4*>(hi + o);
    const uint4 l = *reinterpret_cast<const uint4*>(lo + o);
    const uint32_t hw[4] = {h.x, h.y, h.z, h.w}, lw[4] = {l.x, l.y, l.z, l.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        v[2 * q] = dec16(hw[q] & 0xFFFFu, f16) + dec16(lw[q] & 0xFFFFu, f16);
        v[2 * q + 1] = dec16(hw[q] >> 16, f16) + dec16(lw[q] >> 16, f16);
    }
}

// Eight floats as a hi/lo plane pair of 16-bit values (16-byte stores).
__device__ __forceinline__ void st16x8(__nv_bfloat16* hi, __nv_bfloat16* lo, int64_t o, bool f16,
                                       const float (&v)[8]) {
    uint32_t hw[4], lw[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) split16x2(v[2 * q], v[2 * q + 1], f16, hw[q], lw[q]);
    *reinterpret_cast<uint4*>(hi + o) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
    *reinterpret_cast<uint4*>(lo + o) = make_uint4(lw[0], lw[1], lw[2], lw[3]);
}

// Q (fp16 hi/lo planes in buffer final_buf) -> bf16 hi/lo planes in the other buffer, the
// operand type of Delta's planes (one MMA never mixes fp16 and bf16).  Eight elements per
// thread over the padded rows (ld is a multiple of 8; padding columns are never read as data).
__global__ void __launch_bounds__(256) k_clip_q_bf16(const MatDesc* __restrict__ mats,
                                                     const MatState* __restrict__ state,
                                                     __nv_bfloat16* xh0, __nv_bfloat16* xl0,
                                                     __nv_bfloat16* xh1, __nv_bfloat16* xl1) {
    const int mi = blockIdx.y;
    const int fb = state[mi].final_buf;
    if (fb > 1) return;
    const MatDesc md = mats[mi];
    const __nv_bfloat16* sh = fb ? xh1 : xh0;
    const __nv_bfloat16* sl = fb ? xl1 : xl0;
    __nv_bfloat16* dh = fb ? xh0 : xh1;
    __nv_bfloat16* dl = fb ? xl0 : xl1;
    const int64_t groups = static_cast<int64_t>(md.rows) * md.ld / 8;
    for (int64_t g = blockIdx.x * 256 + threadIdx.x; g < groups; g += static_cast<int64_t>(gridDim.x) * 256) {
        const int64_t o = md.slot + 8 * g;
        float v[8];
        ld16x8(sh, sl, o, true, v);
        st16x8(dh, dl, o, false, v);
    }
}

// The n x n kernels below run eight consecutive columns per thread over rows padded to a
// multiple of 8 (ld_n); padding columns are never read as data.

// A' = H / sigma_bar - I into the auxiliary plan's input planes (bf16 hi/lo), H summed from
// the fp32 split-K partials of the H GEMM; a matrix whose Q is 0 (Delta = 0) gets A' = 0.
__global__ void __launch_bounds__(256) k_clip_form_a(const MatDesc* __restrict__ mats,
                                                     const MatState* __restrict__ state,
                                                     const float* __restrict__ hbuf,
                                                     const int64_t* __restrict__ hoff,
                                                     const int64_t* __restrict__ hsstride,
                                                     const int* __restrict__ nsplit,
                                                     const MatDesc* __restrict__ amats,
                                                     const int* __restrict__ aux_of,
                                                     __nv_bfloat16* __restrict__ ah,
                                                     __nv_bfloat16* __restrict__ al) {
    const int mi = blockIdx.y;
    const MatDesc md = mats[mi];
    const MatDesc amd = amats[aux_of[mi]];
    const float sbar = state[mi].sigma_bar;
    const bool zero = state[mi].final_buf > 1 || !(sbar > 0.f);
    const float inv = zero ? 0.f : 1.f / sbar;
    const int ld = md.ld_n, splits = nsplit[mi];
    const float* h0 = hbuf + hoff[mi];
    const int64_t ss = hsstride[mi];
    const int64_t groups = static_cast<int64_t>(md.n) * ld / 8;
    for (int64_t g = blockIdx.x * 256 + threadIdx.x; g < groups; g += static_cast<int64_t>(gridDim.x) * 256) {
        const int64_t e = 8 * g;
        const int r = static_cast<int>(e / ld), c = static_cast<int>(e % ld);
        float v[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        if (!zero) {
            for (int sp = 0; sp < splits; ++sp) {
                const float4 x = *reinterpret_cast<const float4*>(h0 + sp * ss + e);
                const float4 y = *reinterpret_cast<const float4*>(h0 + sp * ss + e + 4);
                v[0] += x.x; v[1] += x.y; v[2] += x.z; v[3] += x.w;
                v[4] += y.x; v[5] += y.y; v[6] += y.z; v[7] += y.w;
            }
#pragma unroll
            for (int q = 0; q < 8; ++q) v[q] = v[q] * inv - (c + q == r ? 1.f : 0.f);
        }
        st16x8(ah, al, amd.slot + static_cast<int64_t>(r) * amd.ld + c, false, v);
    }
}

// P = (I + sgn Q_A) / 2 (sgn = -1: P_lo for clip_high, +1: P_hi for clip_low) as bf16 hi/lo
// planes in the auxiliary buffer that does not hold Q_A (fp16 planes).  Grid.y runs over the
// auxiliary matrices; those with Q_A = 0 (A' = 0) are skipped (S' = I for them).
__global__ void __launch_bounds__(256) k_clip_form_p(const MatDesc* __restrict__ amats,
                                                     const MatState* __restrict__ astate,
                                                     __nv_bfloat16* axh0, __nv_bfloat16* axl0,
                                                     __nv_bfloat16* axh1, __nv_bfloat16* axl1, float sgn) {
    const int ai = blockIdx.y;
    const int fa = astate[ai].final_buf;
    if (fa > 1) return;
    const MatDesc amd = amats[ai];
    const __nv_bfloat16* qh = fa ? axh1 : axh0;
    const __nv_bfloat16* ql = fa ? axl1 : axl0;
    __nv_bfloat16* ph = fa ? axh0 : axh1;
    __nv_bfloat16* pl = fa ? axl0 : axl1;
    const int ld = amd.ld;
    const int64_t groups = static_cast<int64_t>(amd.n) * ld / 8;
    for (int64_t g = blockIdx.x * 256 + threadIdx.x; g < groups; g += static_cast<int64_t>(gridDim.x) * 256) {
        const int64_t e = 8 * g;
        const int r = static_cast<int>(e / ld), c = static_cast<int>(e % ld);
        float v[8];
        ld16x8(qh, ql, amd.slot + e, true, v);
#pragma unroll
        for (int q = 0; q < 8; ++q) v[q] = 0.5f * ((c + q == r ? 1.f : 0.f) + sgn * v[q]);
        st16x8(ph, pl, amd.slot + e, false, v);
    }
}

// S' = I + (P A' P) from the auxiliary plan's P planes (bf16 hi/lo) into this plan's P
// planes as fp16 hi/lo (the operand type of Q); S' = I where Q_A = 0.  The auxiliary
// iteration's error flags join the plan's.
__global__ void __launch_bounds__(256) k_clip_form_s(const MatDesc* __restrict__ mats,
                                                     const MatDesc* __restrict__ amats,
                                                     const int* __restrict__ aux_of,
                                                     const MatState* __restrict__ astate,
                                                     const __nv_bfloat16* __restrict__ aph,
                                                     const __nv_bfloat16* __restrict__ apl,
                                                     __nv_bfloat16* __restrict__ ph, __nv_bfloat16* __restrict__ pl,
                                                     const uint32_t* __restrict__ aerr, uint32_t* __restrict__ err) {
    if (blockIdx.x == 0 && blockIdx.y == 0 && threadIdx.x == 0) {
        const uint32_t f = *aerr;
        if (f) atomicOr(err, f);
    }
    const int mi = blockIdx.y;
    const MatDesc md = mats[mi];
    const int ai = aux_of[mi];
    const MatDesc amd = amats[ai];
    const bool ident = astate[ai].final_buf > 1;
    const int ld = md.ld_n;
    const int64_t groups = static_cast<int64_t>(md.n) * ld / 8;
    for (int64_t g = blockIdx.x * 256 + threadIdx.x; g < groups; g += static_cast<int64_t>(gridDim.x) * 256) {
        const int64_t e = 8 * g;
        const int r = static_cast<int>(e / ld), c = static_cast<int>(e % ld);
        float v[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        if (!ident) ld16x8(aph, apl, amd.gslot + e, false, v);
#pragma unroll
        for (int q = 0; q < 8; ++q) v[q] += (c + q == r ? 1.f : 0.f);
        st16x8(ph, pl, md.gslot + e, true, v);
    }
}

// Q S' now sits in the other ping-pong buffer: point final_buf at it.
__global__ void k_clip_flip(MatState* __restrict__ state, int nmat) {
    const int mi = blockIdx.x * blockDim.x + threadIdx.x;
    if (mi < nmat && state[mi].final_buf <= 1) state[mi].final_buf = 1 - state[mi].final_buf;
}

}  // namespace isoloco
