// gramside.cu -- the Gram-side polar iteration of very tall matrices (rows >= 8 cols: the
// embedding and the output head).
//
// The polar factor of a tall Delta is Delta (Delta^T Delta)^(-1/2).  The iteration
// X_{t+1} = X_t p_t(X_t^T X_t) from X_1 = Delta_n P_0 (Delta_n = Delta / s) keeps X_t = Delta_n Z_t
// with Z_t an n x n polynomial in A = Delta_n^T Delta_n, so it can run on the n x n matrices
// alone: G_t = X_t^T X_t = Z_t (A Z_t), Z_{t+1} = Z_t p_t(G_t), and Q = Delta_n Z_T once at
// the end.  A step costs ~8 n^3 instead of 4 rows n^2 + 2 n^3.  Iteration 0 is shared with the
// other matrices (the Gram Delta^T Delta, the control step and P_0); then
//   k_gs_init       : A = (Delta^T Delta) / s^2 from the Gram's fp32 split-K partials, as fp16
//                     hi/lo planes (22 bits), and Z_1 = P_0 (bf16 -> fp16 planes), in the first
//                     n rows of the ping-pong buffer the update would have written;
//   (GEMMs)          W = A Z_t, G_t = Z_t W, P_t as usual, Z_{t+1} = Z_t P_t;
//   k_gs_final_prep : (1 / s) Z_T -> bf16 planes (the type of Delta's planes);
//   (GEMM)           Q = Delta (Z_T / s) into the other ping-pong buffer;
//   k_gs_final_flip : final_buf points at Q.
#include "common.cuh"
#include "types.h"

namespace isoloco {

// grid (x: 256-element blocks of the n x n matrix, grid-stride beyond 65535 blocks; y: the
// Gram-side matrices listed in gs_list).
__global__ void __launch_bounds__(256) k_gs_init(const MatDesc* __restrict__ mats, MatState* __restrict__ state,
                                                 const int* __restrict__ gs_list,
                                                 const float* __restrict__ gpart,
                                                 const int64_t* __restrict__ gpart_off,
                                                 const int64_t* __restrict__ gpart_sstride,
                                                 const int* __restrict__ nsplit, __nv_bfloat16* __restrict__ anhi,
                                                 __nv_bfloat16* __restrict__ anlo, __nv_bfloat16* __restrict__ zhi,
                                                 __nv_bfloat16* __restrict__ zlo, const __nv_bfloat16* __restrict__ phi,
                                                 const __nv_bfloat16* __restrict__ plo) {
    const int mi = gs_list[blockIdx.y];
    const MatState& st = state[mi];
    if (st.mode == 0) return;  // Delta = 0 or unusable: nothing to iterate
    const MatDesc md = mats[mi];
    const int n = md.n, ld = md.ld_n;
    const float xs = st.xscale;  // 1 / sqrt(s2) at iteration 0
    const float gscale = xs * xs;
    if (blockIdx.x == 0 && threadIdx.x == 0) state[mi].xs0 = xs;
    const int64_t poff = gpart_off[mi], sstride = gpart_sstride[mi];
    const int splits = nsplit[mi];
    for (int64_t e = blockIdx.x * 256 + threadIdx.x; e < static_cast<int64_t>(n) * n; e += gridDim.x * 256) {
        const int r = static_cast<int>(e / n), c = static_cast<int>(e % n);
        const int64_t o = static_cast<int64_t>(r) * ld + c;
        float a = 0.f;
        for (int sp = 0; sp < splits; ++sp) a += gpart[poff + sp * sstride + o];
        a *= gscale;
        uint32_t hw, lw;
        split16x2(a, 0.f, true, hw, lw);
        reinterpret_cast<uint16_t*>(anhi)[md.gsslot + o] = static_cast<uint16_t>(hw & 0xFFFFu);
        reinterpret_cast<uint16_t*>(anlo)[md.gsslot + o] = static_cast<uint16_t>(lw & 0xFFFFu);
        const float z = __bfloat162float(phi[md.gslot + o]) + __bfloat162float(plo[md.gslot + o]);
        split16x2(z, 0.f, true, hw, lw);
        const int64_t zo = md.slot + static_cast<int64_t>(r) * md.ld + c;
        reinterpret_cast<uint16_t*>(zhi)[zo] = static_cast<uint16_t>(hw & 0xFFFFu);
        reinterpret_cast<uint16_t*>(zlo)[zo] = static_cast<uint16_t>(lw & 0xFFFFu);
    }
}

// (1 / s) Z_T (Z_T: fp16 hi/lo in the first n rows of ping-pong buffer final_buf) -> bf16
// hi/lo planes w, the B operand of the final product.
__global__ void __launch_bounds__(256) k_gs_final_prep(const MatDesc* __restrict__ mats,
                                                       MatState* __restrict__ state,
                                                       const int* __restrict__ gs_list,
                                                       const __nv_bfloat16* __restrict__ xh0,
                                                       const __nv_bfloat16* __restrict__ xl0,
                                                       const __nv_bfloat16* __restrict__ xh1,
                                                       const __nv_bfloat16* __restrict__ xl1,
                                                       __nv_bfloat16* __restrict__ whi, __nv_bfloat16* __restrict__ wlo) {
    const int mi = gs_list[blockIdx.y];
    const int fb = state[mi].final_buf;
    if (fb > 1) return;
    // the final product Q = Delta (Z / s) sums tr(Q^T Delta) in its epilogue
    if (blockIdx.x == 0 && threadIdx.x == 0) state[mi].trace_fused = 1;
    const MatDesc md = mats[mi];
    const int n = md.n;
    const float xs0 = state[mi].xs0;
    const uint16_t* zh = reinterpret_cast<const uint16_t*>(fb ? xh1 : xh0) + md.slot;
    const uint16_t* zl = reinterpret_cast<const uint16_t*>(fb ? xl1 : xl0) + md.slot;
    for (int64_t e = blockIdx.x * 256 + threadIdx.x; e < static_cast<int64_t>(n) * n; e += gridDim.x * 256) {
        const int r = static_cast<int>(e / n), c = static_cast<int>(e % n);
        const int64_t zo = static_cast<int64_t>(r) * md.ld + c;
        const float z = xs0 * (dec16(zh[zo], true) + dec16(zl[zo], true));
        uint32_t hw, lw;
        split16x2(z, 0.f, false, hw, lw);
        const int64_t o = md.gsslot + static_cast<int64_t>(r) * md.ld_n + c;
        reinterpret_cast<uint16_t*>(whi)[o] = static_cast<uint16_t>(hw & 0xFFFFu);
        reinterpret_cast<uint16_t*>(wlo)[o] = static_cast<uint16_t>(lw & 0xFFFFu);
    }
}

// After Q = (1 / s) Delta Z_T went to the other buffer: final_buf points at Q.
__global__ void k_gs_final_flip(MatState* __restrict__ state, const int* __restrict__ gs_list, int ngs) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= ngs) return;
    MatState& st = state[gs_list[i]];
    if (st.final_buf < 2) st.final_buf ^= 1;
}

}  // namespace isoloco
