// gemm.cu -- batched split-precision GEMM on tcgen05 tensor cores (sm_103a).
//
// Computes, for every matrix b of a group and every BM x BN output tile,
//     D[b](i, j) = sum_k A[b](i, k) B[b](j, k)
// where each fp32 operand is carried as two bf16 planes (hi = bf16(x),
// lo = bf16(x - hi)) and the product is hi*hi + hi*lo + lo*hi, accumulated in fp32
// in tensor memory: about 16 significant bits per operand, the precision the polar
// iteration needs (a single bf16 pass would perturb the polar factor by ~1e-3).
//
// Roles (192 threads): warp 0 issues TMA loads into a kStages-deep ring of shared
// memory stages; warp 1 owns the tensor-memory accumulator and issues tcgen05.mma
// from one thread; warps 2..5 drain the accumulator (tcgen05.ld) and run the
// epilogue.  Stage hand-off uses mbarriers: `full` (TMA bytes landed), `empty`
// (the MMAs reading a stage finished, via tcgen05.commit), `acc` (all MMAs done).
//
// Operand layouts: K-major operands (K contiguous in global memory) use 64-byte
// swizzled tiles BK = 32 deep; MN-major operands (M or N contiguous) use 128-byte
// swizzled tiles of 64 MN-elements x BK rows, two (A) or four (B) boxes per stage.
// This lets X^T X, X P and P X all read the row-major iterate without transposes.
#include <cstdio>

#include "common.cuh"
#include "types.h"

namespace isoloco {

namespace {

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
    return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

// Descriptors of one operand plane for the k-th 16-deep slice of a stage.
template <bool MN>
__device__ __forceinline__ uint64_t operand_desc(uint32_t plane_addr, int ks) {
    if (MN) {
        // 128B swizzle, MN-major: 64-element MN chunks are BK*128 bytes apart (LBO),
        // 8-row K groups are 1024 bytes apart (SBO); a 16-deep K slice is 2048 bytes.
        return make_sdesc(plane_addr + ks * 2048, BK * 128, 1024, 2);
    } else {
        // 64B swizzle, K-major: 8-row groups are 512 bytes apart (SBO); a 16-deep
        // K slice is 32 bytes into the 64-byte row.
        return make_sdesc(plane_addr + ks * 32, 16, 512, 4);
    }
}

__device__ __forceinline__ void store_bf16_row(__nv_bfloat16* hi_row, __nv_bfloat16* lo_row,
                                               const float* v, int ncols_valid) {
    if (ncols_valid >= 32) {
        uint32_t h[16], l[16];
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            __nv_bfloat16 h0, l0, h1, l1;
            split_bf16(v[2 * j], h0, l0);
            split_bf16(v[2 * j + 1], h1, l1);
            h[j] = pack_bf16x2(h0, h1);
            l[j] = pack_bf16x2(l0, l1);
        }
        uint4* hp = reinterpret_cast<uint4*>(hi_row);
        uint4* lp = reinterpret_cast<uint4*>(lo_row);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            hp[q] = make_uint4(h[4 * q], h[4 * q + 1], h[4 * q + 2], h[4 * q + 3]);
            lp[q] = make_uint4(l[4 * q], l[4 * q + 1], l[4 * q + 2], l[4 * q + 3]);
        }
    } else {
#pragma unroll
        for (int j = 0; j < 32; ++j) {
            if (j < ncols_valid) {
                __nv_bfloat16 h0, l0;
                split_bf16(v[j], h0, l0);
                hi_row[j] = h0;
                lo_row[j] = l0;
            }
        }
    }
}

}  // namespace

template <bool A_MN, bool B_MN>
__global__ void __launch_bounds__(kGemmThreads, 1) k_gemm_bf16x3(const __grid_constant__ GemmParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = align1024(smem_raw);
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + kStages * kStageBytes);
    uint64_t* empty = full + kStages;
    uint64_t* accbar = empty + kStages;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(accbar + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    // ---- locate (group, matrix, tile, split) of this CTA
    int gi = 0;
    while (gi + 1 < p.num_groups && static_cast<int>(blockIdx.x) >= p.g[gi + 1].cta_begin) ++gi;
    const GemmGroup& g = p.g[gi];
    int local = static_cast<int>(blockIdx.x) - g.cta_begin;
    const int split = local % g.splits;
    local /= g.splits;
    const int ntiles = g.tiles_m * g.tiles_n;
    const int tile = local % ntiles;
    const int b = local / ntiles;
    if (b >= g.batch) return;
    const int m0 = (tile / g.tiles_n) * BM;
    const int n0 = (tile % g.tiles_n) * BN;
    const int mat = g.mat_base + b;

    bool run_mma = true;
    float ca = 0.f, cb = 0.f, cc = 1.f, xs = 1.f;
    if (p.gate != kGateNone) {
        const MatState& st = p.state[mat];
        if (p.gate == kGateActive) {
            if (st.done) return;
        } else {
            if (st.mode == 0) return;
            if (p.epi == kEpiPoly && st.mode == 2) run_mma = false;  // cubic polish: no G^2
        }
        ca = st.a;
        cb = st.b;
        cc = st.c;
        xs = st.xscale;
    }

    const int total_kb = (g.K + BK - 1) / BK;
    const int kb_begin = split * g.kblocks_per_split;
    const int kb_end = min(total_kb, kb_begin + g.kblocks_per_split);
    if (kb_begin >= kb_end) run_mma = false;

    // ---- setup: barriers, tensor memory
    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(accbar, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 0 && lane == 0 && run_mma) {
        tma_prefetch_desc(g.a_hi);
        tma_prefetch_desc(g.a_lo);
        tma_prefetch_desc(g.b_hi);
        tma_prefetch_desc(g.b_lo);
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    if (warp == 0) {
        // ================= TMA producer
        if (lane == 0 && run_mma) {
            int stage = 0;
            uint32_t phase = 0;
            uint32_t issued_mask = 0, issued_parity = 0;
            for (int kb = kb_begin; kb < kb_end; ++kb) {
                if (*abort_flag) break;
                if (!mbar_wait(&empty[stage], phase ^ 1u)) {
                    *abort_flag = 1;
                    atomicOr(p.err, kErrTimeout);
                    break;
                }
                uint8_t* sa_hi = smem + stage * kStageBytes;
                uint8_t* sa_lo = sa_hi + kTileABytes;
                uint8_t* sb_hi = sa_lo + kTileABytes;
                uint8_t* sb_lo = sb_hi + kTileBBytes;
                mbar_arrive_expect_tx(&full[stage], kStageBytes);
                const int k0 = kb * BK;
                if (A_MN) {
#pragma unroll
                    for (int c = 0; c < BM / 64; ++c) {
                        tma_load_3d(sa_hi + c * (BK * 128), g.a_hi, &full[stage], m0 + 64 * c, k0, b);
                        tma_load_3d(sa_lo + c * (BK * 128), g.a_lo, &full[stage], m0 + 64 * c, k0, b);
                    }
                } else {
                    tma_load_3d(sa_hi, g.a_hi, &full[stage], k0, m0, b);
                    tma_load_3d(sa_lo, g.a_lo, &full[stage], k0, m0, b);
                }
                if (B_MN) {
#pragma unroll
                    for (int c = 0; c < BN / 64; ++c) {
                        tma_load_3d(sb_hi + c * (BK * 128), g.b_hi, &full[stage], n0 + 64 * c, k0, b);
                        tma_load_3d(sb_lo + c * (BK * 128), g.b_lo, &full[stage], n0 + 64 * c, k0, b);
                    }
                } else {
                    tma_load_3d(sb_hi, g.b_hi, &full[stage], k0, n0, b);
                    tma_load_3d(sb_lo, g.b_lo, &full[stage], k0, n0, b);
                }
                issued_mask |= 1u << stage;
                issued_parity = (issued_parity & ~(1u << stage)) | (phase << stage);
                if (++stage == kStages) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            if (*abort_flag) {
                // Let the copies already in flight land before the CTA exits.
                for (int s = 0; s < kStages; ++s)
                    if (issued_mask & (1u << s)) (void)mbar_wait(&full[s], (issued_parity >> s) & 1u);
            }
        }
    } else if (warp == 1) {
        // ================= MMA issuer (one thread)
        if (lane == 0) {
            if (run_mma) {
                constexpr uint32_t idesc = make_idesc_bf16(BM, BN, A_MN, B_MN);
                int stage = 0;
                uint32_t phase = 0;
                for (int kb = kb_begin; kb < kb_end; ++kb) {
                    if (*abort_flag) break;
                    if (!mbar_wait(&full[stage], phase)) {
                        *abort_flag = 1;
                        atomicOr(p.err, kErrTimeout);
                        break;
                    }
                    tc_fence_after();
                    const uint32_t sa_hi = smem_u32(smem + stage * kStageBytes);
                    const uint32_t sa_lo = sa_hi + kTileABytes;
                    const uint32_t sb_hi = sa_lo + kTileABytes;
                    const uint32_t sb_lo = sb_hi + kTileBBytes;
#pragma unroll
                    for (int ks = 0; ks < BK / 16; ++ks) {
                        const uint64_t dah = operand_desc<A_MN>(sa_hi, ks);
                        const uint64_t dal = operand_desc<A_MN>(sa_lo, ks);
                        const uint64_t dbh = operand_desc<B_MN>(sb_hi, ks);
                        const uint64_t dbl = operand_desc<B_MN>(sb_lo, ks);
                        const uint32_t acc = (kb > kb_begin || ks > 0) ? 1u : 0u;
                        umma_bf16(tmem_base, dah, dbh, idesc, acc);
                        umma_bf16(tmem_base, dah, dbl, idesc, 1u);
                        umma_bf16(tmem_base, dal, dbh, idesc, 1u);
                    }
                    umma_commit(&empty[stage]);
                    if (++stage == kStages) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
            umma_commit(accbar);  // completes once every MMA above has finished
        }
    } else {
        // ================= epilogue (warps 2..5)
        const int eg = warp & 3;  // tensor-memory lane quarter this warp may access
        const bool ok = __all_sync(0xffffffffu, mbar_wait(accbar, 0));
        if (!ok && lane == 0) atomicOr(p.err, kErrTimeout);
        __syncwarp();
        tc_fence_after();
        const int row = m0 + eg * 32 + lane;
        const bool row_ok = row < g.M;
        for (int c32 = 0; c32 < BN / 32; ++c32) {
            const int col0 = n0 + c32 * 32;
            if (col0 >= g.N) break;
            float v[32];
            __syncwarp();
            if (run_mma && ok) {
                uint32_t r[32];
                tmem_ld32(tmem_base + (static_cast<uint32_t>(eg * 32) << 16) + c32 * 32, r);
                tmem_ld_wait();
#pragma unroll
                for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
            } else {
#pragma unroll
                for (int j = 0; j < 32; ++j) v[j] = 0.f;
            }
            if (row_ok) {
            const int nvalid = min(32, g.N - col0);
            if (p.epi == kEpiF32) {
                float* out = g.out_f32 + split * g.f32_split_stride + b * g.f32_batch_stride +
                             static_cast<int64_t>(row) * g.ld_f32 + col0;
                if (nvalid == 32 && (g.ld_f32 & 3) == 0) {
                    float4* o4 = reinterpret_cast<float4*>(out);
#pragma unroll
                    for (int q = 0; q < 8; ++q)
                        o4[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
                } else {
#pragma unroll
                    for (int j = 0; j < 32; ++j)
                        if (j < nvalid) out[j] = v[j];
                }
            } else {
                if (p.epi == kEpiPoly) {
                    const float* grow = g.g_f32 + b * g.g_batch_stride + static_cast<int64_t>(row) * g.ld_g + col0;
                    if (nvalid == 32 && (g.ld_g & 3) == 0) {
                        const float4* g4 = reinterpret_cast<const float4*>(grow);
#pragma unroll
                        for (int q = 0; q < 8; ++q) {
                            const float4 t = g4[q];
                            v[4 * q] = cc * v[4 * q] + cb * t.x;
                            v[4 * q + 1] = cc * v[4 * q + 1] + cb * t.y;
                            v[4 * q + 2] = cc * v[4 * q + 2] + cb * t.z;
                            v[4 * q + 3] = cc * v[4 * q + 3] + cb * t.w;
                        }
                    } else {
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            if (j < nvalid) v[j] = cc * v[j] + cb * grow[j];
                    }
                    const int d = row - col0;
                    if (d >= 0 && d < 32) {
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            if (j == d) v[j] += ca;
                    }
                } else {
#pragma unroll
                    for (int j = 0; j < 32; ++j) v[j] *= xs;
                }
                const int64_t off = b * g.bf_batch_stride + static_cast<int64_t>(row) * g.ld_bf + col0;
                store_bf16_row(g.out_hi + off, g.out_lo + off, v, nvalid);
            }
            }  // row_ok
        }
    }

    // ---- teardown: no tcgen05 op may be in flight when the accumulator is freed
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem_base, kTmemCols);
    }
}

// ------------------------------------------------------------------ host launcher
template <bool A_MN, bool B_MN>
static cudaError_t launch_gemm_t(const GemmParams& p, int grid, cudaStream_t stream) {
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(k_gemm_bf16x3<A_MN, B_MN>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             kGemmSmemBytes);
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    k_gemm_bf16x3<A_MN, B_MN><<<grid, kGemmThreads, kGemmSmemBytes, stream>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_gemm(const GemmParams& p, bool a_mn, bool b_mn, cudaStream_t stream) {
    int grid = 0;
    for (int i = 0; i < p.num_groups; ++i) {
        const GemmGroup& g = p.g[i];
        grid = g.cta_begin + g.batch * g.tiles_m * g.tiles_n * g.splits;
    }
    if (grid <= 0) return cudaSuccess;
    if (!a_mn && !b_mn) return launch_gemm_t<false, false>(p, grid, stream);
    if (a_mn && b_mn) return launch_gemm_t<true, true>(p, grid, stream);
    if (!a_mn && b_mn) return launch_gemm_t<false, true>(p, grid, stream);
    return launch_gemm_t<true, false>(p, grid, stream);
}

}  // namespace isoloco
