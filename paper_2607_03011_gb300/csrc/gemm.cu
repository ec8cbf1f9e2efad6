// gemm.cu -- batched split-precision GEMM on tcgen05 tensor cores (sm_103a).
//
// Computes, for every matrix b of a group and every BM x BN output tile,
//     D[b](i, j) = sum_k A[b](i, k) B[b](j, k)
// where an fp32 operand is carried as 16-bit planes hi = round(x), lo = round(x - hi)
// (bf16 or fp16, chosen per launch).  The tensor core sums hi*hi, plus hi*lo_B when B
// carries a lo plane and lo_A*hi when A does, into an fp32 accumulator in tensor memory:
// three passes give ~16 (bf16) or ~22 (fp16) significant bits per operand, two passes
// keep one operand at 11 bits (fp16).  The polar iteration uses three bf16 passes on
// the unnormalised pseudo-gradient (iteration 0) and on the final polish step, and two
// fp16 passes elsewhere (the operand that is not split only perturbs the iterate's
// spectrum, which later steps correct).
//
// Roles (320 threads): warp 0 issues TMA loads into a ring of shared
// memory stages; warp 1 owns the tensor-memory accumulator and issues tcgen05.mma
// from one thread; warps 2..9 drain the accumulator (tcgen05.ld) and run the
// epilogue.  Stage hand-off uses mbarriers: `full` (TMA bytes landed), `empty`
// (the MMAs reading a stage finished, via tcgen05.commit), `acc` (all MMAs done).
//
// Operand layouts: K-major operands (K contiguous in global memory) use swizzled
// tiles BK deep; MN-major operands (M or N contiguous) use 128-byte swizzled tiles of
// 64 MN-elements x BK rows, two (A) or four (B) boxes per stage.  This lets X^T X,
// X P and P X all read the row-major iterate without transposes.  The layout is a
// property of each group, so one launch can mix them (the Grams X^T X of tall and
// X X^T of wide matrices share a launch).
#include <cstdio>

#include "common.cuh"
#include "ns_schedule.h"
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
        // K-major, rows of BK bf16 (64 or 128 bytes) with the matching swizzle: 8-row
        // groups are 8 * BK * 2 bytes apart (SBO); a 16-deep K slice is 32 bytes into the row.
        return make_sdesc(plane_addr + ks * 32, 16, 8 * BK * 2, BK * 2 == 128 ? 2 : 4);
    }
}

// Symmetric outputs: the t-th of the tiles that touch the upper triangle (col >= row),
// in row-major order of tiles.
__device__ __forceinline__ void sym_tile(int t, int tiles_m, int tiles_n, int& tm, int& tn) {
    for (tm = 0; tm < tiles_m; ++tm) {
        const int lo = sym_first_tile_n(tm);
        const int cnt = tiles_n - lo;
        if (t < cnt) {
            tn = lo + t;
            return;
        }
        t -= cnt;
    }
    tm = tiles_m - 1;
    tn = tiles_n - 1;
}

}  // namespace

// Everything a role needs to know about one output tile; every role decodes the same
// sequence of tile indices, so the three warps agree without communicating.
struct TileInfo {
    int gi, b, tile, split, m0, n0, mat, kb_begin, kb_end;
    bool run_mma, a_split, b_split;
    bool horner;     // kEpiPoly: P = acc + a I (the MMA computed G Y); else P = a I + b G + c acc
    bool hi_only;    // write the hi plane only (a single-pass Gram's G; an update's X whose lo
                     // plane no later step reads)
    bool trace;      // the output is a matrix's final Q: also sum Q o Delta (GemmGroup::d_hi)
    float ca, cb, cc, xs;
    float yb, yc;    // kEpiGram with p.gram_y: Y = yb I + yc G for the next quintic step
};

// Active-tile prefix of the launch: group i owns active tiles [pre[i], pre[i + 1]).
__device__ __forceinline__ void active_prefix(const GemmParams& p, int* pre) {
    pre[0] = 0;
    for (int i = 0; i < p.num_groups; ++i) {
        const GemmGroup& g = p.g[i];
        const int mats = p.list ? p.cnt[g.bucket] : g.batch;
        pre[i + 1] = pre[i] + mats * (g.sym ? g.tiles_sym : g.tiles_m * g.tiles_n) * g.splits;
    }
}

// Decodes active tile t for the CTA of rank `crank` in its pair (0 without pairs).
// Returns false when the matrix does no work in this launch.
__device__ __forceinline__ bool decode_tile(const GemmParams& p, const int* pre, int t, uint32_t crank,
                                            TileInfo& ti) {
    int gi = 0;
    while (gi + 1 < p.num_groups && t >= pre[gi + 1]) ++gi;
    const GemmGroup& g = p.g[gi];
    int local = t - pre[gi];
    ti.gi = gi;
    ti.split = local % g.splits;
    local /= g.splits;
    const int ntiles = g.sym ? g.tiles_sym : g.tiles_m * g.tiles_n;
    ti.tile = local % ntiles;
    const int j = local / ntiles;
    ti.b = p.list ? p.list[g.mat_base + j] : j;
    if (ti.b >= g.batch) return false;
    int tm, tn;
    if (g.sym) {
        sym_tile(ti.tile, g.tiles_m, g.tiles_n, tm, tn);
    } else {
        tm = ti.tile / g.tiles_n;
        tn = ti.tile % g.tiles_n;
    }
    ti.m0 = tm * kTileM + static_cast<int>(crank) * BM;  // this CTA's rows of the tile
    ti.n0 = tn * BN;
    ti.mat = g.mat_base + ti.b;
    ti.run_mma = true;
    ti.a_split = g.a_split != 0;
    ti.b_split = g.b_split != 0;
    ti.ca = 0.f, ti.cb = 0.f, ti.cc = 1.f, ti.xs = 1.f, ti.yb = 0.f, ti.yc = 0.f;
    ti.horner = false;
    ti.hi_only = false;
    // the final Q of a matrix: the polish update, or an ungated launch (the Gram side's
    // Q = Delta Z, which writes only matrices that have a Q)
    ti.trace = p.epi == kEpiXSplit && g.d_hi != nullptr && p.gate == kGateNone;
    if (g.gate_fb && p.state[ti.mat].final_buf != g.gate_fb - 1) return false;
    if (p.gate != kGateNone) {
        const MatState& st = p.state[ti.mat];
        if (p.gate == kGateActive) {
            if (st.done) return false;
            if (p.gram_y) {  // coefficients of the quintic step this Gram may lead to
                ti.yb = st.yb;
                ti.yc = st.yc;
            }
        } else {
            if (st.mode == 0) return false;
            if (p.gate == kGateQuintic && st.mode != 1) return false;
            if (p.gate == kGatePolish && st.mode != 2) return false;
            if (p.epi == kEpiPoly && st.mode == 2) ti.run_mma = false;  // cubic polish: no G^2
            ti.horner = (p.epi == kEpiPoly && p.poly_horner && st.mode == 1);
            if (p.split_on_polish && st.mode == 2) ti.a_split = ti.b_split = true;  // final step: 3 passes
            ti.trace = p.epi == kEpiXSplit && g.d_hi != nullptr && p.gate == kGateStep && st.mode == 2;
        }
        // precision schedule: single-pass steps.  A Gram only after iteration 0's and only
        // while the last residual is large (>= kOnePassGramResid): a Gram whose test can pass
        // feeds the final polish, which nothing corrects afterwards, so it keeps its passes.
        const int k = (p.epi == kEpiGram) ? st.step : st.step - 1;
        if (k >= g.one_from && k < g.one_to &&
            ((p.epi == kEpiGram) ? (st.step > 0 && st.resid >= kOnePassGramResid) : st.mode == 1)) {
            ti.a_split = ti.b_split = false;
            // a single-pass Gram never feeds the polish and its polynomial reads G's hi only
            if (p.epi == kEpiGram) ti.hi_only = true;
        }
        if (p.epi == kEpiXSplit && p.gate == kGateStep && st.mode == 1 && st.x_hi_only) ti.hi_only = true;
        ti.ca = st.a;
        ti.cb = st.b;
        ti.cc = st.c;
        ti.xs = p.unit_scale ? 1.f : st.xscale;
    }
    const int total_kb = (g.K + BK - 1) / BK;
    ti.kb_begin = ti.split * g.kblocks_per_split;
    ti.kb_end = min(total_kb, ti.kb_begin + g.kblocks_per_split);
    if (ti.kb_begin >= ti.kb_end) ti.run_mma = false;
    return true;
}

// Byte offset of element (r, c) in a 32 x 32 block of 16-bit values stored with 64-byte
// rows and the 64-byte swizzle (16-byte chunk index XOR (r / 2) mod 4), the layout a TMA
// store with CU_TENSOR_MAP_SWIZZLE_64B reads.
__device__ __forceinline__ uint32_t stg_off(int r, int c) {
    return static_cast<uint32_t>(r * 64 + ((((c >> 3) ^ (r >> 1)) & 3) << 4) + (c & 7) * 2);
}

// One warp writes a 32 x 32 block of 16-bit values (lane = row, w = the lane's 32 values
// packed in pairs) to staging and stores it with TMA at (col0, row_base, b): the diagonal
// block is symmetrised in shared memory; an off-diagonal block of a symmetric output is
// also stored transposed at (row_base, col0, b).  `stg` holds the warp's kStageBlocks
// blocks and `seq` counts its stores (one bulk group each): a symmetric store takes the
// pair (seq & 1) once the store before the previous one has read it, any other store the
// block (seq & 3) once the store four back has.
__device__ __forceinline__ void stage_store_block(const uint32_t (&w)[16], const CUtensorMap* map, uint8_t* stg,
                                                  uint32_t& seq, bool diag, bool sym, int lane, int col0,
                                                  int row_base, int b) {
    static_assert(kStageBlocks == 4 || kStageBlocks == 2, "block rotation below handles two or four blocks");
    uint8_t* sd;
    if (kStageBlocks == 4) {
        if (sym) {
            sd = stg + (seq & 1u) * 2u * kStageBlockBytes;
            if (lane == 0) bulk_wait_read1();
        } else {
            sd = stg + (seq & 3u) * kStageBlockBytes;
            if (lane == 0) bulk_wait_read3();
        }
    } else {
        if (sym) {
            sd = stg;
            if (lane == 0) bulk_wait_read0();
        } else {
            sd = stg + (seq & 1u) * kStageBlockBytes;
            if (lane == 0) bulk_wait_read1();
        }
    }
    uint8_t* sm = sd + kStageBlockBytes;  // transposed block (symmetric outputs only)
    ++seq;
    __syncwarp();
    if (diag) {
#pragma unroll
        for (int j = 0; j < 32; ++j) {
            const uint16_t x = static_cast<uint16_t>((j & 1) ? (w[j >> 1] >> 16) : (w[j >> 1] & 0xFFFFu));
            if (j >= lane) *reinterpret_cast<uint16_t*>(sd + stg_off(lane, j)) = x;
            if (j > lane) *reinterpret_cast<uint16_t*>(sd + stg_off(j, lane)) = x;
        }
    } else {
#pragma unroll
        for (int q = 0; q < 4; ++q)
            *reinterpret_cast<uint4*>(sd + lane * 64 + ((((q ^ (lane >> 1)) & 3)) << 4)) =
                make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
        if (sym) {
            // transposed block T(r, c) = value of lane c at column r: for rows 2i and 2i + 1,
            // even lanes c form (own, partner) column 2i and odd lanes (partner, own) column
            // 2i + 1 from the packed pair w[i] and the partner lane's, one 32-bit store each
            const uint32_t sel = (lane & 1) ? 0x3276u : 0x5410u;
            const int r_odd = lane & 1, c_even = lane & ~1;
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                const uint32_t other = __shfl_xor_sync(0xffffffffu, w[i], 1);
                *reinterpret_cast<uint32_t*>(sm + stg_off(2 * i + r_odd, c_even)) = __byte_perm(w[i], other, sel);
            }
        }
    }
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) {
        tma_store_3d(map, sd, col0, row_base, b);
        if (sym && !diag) tma_store_3d(map, sm, row_base, col0, b);
        bulk_commit();
    }
}

// Epilogue of one tile's column half, run by four warps (thread (eg, lane) owns
// output row m0 + 32 eg + lane).  `tacc` is the tensor-memory accumulator of the tile.
// 16-bit outputs leave through the warp's shared-memory staging blocks `stg` and TMA
// stores, one 32 x 32 block at a time.  In symmetric mode (Gram, G^2) blocks below the
// diagonal are skipped, a block above it is also stored transposed at (col, row), and the
// diagonal block is made symmetric in shared memory (its upper half mirrored) before its
// single store, so every entry is written once and the matrix is bitwise symmetric.
__device__ __forceinline__ void tile_epilogue(const GemmParams& p, const TileInfo& ti, uint32_t tacc, bool ok,
                                              int eg, int half, int lane, uint32_t crank, uint8_t* stg,
                                              uint32_t& sseq) {
    const GemmGroup& g = p.g[ti.gi];
    const int b = ti.b, m0 = ti.m0, n0 = ti.n0, split = ti.split;
    const float ca = ti.ca, cb = ti.cb, cc = ti.cc, xs = ti.xs;
    const int row_base = m0 + eg * 32;
    const int row = row_base + lane;
    const bool row_ok = row < g.M;
    const bool sym = g.sym != 0;
    const bool f32_out = (p.epi == kEpiF32) || (p.epi == kEpiGram && g.splits > 1);
    const bool gram_fused = (p.epi == kEpiGram && g.splits == 1);
    const bool of16 = p.out_f16 != 0;
    // planes written: hi, lo (if kept; not for a Horner-form P, whose lo plane nobody reads),
    // and for the Gram with p.gram_y the plane Y = yb I + yc G (hi only)
    const bool write_y = (p.epi == kEpiGram && p.gram_y);
    const int nplanes = (ti.horner || ti.hi_only || g.st_lo == nullptr) ? 1 : 2;
    float s_sq = 0.f, s_tr = 0.f, s_dev = 0.f;
    float s_tq = 0.f;  // share of tr(Q^T Delta) (ti.trace)
    for (int c32 = half * (BN / 64); c32 < (half + 1) * (BN / 64); ++c32) {
        const int col0 = n0 + c32 * 32;
        if (col0 >= g.N) break;
        if (sym && col0 < row_base) continue;  // block below the diagonal (warp-uniform)
        const bool diag = sym && col0 == row_base;
        float v[32];
        __syncwarp();
        if (ti.run_mma && ok) {
            uint32_t r[32];
            tmem_ld32(tacc + (static_cast<uint32_t>(eg * 32) << 16) + c32 * 32, r);
            tmem_ld_wait();
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
        } else {
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] = 0.f;
        }
        const int nvalid = min(32, g.N - col0);
        const int d = row - col0;  // column index of this lane's diagonal entry in the block
        if (ti.horner) {
#pragma unroll
            for (int j = 0; j < 32; ++j)
                if (j == d) v[j] += ca;
        } else if (p.epi == kEpiPoly && row_ok) {
            const int64_t goff = b * g.bf_batch_stride + static_cast<int64_t>(row) * g.ld_bf + col0;
            const uint16_t* gh = reinterpret_cast<const uint16_t*>(g.g_hi) + goff;
            const uint16_t* gl = reinterpret_cast<const uint16_t*>(g.g_lo) + goff;
            const bool gf16 = p.in_f16 != 0;
            if (nvalid == 32) {
                const uint4* h4 = reinterpret_cast<const uint4*>(gh);
                const uint4* l4 = reinterpret_cast<const uint4*>(gl);
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const uint4 hh = h4[q], ll = l4[q];
                    const uint32_t hw[4] = {hh.x, hh.y, hh.z, hh.w};
                    const uint32_t lw[4] = {ll.x, ll.y, ll.z, ll.w};
#pragma unroll
                    for (int w = 0; w < 4; ++w) {
                        const float g0 = dec16(hw[w] & 0xFFFFu, gf16) + dec16(lw[w] & 0xFFFFu, gf16);
                        const float g1 = dec16(hw[w] >> 16, gf16) + dec16(lw[w] >> 16, gf16);
                        v[8 * q + 2 * w] = cc * v[8 * q + 2 * w] + cb * g0;
                        v[8 * q + 2 * w + 1] = cc * v[8 * q + 2 * w + 1] + cb * g1;
                    }
                }
            } else {
#pragma unroll
                for (int j = 0; j < 32; ++j)
                    if (j < nvalid) v[j] = cc * v[j] + cb * (dec16(gh[j], gf16) + dec16(gl[j], gf16));
            }
#pragma unroll
            for (int j = 0; j < 32; ++j)
                if (j == d) v[j] += ca;
        } else if (p.epi == kEpiXSplit) {
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] *= xs;
            if (ti.trace && row_ok) {
                // this row's share of tr(Q^T Delta): Q in fp32 as stored (before its split
                // into planes), Delta from its bf16 hi/lo planes
                const int64_t doff = b * g.bf_batch_stride + static_cast<int64_t>(row) * g.ld_bf + col0;
                const uint16_t* dh = reinterpret_cast<const uint16_t*>(g.d_hi) + doff;
                const uint16_t* dl = reinterpret_cast<const uint16_t*>(g.d_lo) + doff;
                if (nvalid == 32) {
                    const uint4* h4 = reinterpret_cast<const uint4*>(dh);
                    const uint4* l4 = reinterpret_cast<const uint4*>(dl);
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        const uint4 hh = h4[q], ll = l4[q];
                        const uint32_t hw[4] = {hh.x, hh.y, hh.z, hh.w};
                        const uint32_t lw[4] = {ll.x, ll.y, ll.z, ll.w};
#pragma unroll
                        for (int w = 0; w < 4; ++w) {
                            const float d0 = __uint_as_float(hw[w] << 16) + __uint_as_float(lw[w] << 16);
                            const float d1 = __uint_as_float(hw[w] & 0xFFFF0000u) + __uint_as_float(lw[w] & 0xFFFF0000u);
                            s_tq = fmaf(v[8 * q + 2 * w], d0, s_tq);
                            s_tq = fmaf(v[8 * q + 2 * w + 1], d1, s_tq);
                        }
                    }
                } else {
#pragma unroll
                    for (int j = 0; j < 32; ++j)
                        if (j < nvalid)
                            s_tq = fmaf(v[j], __uint_as_float(static_cast<uint32_t>(dh[j]) << 16) +
                                                  __uint_as_float(static_cast<uint32_t>(dl[j]) << 16), s_tq);
                }
            }
        }
        if (gram_fused && row_ok && sym && !diag && nvalid == 32) {
            // block strictly above the diagonal: every entry counts twice and (G - I) = G
            float ss = 0.f;
#pragma unroll
            for (int j = 0; j < 32; ++j) ss = fmaf(v[j], v[j], ss);
            s_sq = fmaf(2.f, ss, s_sq);
            s_dev = fmaf(2.f, ss, s_dev);
        } else if (gram_fused && row_ok) {
#pragma unroll
            for (int j = 0; j < 32; ++j) {
                if (j < nvalid && (!sym || j >= d)) {
                    const float x = v[j];
                    const float e = (j == d) ? x - 1.f : x;
                    const float w = (sym && j > d) ? 2.f : 1.f;  // mirrored entry counts twice
                    s_sq = fmaf(w * x, x, s_sq);
                    s_dev = fmaf(w * e, e, s_dev);
                    if (j == d) s_tr += x;
                }
            }
        }
        if (f32_out) {
            if (!row_ok) continue;
            float* base = g.out_f32 + split * g.f32_split_stride + b * g.f32_batch_stride;
            float* out = base + static_cast<int64_t>(row) * g.ld_f32 + col0;
            if (!diag && nvalid == 32 && (g.ld_f32 & 3) == 0) {
                float4* o4 = reinterpret_cast<float4*>(out);
#pragma unroll
                for (int q = 0; q < 8; ++q) o4[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
            } else {
#pragma unroll
                for (int j = 0; j < 32; ++j)
                    if (j < nvalid && (!sym || j >= d)) out[j] = v[j];
            }
            if (sym) {
#pragma unroll
                for (int j = 0; j < 32; ++j)
                    if (j < nvalid && j > d) base[static_cast<int64_t>(col0 + j) * g.ld_f32 + row] = v[j];
            }
            continue;
        }
        // ---- 16-bit planes through shared memory and TMA stores
        uint32_t hw[16], lw[16];
#pragma unroll
        for (int j = 0; j < 16; ++j) split16x2(v[2 * j], v[2 * j + 1], of16, hw[j], lw[j]);
        stage_store_block(hw, g.st_hi, stg, sseq, diag, sym, lane, col0, row_base, b);
        if (nplanes > 1) stage_store_block(lw, g.st_lo, stg, sseq, diag, sym, lane, col0, row_base, b);
        if (write_y) {
            // Y = yb I + yc G, hi plane only (it is the single operand of G Y)
            if (diag) {
#pragma unroll
                for (int j = 0; j < 16; ++j)
                    lw[j] = round16x2(ti.yc * v[2 * j] + (2 * j == d ? ti.yb : 0.f),
                                      ti.yc * v[2 * j + 1] + (2 * j + 1 == d ? ti.yb : 0.f), of16);
            } else {
#pragma unroll
                for (int j = 0; j < 16; ++j) lw[j] = round16x2(ti.yc * v[2 * j], ti.yc * v[2 * j + 1], of16);
            }
            stage_store_block(lw, g.st_y, stg, sseq, diag, sym, lane, col0, row_base, b);
        }
    }
    if (ti.trace) {
        // fixed-order warp reduction into this warp's slot of the tile (every slot of every
        // tile of the matrix is written by the launch that writes its Q)
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) s_tq += __shfl_xor_sync(0xffffffffu, s_tq, o);
        if (lane == 0)
            g.tf_part[(static_cast<int64_t>(b) * (g.tiles_m * g.tiles_n) + ti.tile) * kPartSlots +
                      static_cast<int>(crank) * kEpiWarps + half * 4 + eg] = static_cast<double>(s_tq);
    }
    if (gram_fused) {
        // fixed-order warp reduction; each epilogue warp owns one of the tile's kEpiWarps slots
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            s_sq += __shfl_xor_sync(0xffffffffu, s_sq, o);
            s_tr += __shfl_xor_sync(0xffffffffu, s_tr, o);
            s_dev += __shfl_xor_sync(0xffffffffu, s_dev, o);
        }
        if (lane == 0) {
            const int ntiles = sym ? g.tiles_sym : g.tiles_m * g.tiles_n;
            float* slot = g.part + ((g.part_base + static_cast<int64_t>(b) * ntiles + ti.tile) * kPartSlots +
                                    static_cast<int>(crank) * kEpiWarps + half * 4 + eg) * 3;
            slot[0] = s_sq;
            slot[1] = s_tr;
            slot[2] = s_dev;
        }
    }
}

// Persistent kernel.  Without pairs, CTA c starts with tile c and claims further tiles
// from the launch's counter.  With kPairMma the grid is made of clusters of two CTAs
// (ranks 0 and 1, on neighbouring SMs); cluster c processes tiles c, c + clusters, ...
// and both CTAs walk that sequence together: each loads its rows of A and its half of B,
// the TMA bytes of both complete on rank 0's `full` barrier, rank 0 alone issues the
// cta_group::2 MMAs, whose commits arrive on the `empty` / `tfull` barriers of both CTAs,
// and each CTA's epilogue drains its own half of the accumulator and reports to rank 0's
// `tempty`.  The TMA ring runs continuously across tile boundaries, and the accumulator
// is double buffered in tensor memory (2 x 256 columns): the epilogue of one tile
// overlaps the MMAs of the next.
__global__ void __launch_bounds__(kGemmThreads, 1) k_gemm_split(const __grid_constant__ GemmParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = align1024(smem_raw);
    uint8_t* staging = smem + kRingBytes;  // kEpiWarps x (direct, mirror) blocks
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + kRingBytes + kEpiStagingBytes);
    uint64_t* empty = full + kMaxStages;
    uint64_t* tfull = empty + kMaxStages;  // [2] accumulator buffer ready for the epilogue
    uint64_t* tempty = tfull + 2;        // [2] accumulator buffer released by the epilogue
    uint64_t* drain = tempty + 2;        // teardown: every issued MMA has completed
    uint64_t* tq_full = drain + 1;       // [kTileQueue] tile index written by the producer
    uint64_t* tq_empty = tq_full + kTileQueue;  // [kTileQueue] read by the MMA and epilogue warps
    int* tq_tile = reinterpret_cast<int*>(tq_empty + kTileQueue);
    int* pre = tq_tile + kTileQueue;     // [kMaxGroups + 1] active-tile prefix
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(pre + kMaxGroups + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const uint32_t crank = kPairMma ? cluster_ctarank() : 0u;  // rank in the CTA pair
    const bool leader = crank == 0;                              // issues the MMAs
    // ring geometry of this launch: room for the planes its tiles can load
    const uint32_t stage_stride = kTileABytes * (p.a_split || p.split_on_polish ? 2u : 1u) +
                                  kTileBBytes * (p.b_split || p.split_on_polish ? 2u : 1u);
    const int nstages = min(kMaxStages, static_cast<int>(kRingBytes / stage_stride));

    if (threadIdx.x == 0) {
        for (int s = 0; s < nstages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&tfull[i], 1);
            mbar_init(&tempty[i], kEpiWarps * (kPairMma ? 2 : 1));  // one arrival per epilogue warp of the pair
        }
        mbar_init(drain, 1);
        for (int q = 0; q < kTileQueue; ++q) {
            mbar_init(&tq_full[q], 1);
            mbar_init(&tq_empty[q], 1 + kEpiWarps);  // the MMA thread and one lane per epilogue warp
        }
        active_prefix(p, pre);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        if (kPairMma) {
            tmem_alloc_pair(tmem_slot, 2 * kTmemCols);
            tmem_relinquish_pair();
        } else {
            tmem_alloc(tmem_slot, 2 * kTmemCols);
            tmem_relinquish();
        }
    }
    tc_fence_before();
    __syncthreads();
    if (kPairMma) cluster_sync();  // both CTAs' barriers exist before either signals the other's
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    if (warp == 0) {
        // ================= TMA producer
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            uint32_t issued_mask = 0, issued_parity = 0;
            int prefetched = -1;
            const int T = pre[p.num_groups];
            int q = 0;
            uint32_t qphase = 0;
            // first tile; without pairs later ones come from the launch's counter, with pairs
            // cluster c takes tiles c, c + clusters, ... (both CTAs of the pair agree)
            const int tile_stride = kPairMma ? static_cast<int>(gridDim.x >> 1) : 0;
            int t = kPairMma ? static_cast<int>(blockIdx.x >> 1) : static_cast<int>(blockIdx.x);
            for (;;) {
                // publish the next tile (or -1: no more) to the MMA and epilogue warps
                const int tile = (t < T && !*abort_flag) ? t : -1;
                if (!mbar_wait(&tq_empty[q], qphase ^ 1u)) {
                    *abort_flag = 1;
                    atomicOr(p.err, kErrTimeout);
                    break;
                }
                tq_tile[q] = tile;
                mbar_arrive(&tq_full[q]);
                if (++q == kTileQueue) {
                    q = 0;
                    qphase ^= 1u;
                }
                if (tile < 0) break;
                if (kPairMma)
                    t += tile_stride;
                else
                    t = atomicAdd(p.counter, 1) + static_cast<int>(gridDim.x);  // claimed early
                TileInfo ti;
                if (!decode_tile(p, pre, tile, crank, ti) || !ti.run_mma) continue;
                const GemmGroup& g = p.g[ti.gi];
                if (prefetched != ti.gi) {
                    tma_prefetch_desc(g.a_hi);
                    tma_prefetch_desc(g.b_hi);
                    if (ti.a_split) tma_prefetch_desc(g.a_lo);
                    if (ti.b_split) tma_prefetch_desc(g.b_lo);
                    prefetched = ti.gi;
                }
                const uint32_t stage_bytes =
                    kTileABytes * (ti.a_split ? 2u : 1u) + kTileBBytes * (ti.b_split ? 2u : 1u);
                const int nb0 = ti.n0 + static_cast<int>(crank) * kBRows;  // this CTA's rows of B
                for (int kb = ti.kb_begin; kb < ti.kb_end; ++kb) {
                    if (!mbar_wait(&empty[stage], phase ^ 1u)) {
                        *abort_flag = 1;
                        atomicOr(p.err, kErrTimeout);
                        break;
                    }
                    uint8_t* sa_hi = smem + stage * stage_stride;
                    uint8_t* sa_lo = sa_hi + kTileABytes;
                    uint8_t* sb_hi = sa_hi + kTileABytes * (ti.a_split ? 2u : 1u);
                    uint8_t* sb_lo = sb_hi + kTileBBytes;
                    // rank 0's barrier expects the bytes of both CTAs of the pair
                    if (leader) mbar_arrive_expect_tx(&full[stage], stage_bytes * (kPairMma ? 2u : 1u));
                    const uint32_t fbar = kPairMma ? mapa_shared(smem_u32(&full[stage]), 0) : 0u;
                    auto load = [&](uint8_t* dst, const CUtensorMap* map, int c0, int c1) {
                        if (kPairMma)
                            tma_load_3d_pair(dst, map, fbar, c0, c1, ti.b);
                        else
                            tma_load_3d(dst, map, &full[stage], c0, c1, ti.b);
                    };
                    const int k0 = kb * BK;
                    if (g.a_mn) {
#pragma unroll
                        for (int c = 0; c < BM / 64; ++c) {
                            load(sa_hi + c * (BK * 128), g.a_hi, ti.m0 + 64 * c, k0);
                            if (ti.a_split) load(sa_lo + c * (BK * 128), g.a_lo, ti.m0 + 64 * c, k0);
                        }
                    } else {
                        load(sa_hi, g.a_hi, k0, ti.m0);
                        if (ti.a_split) load(sa_lo, g.a_lo, k0, ti.m0);
                    }
                    if (g.b_mn) {
#pragma unroll
                        for (int c = 0; c < kBRows / 64; ++c) {
                            load(sb_hi + c * (BK * 128), g.b_hi, nb0 + 64 * c, k0);
                            if (ti.b_split) load(sb_lo + c * (BK * 128), g.b_lo, nb0 + 64 * c, k0);
                        }
                    } else {
                        load(sb_hi, g.b_hi, k0, nb0);
                        if (ti.b_split) load(sb_lo, g.b_lo, k0, nb0);
                    }
                    issued_mask |= 1u << stage;
                    issued_parity = (issued_parity & ~(1u << stage)) | (phase << stage);
                    if (++stage == nstages) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
            if (*abort_flag) {
                // Let the copies already in flight land before the CTA exits (rank 0's
                // barriers also count rank 1's copies; rank 1 cannot observe its own, so it
                // leaves them a generous margin).
                if (leader) {
                    for (int s = 0; s < nstages; ++s)
                        if (issued_mask & (1u << s)) (void)mbar_wait(&full[s], (issued_parity >> s) & 1u);
                } else {
                    const uint64_t t0 = globaltimer_ns();
                    while (globaltimer_ns() - t0 < 100000ull) {
                    }
                }
            }
        }
    } else if (warp == 1) {
        // ================= MMA issuer (one thread; with pairs only in rank 0)
        if (lane == 0 && kPairMma && !leader) {
            // rank 1 issues no MMAs; it only keeps its tile queue moving
            int q = 0;
            uint32_t qphase = 0;
            for (;;) {
                if (!mbar_wait(&tq_full[q], qphase)) {
                    *abort_flag = 1;
                    atomicOr(p.err, kErrTimeout);
                    break;
                }
                const int tile = tq_tile[q];
                mbar_arrive(&tq_empty[q]);
                if (++q == kTileQueue) {
                    q = 0;
                    qphase ^= 1u;
                }
                if (tile < 0) break;
            }
        } else if (lane == 0) {
            const uint32_t sbase = smem_u32(smem);
            int stage = 0;
            uint32_t phase = 0;
            uint32_t n = 0;  // active tiles processed
            int q = 0;
            uint32_t qphase = 0;
            for (;;) {
                if (!mbar_wait(&tq_full[q], qphase)) {
                    *abort_flag = 1;
                    atomicOr(p.err, kErrTimeout);
                    break;
                }
                const int tile = tq_tile[q];
                mbar_arrive(&tq_empty[q]);
                if (++q == kTileQueue) {
                    q = 0;
                    qphase ^= 1u;
                }
                if (tile < 0 || *abort_flag) break;
                TileInfo ti;
                if (!decode_tile(p, pre, tile, crank, ti)) continue;
                const uint32_t buf = n & 1u, use = n >> 1;
                ++n;
                if (!mbar_wait(&tempty[buf], (use & 1u) ^ 1u)) {
                    *abort_flag = 1;
                    atomicOr(p.err, kErrTimeout);
                    break;
                }
                tc_fence_after();
                const uint32_t tacc = tmem_base + buf * kTmemCols;
                if (ti.run_mma) {
                    // instruction and operand descriptors for the layouts of this tile's group
                    const bool a_mn = p.g[ti.gi].a_mn != 0, b_mn = p.g[ti.gi].b_mn != 0;
                    const uint32_t idesc = make_idesc_16bit(kTileM, BN, a_mn, b_mn, p.in_f16 != 0);
                    const uint64_t desc_a0 = a_mn ? operand_desc<true>(sbase, 0) : operand_desc<false>(sbase, 0);
                    const uint64_t desc_b0 = b_mn ? operand_desc<true>(sbase, 0) : operand_desc<false>(sbase, 0);
                    // start-address step of one 16-deep K slice: 2048 bytes MN-major, 32 bytes K-major
                    const uint64_t step_a = a_mn ? (2048 >> 4) : (32 >> 4);
                    const uint64_t step_b = b_mn ? (2048 >> 4) : (32 >> 4);
                    // descriptors of this tile's planes in stage 0; a stage or a 16-deep K
                    // slice only moves the start address (14-bit field in 16-byte units; every
                    // shared address is below 256 KB, so the sum never carries out of it)
                    const uint64_t a_hi0 = desc_a0;
                    const uint64_t a_lo0 = desc_a0 + (kTileABytes >> 4);
                    const uint64_t b_hi0 = desc_b0 + ((kTileABytes * (ti.a_split ? 2u : 1u)) >> 4);
                    const uint64_t b_lo0 = b_hi0 + (kTileBBytes >> 4);
                    const bool bs = ti.b_split, as = ti.a_split;
                    uint32_t acc = 0u;
                    for (int kb = ti.kb_begin; kb < ti.kb_end; ++kb) {
                        if (!mbar_wait(&full[stage], phase)) {
                            *abort_flag = 1;
                            atomicOr(p.err, kErrTimeout);
                            break;
                        }
                        tc_fence_after();
                        const uint64_t so = static_cast<uint64_t>(stage) * (stage_stride >> 4);
#pragma unroll
                        for (int ks = 0; ks < BK / 16; ++ks) {
                            const uint64_t da = so + ks * step_a, db = so + ks * step_b;
                            if (kPairMma) {
                                umma_16bit_pair(tacc, a_hi0 + da, b_hi0 + db, idesc, acc);
                                if (bs) umma_16bit_pair(tacc, a_hi0 + da, b_lo0 + db, idesc, 1u);
                                if (as) umma_16bit_pair(tacc, a_lo0 + da, b_hi0 + db, idesc, 1u);
                            } else {
                                umma_16bit(tacc, a_hi0 + da, b_hi0 + db, idesc, acc);
                                if (bs) umma_16bit(tacc, a_hi0 + da, b_lo0 + db, idesc, 1u);
                                if (as) umma_16bit(tacc, a_lo0 + da, b_hi0 + db, idesc, 1u);
                            }
                            acc = 1u;
                        }
                        // the stage is free in both CTAs once these MMAs have read it
                        if (kPairMma)
                            umma_commit_pair_mc(&empty[stage], 0x3);
                        else
                            umma_commit(&empty[stage]);
                        if (++stage == nstages) {
                            stage = 0;
                            phase ^= 1u;
                        }
                    }
                }
                // completes once every MMA of this tile has finished (in both CTAs' barriers)
                if (kPairMma)
                    umma_commit_pair_mc(&tfull[buf], 0x3);
                else
                    umma_commit(&tfull[buf]);
            }
            if (kPairMma)
                umma_commit_pair(drain);
            else
                umma_commit(drain);
            (void)mbar_wait(drain, 0);
        }
    } else {
        // ================= epilogue (warps 2..9): warp w reads TMEM lanes 32 (w % 4) ..,
        // warps 2..5 take columns 0..127 of the tile and warps 6..9 columns 128..255
        const int eg = warp & 3;  // tensor-memory lane quarter this warp may access
        const int half = (warp - 2) >> 2;
        uint32_t n = 0;
        uint32_t sseq = 0;  // this warp's staged stores so far (staging block rotation)
        int q = 0;
        uint32_t qphase = 0;
        for (;;) {
            int tile = -1;
            int got = 1;
            if (lane == 0) {
                got = mbar_wait(&tq_full[q], qphase) ? 1 : 0;
                if (got) {
                    tile = tq_tile[q];
                    mbar_arrive(&tq_empty[q]);
                }
            }
            tile = __shfl_sync(0xffffffffu, tile, 0);
            got = __shfl_sync(0xffffffffu, got, 0);
            if (++q == kTileQueue) {
                q = 0;
                qphase ^= 1u;
            }
            if (!got) {
                if (lane == 0) atomicOr(p.err, kErrTimeout);
                break;
            }
            if (tile < 0) break;
            TileInfo ti;
            if (!decode_tile(p, pre, tile, crank, ti)) continue;
            const uint32_t buf = n & 1u, use = n >> 1;
            ++n;
            const bool ok = __all_sync(0xffffffffu, mbar_wait(&tfull[buf], use & 1u));
            if (!ok) {
                if (lane == 0) atomicOr(p.err, kErrTimeout);
                break;
            }
            __syncwarp();
            tc_fence_after();
            tile_epilogue(p, ti, tmem_base + buf * kTmemCols, ok, eg, half, lane, crank,
                          staging + (warp - 2) * kStageBlocks * kStageBlockBytes, sseq);
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {
                if (leader)
                    mbar_arrive(&tempty[buf]);
                else
                    mbar_arrive_cluster(mapa_shared(smem_u32(&tempty[buf]), 0));  // rank 0 issues the MMAs
            }
        }
        if (lane == 0) bulk_wait0();  // this warp's TMA stores have completed
        __syncwarp();
    }

    // ---- teardown: the MMA thread has waited for all its MMAs (drain barrier); with
    // pairs neither CTA leaves (or frees tensor memory) while rank 0's MMAs could still
    // read rank 1's shared memory or write its tensor memory
    tc_fence_before();
    __syncthreads();
    if (kPairMma) cluster_sync();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        if (kPairMma)
            tmem_dealloc_pair(tmem_base, 2 * kTmemCols);
        else
            tmem_dealloc(tmem_base, 2 * kTmemCols);
    }
}

// ------------------------------------------------------------------ host launcher
// Launches one persistent GEMM over the groups of `p` (p.total_tiles output tiles) on at
// most `max_ctas` CTAs (one per SM; with kPairMma, clusters of two CTAs per tile).
cudaError_t launch_gemm(const GemmParams& p, int max_ctas, cudaStream_t stream) {
    if (p.total_tiles <= 0) return cudaSuccess;
    static int max_clusters = 0;  // clusters of two that can be resident at once
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(k_gemm_split, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             kGemmSmemBytes);
        if (e != cudaSuccess) return e;
        if (kPairMma) {
            cudaLaunchConfig_t cfg = {};
            cudaLaunchAttribute at[1];
            at[0].id = cudaLaunchAttributeClusterDimension;
            at[0].val.clusterDim.x = 2;
            at[0].val.clusterDim.y = 1;
            at[0].val.clusterDim.z = 1;
            cfg.gridDim = dim3(static_cast<unsigned>(max_ctas & ~1));
            cfg.blockDim = dim3(kGemmThreads);
            cfg.dynamicSmemBytes = kGemmSmemBytes;
            cfg.attrs = at;
            cfg.numAttrs = 1;
            int n = 0;
            e = cudaOccupancyMaxActiveClusters(&n, k_gemm_split, &cfg);
            if (e != cudaSuccess) return e;
            max_clusters = n > 0 ? n : 1;
        }
        attr_set = true;
    }
    if (!kPairMma) {
        const int grid = p.total_tiles < max_ctas ? p.total_tiles : max_ctas;
        k_gemm_split<<<grid, kGemmThreads, kGemmSmemBytes, stream>>>(p);
        return cudaGetLastError();
    }
    int clusters = p.total_tiles;
    clusters = clusters < max_clusters ? clusters : max_clusters;
    clusters = clusters < max_ctas / 2 ? clusters : (max_ctas / 2 > 0 ? max_ctas / 2 : 1);
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = 2;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.gridDim = dim3(static_cast<unsigned>(2 * clusters));
    cfg.blockDim = dim3(kGemmThreads);
    cfg.dynamicSmemBytes = kGemmSmemBytes;
    cfg.stream = stream;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, k_gemm_split, p);
}

}  // namespace isoloco
