// types.h -- structures shared by the host plan code and the kernels.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <stdint.h>

namespace isoloco {

// ------------------------------------------------------------------ GEMM tiles
// One CTA holds a BM x BN fp32 tile in tensor memory, computed from 16-bit hi/lo
// operand planes staged BK deep per pipeline stage.  With kPairMma a pair of CTAs on
// neighbouring SMs (a cluster of two) computes one kTileM x BN = 256 x 256 output tile
// with tcgen05 cta_group::2: each CTA stages its own BM rows of A and half of B's BN
// rows, so an SM loads and stages 8 KB instead of 12 KB per 16-deep MMA step.
// BK = 64: one TMA instruction moves twice the bytes of a 32-deep stage; with 32-deep
// stages the single producer thread's issue rate held back the MN-major operands (a Gram
// stage needs six 64 x 32 boxes).
constexpr bool kPairMma = true;
constexpr int BM = 128;
constexpr int BN = 256;
constexpr int BK = 64;
constexpr int kTileM = kPairMma ? 2 * BM : BM;  // rows of one output tile
constexpr int kBRows = kPairMma ? BN / 2 : BN;  // rows of B (N extent) staged by one CTA
// Shared-memory ring of the persistent GEMM (one CTA per SM): as many stages of the
// launch's plane set as fit in kRingBytes, at most kMaxStages.
constexpr int kMaxStages = 12;
constexpr int kRingBytes = 192 * 1024;
constexpr int kTileABytes = BM * BK * 2;                       // one bf16 plane of A
constexpr int kTileBBytes = kBRows * BK * 2;                   // one bf16 plane of this CTA's B

constexpr int kEpiWarps = 8;       // two warps per tensor-memory lane quarter
constexpr int kPartSlots = kEpiWarps * (kPairMma ? 2 : 1);  // Gram partial sums per output tile
constexpr int kGemmThreads = 64 + 32 * kEpiWarps;  // warp 0 TMA, warp 1 MMA, warps 2.. epilogue
constexpr int kTmemCols = 256;     // one accumulator; the kernel double-buffers (512 columns)
constexpr int kMaxGroups = 8;
constexpr int kControlThreads = 256;  // k_control block: one warp per matrix
constexpr int kFinRows = 32;  // rows of one k_gram_finalize tile (x BN columns)
constexpr int kSvdThreads = 1024;  // k_svd_tridiag block: one CTA per matrix
// Tall matrices with rows >= kGramSideRatio * cols iterate on n x n matrices (Gram side):
// X_t = Delta_n Z_t with G_t = Z_t A Z_t, A = Delta_n^T Delta_n, instead of on the rows x cols
// iterate; a step then costs ~8 n^3 instead of 4 rows n^2 + 2 n^3.
constexpr int kGramSideRatio = 8;
// A Gram of the precision schedule's single-pass steps runs one pass only when the previous
// residual ||X^T X - I||_F / sqrt(n) is at least this: one quintic step cannot bring such a
// residual below the convergence tolerance, so the Gram cannot be the one the polish uses.
constexpr float kOnePassGramResid = 0.5f;
// Epilogue staging: per epilogue warp kStageBlocks blocks of 32 x 32 16-bit values (2 KB,
// 64-byte swizzled rows), written to global memory by TMA stores.  With four, a symmetric
// output uses them as two (direct, transposed) pairs and anything else as four single
// blocks, so that a warp fills one while the TMA stores of the others still read shared
// memory; with two (the setting: the epilogue keeps up with the main loop, and the ring
// gets the 32 KB), one pair, or two alternating single blocks.
constexpr int kStageBlockBytes = 32 * 32 * 2;
constexpr int kStageBlocks = 2;
constexpr int kEpiStagingBytes = kEpiWarps * kStageBlocks * kStageBlockBytes;
constexpr int kTileQueue = 8;  // tiles handed from the producer warp to the MMA and epilogue warps
constexpr int kGemmSmemBytes = kRingBytes + kEpiStagingBytes + 1024 /*align*/ + 512 /*barriers, queues*/;

// Epilogue of the split-precision GEMM.
enum EpiMode : int {
    kEpiF32 = 0,     // store the fp32 accumulator (tests; split-K Gram partial products)
    kEpiPoly = 1,    // P = a I + b G + c acc  -> bf16 hi/lo planes
    kEpiXSplit = 2,  // X = xscale * acc       -> bf16 hi/lo planes
    kEpiGram = 3,    // G = acc -> bf16 hi/lo planes + per-tile sums of G^2, diag G, (G-I)^2;
                     // with split-K (splits > 1) behaves as kEpiF32 and k_gram_finalize follows
};

// Which matrices a GEMM launch works on, read from the per-matrix state.
enum GateMode : int {
    kGateNone = 0,    // all (debug GEMM)
    kGateActive = 1,  // matrices not yet done (Gram)
    kGateStep = 2,    // matrices whose mode this iteration is quintic or polish
    kGateQuintic = 3, // matrices taking a quintic step
    kGatePolish = 4,  // matrices taking the final polish step
};

// First tile column of tile row tm that touches the upper triangle of a square output.
__host__ __device__ constexpr int sym_first_tile_n(int tm) {
    return (tm * kTileM - BN + 1) <= 0 ? 0 : (tm * kTileM - BN + 1 + BN - 1) / BN;
}

struct GemmGroup {
    const CUtensorMap* a_hi;
    const CUtensorMap* a_lo;
    const CUtensorMap* b_hi;
    const CUtensorMap* b_lo;
    int M, N, K;  // output tile space M x N, reduction length K
    int batch;    // matrices in this group
    int tiles_m, tiles_n, splits, kblocks_per_split;
    int sym;        // square symmetric output: compute only tiles touching col >= row
    int tiles_sym;  // number of such tiles per matrix
    int cta_begin;  // (host bookkeeping) first tile of the group when every matrix is active
    int mat_base;   // index of the group's first matrix in the state array
    int bucket;     // shape bucket: index into the work-list counts
    int gate_fb;    // 0: no condition; f > 0: only matrices whose Q is in buffer f - 1 (final_buf)
    int a_mn, b_mn; // operand layout: 1 MN-major (M or N index contiguous), 0 K-major
    int a_split, b_split;  // operand carries a lo plane in this group (one tensor pass each)
    // quintic steps whose index k lies in [one_from, one_to) run a single pass (no lo planes);
    // k = the matrix's step count for a Gram (the step it leads to), the step count - 1 for
    // the polynomial and the update (the step they form)
    int one_from, one_to;
    // fp32 output (kEpiF32): out_f32 + split*split_stride + b*batch_stride + row*ld + col
    float* out_f32;
    int64_t f32_split_stride, f32_batch_stride;
    int ld_f32;
    // 16-bit hi/lo output planes (kEpiGram, kEpiPoly, kEpiXSplit) and their TMA store maps
    // (32 x 32 boxes, 64-byte swizzle); out_lo/st_lo may be null when no lo plane is kept
    __nv_bfloat16* out_hi;
    __nv_bfloat16* out_lo;
    const CUtensorMap* st_hi;
    const CUtensorMap* st_lo;
    const CUtensorMap* st_y;  // kEpiGram with gram_y: store map of the Y plane
    int64_t bf_batch_stride;
    int ld_bf;
    // kEpiPoly: the Gram matrix G as bf16 hi/lo planes (same indexing as the output)
    const __nv_bfloat16* g_hi;
    const __nv_bfloat16* g_lo;
    // kEpiGram: per-tile partial sums, 3 floats at part[(part_base + b * tiles + tile) * 3]
    float* part;
    int64_t part_base;
    // kEpiXSplit: when the tile writes a matrix's final Q (the polish update, the Gram side's
    // Q = Delta Z), the tile's share of tr(Q^T Delta) = sum of Q o Delta, with Delta's bf16
    // hi/lo planes indexed like the output; one double per epilogue warp and CTA at
    // tf_part[(b * tiles + tile) * kPartSlots + slot].  Null d_hi: no trace here.
    const __nv_bfloat16* d_hi;
    const __nv_bfloat16* d_lo;
    double* tf_part;
};

// Per-matrix state of the polar iteration (device memory, one per 2-D tensor).
struct MatState {
    float a, b, c;    // P = a I + b G + c G^2 for this iteration
    float xscale;     // X_{t+1} = xscale * X_t P
    float resid;      // last ||X^T X - I||_F / sqrt(n)
    float sigma_bar;  // tr(Q^T Delta) / n
    int mode;         // 0 none, 1 quintic step, 2 final cubic polish
    int step;         // quintic steps taken
    int iters;        // GEMM iterations used
    int done;         // 1 once finished
    int final_buf;    // ping-pong buffer holding Q (0/1), or 2 when Q = 0
    float yb, yc;     // Y = yb I + yc G for the quintic step the next Gram leads to
    int status;       // 0, or kErrNotConverged
    float lift;       // product of the linear coefficients of the steps taken: the factor
                      // by which a singular value near 0 (relative to the normalisation) has grown
    float lift_round; // lift when the current round of the schedule started
    float xs0;        // 1 / s at iteration 0 (Gram-side matrices: Q = xs0 Delta Z at the end)
    int x_hi_only;    // this step's update writes X's hi plane only: the next Gram and update
                      // run single-pass and the next iteration cannot end the polar loop
    double trace;     // tr(Q^T Delta)
    int trace_fused;  // 1: the GEMM that wrote Q also summed tr(Q^T Delta) (its tf_part slots)
};

struct GemmParams {
    GemmGroup g[kMaxGroups];
    int num_groups;
    int total_tiles;      // tiles of all groups when every matrix is active (grid sizing)
    // Work list of this launch (null: every matrix of every group): for group i, the
    // matrices list[g.mat_base + j], j < cnt[g.bucket] (indices within the group).
    const int* list;
    const int* cnt;
    int* counter;         // dynamic tile scheduler of this launch (zeroed before the step)
    int epi;
    int gate;
    int in_f16;           // operand planes are fp16 (else bf16); also the G planes of kEpiPoly
    int out_f16;          // hi/lo output planes are fp16 (else bf16)
    int a_split, b_split; // some group's operand carries a lo plane (sizes the ring's stages)
    int split_on_polish;  // matrices in the polish step use both lo planes
    int gram_y;           // kEpiGram: also write Y = b I + c G for the next quintic step
    int poly_horner;      // kEpiPoly: B is Y, so P = G Y + a I (quintic steps)
    int unit_scale;       // kEpiXSplit: no xscale (the Gram-side W = A Z, launched before the
                          // iteration's control step has reset xscale to 1)
    MatState* state;
    uint32_t* err;
};

// Description of one 2-D tensor in the workspace (device array, one per matrix).
struct MatDesc {
    int64_t param_offset;  // offset in the flat parameter buffers
    int64_t slot;          // element offset of the matrix in the bucket's planes
    int rows, cols, ld;    // row-major, leading dimension ld (multiple of 8)
    int n;                 // min(rows, cols): size of the Gram matrix
    int ld_n;              // leading dimension of the n x n planes
    int bucket;
    int64_t gslot;         // element offset of the matrix in the n x n planes
    int64_t gpart_slot;    // first partial (3 floats each) of the finalize pass
    int64_t trace_part;    // first partial of the trace pass
    int n_gtiles;          // groups of kPartSlots Gram partial sums of this matrix
    int deep;              // 1: near-square, polar steps from the deep schedule
    int n_tchunks;         // trace chunks of this matrix
    int gs;                // 1: Gram-side iteration (tall with rows >= kGramSideRatio * cols)
    int64_t gsslot;        // element offset of the matrix in the Gram-side n x n planes
    int64_t tf_part;       // first of the matrix's fused-trace slots (GemmGroup::tf_part)
    int tf_slots;          // their number: output tiles x kPartSlots
};

// A contiguous range of one parameter handled by one streaming CTA.
struct Chunk {
    int64_t flat_begin;  // first element in the flat buffers
    int32_t count;       // elements
    int32_t param;       // index in the parameter table
    int32_t matrix;      // index of the 2-D tensor, or -1 for 1-D
    int32_t elem_begin;  // first element within the parameter
    int64_t dst;         // 1-D: offset in the 1-D workspace; 2-D: unused
};

// Sources of the update direction U read by the apply pass.
struct UpdateSrc {
    const __nv_bfloat16* qh[2];  // hi planes of the two ping-pong iterate buffers
    const __nv_bfloat16* ql[2];  // lo planes
    const float* d1d;            // mean pseudo-gradient of the 1-D tensors
};

constexpr int kMaxK = 64;
struct ReplicaPtrs {
    const void* p[kMaxK];
};

}  // namespace isoloco
