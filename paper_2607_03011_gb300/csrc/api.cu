// api.cu -- plan (bucketing, workspace, TMA descriptors), launch sequencing and the
// C ABI declared in include/isoloco.h.
//
// One IsoLoCo outer step (Alg. 2) on a stream:
//   k_reset_state -> k_reduce (Delta, all tensors)
//   for t = 0..max_iter:   Gram X^T X (tcgen05) -> k_gram_finalize -> k_control
//                          -> G^2 with P = a I + b G + c G^2 epilogue (tcgen05)
//                          -> X P (tcgen05)  [matrices that finished exit at once; the
//                             polish's epilogue also sums tr(Q^T Delta)]
//   k_trace_partial (matrices left unconverged) -> k_trace_final (sigma_bar)
//   -> k_apply (Nesterov) -> status copy
// Every kernel reads its per-matrix decisions from device memory: the host never
// waits inside a step.
#include <algorithm>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <map>
#include <mutex>
#include <string>
#include <vector>

#include "common.cuh"
#include "isoloco.h"
#include "types.h"

namespace isoloco {

// Guard bytes around each workspace region (the plan's bounds check: a kernel that writes
// past either end of its region changes them; isoloco_check_guards compares them).
constexpr size_t kGuardBytes = 256;
constexpr int kGuardByte = 0xA5;

// kernels defined in the other translation units
cudaError_t launch_gemm(const GemmParams& p, int max_ctas, cudaStream_t stream);
__global__ void k_gram_finalize(const MatDesc*, const int2*, const MatState*, const float*, const int64_t*,
                                const int64_t*, const int*, __nv_bfloat16*, __nv_bfloat16*, float*, int,
                                __nv_bfloat16*, int);
__global__ void k_gs_init(const MatDesc*, MatState*, const int*, const float*, const int64_t*, const int64_t*,
                          const int*, __nv_bfloat16*, __nv_bfloat16*, __nv_bfloat16*, __nv_bfloat16*,
                          const __nv_bfloat16*, const __nv_bfloat16*);
__global__ void k_gs_final_prep(const MatDesc*, MatState*, const int*, const __nv_bfloat16*, const __nv_bfloat16*,
                                const __nv_bfloat16*, const __nv_bfloat16*, __nv_bfloat16*, __nv_bfloat16*);
__global__ void k_gs_final_flip(MatState*, const int*, int);
__global__ void k_control(const MatDesc*, int, MatState*, const float*, int, int, float, uint32_t*, const int*,
                          const int*, int, int*, int*, int*, int*, cudaGraphConditionalHandle, int, long long*,
                          int, int*, int4, int4, int);
__global__ void k_trace_partial(const MatDesc*, const int4*, int, const MatState*, const __nv_bfloat16*,
                                const __nv_bfloat16*, const __nv_bfloat16*, const __nv_bfloat16*,
                                const __nv_bfloat16*, const __nv_bfloat16*, double*);
__global__ void k_trace_final(const MatDesc*, int, MatState*, const double*, const double*);
__global__ void k_reset_state(MatState*, int, uint32_t*, const MatDesc*, const int*, const int*, int, int*, int*,
                              int*, int);
__global__ void k_reduce(const Chunk*, const MatDesc*, ReplicaPtrs, int, int, const float*, float,
                         __nv_bfloat16*, __nv_bfloat16*, float*, uint32_t*);
__global__ void k_reduce_f32(const Chunk*, const MatDesc*, ReplicaPtrs, int, const float*, float, __nv_bfloat16*,
                             __nv_bfloat16*, float*, uint32_t*);
__global__ void k_reduce_p(const Chunk*, const MatDesc*, ReplicaPtrs, int, int, const float*, float,
                           __nv_bfloat16*, __nv_bfloat16*, float*, uint32_t*, int, float, const float*, float*);
__global__ void k_apply(const Chunk*, const MatDesc*, const MatState*, UpdateSrc, int, float, float, float,
                        float*, float*, const float*, float*, float*, const uint32_t*, int, int, int, const float*);
__global__ void k_clip_q_bf16(const MatDesc*, const MatState*, __nv_bfloat16*, __nv_bfloat16*, __nv_bfloat16*,
                              __nv_bfloat16*);
__global__ void k_clip_form_a(const MatDesc*, const MatState*, const float*, const int64_t*, const int64_t*,
                              const int*, const MatDesc*, const int*, __nv_bfloat16*, __nv_bfloat16*);
__global__ void k_clip_form_p(const MatDesc*, const MatState*, __nv_bfloat16*, __nv_bfloat16*, __nv_bfloat16*,
                              __nv_bfloat16*, float);
__global__ void k_clip_form_s(const MatDesc*, const MatDesc*, const int*, const MatState*, const __nv_bfloat16*,
                              const __nv_bfloat16*, __nv_bfloat16*, __nv_bfloat16*, const uint32_t*, uint32_t*);
__global__ void k_clip_flip(MatState*, int);
__global__ void k_svd_tridiag(const MatDesc*, const MatState*, float*, const int64_t*, const int64_t*, const int*,
                              float*, const int64_t*);
__global__ void k_svd_bisect(const MatDesc*, const float*, const int64_t*, float*, const int64_t*);
__global__ void k_svd_sigma_bar(const MatDesc*, int, MatState*, const float*, const int64_t*);
__global__ void k_diloco(ReplicaPtrs, int, int, float*, float*, int64_t, float, float, float, uint32_t*);
__global__ void k_dare(ReplicaPtrs, int, int, float*, float*, int64_t, float, uint32_t, float, unsigned int,
                       uint64_t, float, float, uint32_t*);
__global__ void k_ties_init(int, uint64_t, uint64_t, uint64_t, unsigned long long*, uint64_t*, uint64_t*, uint64_t*,
                            uint64_t*, uint64_t*, uint64_t*, unsigned long long*, int*);
__global__ void k_ties_sample(ReplicaPtrs, int, int, const float*, int64_t, int64_t, uint32_t*);
__global__ void k_ties_hist_buf(const uint32_t*, const uint32_t*, int, int64_t, int, int, int, const uint64_t*,
                                unsigned long long*);
__global__ void k_ties_bracket(ReplicaPtrs, int, int, const float*, int64_t, const uint64_t*, uint32_t*, uint32_t*,
                               int64_t, unsigned long long*);
__global__ void k_ties_check(int, int, int64_t, uint64_t, const unsigned long long*, const uint32_t*, uint64_t*,
                             int*);
__global__ void k_ties_hist(ReplicaPtrs, int, int, const float*, int64_t, int, const uint64_t*, unsigned long long*,
                            const int*);
__global__ void k_ties_select(int, int, unsigned long long*, uint64_t*, uint64_t*, const int*);
__global__ void k_ties_merge(ReplicaPtrs, int, int, float*, float*, int64_t, const uint64_t*, const uint64_t*,
                             const int*, float, float, uint32_t*);
__global__ void k_split_planes(const float*, int64_t, int, int, int, __nv_bfloat16*, __nv_bfloat16*, int);
__global__ void k_debug_wait(uint32_t*, uint64_t, unsigned long long*);

constexpr int kChunkElems = 16384;
constexpr int kTraceChunkElems = 16384;
constexpr int kDefaultMaxIter = 28;
constexpr int kLaunchCounters = 4096;  // dynamic-scheduler counters, one per GEMM launch of a step
constexpr float kDefaultTol = 4e-3f;

// Roles of the tensor maps of one bucket.
enum MapRole { kRoleKA = 0, kRoleKB = 1, kRoleMN = 2, kRoleST = 3 };
// 3 sources x 3 roles x 2 planes + G (2x2) + P (2x2) + store maps (X0, X1, G, P) x 2 planes
// + Y (operand KB, store)
// + Gram-side buckets: Z in the first n rows of X0 / X1 (operand K-major A, MN-major, store)
// x 2 planes, A (K-major A), W (MN-major, store) x 2 planes
constexpr int kMapsPerBucket = 54;
inline int src_map(int src, int role, int plane) { return (src * 3 + role) * 2 + plane; }
inline int g_map(int role, int plane) { return 18 + role * 2 + plane; }
inline int p_map(int role, int plane) { return 22 + role * 2 + plane; }
// store maps (32 x 32 boxes): which 0 = X0, 1 = X1, 2 = G, 3 = P
inline int st_map(int which, int plane) { return 26 + which * 2 + plane; }
// Gram-side maps; Z's roles: 0 K-major A, 1 MN-major, 2 store
inline int z_map(int buf, int role, int plane) { return 36 + buf * 6 + role * 2 + plane; }
inline int an_map(int plane) { return 48 + plane; }
inline int w_mn_map(int plane) { return 50 + plane; }
inline int w_st_map(int plane) { return 52 + plane; }
inline int y_map() { return 34; }     // Y as the B operand (K-major, 256 rows)
inline int y_st_map() { return 35; }  // Y store map

struct Bucket {
    int rows, cols, ld, n, ld_n, count;
    bool tall;
    int mat_base;
    int64_t plane_off, gplane_off, gpart_off;
    int splits;
    bool gs;         // Gram-side iteration (gramside.cu)
    int64_t gs_off;  // offset of the bucket in the Gram-side n x n planes (A, W)
    int64_t tf_base; // first fused-trace slot of the bucket (GemmGroup::tf_part)
    int tf_tiles;    // output tiles of one matrix (rows x cols)
};

}  // namespace isoloco

using namespace isoloco;

struct isoloco_plan {
    int device = 0;
    int num_sms = 148;
    int K = 0;
    int dtype = 0;
    int64_t N = 0;
    std::vector<isoloco_param_t> table;
    std::vector<int> mat_param;
    std::vector<MatDesc> mats_h;
    std::vector<Bucket> buckets;
    int nmat = 0, nchunks = 0, nftiles = 0, ntchunks = 0;
    int nftiles_reg = 0;  // finalize tiles of matrices that are not Gram-side
    int64_t plane_elems = 0, gplane_elems = 0, gpart_elems = 0, n1d = 0;
    // device workspace
    std::vector<void*> allocs;
    // every workspace region sits between guard bytes (dalloc): allocation base, region bytes
    std::vector<std::pair<uint8_t*, size_t>> guards;
    int64_t ws_bytes = 0;
    __nv_bfloat16 *dhi = nullptr, *dlo = nullptr, *xhi[2] = {nullptr, nullptr}, *xlo[2] = {nullptr, nullptr};
    __nv_bfloat16 *ghi = nullptr, *glo = nullptr, *phi = nullptr, *plo = nullptr;
    __nv_bfloat16* ypl = nullptr;  // Y = b I + c G of the next quintic step (hi plane only)
    // Gram-side buckets: A = Delta_n^T Delta_n and W = A Z (n x n, hi/lo), their matrices' list
    __nv_bfloat16 *anhi = nullptr, *anlo = nullptr, *whi = nullptr, *wlo = nullptr;
    int* gs_list = nullptr;
    int n_gs = 0;
    int gs_blocks = 1;  // 256-thread blocks per Gram-side matrix in k_gs_init / k_gs_final_prep (one per 256 elements)
    int64_t gs_slot_first = 0, gs_slot_count = 0;  // Gram partial slots of the Gram-side matrices
    float* gpart = nullptr;
    float* d1d = nullptr;
    float* fin_part = nullptr;
    int2* ftiles = nullptr;
    double* tpart = nullptr;
    double* tfpart = nullptr;  // fused-trace slots (GemmGroup::tf_part), tf_slots doubles
    int64_t tf_slots = 0;
    int4* tchunks = nullptr;
    MatState* state = nullptr;
    MatDesc* mats_d = nullptr;
    // work lists (per shape bucket) rebuilt by k_control, and the GEMM tile counters
    int* bucket_first_d = nullptr;
    int* bucket_count_d = nullptr;
    int* list_gram = nullptr;
    int* cnt_gram = nullptr;
    int* list_step = nullptr;
    int* cnt_step = nullptr;
    int* counters = nullptr;
    int launch_seq = 0;
    int64_t* gpart_off_d = nullptr;
    int64_t* gpart_sstride_d = nullptr;
    int* nsplit_d = nullptr;
    Chunk* chunks_d = nullptr;
    uint32_t* err_d = nullptr;
    uint32_t* err_h = nullptr;  // pinned
    CUtensorMap* tmaps_d = nullptr;
    cudaEvent_t done_ev = nullptr;
    // iterations 1, 2, ... of the polar loop as one CUDA graph: a while-conditional node
    // whose body (two iterations) runs until k_control reports no matrix left to iterate
    cudaStream_t cap_st = nullptr;  // private stream the body is captured on
    cudaGraph_t graph = nullptr;
    cudaGraphExec_t gexec = nullptr;
    int g_max_iter = -1;
    float g_tol = 0.f;
    int g_fast = -1;
    int g_full = -1;
    long long g_prec = -2;
    // precision schedule of this call (isoloco_opts_t::precision_schedule, decoded): per
    // schedule kind (0 standard, 1 deep) the quintic steps [from, to) whose Gram and
    // polynomial, and those whose update, run a single pass
    long long prec_code = 0;
    int gp_from[2] = {0, 0}, gp_to[2] = {0, 0}, up_from[2] = {0, 0}, up_to[2] = {0, 0};
    bool per_launch = false;        // polar iterations as plain launches (no graph), with early stop
    bool full_prec = false;         // every polar step with three passes and no Horner form
                                    // (the clip variants' sign iteration)
    int fast_steps = 0;             // this call's fast-variant step count (0: exact Iso-C)
    bool skip_trace = false;        // this call needs no tr(Q^T Delta) (fast variant, spectral scale)
    float* bnew = nullptr;          // B' of the orthogonalise-P ablation (allocated on first use)
    int64_t body_launches = 0;      // kernels in one run of the body
    long long* loopc = nullptr;     // device: [0] body runs in this call, [1] body runs ever
    // phase timing (isoloco_profile_enable) and launch counting
    bool prof = false;
    std::vector<std::pair<cudaEvent_t, cudaEvent_t>> pend[ISOLOCO_NUM_PHASES];
    std::vector<cudaEvent_t> ev_pool;
    double prof_ms[ISOLOCO_NUM_PHASES] = {0};
    int64_t prof_n[ISOLOCO_NUM_PHASES] = {0};
    int64_t launches = 0;
    // clip variants (Sec. 4.5), allocated on first use: the plan of the n x n matrices
    // H - sigma_bar I whose polar factors are sign(H - sigma_bar I); fp32 H (split-K
    // partials) with per-matrix offsets and split strides; aux matrix index of each matrix
    isoloco_plan* aux = nullptr;
    float* hbuf = nullptr;
    int64_t* hoff_d = nullptr;
    int64_t* hss_d = nullptr;
    int* aux_of_d = nullptr;
    std::vector<int64_t> hbucket_off;
    // exact singular values (spectrum_kind 3): tridiagonal (d, e) and sigma_i per matrix
    float* tri = nullptr;
    int64_t* tri_off_d = nullptr;
    float* sv = nullptr;
    int64_t* sv_off_d = nullptr;
    std::vector<int64_t> sv_off_h;  // by matrix index (plan order)
    // TIES trim (allocated on first use): radix-select histograms [2K][256]; ranks and key
    // prefixes of the sample (2 per worker), candidate and fallback selections; the keys
    // above each bracket; the fallback flag; the sample [K][S]; the candidate segments
    // [K][ties_nseg][ties_segcap] and their counts
    unsigned long long* ties_hist = nullptr;
    uint64_t *ties_rank_s = nullptr, *ties_prefix_s = nullptr, *ties_rank_c = nullptr, *ties_prefix_c = nullptr;
    uint64_t *ties_rank_f = nullptr, *ties_prefix_f = nullptr;
    unsigned long long* ties_above = nullptr;
    int* ties_fail = nullptr;
    uint32_t* ties_samp = nullptr;
    uint32_t* ties_cand = nullptr;
    uint32_t* ties_cnt = nullptr;
    int64_t ties_S = 0, ties_segcap = 0;
    int ties_nseg = 0;
    // staging for the host-buffer entry point (allocated on first use); with pinned inputs
    // the replicas are read in place and theta / B are copied on side_st during the polar
    // iteration
    float* st_theta = nullptr;
    float* st_mom = nullptr;
    void* st_reps = nullptr;
    cudaStream_t side_st = nullptr;
    cudaEvent_t ev_reduced = nullptr, ev_copied = nullptr;
};

// ------------------------------------------------------------------ errors
static thread_local std::string g_last_error;

static int fail(int code, const std::string& msg) {
    g_last_error = msg;
    return code;
}

#define CUDA_TRY(expr)                                                                        \
    do {                                                                                      \
        cudaError_t _e = (expr);                                                              \
        if (_e != cudaSuccess)                                                                \
            return fail(ISOLOCO_ERR_CUDA, std::string(#expr) + ": " + cudaGetErrorString(_e)); \
    } while (0)

// ------------------------------------------------------------------ tensor maps
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    }
    return fn;
}

// 3-D bf16 map over [count][rows][ld] with logical extent cols x rows x count; batch_elems > 0
// gives a batch stride other than rows * ld (an n x n matrix in the first rows of a taller slot).
static bool make_map(CUtensorMap* m, const void* base, int cols, int rows, int count, int ld, int role,
                     int64_t batch_elems = -1) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[3] = {(cuuint64_t)cols, (cuuint64_t)rows, (cuuint64_t)count};
    cuuint64_t strides[2] = {(cuuint64_t)ld * 2,
                             (cuuint64_t)(batch_elems > 0 ? batch_elems : (int64_t)rows * ld) * 2};
    cuuint32_t box[3];
    CUtensorMapSwizzle sw;
    if (role == kRoleMN) {
        box[0] = 64; box[1] = BK; sw = CU_TENSOR_MAP_SWIZZLE_128B;
    } else if (role == kRoleST) {
        box[0] = 32; box[1] = 32; sw = CU_TENSOR_MAP_SWIZZLE_64B;
    } else {
        box[0] = BK; box[1] = (role == kRoleKA) ? BM : kBRows;
        sw = (BK * 2 == 128) ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B;
    }
    box[2] = 1;
    cuuint32_t es[3] = {1, 1, 1};
    CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, es,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

static inline int64_t round_up(int64_t x, int64_t a) { return (x + a - 1) / a * a; }

// Output tiles of an n x n symmetric product that touch the upper triangle.
static int sym_tiles(int n) {
    const int tm_n = (n + kTileM - 1) / kTileM, tn_n = (n + BN - 1) / BN;
    int c = 0;
    for (int tm = 0; tm < tm_n; ++tm) c += tn_n - sym_first_tile_n(tm);
    return c;
}


template <typename T>
static int dalloc(isoloco_plan* p, T** ptr, int64_t count) {
    *ptr = nullptr;
    if (count <= 0) count = 1;
    const size_t bytes = static_cast<size_t>(count) * sizeof(T);
    // [guard | region | pad to 256 | guard]: the region keeps cudaMalloc's 256-byte alignment
    const size_t body = (bytes + kGuardBytes - 1) / kGuardBytes * kGuardBytes;
    uint8_t* base = nullptr;
    cudaError_t e = cudaMalloc(reinterpret_cast<void**>(&base), body + 2 * kGuardBytes);
    if (e != cudaSuccess) {
        (void)cudaGetLastError();
        return fail(ISOLOCO_ERR_OOM, std::string("cudaMalloc of ") + std::to_string(bytes) + " bytes failed");
    }
    if (cudaMemset(base, kGuardByte, kGuardBytes) != cudaSuccess ||
        cudaMemset(base + kGuardBytes + bytes, kGuardByte, body - bytes + kGuardBytes) != cudaSuccess) {
        cudaFree(base);
        return fail(ISOLOCO_ERR_CUDA, "guard fill failed");
    }
    *ptr = reinterpret_cast<T*>(base + kGuardBytes);
    p->allocs.push_back(base);
    p->guards.push_back({base, bytes});
    p->ws_bytes += static_cast<int64_t>(body + 2 * kGuardBytes);
    return ISOLOCO_OK;
}

static void free_plan(isoloco_plan* p) {
    if (!p) return;
    if (p->aux) free_plan(p->aux);
    for (void* a : p->allocs) cudaFree(a);
    for (int ph = 0; ph < ISOLOCO_NUM_PHASES; ++ph)
        for (auto& pr : p->pend[ph]) {
            cudaEventDestroy(pr.first);
            cudaEventDestroy(pr.second);
        }
    for (cudaEvent_t e : p->ev_pool) cudaEventDestroy(e);
    if (p->err_h) cudaFreeHost(p->err_h);
    if (p->done_ev) cudaEventDestroy(p->done_ev);
    if (p->gexec) cudaGraphExecDestroy(p->gexec);
    if (p->graph) cudaGraphDestroy(p->graph);
    if (p->cap_st) cudaStreamDestroy(p->cap_st);
    if (p->side_st) cudaStreamDestroy(p->side_st);
    if (p->ev_reduced) cudaEventDestroy(p->ev_reduced);
    if (p->ev_copied) cudaEventDestroy(p->ev_copied);
    delete p;
}

static bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Records CUDA events around the launches of one phase when profiling is on, and
// counts the launches either way.
struct PhaseTimer {
    isoloco_plan* p;
    int phase;
    cudaStream_t st;
    cudaEvent_t e0 = nullptr;
    static cudaEvent_t get(isoloco_plan* p) {
        if (!p->ev_pool.empty()) {
            cudaEvent_t e = p->ev_pool.back();
            p->ev_pool.pop_back();
            return e;
        }
        cudaEvent_t e = nullptr;
        cudaEventCreate(&e);
        return e;
    }
    PhaseTimer(isoloco_plan* p_, int ph, cudaStream_t s, int nlaunch = 1) : p(p_), phase(ph), st(s) {
        p->launches += nlaunch;
        p->prof_n[phase] += nlaunch;
        if (p->prof) {
            e0 = get(p);
            cudaEventRecord(e0, st);
        }
    }
    ~PhaseTimer() {
        if (e0) {
            cudaEvent_t e1 = get(p);
            cudaEventRecord(e1, st);
            p->pend[phase].emplace_back(e0, e1);
        }
    }
};

// ------------------------------------------------------------------ plan creation
static int build_plan(isoloco_plan* p, const isoloco_param_t* table, int n_params) {
    // --- matrices and buckets
    std::map<std::pair<int, int>, int> bucket_of;
    std::vector<std::vector<int>> members;
    for (int i = 0; i < n_params; ++i) {
        const isoloco_param_t& t = table[i];
        if (t.cols > 0) {
            auto key = std::make_pair((int)t.rows, (int)t.cols);
            auto it = bucket_of.find(key);
            int b;
            if (it == bucket_of.end()) {
                b = (int)p->buckets.size();
                bucket_of[key] = b;
                Bucket bk{};
                bk.rows = t.rows;
                bk.cols = t.cols;
                bk.ld = (int)round_up(t.cols, 8);
                bk.n = std::min(t.rows, t.cols);
                bk.ld_n = (int)round_up(bk.n, 8);
                bk.tall = t.rows >= t.cols;
                bk.gs = bk.tall && t.rows >= kGramSideRatio * t.cols && t.rows >= 2 * BK;
                bk.gs_off = 0;
                p->buckets.push_back(bk);
                members.emplace_back();
            } else {
                b = it->second;
            }
            members[b].push_back(i);
        }
    }
    // matrices ordered bucket by bucket so each bucket's slots are contiguous
    std::vector<int> mat_of_param(n_params, -1);
    int64_t plane = 0, gplane = 0, gpart = 0, fin = 0, tr = 0, tf = 0;
    std::vector<int2> ftiles;
    std::vector<int4> tchunks;
    std::vector<int64_t> gpoff, gpss;
    std::vector<int> nsp;
    std::vector<int> gs_mats;
    int64_t gs_elems = 0;
    auto g_elems_of = [](const Bucket& b) { return (int64_t)b.n * b.ld_n; };
    for (size_t b = 0; b < p->buckets.size(); ++b) {
        Bucket& bk = p->buckets[b];
        bk.count = (int)members[b].size();
        bk.mat_base = (int)p->mats_h.size();
        bk.plane_off = plane;
        bk.gplane_off = gplane;
        bk.gpart_off = gpart;
        bk.tf_base = tf;
        bk.tf_tiles = ((bk.rows + kTileM - 1) / kTileM) * ((bk.cols + BN - 1) / BN);
        // split-K for the Gram when the bucket has few output tiles
        const int tiles = sym_tiles(bk.n) * bk.count;
        const int kdim = bk.tall ? bk.rows : bk.cols;
        const int kblocks = (kdim + BK - 1) / BK;
        // split-K for long reductions: at most 256 k-blocks per split, and more splits
        // (down to 32 k-blocks each) only while the bucket alone would not fill the GPU
        // (two output tiles per SM, or per pair of SMs with pair MMAs)
        const int slots = 2 * p->num_sms / (kPairMma ? 2 : 1);
        int splits = std::max(1, (kblocks + 255) / 256);
        if (tiles * splits < slots) splits = std::max(splits, std::min(slots / std::max(1, tiles), kblocks / 32));
        if (bk.gs) splits = std::max(splits, 2);  // iteration 0's Gram stays in fp32 partials (k_gs_init)
        int kper = (kblocks + splits - 1) / splits;
        splits = (kblocks + kper - 1) / kper;  // no empty split
        bk.splits = splits;
        const int64_t mat_elems = (int64_t)bk.rows * bk.ld;
        const int64_t g_elems = (int64_t)bk.n * bk.ld_n;
        // Gram partial sums per matrix, in groups of kPartSlots slots: one group per computed
        // Gram tile (upper-triangle tiles) when the Gram's epilogue produces them; with
        // split-K one slot per finalize tile, packed, the rest of the last group zero
        const int nft = splits > 1 ? ((bk.n + kFinRows - 1) / kFinRows) * ((bk.n + BN - 1) / BN) : 0;
        int gtiles = splits > 1 ? (nft + kPartSlots - 1) / kPartSlots : sym_tiles(bk.n);
        // Gram-side: later Grams are n x n products with one slot group per upper tile
        if (bk.gs) gtiles = std::max(gtiles, sym_tiles(bk.n));
        if (bk.gs) {
            bk.gs_off = gs_elems;
            gs_elems += round_up((int64_t)bk.count * g_elems_of(bk), 128);
            if (gs_mats.empty()) p->gs_slot_first = fin;
            p->gs_slot_count = fin + (int64_t)bk.count * gtiles - p->gs_slot_first;
        }
        for (int j = 0; j < bk.count; ++j) {
            const int pi = members[b][j];
            MatDesc md{};
            md.param_offset = table[pi].offset;
            md.slot = plane + j * mat_elems;
            md.rows = bk.rows;
            md.cols = bk.cols;
            md.ld = bk.ld;
            md.n = bk.n;
            md.ld_n = bk.ld_n;
            md.bucket = (int)b;
            md.gslot = gplane + j * g_elems;
            md.gpart_slot = fin;
            md.n_gtiles = gtiles;
            // near-square (|rows - cols| < min / 16): the deep polar schedule
            md.deep = (std::abs(bk.rows - bk.cols) * 16 < bk.n) ? 1 : 0;
            md.gs = bk.gs ? 1 : 0;
            md.gsslot = bk.gs_off + j * g_elems;
            if (bk.gs) gs_mats.push_back((int)p->mats_h.size());
            md.trace_part = tr;
            md.tf_part = tf;
            md.tf_slots = bk.tf_tiles * kPartSlots;
            tf += md.tf_slots;
            const int rows_per = std::max(1, kTraceChunkElems / bk.cols);
            md.n_tchunks = (bk.rows + rows_per - 1) / rows_per;
            const int mi = (int)p->mats_h.size();
            if (splits > 1)
                for (int t = 0; t < nft; ++t) ftiles.push_back(make_int2(mi, t));
            for (int c = 0; c < md.n_tchunks; ++c) {
                const int r0 = c * rows_per;
                tchunks.push_back(make_int4(mi, r0, std::min(rows_per, bk.rows - r0), c));
            }
            fin += md.n_gtiles;
            tr += md.n_tchunks;
            gpoff.push_back(gpart + j * g_elems);
            gpss.push_back((int64_t)bk.count * g_elems);
            nsp.push_back(splits);
            mat_of_param[pi] = mi;
            p->mat_param.push_back(pi);
            p->mats_h.push_back(md);
        }
        plane += round_up((int64_t)bk.count * mat_elems, 128);
        gplane += round_up((int64_t)bk.count * g_elems, 128);
        gpart += round_up((int64_t)splits * bk.count * g_elems, 128);
    }
    p->nmat = (int)p->mats_h.size();
    p->n_gs = (int)gs_mats.size();
    for (int mi : gs_mats)
        p->gs_blocks = std::max<int>(p->gs_blocks, (int)std::min<int64_t>(65535, ((int64_t)p->mats_h[mi].n * p->mats_h[mi].n + 255) / 256));
    p->plane_elems = plane;
    p->gplane_elems = gplane;
    p->gpart_elems = gpart;
    p->nftiles = (int)ftiles.size();
    for (const int2& f : ftiles) p->nftiles_reg += p->mats_h[f.x].gs ? 0 : 1;
    p->ntchunks = (int)tchunks.size();
    p->tf_slots = tf;

    // --- streaming chunks (table order) and the 1-D workspace
    std::vector<Chunk> chunks;
    int64_t d1 = 0;
    for (int i = 0; i < n_params; ++i) {
        const isoloco_param_t& t = table[i];
        const int64_t len = (int64_t)t.rows * (t.cols > 0 ? t.cols : 1);
        int64_t dst = 0;
        if (t.cols == 0) {
            dst = d1;
            d1 += round_up(len, 4);
        }
        for (int64_t e = 0; e < len; e += kChunkElems) {
            Chunk c{};
            c.flat_begin = t.offset + e;
            c.count = (int32_t)std::min<int64_t>(kChunkElems, len - e);
            c.param = i;
            c.matrix = mat_of_param[i];
            c.elem_begin = (int32_t)e;
            c.dst = dst + e;
            chunks.push_back(c);
        }
    }
    p->n1d = d1;
    p->nchunks = (int)chunks.size();

    // --- allocations
    int rc;
    if ((rc = dalloc(p, &p->dhi, plane)) || (rc = dalloc(p, &p->dlo, plane)) || (rc = dalloc(p, &p->xhi[0], plane)) ||
        (rc = dalloc(p, &p->xlo[0], plane)) || (rc = dalloc(p, &p->xhi[1], plane)) ||
        (rc = dalloc(p, &p->xlo[1], plane)) ||
        (rc = dalloc(p, &p->ghi, gplane)) || (rc = dalloc(p, &p->glo, gplane)) || (rc = dalloc(p, &p->phi, gplane)) ||
        (rc = dalloc(p, &p->plo, gplane)) || (rc = dalloc(p, &p->ypl, gplane)) || (rc = dalloc(p, &p->gpart, gpart)) || (rc = dalloc(p, &p->d1d, d1)) ||
        (rc = dalloc(p, &p->fin_part, 3 * kPartSlots * fin)) || (rc = dalloc(p, &p->ftiles, (int64_t)ftiles.size())) ||
        (rc = dalloc(p, &p->tpart, tr)) || (rc = dalloc(p, &p->tchunks, tr)) ||
        (rc = dalloc(p, &p->tfpart, std::max<int64_t>(1, tf))) ||
        (rc = dalloc(p, &p->state, p->nmat)) || (rc = dalloc(p, &p->mats_d, p->nmat)) ||
        (rc = dalloc(p, &p->gpart_off_d, p->nmat)) || (rc = dalloc(p, &p->gpart_sstride_d, p->nmat)) ||
        (rc = dalloc(p, &p->nsplit_d, p->nmat)) || (rc = dalloc(p, &p->chunks_d, p->nchunks)) ||
        (rc = dalloc(p, &p->err_d, 1)) || (rc = dalloc(p, &p->list_gram, p->nmat)) ||
        (rc = dalloc(p, &p->list_step, p->nmat)) ||
        (rc = dalloc(p, &p->bucket_first_d, (int64_t)p->buckets.size())) ||
        (rc = dalloc(p, &p->bucket_count_d, (int64_t)p->buckets.size())) ||
        (rc = dalloc(p, &p->cnt_gram, (int64_t)p->buckets.size())) ||
        (rc = dalloc(p, &p->cnt_step, (int64_t)p->buckets.size())) ||
        (rc = dalloc(p, &p->counters, kLaunchCounters + 1)) || (rc = dalloc(p, &p->loopc, 2)) ||
        (rc = dalloc(p, &p->tmaps_d, (int64_t)kMapsPerBucket * std::max<size_t>(1, p->buckets.size()))) ||
        (rc = dalloc(p, &p->anhi, gs_elems)) || (rc = dalloc(p, &p->anlo, gs_elems)) ||
        (rc = dalloc(p, &p->whi, gs_elems)) || (rc = dalloc(p, &p->wlo, gs_elems)) ||
        (rc = dalloc(p, &p->gs_list, (int64_t)gs_mats.size())))
        return rc;
    if (!gs_mats.empty())
        CUDA_TRY(cudaMemcpy(p->gs_list, gs_mats.data(), sizeof(int) * gs_mats.size(), cudaMemcpyHostToDevice));
    CUDA_TRY(cudaHostAlloc(reinterpret_cast<void**>(&p->err_h), sizeof(uint32_t), cudaHostAllocDefault));
    *p->err_h = 0;
    CUDA_TRY(cudaEventCreateWithFlags(&p->done_ev, cudaEventDisableTiming));
    if (p->K * 256 * 4 > 48 * 1024)  // TIES histograms: K (replica passes) or 2K x 256 shared counters
        CUDA_TRY(cudaFuncSetAttribute(k_ties_hist, cudaFuncAttributeMaxDynamicSharedMemorySize, p->K * 256 * 4));
    if (p->K * 256 * 4 > 48 * 1024)  // per-thread counters of the TIES bracket pass
        CUDA_TRY(cudaFuncSetAttribute(k_ties_bracket, cudaFuncAttributeMaxDynamicSharedMemorySize, p->K * 256 * 4));
    if (2 * p->K * 256 * 4 > 48 * 1024)
        CUDA_TRY(cudaFuncSetAttribute(k_ties_hist_buf, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      2 * p->K * 256 * 4));
    CUDA_TRY(cudaStreamCreateWithFlags(&p->cap_st, cudaStreamNonBlocking));
    CUDA_TRY(cudaMemset(p->loopc, 0, 2 * sizeof(long long)));
    // zero the planes once so that padding columns hold zeros
    for (void* a : {(void*)p->dhi, (void*)p->dlo, (void*)p->xhi[0], (void*)p->xlo[0], (void*)p->xhi[1],
                    (void*)p->xlo[1]})
        CUDA_TRY(cudaMemset(a, 0, std::max<int64_t>(1, plane) * 2));
    for (void* a : {(void*)p->ghi, (void*)p->glo, (void*)p->phi, (void*)p->plo, (void*)p->ypl})
        CUDA_TRY(cudaMemset(a, 0, std::max<int64_t>(1, gplane) * 2));
    CUDA_TRY(cudaMemset(p->err_d, 0, 4));
    // Gram partial sums: slots that no kernel writes (the tail of a split-K matrix's last
    // group) must read as zero
    if (fin > 0) CUDA_TRY(cudaMemset(p->fin_part, 0, sizeof(float) * 3 * kPartSlots * fin));
    if (p->nmat) {
        CUDA_TRY(cudaMemcpy(p->mats_d, p->mats_h.data(), sizeof(MatDesc) * p->nmat, cudaMemcpyHostToDevice));
        CUDA_TRY(cudaMemcpy(p->gpart_off_d, gpoff.data(), sizeof(int64_t) * p->nmat, cudaMemcpyHostToDevice));
        CUDA_TRY(cudaMemcpy(p->gpart_sstride_d, gpss.data(), sizeof(int64_t) * p->nmat, cudaMemcpyHostToDevice));
        CUDA_TRY(cudaMemcpy(p->nsplit_d, nsp.data(), sizeof(int) * p->nmat, cudaMemcpyHostToDevice));
        if (!ftiles.empty())
            CUDA_TRY(cudaMemcpy(p->ftiles, ftiles.data(), sizeof(int2) * ftiles.size(), cudaMemcpyHostToDevice));
        CUDA_TRY(cudaMemcpy(p->tchunks, tchunks.data(), sizeof(int4) * tr, cudaMemcpyHostToDevice));
    }
    if (p->nchunks)
        CUDA_TRY(cudaMemcpy(p->chunks_d, chunks.data(), sizeof(Chunk) * p->nchunks, cudaMemcpyHostToDevice));
    if (!p->buckets.empty()) {
        std::vector<int> bf, bc;
        for (const Bucket& bk : p->buckets) {
            bf.push_back(bk.mat_base);
            bc.push_back(bk.count);
        }
        CUDA_TRY(cudaMemcpy(p->bucket_first_d, bf.data(), sizeof(int) * bf.size(), cudaMemcpyHostToDevice));
        CUDA_TRY(cudaMemcpy(p->bucket_count_d, bc.data(), sizeof(int) * bc.size(), cudaMemcpyHostToDevice));
    }

    // --- tensor maps
    if (!p->buckets.empty()) {
        std::vector<CUtensorMap> maps(kMapsPerBucket * p->buckets.size());
        for (size_t b = 0; b < p->buckets.size(); ++b) {
            const Bucket& bk = p->buckets[b];
            CUtensorMap* m = &maps[b * kMapsPerBucket];
            const __nv_bfloat16* src_hi[3] = {p->dhi, p->xhi[0], p->xhi[1]};
            const __nv_bfloat16* src_lo[3] = {p->dlo, p->xlo[0], p->xlo[1]};
            for (int s = 0; s < 3; ++s)
                for (int role = 0; role < 3; ++role)
                    for (int pl = 0; pl < 2; ++pl) {
                        const __nv_bfloat16* base = (pl == 0 ? src_hi[s] : src_lo[s]) + bk.plane_off;
                        if (!make_map(&m[src_map(s, role, pl)], base, bk.cols, bk.rows, bk.count, bk.ld, role))
                            return fail(ISOLOCO_ERR_CUDA, "cuTensorMapEncodeTiled failed (iterate planes)");
                    }
            for (int role = 0; role < 2; ++role)
                for (int pl = 0; pl < 2; ++pl) {
                    if (!make_map(&m[g_map(role, pl)], (pl == 0 ? p->ghi : p->glo) + bk.gplane_off, bk.n, bk.n,
                                  bk.count, bk.ld_n, role) ||
                        !make_map(&m[p_map(role, pl)], (pl == 0 ? p->phi : p->plo) + bk.gplane_off, bk.n, bk.n,
                                  bk.count, bk.ld_n, role))
                        return fail(ISOLOCO_ERR_CUDA, "cuTensorMapEncodeTiled failed (Gram planes)");
                }
            for (int pl = 0; pl < 2; ++pl) {
                if (!make_map(&m[st_map(0, pl)], (pl == 0 ? p->xhi[0] : p->xlo[0]) + bk.plane_off, bk.cols, bk.rows,
                              bk.count, bk.ld, kRoleST) ||
                    !make_map(&m[st_map(1, pl)], (pl == 0 ? p->xhi[1] : p->xlo[1]) + bk.plane_off, bk.cols, bk.rows,
                              bk.count, bk.ld, kRoleST) ||
                    !make_map(&m[st_map(2, pl)], (pl == 0 ? p->ghi : p->glo) + bk.gplane_off, bk.n, bk.n, bk.count,
                              bk.ld_n, kRoleST) ||
                    !make_map(&m[st_map(3, pl)], (pl == 0 ? p->phi : p->plo) + bk.gplane_off, bk.n, bk.n, bk.count,
                              bk.ld_n, kRoleST))
                    return fail(ISOLOCO_ERR_CUDA, "cuTensorMapEncodeTiled failed (store maps)");
            }
            if (!make_map(&m[y_map()], p->ypl + bk.gplane_off, bk.n, bk.n, bk.count, bk.ld_n, kRoleKB) ||
                !make_map(&m[y_st_map()], p->ypl + bk.gplane_off, bk.n, bk.n, bk.count, bk.ld_n, kRoleST))
                return fail(ISOLOCO_ERR_CUDA, "cuTensorMapEncodeTiled failed (Y maps)");
            if (bk.gs) {
                // Z in the first n rows of each matrix's slot of X0 / X1 (tall: ld = ld_n)
                const int zroles[3] = {kRoleKA, kRoleMN, kRoleST};
                for (int buf = 0; buf < 2; ++buf)
                    for (int r = 0; r < 3; ++r)
                        for (int pl = 0; pl < 2; ++pl)
                            if (!make_map(&m[z_map(buf, r, pl)], (pl == 0 ? p->xhi[buf] : p->xlo[buf]) + bk.plane_off,
                                          bk.n, bk.n, bk.count, bk.ld, zroles[r], (int64_t)bk.rows * bk.ld))
                                return fail(ISOLOCO_ERR_CUDA, "cuTensorMapEncodeTiled failed (Gram-side Z maps)");
                for (int pl = 0; pl < 2; ++pl) {
                    const __nv_bfloat16* a = (pl == 0 ? p->anhi : p->anlo) + bk.gs_off;
                    const __nv_bfloat16* w = (pl == 0 ? p->whi : p->wlo) + bk.gs_off;
                    if (!make_map(&m[an_map(pl)], a, bk.n, bk.n, bk.count, bk.ld_n, kRoleKA) ||
                        !make_map(&m[w_mn_map(pl)], w, bk.n, bk.n, bk.count, bk.ld_n, kRoleMN) ||
                        !make_map(&m[w_st_map(pl)], w, bk.n, bk.n, bk.count, bk.ld_n, kRoleST))
                        return fail(ISOLOCO_ERR_CUDA, "cuTensorMapEncodeTiled failed (Gram-side A / W maps)");
                }
            }
        }
        CUDA_TRY(cudaMemcpy(p->tmaps_d, maps.data(), sizeof(CUtensorMap) * maps.size(), cudaMemcpyHostToDevice));
    }
    CUDA_TRY(cudaDeviceSynchronize());
    return ISOLOCO_OK;
}

// ------------------------------------------------------------------ launch helpers
static void set_group_common(GemmGroup& g, int M, int N, int K, int batch, int splits, int mat_base) {
    g.M = M;
    g.N = N;
    g.K = K;
    g.batch = batch;
    g.tiles_m = (M + kTileM - 1) / kTileM;
    g.tiles_n = (N + BN - 1) / BN;
    const int kblocks = (K + BK - 1) / BK;
    g.kblocks_per_split = (kblocks + splits - 1) / splits;
    g.splits = splits;
    g.mat_base = mat_base;
}

// Groups (one per shape bucket) of one GEMM phase; launched kMaxGroups at a time.
static void set_sym(GemmGroup& g, int n) {
    g.sym = 1;
    g.tiles_sym = sym_tiles(n);
}

// Output tiles of one matrix of a group.
static int group_tiles(const GemmGroup& g) { return g.sym ? g.tiles_sym : g.tiles_m * g.tiles_n; }

struct LaunchSet {
    GemmParams p;
    std::vector<GemmGroup> groups;
    // a_mn / b_mn: the operands' layouts in this group (MN-major or K-major); the operands
    // carry lo planes as the set's precision says
    void add(GemmGroup g, bool a_mn, bool b_mn) { add(g, a_mn, b_mn, p.a_split != 0, p.b_split != 0); }
    // ... or as given for this group (the launch's stages take room for either)
    void add(GemmGroup g, bool a_mn, bool b_mn, bool a_split, bool b_split) {
        g.a_mn = a_mn ? 1 : 0;
        g.b_mn = b_mn ? 1 : 0;
        g.a_split = a_split ? 1 : 0;
        g.b_split = b_split ? 1 : 0;
        p.a_split |= g.a_split;
        p.b_split |= g.b_split;
        groups.push_back(g);
    }
};

// Precision of a GEMM launch: operand and output plane types and which operands carry
// a lo plane.  Iteration 0 multiplies the unnormalised Delta: three bf16 passes.  Later
// iterates are normalised and use fp16 planes with two passes (A or B split); the update
// of a matrix's final polish step uses three.
struct Precision {
    int in_f16, out_f16, a_split, b_split, split_on_polish;
};

// Iterations after the first write Y = b I + c G in the Gram epilogue and form
// P = a I + G Y (Horner) in the G^2 launch: no G reads in that epilogue.

static void init_set(LaunchSet& s, int epi, int gate, isoloco_plan* pl, Precision pr) {
    memset(&s.p, 0, sizeof(s.p));
    s.groups.clear();
    s.p.in_f16 = pr.in_f16;
    s.p.out_f16 = pr.out_f16;
    s.p.a_split = pr.a_split;
    s.p.b_split = pr.b_split;
    s.p.split_on_polish = pr.split_on_polish;
    s.p.epi = epi;
    s.p.gate = gate;
    s.p.list = (gate == kGateActive) ? pl->list_gram : pl->list_step;
    s.p.cnt = (gate == kGateActive) ? pl->cnt_gram : pl->cnt_step;
    s.p.state = pl->state;
    s.p.err = pl->err_d;
}

static int flush_set(isoloco_plan* pl, int phase, LaunchSet& s, cudaStream_t st) {
    if (s.groups.empty()) return ISOLOCO_OK;
    // longest CTAs first, so that short tiles fill in behind them (less tail)
    std::stable_sort(s.groups.begin(), s.groups.end(), [](const GemmGroup& x, const GemmGroup& y) {
        return x.kblocks_per_split > y.kblocks_per_split;
    });
    PhaseTimer timer(pl, phase, st, (int)((s.groups.size() + kMaxGroups - 1) / kMaxGroups));
    for (size_t first = 0; first < s.groups.size(); first += kMaxGroups) {
        GemmParams p = s.p;
        p.num_groups = 0;
        int cta = 0;
        for (size_t i = first; i < s.groups.size() && p.num_groups < kMaxGroups; ++i) {
            GemmGroup g = s.groups[i];
            g.cta_begin = cta;
            cta += g.batch * group_tiles(g) * g.splits;
            p.g[p.num_groups++] = g;
        }
        p.total_tiles = cta;
        p.counter = pl->counters + (pl->launch_seq++ % kLaunchCounters);
        CUDA_TRY(launch_gemm(p, pl->num_sms, st));
    }
    return ISOLOCO_OK;
}

// The library's default precision schedule (isoloco_opts_t::precision_schedule = 0), chosen
// by measuring each bucket's Iso-C error against the oracle at 180M K = 8 (every matrix):
// standard schedule (steps 0 .. 5 quintic): Gram and polynomial of steps 1 .. 5 and the
// update of steps 2 .. 5 single-pass; deep schedule (0 .. 10): Gram and polynomial of steps
// 9, 10 and the update of step 10.  Symmetric (Gram, polynomial) roundings only perturb the
// spectrum, which later steps correct; a single-pass update rounds X itself, which turns
// singular vectors for good, so it is kept to the steps where the singular values are
// already clustered near 1.
constexpr long long kDefaultPrecisionSchedule =
    (1ll << 0) | (6ll << 5) | (2ll << 10) | (6ll << 15) | (9ll << 20) | (11ll << 25) | (10ll << 30) | (11ll << 35);

// Decodes a precision schedule code into the plan's per-kind step ranges.
static void set_precision_schedule(isoloco_plan* p, long long code) {
    if (code == 0) code = kDefaultPrecisionSchedule;
    for (int kind = 0; kind < 2; ++kind) {
        int f[4] = {0, 0, 0, 0};
        if (code > 0)
            for (int i = 0; i < 4; ++i) f[i] = static_cast<int>((code >> (5 * (4 * kind + i))) & 31);
        p->gp_from[kind] = f[0];
        p->gp_to[kind] = f[1];
        p->up_from[kind] = f[2];
        p->up_to[kind] = f[3];
    }
    p->prec_code = code;
}

// Bound `end` (0 from, 1 to) of the single-pass Gram / polynomial steps of a schedule kind
// (0 standard, 1 deep); an empty range in the full-precision paths.
static int gp_one(const isoloco_plan* p, int kind, int end) {
    if (p->fast_steps > 0 || p->full_prec) return 0;
    return end ? p->gp_to[kind] : p->gp_from[kind];
}

// The same for the update's single-pass steps.
static int up_one(const isoloco_plan* p, int kind, int end) {
    if (p->fast_steps > 0 || p->full_prec) return 0;
    return end ? p->up_to[kind] : p->up_from[kind];
}

// Single-pass step range of a group (precision schedule; none in the full-precision paths).
static void set_one_pass(const isoloco_plan* p, GemmGroup& g, const Bucket& bk, bool update) {
    const int kind = (std::abs(bk.rows - bk.cols) * 16 < bk.n) ? 1 : 0;  // deep schedule (as MatDesc::deep)
    const bool full = p->fast_steps > 0 || p->full_prec || bk.gs;  // Gram-side steps keep their passes
    g.one_from = full ? 0 : (update ? p->up_from[kind] : p->gp_from[kind]);
    g.one_to = full ? 0 : (update ? p->up_to[kind] : p->gp_to[kind]);
}

// Iteration t of the polar loop for every matrix still active: Gram, convergence test
// and choice of the step (k_control), polynomial, update.  With set_cond, k_control also
// sets the graph condition `cond` (graph body only).
static int polar_iteration(isoloco_plan* p, int t, int max_iter, float tol, cudaStream_t st,
                           cudaGraphConditionalHandle cond, int set_cond) {
    const CUtensorMap* maps = p->tmaps_d;
    {
        const int src = (t == 0) ? 0 : 1 + (t & 1);  // Delta, X0 or X1 as the current iterate
        const int dst = (t + 1) & 1;
        // ---- Gram G = X^T X (tall, MN-major operands) or X X^T (wide, K-major)
        const bool first = (t == 0);
        // The fast variant stops after a fixed number of steps, so nothing corrects a step's
        // rounding afterwards: every step splits both operands (fp16 three passes) and the
        // polynomial is formed from G's hi/lo planes (no single-plane Y).  So does the clip
        // variants' sign iteration (full_prec): there a single-plane rounding perturbs the
        // invariant subspaces the result must separate, which later steps do not undo.  The
        // converging path keeps one operand single from iteration 1 on (its rounding only
        // perturbs the spectrum, which later steps correct).
        const bool full = p->fast_steps > 0 || p->full_prec;
        const bool gs_on = p->n_gs > 0 && !full;  // Gram-side buckets iterate on n x n matrices
        const Precision gram_pr = first ? Precision{0, 0, 1, 1, 0}
                                        : (full ? Precision{1, 1, 1, 1, 0} : Precision{1, 1, 1, 0, 0});
        // Tall and wide matrices share one launch (their tiles pack into fewer waves).
        LaunchSet gram;
        init_set(gram, kEpiGram, kGateActive, p, gram_pr);
        gram.p.gram_y = (first || full) ? 0 : 1;
        // Gram-side buckets after iteration 0 (gramside.cu): W = A Z, then G = Z^T W, both with
        // three passes in launches of their own (a split B operand would thin the main Gram's ring)
        const bool gs_iter = gs_on && !first;
        LaunchSet wset, gsg;
        if (gs_iter) {
            init_set(wset, kEpiXSplit, kGateActive, p, Precision{1, 1, 1, 1, 0});
            wset.p.unit_scale = 1;
            init_set(gsg, kEpiGram, kGateActive, p, Precision{1, 1, 1, 1, 0});
            gsg.p.gram_y = 1;
        }
        for (size_t b = 0; b < p->buckets.size(); ++b) {
            const Bucket& bk = p->buckets[b];
            const CUtensorMap* m = maps + b * kMapsPerBucket;
            GemmGroup g{};
            if (gs_iter && bk.gs) {
                const int zb = t & 1;  // ping-pong buffer holding Z_t
                GemmGroup w{};
                w.a_hi = m + an_map(0);
                w.a_lo = m + an_map(1);
                w.b_hi = m + z_map(zb, 1, 0);
                w.b_lo = m + z_map(zb, 1, 1);
                set_group_common(w, bk.n, bk.n, bk.n, bk.count, 1, bk.mat_base);
                w.bucket = (int)b;
                w.out_hi = p->whi + bk.gs_off;
                w.out_lo = p->wlo + bk.gs_off;
                w.st_hi = m + w_st_map(0);
                w.st_lo = m + w_st_map(1);
                w.bf_batch_stride = (int64_t)bk.n * bk.ld_n;
                w.ld_bf = bk.ld_n;
                wset.add(w, false, true);
                g.a_hi = m + z_map(zb, 1, 0);
                g.a_lo = m + z_map(zb, 1, 1);
                g.b_hi = m + w_mn_map(0);
                g.b_lo = m + w_mn_map(1);
                set_group_common(g, bk.n, bk.n, bk.n, bk.count, 1, bk.mat_base);
                g.bucket = (int)b;
                g.out_hi = p->ghi + bk.gplane_off;
                g.out_lo = p->glo + bk.gplane_off;
                g.st_hi = m + st_map(2, 0);
                g.st_lo = m + st_map(2, 1);
                g.st_y = m + y_st_map();
                g.bf_batch_stride = (int64_t)bk.n * bk.ld_n;
                g.ld_bf = bk.ld_n;
                g.part = p->fin_part;
                g.part_base = p->mats_h[bk.mat_base].gpart_slot;
                set_sym(g, bk.n);
                gsg.add(g, true, true);
                continue;
            }
            const int role_a = bk.tall ? kRoleMN : kRoleKA;
            const int role_b = bk.tall ? kRoleMN : kRoleKB;
            g.a_hi = m + src_map(src, role_a, 0);
            g.a_lo = m + src_map(src, role_a, 1);
            g.b_hi = m + src_map(src, role_b, 0);
            g.b_lo = m + src_map(src, role_b, 1);
            set_group_common(g, bk.n, bk.n, bk.tall ? bk.rows : bk.cols, bk.count, bk.splits, bk.mat_base);
            g.bucket = (int)b;
            g.out_f32 = p->gpart + bk.gpart_off;
            g.f32_batch_stride = (int64_t)bk.n * bk.ld_n;
            g.f32_split_stride = (int64_t)bk.count * bk.n * bk.ld_n;
            g.ld_f32 = bk.ld_n;
            g.out_hi = p->ghi + bk.gplane_off;
            g.out_lo = p->glo + bk.gplane_off;
            g.st_hi = m + st_map(2, 0);
            g.st_lo = m + st_map(2, 1);
            g.st_y = m + y_st_map();
            g.bf_batch_stride = (int64_t)bk.n * bk.ld_n;
            g.ld_bf = bk.ld_n;
            g.part = p->fin_part;
            g.part_base = p->mats_h[bk.mat_base].gpart_slot;
            set_sym(g, bk.n);
            set_one_pass(p, g, bk, false);
            gram.add(g, bk.tall, bk.tall);
        }
        int rc;
        if (gs_iter && ((rc = flush_set(p, ISOLOCO_PHASE_GRAM, wset, st)) ||
                        (rc = flush_set(p, ISOLOCO_PHASE_GRAM, gsg, st))))
            return rc;
        if ((rc = flush_set(p, ISOLOCO_PHASE_GRAM, gram, st))) return rc;
        // after iteration 0 the Gram-side matrices need no finalize: skip an empty launch
        if (p->nftiles && (first || !gs_on || p->nftiles_reg > 0)) {
            PhaseTimer tm(p, ISOLOCO_PHASE_FINALIZE, st);
            k_gram_finalize<<<p->nftiles, 256, 0, st>>>(p->mats_d, p->ftiles, p->state, p->gpart, p->gpart_off_d,
                                                        p->gpart_sstride_d, p->nsplit_d, p->ghi, p->glo,
                                                        p->fin_part, first ? 0 : 1, (first || full) ? nullptr : p->ypl,
                                                        (!first && gs_on) ? 1 : 0);
            CUDA_TRY(cudaGetLastError());
        }
        { PhaseTimer tm(p, ISOLOCO_PHASE_CONTROL, st);
        k_control<<<(p->nmat + kControlThreads / 32 - 1) / (kControlThreads / 32), kControlThreads, 0, st>>>(p->mats_d, p->nmat, p->state, p->fin_part, t, max_iter, tol, p->err_d,
                                      p->bucket_first_d, p->bucket_count_d, (int)p->buckets.size(), p->list_gram,
                                      p->cnt_gram, p->list_step, p->cnt_step, cond, set_cond, p->loopc,
                                      p->fast_steps, p->counters + kLaunchCounters,
                                      make_int4(gp_one(p, 0, 0), gp_one(p, 0, 1), gp_one(p, 1, 0), gp_one(p, 1, 1)),
                                      make_int4(up_one(p, 0, 0), up_one(p, 0, 1), up_one(p, 1, 0), up_one(p, 1, 1)), gs_on ? 1 : 0); }
        CUDA_TRY(cudaGetLastError());
        // ---- P = a I + b G + c G^2
        LaunchSet poly;
        init_set(poly, kEpiPoly, kGateStep, p,
                 first ? Precision{0, 0, 1, 1, 0} : (full ? Precision{1, 1, 1, 1, 0} : Precision{1, 1, 1, 0, 0}));
        poly.p.poly_horner = (first || full) ? 0 : 1;
        for (size_t b = 0; b < p->buckets.size(); ++b) {
            const Bucket& bk = p->buckets[b];
            const CUtensorMap* m = maps + b * kMapsPerBucket;
            GemmGroup g{};
            g.a_hi = m + g_map(kRoleKA, 0);
            g.a_lo = m + g_map(kRoleKA, 1);
            g.b_hi = (first || full) ? m + g_map(kRoleKB, 0) : m + y_map();  // G G or G Y (Horner)
            g.b_lo = m + g_map(kRoleKB, 1);
            set_group_common(g, bk.n, bk.n, bk.n, bk.count, 1, bk.mat_base);
            g.bucket = (int)b;
            g.out_hi = p->phi + bk.gplane_off;
            g.out_lo = p->plo + bk.gplane_off;
            g.st_hi = m + st_map(3, 0);
            g.st_lo = m + st_map(3, 1);
            g.bf_batch_stride = (int64_t)bk.n * bk.ld_n;
            g.ld_bf = bk.ld_n;
            g.g_hi = p->ghi + bk.gplane_off;
            g.g_lo = p->glo + bk.gplane_off;
            set_sym(g, bk.n);
            set_one_pass(p, g, bk, false);
            poly.add(g, false, false);
        }
        if ((rc = flush_set(p, ISOLOCO_PHASE_POLY, poly, st))) return rc;
        // ---- X_{t+1} = xscale * X_t P (tall) or P X_t (wide), one launch
        // X_{t+1} is always written as fp16 planes; X is the split operand (A when tall,
        // B when wide), P the single one except in the polish step (3 passes) and in
        // iteration 0 and the full-precision paths (both split)
        LaunchSet upd;
        init_set(upd, kEpiXSplit, kGateStep, p,
                 first ? Precision{0, 1, 0, 0, 0} : (full ? Precision{1, 1, 0, 0, 0} : Precision{1, 1, 0, 0, 1}));
        const bool p_split = first || full;
        for (size_t b = 0; b < p->buckets.size(); ++b) {
            const Bucket& bk = p->buckets[b];
            const CUtensorMap* m = maps + b * kMapsPerBucket;
            GemmGroup g{};
            if (gs_on && bk.gs) {
                if (first) continue;  // Z_1 = P_0: k_gs_init below
                // Z_{t+1} = Z_t P_t in the first n rows of the other buffer
                g.a_hi = m + z_map(t & 1, 0, 0);
                g.a_lo = m + z_map(t & 1, 0, 1);
                g.b_hi = m + p_map(kRoleKB, 0);
                g.b_lo = m + p_map(kRoleKB, 1);
                set_group_common(g, bk.n, bk.n, bk.n, bk.count, 1, bk.mat_base);
                g.bucket = (int)b;
                g.out_hi = p->xhi[dst] + bk.plane_off;
                g.out_lo = p->xlo[dst] + bk.plane_off;
                g.st_hi = m + z_map(dst, 2, 0);
                g.st_lo = m + z_map(dst, 2, 1);
                g.bf_batch_stride = (int64_t)bk.rows * bk.ld;
                g.ld_bf = bk.ld;
                upd.add(g, false, false, true, p_split);
                continue;
            }
            if (bk.tall) {
                g.a_hi = m + src_map(src, kRoleKA, 0);
                g.a_lo = m + src_map(src, kRoleKA, 1);
                g.b_hi = m + p_map(kRoleKB, 0);
                g.b_lo = m + p_map(kRoleKB, 1);
            } else {
                g.a_hi = m + p_map(kRoleKA, 0);
                g.a_lo = m + p_map(kRoleKA, 1);
                g.b_hi = m + src_map(src, kRoleMN, 0);
                g.b_lo = m + src_map(src, kRoleMN, 1);
            }
            set_group_common(g, bk.rows, bk.cols, bk.n, bk.count, 1, bk.mat_base);
            g.bucket = (int)b;
            g.out_hi = p->xhi[dst] + bk.plane_off;
            g.out_lo = p->xlo[dst] + bk.plane_off;
            g.st_hi = m + st_map(dst, 0);
            g.st_lo = m + st_map(dst, 1);
            g.bf_batch_stride = (int64_t)bk.rows * bk.ld;
            g.ld_bf = bk.ld;
            set_one_pass(p, g, bk, true);
            // the polish writes the final Q: its epilogue also sums tr(Q^T Delta)
            g.d_hi = p->dhi + bk.plane_off;
            g.d_lo = p->dlo + bk.plane_off;
            g.tf_part = p->tfpart + bk.tf_base;
            if (bk.tall)
                upd.add(g, false, false, true, p_split);
            else
                upd.add(g, false, true, p_split, true);
        }
        if ((rc = flush_set(p, ISOLOCO_PHASE_UPDATE, upd, st)))
            return rc;
        if (gs_on && first) {
            // Gram-side: A = Delta^T Delta / s^2 from the fp32 partials, Z_1 = P_0
            PhaseTimer tm(p, ISOLOCO_PHASE_UPDATE, st);
            k_gs_init<<<dim3(p->gs_blocks, p->n_gs), 256, 0, st>>>(p->mats_d, p->state, p->gs_list, p->gpart, p->gpart_off_d,
                                                         p->gpart_sstride_d, p->nsplit_d, p->anhi, p->anlo,
                                                         p->xhi[1], p->xlo[1], p->phi, p->plo);
            CUDA_TRY(cudaGetLastError());
        }
    }
    return ISOLOCO_OK;
}

// Captures iterations 1 and 2 (the buffer parity of every later odd / even pair) as the
// body of a while-conditional graph node; the body's second k_control keeps the loop
// going while some matrix is not done.  Built once per plan and (max_iter, tol).
static int build_polar_graph(isoloco_plan* p, int max_iter, float tol) {
    if (p->gexec) cudaGraphExecDestroy(p->gexec);
    if (p->graph) cudaGraphDestroy(p->graph);
    p->gexec = nullptr;
    p->graph = nullptr;
    p->g_max_iter = -1;
    cudaGraph_t g = nullptr;
    CUDA_TRY(cudaGraphCreate(&g, 0));
    cudaGraphConditionalHandle h;
    cudaError_t e = cudaGraphConditionalHandleCreate(&h, g, 1, cudaGraphCondAssignDefault);
    cudaGraphNodeParams np = {cudaGraphNodeTypeConditional};
    np.conditional.handle = h;
    np.conditional.type = cudaGraphCondTypeWhile;
    np.conditional.size = 1;
    cudaGraphNode_t node = nullptr;
    if (e == cudaSuccess) e = cudaGraphAddNode(&node, g, nullptr, nullptr, 0, &np);
    if (e != cudaSuccess) {
        cudaGraphDestroy(g);
        return fail(ISOLOCO_ERR_CUDA, std::string("polar graph: ") + cudaGetErrorString(e));
    }
    cudaGraph_t body = np.conditional.phGraph_out[0];
    // the captured launches are counted per run of the body, not at capture time
    const int64_t launches0 = p->launches;
    int64_t prof_n0[ISOLOCO_NUM_PHASES];
    memcpy(prof_n0, p->prof_n, sizeof(prof_n0));
    e = cudaStreamBeginCaptureToGraph(p->cap_st, body, nullptr, nullptr, 0, cudaStreamCaptureModeThreadLocal);
    int rc = ISOLOCO_OK;
    if (e == cudaSuccess) {
        rc = polar_iteration(p, 1, max_iter, tol, p->cap_st, h, 0);
        if (rc == ISOLOCO_OK) rc = polar_iteration(p, 2, max_iter, tol, p->cap_st, h, 1);
        cudaGraph_t captured = nullptr;
        const cudaError_t e2 = cudaStreamEndCapture(p->cap_st, &captured);
        if (e2 != cudaSuccess && rc == ISOLOCO_OK) rc = fail(ISOLOCO_ERR_CUDA, std::string("polar graph capture: ") + cudaGetErrorString(e2));
    } else {
        rc = fail(ISOLOCO_ERR_CUDA, std::string("polar graph capture: ") + cudaGetErrorString(e));
    }
    p->body_launches = p->launches - launches0;
    p->launches = launches0;
    memcpy(p->prof_n, prof_n0, sizeof(prof_n0));
    if (rc == ISOLOCO_OK) {
        e = cudaGraphInstantiate(&p->gexec, g, 0);
        if (e != cudaSuccess) rc = fail(ISOLOCO_ERR_CUDA, std::string("polar graph instantiate: ") + cudaGetErrorString(e));
    }
    if (rc != ISOLOCO_OK) {
        (void)cudaGetLastError();
        cudaGraphDestroy(g);
        p->gexec = nullptr;
        return rc;
    }
    p->graph = g;
    p->g_max_iter = max_iter;
    p->g_tol = tol;
    p->g_fast = p->fast_steps;
    p->g_full = p->full_prec ? 1 : 0;
    p->g_prec = p->prec_code;
    return ISOLOCO_OK;
}

// The polar iteration for every matrix, from Delta (planes dhi/dlo) to Q and sigma_bar.
// Iteration 0 is launched directly; the rest run as one graph launch that stops as soon
// as every matrix is done.  With phase profiling on (events cannot sit inside the graph
// body), or when `st` is itself being captured, iterations 1 .. max_iter are launched one
// by one instead (empty launches once every matrix is done).
// Gram-side matrices after the loop: Q = Delta (Z_T / s) into the ping-pong buffer that
// does not hold Z_T (bf16 operands, three passes), and final_buf pointed at it.
static int gs_final(isoloco_plan* p, cudaStream_t st) {
    const CUtensorMap* maps = p->tmaps_d;
    { PhaseTimer tm(p, ISOLOCO_PHASE_UPDATE, st);
    k_gs_final_prep<<<dim3(p->gs_blocks, p->n_gs), 256, 0, st>>>(p->mats_d, p->state, p->gs_list, p->xhi[0], p->xlo[0],
                                                       p->xhi[1], p->xlo[1], p->whi, p->wlo); }
    CUDA_TRY(cudaGetLastError());
    LaunchSet fq;
    init_set(fq, kEpiXSplit, kGateNone, p, Precision{0, 1, 1, 1, 0});
    fq.p.list = nullptr;
    fq.p.cnt = nullptr;
    for (size_t b = 0; b < p->buckets.size(); ++b) {
        const Bucket& bk = p->buckets[b];
        if (!bk.gs) continue;
        const CUtensorMap* m = maps + b * kMapsPerBucket;
        for (int fb = 0; fb < 2; ++fb) {
            GemmGroup g{};
            g.a_hi = m + src_map(0, kRoleKA, 0);
            g.a_lo = m + src_map(0, kRoleKA, 1);
            g.b_hi = m + w_mn_map(0);
            g.b_lo = m + w_mn_map(1);
            set_group_common(g, bk.rows, bk.cols, bk.n, bk.count, 1, bk.mat_base);
            g.bucket = (int)b;
            g.gate_fb = fb + 1;
            g.out_hi = p->xhi[1 - fb] + bk.plane_off;
            g.out_lo = p->xlo[1 - fb] + bk.plane_off;
            g.st_hi = m + st_map(1 - fb, 0);
            g.st_lo = m + st_map(1 - fb, 1);
            g.bf_batch_stride = (int64_t)bk.rows * bk.ld;
            g.ld_bf = bk.ld;
            g.d_hi = p->dhi + bk.plane_off;  // Q is final: tr(Q^T Delta) in the epilogue
            g.d_lo = p->dlo + bk.plane_off;
            g.tf_part = p->tfpart + bk.tf_base;
            fq.add(g, false, true);
        }
    }
    int rc = flush_set(p, ISOLOCO_PHASE_UPDATE, fq, st);
    if (rc) return rc;
    { PhaseTimer tm(p, ISOLOCO_PHASE_UPDATE, st);
    k_gs_final_flip<<<(p->n_gs + 255) / 256, 256, 0, st>>>(p->state, p->gs_list, p->n_gs); }
    CUDA_TRY(cudaGetLastError());
    return ISOLOCO_OK;
}

static int run_polar(isoloco_plan* p, int max_iter, float tol, cudaStream_t st) {
    if (p->nmat == 0) return ISOLOCO_OK;
    // the Gram partial slots of Gram-side matrices: iteration 0's finalize fills fewer of them
    // than the later n x n Grams do, and the control step sums them all
    if (p->n_gs)
        CUDA_TRY(cudaMemsetAsync(p->fin_part + p->gs_slot_first * kPartSlots * 3, 0,
                                 sizeof(float) * p->gs_slot_count * kPartSlots * 3, st));
    int rc = polar_iteration(p, 0, max_iter, tol, st, 0, 0);
    if (rc) return rc;
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    CUDA_TRY(cudaStreamIsCapturing(st, &cs));
    const bool use_graph = kPairMma && !p->prof && !p->per_launch && cs == cudaStreamCaptureStatusNone;
    if (use_graph) {
        if (!p->gexec || p->g_max_iter != max_iter || p->g_tol != tol || p->g_fast != p->fast_steps ||
            p->g_full != (p->full_prec ? 1 : 0) || p->g_prec != p->prec_code)
            if ((rc = build_polar_graph(p, max_iter, tol))) return rc;
        CUDA_TRY(cudaGraphLaunch(p->gexec, st));
    } else {
        std::vector<int> cnt(p->buckets.size());
        for (int t = 1; t <= max_iter; ++t) {
            if ((rc = polar_iteration(p, t, max_iter, tol, st, 0, 0))) return rc;
            if ((p->prof || p->per_launch) && cs == cudaStreamCaptureStatusNone && !cnt.empty()) {
                // profiling: stop, as the graph does, once no matrix is left (the wait for
                // the count lies between the phases' events)
                CUDA_TRY(cudaMemcpyAsync(cnt.data(), p->cnt_gram, sizeof(int) * cnt.size(), cudaMemcpyDeviceToHost, st));
                CUDA_TRY(cudaStreamSynchronize(st));
                int active = 0;
                for (int c : cnt) active += c;
                if (active == 0) break;
            }
        }
    }
    if (p->n_gs && !(p->fast_steps > 0 || p->full_prec) && (rc = gs_final(p, st))) return rc;
    if (p->skip_trace) return ISOLOCO_OK;  // sigma_bar from ||Delta||_F (fast) or not used (spectral)
    { PhaseTimer tm(p, ISOLOCO_PHASE_TRACE, st, 2);
    // windows of 32 chunks: converged matrices' chunks (summed in their GEMM epilogue) cost a
    // flag read each
    k_trace_partial<<<std::max(1, std::min((p->ntchunks + 31) / 32, 4 * p->num_sms)), 256, 0, st>>>(
        p->mats_d, p->tchunks, p->ntchunks, p->state, p->dhi, p->dlo, p->xhi[0],
                                                 p->xlo[0], p->xhi[1], p->xlo[1], p->tpart);
    CUDA_TRY(cudaGetLastError());
    k_trace_final<<<p->nmat, 256, 0, st>>>(p->mats_d, p->nmat, p->state, p->tpart, p->tfpart); }
    CUDA_TRY(cudaGetLastError());
    return ISOLOCO_OK;
}

static int finish_call(isoloco_plan* p, cudaStream_t st, int sync) {
    CUDA_TRY(cudaMemcpyAsync(p->err_h, p->err_d, sizeof(uint32_t), cudaMemcpyDeviceToHost, st));
    CUDA_TRY(cudaEventRecord(p->done_ev, st));
    if (!sync) return ISOLOCO_OK;
    return isoloco_last_status(p, st);
}

// ---------------------------------------------------------------- TIES trim buffers
// Sized once for the plan: a sample of S = min(N, 2^20) keys per worker, and candidate
// segments (one per CTA of the bracket pass) for the widest bracket (sparsity 1/2), with 4x
// headroom over the expected count per CTA.
static int ensure_ties(isoloco_plan* p, int nseg) {
    if (p->ties_hist) return ISOLOCO_OK;
    const int K = p->K;
    const int64_t S = std::min<int64_t>(p->N, int64_t(1) << 20);
    const double m = 8.0 * std::sqrt((double)S * 0.25) + 16.0;
    const double expected = (2.0 * m + 1.0) / (double)S * (double)p->N;  // candidates per worker
    const int64_t segcap = round_up((int64_t)std::ceil(4.0 * expected / nseg) + 256, 4);
    int rc;
    if ((rc = dalloc(p, &p->ties_hist, (int64_t)2 * K * 256)) || (rc = dalloc(p, &p->ties_rank_s, 2 * K)) ||
        (rc = dalloc(p, &p->ties_prefix_s, 2 * K)) || (rc = dalloc(p, &p->ties_rank_c, K)) ||
        (rc = dalloc(p, &p->ties_prefix_c, K)) || (rc = dalloc(p, &p->ties_rank_f, K)) ||
        (rc = dalloc(p, &p->ties_prefix_f, K)) || (rc = dalloc(p, &p->ties_above, K)) ||
        (rc = dalloc(p, &p->ties_fail, 1)) || (rc = dalloc(p, &p->ties_samp, (int64_t)K * S)) ||
        (rc = dalloc(p, &p->ties_cand, (int64_t)K * nseg * segcap)) ||
        (rc = dalloc(p, &p->ties_cnt, (int64_t)K * nseg))) {
        p->ties_hist = nullptr;
        return rc;
    }
    p->ties_S = S;
    p->ties_segcap = segcap;
    p->ties_nseg = nseg;
    return ISOLOCO_OK;
}

// ---------------------------------------------------------------- clip variants (Sec. 4.5)
// Creates, on first use, the auxiliary plan (one n x n matrix per matrix of the plan, the
// same n) and the fp32 buffer of H.
// The fp32 n x n matrices H = Q^T Delta (per split for split-K buckets) and their offsets.
static int ensure_hbuf(isoloco_plan* p) {
    if (p->hbuf) return ISOLOCO_OK;
    std::vector<int64_t> hoff(p->nmat), hss(p->nmat);
    int64_t hb = 0;
    p->hbucket_off.clear();
    for (const Bucket& bk : p->buckets) {
        const int64_t g = (int64_t)bk.n * bk.ld_n;
        p->hbucket_off.push_back(hb);
        for (int j = 0; j < bk.count; ++j) {
            hoff[bk.mat_base + j] = hb + j * g;
            hss[bk.mat_base + j] = (int64_t)bk.count * g;
        }
        hb += round_up((int64_t)bk.splits * bk.count * g, 128);
    }
    int rc;
    if ((rc = dalloc(p, &p->hbuf, hb)) || (rc = dalloc(p, &p->hoff_d, p->nmat)) || (rc = dalloc(p, &p->hss_d, p->nmat)))
        return rc;
    CUDA_TRY(cudaMemcpy(p->hoff_d, hoff.data(), sizeof(int64_t) * p->nmat, cudaMemcpyHostToDevice));
    CUDA_TRY(cudaMemcpy(p->hss_d, hss.data(), sizeof(int64_t) * p->nmat, cudaMemcpyHostToDevice));
    return ISOLOCO_OK;
}

static int ensure_clip(isoloco_plan* p) {
    if (p->aux) return ISOLOCO_OK;
    int rc0 = ensure_hbuf(p);
    if (rc0) return rc0;
    std::vector<isoloco_param_t> t(p->nmat);
    int64_t off = 0;
    for (int i = 0; i < p->nmat; ++i) {
        const int n = p->mats_h[i].n;
        t[i].offset = off;
        t[i].rows = n;
        t[i].cols = n;
        off += (int64_t)n * n;
    }
    isoloco_plan_t a = nullptr;
    int rc = isoloco_plan_create(&a, t.data(), (int)t.size(), off, 1, ISOLOCO_F32);
    if (rc) return rc;
    // aux matrix i holds aux parameter aux->mat_param[i], i.e. this plan's matrix of that index
    std::vector<int> aux_of(p->nmat);
    for (int j = 0; j < a->nmat; ++j) aux_of[a->mat_param[j]] = j;
    if ((rc = dalloc(p, &p->aux_of_d, p->nmat))) {
        isoloco_plan_destroy(a);
        return rc;
    }
    p->aux = a;
    CUDA_TRY(cudaMemcpy(p->aux_of_d, aux_of.data(), sizeof(int) * p->nmat, cudaMemcpyHostToDevice));
    return ISOLOCO_OK;
}

// H = Qb^T Delta (tall, MN-major operands) or Delta Qb^T (wide, K-major), fp32, upper-triangle
// tiles mirrored, split-K partials for split buckets; Qb is Q converted to bf16 (the type of
// Delta's planes) in the ping-pong buffer that does not hold Q.  One GEMM launch per set.
static int form_h(isoloco_plan* p, cudaStream_t st) {
    const CUtensorMap* maps = p->tmaps_d;
    const dim3 grid(64, p->nmat);
    { PhaseTimer tm(p, ISOLOCO_PHASE_CLIP, st);
    k_clip_q_bf16<<<grid, 256, 0, st>>>(p->mats_d, p->state, p->xhi[0], p->xlo[0], p->xhi[1], p->xlo[1]); }
    CUDA_TRY(cudaGetLastError());
    LaunchSet hs;
    init_set(hs, kEpiF32, kGateNone, p, Precision{0, 0, 1, 1, 0});
    hs.p.list = nullptr;
    hs.p.cnt = nullptr;
    for (size_t b = 0; b < p->buckets.size(); ++b) {
        const Bucket& bk = p->buckets[b];
        const CUtensorMap* m = maps + b * kMapsPerBucket;
        for (int fb = 0; fb < 2; ++fb) {
            const int qsrc = 1 + (1 - fb);  // the bf16 copy of Q sits in the other buffer
            GemmGroup g{};
            if (bk.tall) {
                g.a_hi = m + src_map(qsrc, kRoleMN, 0);
                g.a_lo = m + src_map(qsrc, kRoleMN, 1);
                g.b_hi = m + src_map(0, kRoleMN, 0);
                g.b_lo = m + src_map(0, kRoleMN, 1);
            } else {
                g.a_hi = m + src_map(0, kRoleKA, 0);
                g.a_lo = m + src_map(0, kRoleKA, 1);
                g.b_hi = m + src_map(qsrc, kRoleKB, 0);
                g.b_lo = m + src_map(qsrc, kRoleKB, 1);
            }
            set_group_common(g, bk.n, bk.n, bk.tall ? bk.rows : bk.cols, bk.count, bk.splits, bk.mat_base);
            g.bucket = (int)b;
            g.gate_fb = fb + 1;
            g.out_f32 = p->hbuf + p->hbucket_off[b];
            g.f32_batch_stride = (int64_t)bk.n * bk.ld_n;
            g.f32_split_stride = (int64_t)bk.count * bk.n * bk.ld_n;
            g.ld_f32 = bk.ld_n;
            set_sym(g, bk.n);
            hs.add(g, bk.tall, bk.tall);
        }
    }
    return flush_set(p, ISOLOCO_PHASE_CLIP, hs, st);
}

// Buffers of the exact singular values: per matrix the tridiagonal (2 n floats) and sigma_i.
static int ensure_svd(isoloco_plan* p) {
    if (p->sv) return ISOLOCO_OK;
    int rc = ensure_hbuf(p);
    if (rc) return rc;
    std::vector<int64_t> toff(p->nmat), soff(p->nmat);
    int64_t t = 0, v = 0;
    for (int i = 0; i < p->nmat; ++i) {
        toff[i] = t;
        soff[i] = v;
        t += 2 * (int64_t)p->mats_h[i].n;
        v += p->mats_h[i].n;
    }
    if ((rc = dalloc(p, &p->tri, std::max<int64_t>(t, 1))) || (rc = dalloc(p, &p->tri_off_d, p->nmat)) ||
        (rc = dalloc(p, &p->sv, std::max<int64_t>(v, 1))) || (rc = dalloc(p, &p->sv_off_d, p->nmat)))
        return rc;
    CUDA_TRY(cudaMemcpy(p->tri_off_d, toff.data(), sizeof(int64_t) * p->nmat, cudaMemcpyHostToDevice));
    CUDA_TRY(cudaMemcpy(p->sv_off_d, soff.data(), sizeof(int64_t) * p->nmat, cudaMemcpyHostToDevice));
    p->sv_off_h = soff;
    return ISOLOCO_OK;
}

// After the polar iteration and the trace (Q known): sigma_i of every matrix as the
// eigenvalues of H (svd.cu), and sigma_bar = their mean in place of the trace's.
static int run_svd(isoloco_plan* p, cudaStream_t st) {
    if (p->nmat == 0) return ISOLOCO_OK;
    int rc;
    if ((rc = ensure_svd(p)) || (rc = form_h(p, st))) return rc;
    int nmax = 1;
    for (int i = 0; i < p->nmat; ++i) nmax = std::max(nmax, p->mats_h[i].n);
    const size_t smem = sizeof(float) * (4 * (size_t)nmax + 32);
    static bool attr = false;
    if (!attr) {
        CUDA_TRY(cudaFuncSetAttribute(k_svd_tridiag, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024));
        attr = true;
    }
    if (smem > 200 * 1024) return fail(ISOLOCO_ERR_INVALID, "exact singular values: matrices up to 12,792 wide");
    PhaseTimer tm(p, ISOLOCO_PHASE_CLIP, st);
    k_svd_tridiag<<<p->nmat, kSvdThreads, smem, st>>>(p->mats_d, p->state, p->hbuf, p->hoff_d, p->hss_d, p->nsplit_d,
                                                      p->tri, p->tri_off_d);
    CUDA_TRY(cudaGetLastError());
    k_svd_bisect<<<dim3((nmax + 255) / 256, p->nmat), 256, 0, st>>>(p->mats_d, p->tri, p->tri_off_d, p->sv,
                                                                     p->sv_off_d);
    CUDA_TRY(cudaGetLastError());
    k_svd_sigma_bar<<<(p->nmat + 7) / 8, 256, 0, st>>>(p->mats_d, p->nmat, p->state, p->sv, p->sv_off_d);
    CUDA_TRY(cudaGetLastError());
    p->launches += 4;
    return ISOLOCO_OK;
}

// After the polar iteration and sigma_bar's trace (Q and sigma_bar known): Q S' in the ping-pong
// buffer that did not hold Q, and final_buf pointed at it, so that the apply pass forms
// U = alpha sigma_bar Q S' (derivation in spectral.cu).  kind 1: clip_high, 2: clip_low.
static int run_clip(isoloco_plan* p, int kind, int max_iter, float tol, cudaStream_t st) {
    if (p->nmat == 0) return ISOLOCO_OK;
    int rc;
    if ((rc = ensure_clip(p))) return rc;
    isoloco_plan* a = p->aux;
    const CUtensorMap* maps = p->tmaps_d;
    const dim3 grid(64, p->nmat);
    if ((rc = form_h(p, st))) return rc;
    // ---- A' = H / sigma_bar - I -> the auxiliary plan; its polar factor Q_A = sign(A');
    // P = (I -/+ Q_A) / 2; S'' = (P A') P, all in the auxiliary plan's planes
    { PhaseTimer tm(p, ISOLOCO_PHASE_CLIP, st, 0);
    k_reset_state<<<(std::max(1, a->nmat) + 255) / 256, 256, 0, st>>>(
        a->state, a->nmat, a->err_d, a->mats_d, a->bucket_first_d, a->bucket_count_d, (int)a->buckets.size(),
        a->list_gram, a->cnt_gram, a->counters, kLaunchCounters + 1);
    a->launches += 1;
    a->launch_seq = 0;
    CUDA_TRY(cudaGetLastError());
    k_clip_form_a<<<grid, 256, 0, st>>>(p->mats_d, p->state, p->hbuf, p->hoff_d, p->hss_d, p->nsplit_d, a->mats_d,
                                         p->aux_of_d, a->dhi, a->dlo);
    p->launches += 1;
    CUDA_TRY(cudaGetLastError());
    a->fast_steps = 0;
    a->skip_trace = true;
    a->full_prec = true;  // sign(A') is used to first order (P A' P): no single-plane steps
    a->per_launch = p->prof;  // under phase profiling, plain launches as in this plan
    if ((rc = run_polar(a, max_iter, tol, st))) return rc;
    k_clip_form_p<<<dim3(64, a->nmat), 256, 0, st>>>(a->mats_d, a->state, a->xhi[0], a->xlo[0], a->xhi[1],
                                                     a->xlo[1], kind == 1 ? -1.f : 1.f);
    a->launches += 1;
    CUDA_TRY(cudaGetLastError());
    const CUtensorMap* amaps = a->tmaps_d;
    for (int step = 0; step < 2; ++step) {
        // step 0: T = P A' -> G planes; step 1: S'' = T P -> P planes (P and A' symmetric,
        // so their K-major role reads them as they are); bf16, three passes
        LaunchSet ls;
        init_set(ls, kEpiXSplit, kGateNone, a, Precision{0, 0, 1, 1, 0});
        ls.p.list = nullptr;
        ls.p.cnt = nullptr;
        for (size_t b = 0; b < a->buckets.size(); ++b) {
            const Bucket& bk = a->buckets[b];
            const CUtensorMap* m = amaps + b * kMapsPerBucket;
            for (int fa = 0; fa < 2; ++fa) {
                const int psrc = 1 + (1 - fa);  // P sits in the buffer not holding Q_A
                GemmGroup g{};
                if (step == 0) {
                    g.a_hi = m + src_map(psrc, kRoleKA, 0);
                    g.a_lo = m + src_map(psrc, kRoleKA, 1);
                    g.b_hi = m + src_map(0, kRoleKB, 0);
                    g.b_lo = m + src_map(0, kRoleKB, 1);
                    g.out_hi = a->ghi + bk.gplane_off;
                    g.out_lo = a->glo + bk.gplane_off;
                    g.st_hi = m + st_map(2, 0);
                    g.st_lo = m + st_map(2, 1);
                } else {
                    g.a_hi = m + g_map(kRoleKA, 0);
                    g.a_lo = m + g_map(kRoleKA, 1);
                    g.b_hi = m + src_map(psrc, kRoleKB, 0);
                    g.b_lo = m + src_map(psrc, kRoleKB, 1);
                    g.out_hi = a->phi + bk.gplane_off;
                    g.out_lo = a->plo + bk.gplane_off;
                    g.st_hi = m + st_map(3, 0);
                    g.st_lo = m + st_map(3, 1);
                }
                set_group_common(g, bk.n, bk.n, bk.n, bk.count, 1, bk.mat_base);
                g.bucket = (int)b;
                g.gate_fb = fa + 1;
                g.bf_batch_stride = (int64_t)bk.n * bk.ld_n;
                g.ld_bf = bk.ld_n;
                ls.add(g, false, false);
            }
        }
        if ((rc = flush_set(a, ISOLOCO_PHASE_CLIP, ls, st))) return rc;
    } }
    // ---- S' = I + S'' -> this plan's P planes (fp16); X = Q S' (tall) or S' Q (wide) into
    // the other ping-pong buffer (fp16, three passes), which then holds the result
    { PhaseTimer tm(p, ISOLOCO_PHASE_CLIP, st);
    k_clip_form_s<<<grid, 256, 0, st>>>(p->mats_d, a->mats_d, p->aux_of_d, a->state, a->phi, a->plo, p->phi, p->plo,
                                         a->err_d, p->err_d); }
    CUDA_TRY(cudaGetLastError());
    LaunchSet us;
    init_set(us, kEpiXSplit, kGateNone, p, Precision{1, 1, 1, 1, 0});
    us.p.list = nullptr;
    us.p.cnt = nullptr;
    for (size_t b = 0; b < p->buckets.size(); ++b) {
        const Bucket& bk = p->buckets[b];
        const CUtensorMap* m = maps + b * kMapsPerBucket;
        for (int fb = 0; fb < 2; ++fb) {
            const int src = 1 + fb, dst = 1 - fb;
            GemmGroup g{};
            if (bk.tall) {
                g.a_hi = m + src_map(src, kRoleKA, 0);
                g.a_lo = m + src_map(src, kRoleKA, 1);
                g.b_hi = m + p_map(kRoleKB, 0);
                g.b_lo = m + p_map(kRoleKB, 1);
            } else {
                g.a_hi = m + p_map(kRoleKA, 0);
                g.a_lo = m + p_map(kRoleKA, 1);
                g.b_hi = m + src_map(src, kRoleMN, 0);
                g.b_lo = m + src_map(src, kRoleMN, 1);
            }
            set_group_common(g, bk.rows, bk.cols, bk.n, bk.count, 1, bk.mat_base);
            g.bucket = (int)b;
            g.gate_fb = fb + 1;
            g.out_hi = p->xhi[dst] + bk.plane_off;
            g.out_lo = p->xlo[dst] + bk.plane_off;
            g.st_hi = m + st_map(dst, 0);
            g.st_lo = m + st_map(dst, 1);
            g.bf_batch_stride = (int64_t)bk.rows * bk.ld;
            g.ld_bf = bk.ld;
            us.add(g, false, !bk.tall);
        }
    }
    if ((rc = flush_set(p, ISOLOCO_PHASE_CLIP, us, st))) return rc;
    { PhaseTimer tm(p, ISOLOCO_PHASE_CLIP, st);
    k_clip_flip<<<(p->nmat + 255) / 256, 256, 0, st>>>(p->state, p->nmat); }
    CUDA_TRY(cudaGetLastError());
    return ISOLOCO_OK;
}

static int check_opts(const isoloco_opts_t* o, isoloco_opts_t* out) {
    isoloco_opts_default(out);
    if (o) *out = *o;
    if (out->max_iter <= 0) out->max_iter = kDefaultMaxIter;
    if (out->max_iter > 200) return fail(ISOLOCO_ERR_INVALID, "max_iter must be <= 200");
    if (!(out->tol > 0.f)) out->tol = kDefaultTol;
    if (out->fast_steps < 0 || out->fast_steps > 64) return fail(ISOLOCO_ERR_INVALID, "fast_steps must be in 0..64");
    if (out->orth_target < 0 || out->orth_target > 1 || out->momentum_kind < 0 || out->momentum_kind > 1 ||
        out->scale_kind < 0 || out->scale_kind > 1)
        return fail(ISOLOCO_ERR_INVALID, "orth_target, momentum_kind and scale_kind must be 0 or 1");
    if (out->aggregator < 0 || out->aggregator > 2) return fail(ISOLOCO_ERR_INVALID, "aggregator must be 0, 1 or 2");
    if (!(out->sparsity >= 0.f && out->sparsity < 1.f))
        return fail(ISOLOCO_ERR_INVALID, "sparsity must be in [0, 1)");
    if (out->spectrum_kind < 0 || out->spectrum_kind > 3)
        return fail(ISOLOCO_ERR_INVALID, "spectrum_kind must be 0, 1, 2 or 3");
    if (out->full_precision < 0 || out->full_precision > 1)
        return fail(ISOLOCO_ERR_INVALID, "full_precision must be 0 or 1");
    if (out->precision_schedule < -1 || out->precision_schedule >= (1ll << 40))
        return fail(ISOLOCO_ERR_INVALID, "precision_schedule must be -1, 0 or a 40-bit code");
    if (out->spectrum_kind && (out->fast_steps || out->scale_kind))
        return fail(ISOLOCO_ERR_INVALID, "clip_high / clip_low need the exact polar path and sigma_bar "
                                         "(fast_steps = 0, scale_kind = 0)");
    return ISOLOCO_OK;
}

static int check_replicas(isoloco_plan* p, const void* const* reps, ReplicaPtrs& rp) {
    if (!reps) return fail(ISOLOCO_ERR_INVALID, "replicas array is NULL");
    memset(&rp, 0, sizeof(rp));
    for (int k = 0; k < p->K; ++k) {
        if (!reps[k]) return fail(ISOLOCO_ERR_INVALID, "replica pointer is NULL");
        if (!aligned16(reps[k])) return fail(ISOLOCO_ERR_ALIGN, "replica pointer is not 16-byte aligned");
        rp.p[k] = reps[k];
    }
    return ISOLOCO_OK;
}

// The host-buffer entry point with pinned inputs: the reduce reads theta (and B, for the
// orthogonalise-P ablation) from the mapped host buffers; theta and B reach the device
// buffers the step updates by copies on side_st after the reduce (the host link is idle
// while the polar iteration runs), which the apply pass waits for.
struct HostInputs {
    const float* theta_h;
    const float* mom_h;
};

static int run_isoc_step(isoloco_plan* p, int merge, float* theta, float* mom, const void* const* reps,
                         const isoloco_opts_t* opts_in, cudaStream_t st, float* upd_out, const float* base,
                         float* out, float alpha_merge, const HostInputs* hin = nullptr) {
    isoloco_opts_t o;
    int rc;
    if ((rc = check_opts(opts_in, &o))) return rc;
    ReplicaPtrs rp;
    if ((rc = check_replicas(p, reps, rp))) return rc;
    CUDA_TRY(cudaSetDevice(p->device));
    const float* th_src = hin ? hin->theta_h : (merge ? base : theta);
    const float scale = merge ? -1.f : (o.reduce_mean ? 1.f / (float)p->K : 1.f);
    // orthogonalise-P ablation: the reduce pass takes the momentum step on the raw Delta and
    // keeps B' aside, so that a non-finite Delta still leaves B untouched
    const int pmode = (!merge && o.orth_target) ? (o.momentum_kind ? 2 : 1) : 0;
    if (pmode && !p->bnew) {
        const int rc2 = dalloc(p, &p->bnew, p->N);
        if (rc2) return rc2;
    }
    { PhaseTimer tm(p, ISOLOCO_PHASE_OTHER, st);
    k_reset_state<<<(std::max(1, p->nmat) + 255) / 256, 256, 0, st>>>(
        p->state, p->nmat, p->err_d, p->mats_d, p->bucket_first_d, p->bucket_count_d, (int)p->buckets.size(),
        p->list_gram, p->cnt_gram, p->counters, kLaunchCounters + 1); }
    p->launch_seq = 0;
    CUDA_TRY(cudaGetLastError());
    if (p->nchunks) {
        PhaseTimer tm(p, ISOLOCO_PHASE_REDUCE, st);
        if (pmode)
            k_reduce_p<<<p->nchunks, 256, 0, st>>>(p->chunks_d, p->mats_d, rp, p->K, p->dtype, th_src, scale,
                                                   p->dhi, p->dlo, p->d1d, p->err_d, pmode, o.momentum,
                                                   hin ? hin->mom_h : mom, p->bnew);
        else if (p->dtype == ISOLOCO_F32)
            k_reduce_f32<<<p->nchunks, 256, 0, st>>>(p->chunks_d, p->mats_d, rp, p->K, th_src, scale, p->dhi,
                                                     p->dlo, p->d1d, p->err_d);
        else
            k_reduce<<<p->nchunks, 256, 0, st>>>(p->chunks_d, p->mats_d, rp, p->K, p->dtype, th_src, scale, p->dhi,
                                                 p->dlo, p->d1d, p->err_d);
        CUDA_TRY(cudaGetLastError());
    }
    if (hin) {
        CUDA_TRY(cudaEventRecord(p->ev_reduced, st));
        CUDA_TRY(cudaStreamWaitEvent(p->side_st, p->ev_reduced, 0));
        CUDA_TRY(cudaMemcpyAsync(theta, hin->theta_h, p->N * 4, cudaMemcpyHostToDevice, p->side_st));
        CUDA_TRY(cudaMemcpyAsync(mom, hin->mom_h, p->N * 4, cudaMemcpyHostToDevice, p->side_st));
        CUDA_TRY(cudaEventRecord(p->ev_copied, p->side_st));
    }
    p->fast_steps = merge ? 0 : o.fast_steps;
    // the spectrum variants need Q's singular values at 1 to ~2^-20: three passes throughout
    // (a two-pass Gram feeding the polish leaves ~1e-4 in them)
    p->full_prec = !merge && (o.spectrum_kind != 0 || o.full_precision != 0);
    set_precision_schedule(p, merge ? -1 : o.precision_schedule);
    p->skip_trace = !merge && (o.fast_steps > 0 || o.scale_kind == 1);
    if ((rc = run_polar(p, p->fast_steps ? std::max(o.max_iter, o.fast_steps) : o.max_iter, o.tol, st))) return rc;
    const int clip = merge ? 0 : o.spectrum_kind;
    if ((clip == 1 || clip == 2) && (rc = run_clip(p, clip, o.max_iter, o.tol, st))) return rc;
    if (clip == 3 && (rc = run_svd(p, st))) return rc;
    UpdateSrc us;
    us.qh[0] = p->xhi[0];
    us.qh[1] = p->xhi[1];
    us.ql[0] = p->xlo[0];
    us.ql[1] = p->xlo[1];
    us.d1d = p->d1d;
    if (hin) CUDA_TRY(cudaStreamWaitEvent(st, p->ev_copied, 0));
    if (p->nchunks) {
        PhaseTimer tm(p, ISOLOCO_PHASE_APPLY, st);
        if (merge)
            k_apply<<<p->nchunks, 256, 0, st>>>(p->chunks_d, p->mats_d, p->state, us, 1, alpha_merge, 0.f, 0.f,
                                                nullptr, nullptr, base, out, nullptr, p->err_d, 0, 0, 0, nullptr);
        else
            k_apply<<<p->nchunks, 256, 0, st>>>(p->chunks_d, p->mats_d, p->state, us, 0, o.alpha, o.outer_lr,
                                                o.momentum, theta, mom, nullptr, nullptr, upd_out, p->err_d,
                                                o.momentum_kind, pmode, o.scale_kind, p->bnew);
        CUDA_TRY(cudaGetLastError());
    }
    return finish_call(p, st, o.sync);
}

// ================================================================== C ABI
extern "C" {

const char* isoloco_last_error(void) { return g_last_error.c_str(); }

int isoloco_opts_default(isoloco_opts_t* o) {
    if (!o) return fail(ISOLOCO_ERR_INVALID, "opts is NULL");
    o->alpha = 1.f;
    o->outer_lr = 0.7f;
    o->momentum = 0.9f;
    o->reduce_mean = 1;
    o->max_iter = kDefaultMaxIter;
    o->tol = kDefaultTol;
    o->sync = 0;
    o->fast_steps = 0;
    o->orth_target = 0;
    o->momentum_kind = 0;
    o->scale_kind = 0;
    o->aggregator = 0;
    o->sparsity = 0.f;
    o->seed = 0u;
    o->spectrum_kind = 0;
    o->full_precision = 0;
    o->precision_schedule = 0;
    return ISOLOCO_OK;
}

int isoloco_plan_create(isoloco_plan_t* out, const isoloco_param_t* table, int n_params, int64_t n_total, int K,
                        isoloco_dtype_t replica_dtype) {
    if (!out) return fail(ISOLOCO_ERR_INVALID, "plan out-pointer is NULL");
    *out = nullptr;
    if (n_params < 0 || (n_params > 0 && !table)) return fail(ISOLOCO_ERR_INVALID, "bad table");
    if (n_total <= 0) return fail(ISOLOCO_ERR_INVALID, "n_total must be positive");
    if (K < 1 || K > kMaxK) return fail(ISOLOCO_ERR_INVALID, "K must be in 1..64");
    if (replica_dtype != ISOLOCO_F32 && replica_dtype != ISOLOCO_BF16)
        return fail(ISOLOCO_ERR_INVALID, "bad replica dtype");
    std::vector<std::pair<int64_t, int64_t>> spans;
    for (int i = 0; i < n_params; ++i) {
        const isoloco_param_t& t = table[i];
        if (t.rows <= 0 || t.cols < 0 || t.offset < 0) return fail(ISOLOCO_ERR_INVALID, "bad table entry");
        const int64_t len = (int64_t)t.rows * (t.cols > 0 ? t.cols : 1);
        if (len > 2147483647LL || t.offset + len > n_total)
            return fail(ISOLOCO_ERR_INVALID, "table entry outside [0, n_total)");
        spans.emplace_back(t.offset, t.offset + len);
    }
    std::sort(spans.begin(), spans.end());
    for (size_t i = 1; i < spans.size(); ++i)
        if (spans[i].first < spans[i - 1].second) return fail(ISOLOCO_ERR_INVALID, "table entries overlap");
    isoloco_plan* p = new isoloco_plan();
    cudaError_t e = cudaGetDevice(&p->device);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&p->num_sms, cudaDevAttrMultiProcessorCount, p->device);
    if (e != cudaSuccess) {
        delete p;
        return fail(ISOLOCO_ERR_CUDA, std::string("no CUDA device: ") + cudaGetErrorString(e));
    }
    p->K = K;
    p->dtype = (int)replica_dtype;
    p->N = n_total;
    p->table.assign(table, table + n_params);
    int rc = build_plan(p, table, n_params);
    if (rc != ISOLOCO_OK) {
        free_plan(p);
        return rc;
    }
    *out = p;
    return ISOLOCO_OK;
}

void isoloco_plan_destroy(isoloco_plan_t p) {
    if (!p) return;
    cudaSetDevice(p->device);
    cudaDeviceSynchronize();
    free_plan(p);
}

int64_t isoloco_plan_workspace_bytes(isoloco_plan_t p) { return p ? p->ws_bytes : 0; }

int isoloco_plan_num_matrices(isoloco_plan_t p) { return p ? p->nmat : 0; }

int isoloco_outer_step(isoloco_plan_t p, float* theta, float* momentum, const void* const* replicas,
                       const isoloco_opts_t* opts, void* stream, float* update_out) {
    if (!p) return fail(ISOLOCO_ERR_INVALID, "plan is NULL");
    if (!theta || !momentum) return fail(ISOLOCO_ERR_INVALID, "theta or momentum is NULL");
    if (!aligned16(theta) || !aligned16(momentum) || (update_out && !aligned16(update_out)))
        return fail(ISOLOCO_ERR_ALIGN, "theta, momentum and update_out must be 16-byte aligned");
    return run_isoc_step(p, 0, theta, momentum, replicas, opts, static_cast<cudaStream_t>(stream), update_out,
                         nullptr, nullptr, 0.f);
}

int iso_c_merge(isoloco_plan_t p, const float* base, const void* const* experts, float alpha, float* out,
                void* stream) {
    if (!p) return fail(ISOLOCO_ERR_INVALID, "plan is NULL");
    if (!base || !out) return fail(ISOLOCO_ERR_INVALID, "base or out is NULL");
    if (!aligned16(base) || !aligned16(out)) return fail(ISOLOCO_ERR_ALIGN, "base and out must be 16-byte aligned");
    isoloco_opts_t o;
    isoloco_opts_default(&o);
    return run_isoc_step(p, 1, nullptr, nullptr, experts, &o, static_cast<cudaStream_t>(stream), nullptr, base,
                         out, alpha);
}

int diloco_outer_step(isoloco_plan_t p, float* theta, float* momentum, const void* const* replicas,
                      const isoloco_opts_t* opts_in, void* stream) {
    if (!p) return fail(ISOLOCO_ERR_INVALID, "plan is NULL");
    if (!theta || !momentum) return fail(ISOLOCO_ERR_INVALID, "theta or momentum is NULL");
    if (!aligned16(theta) || !aligned16(momentum)) return fail(ISOLOCO_ERR_ALIGN, "theta/momentum not aligned");
    isoloco_opts_t o;
    int rc;
    if ((rc = check_opts(opts_in, &o))) return rc;
    ReplicaPtrs rp;
    if ((rc = check_replicas(p, replicas, rp))) return rc;
    CUDA_TRY(cudaSetDevice(p->device));
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    CUDA_TRY(cudaMemsetAsync(p->err_d, 0, 4, st));
    const float scale = o.reduce_mean ? 1.f / (float)p->K : 1.f;
    const int grid = p->num_sms * 8;
    if (o.aggregator == 0) {
        PhaseTimer tm(p, ISOLOCO_PHASE_DILOCO, st);
        k_diloco<<<grid, 256, 0, st>>>(rp, p->K, p->dtype, theta, momentum, p->N, scale, o.outer_lr, o.momentum,
                                       p->err_d);
    } else if (o.aggregator == 2) {
        PhaseTimer tm(p, ISOLOCO_PHASE_DILOCO, st);
        // keep when top24 >= ceil(p * 2^24) (exact in double); draw numbers step by N * GAMMA
        const uint32_t pthr = (uint32_t)std::ceil((double)o.sparsity * 16777216.0);
        const uint64_t ng = (uint64_t)p->N * 0x9E3779B97F4A7C15ull;
        k_dare<<<grid, 256, 0, st>>>(rp, p->K, p->dtype, theta, momentum, p->N, scale, pthr,
                                     1.f / (1.f - o.sparsity), o.seed, ng, o.outer_lr, o.momentum, p->err_d);
    } else {
        // keep the n_keep largest |Delta_k| of each worker; n_keep = N keeps all (threshold 0)
        const uint64_t n_keep = (uint64_t)(p->N - (int64_t)std::floor((double)o.sparsity * (double)p->N));
        const bool select = n_keep < (uint64_t)p->N;
        if ((rc = ensure_ties(p, grid))) return rc;
        const int K = p->K;
        // sample ranks bracketing the threshold's expected rank n_keep S / N by 8 standard
        // deviations of a sample count (and 16)
        const double S = (double)p->ties_S, q = (double)n_keep / (double)p->N;
        const double r_mid = q * S, m = 8.0 * std::sqrt(S * q * (1.0 - q)) + 16.0;
        const uint64_t r_hi = (uint64_t)std::max(1.0, std::floor(r_mid - m));
        const uint64_t r_lo = (uint64_t)std::min(S, std::ceil(r_mid + m));
        {
            PhaseTimer tm(p, ISOLOCO_PHASE_TRIM, st, select ? 29 : 1);
            k_ties_init<<<1, 256, 0, st>>>(K, n_keep, r_hi, r_lo, p->ties_hist, p->ties_rank_s, p->ties_prefix_s,
                                           p->ties_rank_c, p->ties_prefix_c, p->ties_rank_f, p->ties_prefix_f,
                                           p->ties_above, p->ties_fail);
            if (select) {
                k_ties_sample<<<(unsigned)((p->ties_S + 255) / 256), 256, 0, st>>>(rp, K, p->dtype, theta, p->N,
                                                                                 p->ties_S, p->ties_samp);
                for (int pass = 0; pass < 4; ++pass) {
                    k_ties_hist_buf<<<dim3(1, 256), 256, 2 * K * 256 * 4, st>>>(
                        p->ties_samp, nullptr, 1, p->ties_S, 2 * K, 2, pass, p->ties_prefix_s, p->ties_hist);
                    k_ties_select<<<(2 * K * 32 + 255) / 256, 256, 0, st>>>(2 * K, pass, p->ties_hist, p->ties_rank_s, p->ties_prefix_s,
                                                     nullptr);
                }
                k_ties_bracket<<<p->ties_nseg, 256, K * 256 * 4, st>>>(rp, K, p->dtype, theta, p->N, p->ties_prefix_s,
                                                            p->ties_cand, p->ties_cnt, p->ties_segcap, p->ties_above);
                k_ties_check<<<K, 256, 0, st>>>(K, p->ties_nseg, p->ties_segcap, n_keep, p->ties_above, p->ties_cnt,
                                               p->ties_rank_c, p->ties_fail);
                for (int pass = 0; pass < 4; ++pass) {
                    k_ties_hist_buf<<<dim3(p->ties_nseg, 1), 256, K * 256 * 4, st>>>(
                        p->ties_cand, p->ties_cnt, p->ties_nseg, p->ties_segcap, K, 1, pass, p->ties_prefix_c,
                        p->ties_hist);
                    k_ties_select<<<(K * 32 + 255) / 256, 256, 0, st>>>(K, pass, p->ties_hist, p->ties_rank_c, p->ties_prefix_c,
                                                    nullptr);
                }
                // fallback, only when some bracket missed: the four passes over the replicas
                const int smem = K * 256 * 4;
                for (int pass = 0; pass < 4; ++pass) {
                    k_ties_hist<<<grid, 256, smem, st>>>(rp, K, p->dtype, theta, p->N, pass, p->ties_prefix_f,
                                                         p->ties_hist, p->ties_fail);
                    k_ties_select<<<(K * 32 + 255) / 256, 256, 0, st>>>(K, pass, p->ties_hist, p->ties_rank_f, p->ties_prefix_f,
                                                    p->ties_fail);
                }
            }
        }
        PhaseTimer tm(p, ISOLOCO_PHASE_DILOCO, st);
        k_ties_merge<<<grid, 256, 0, st>>>(rp, p->K, p->dtype, theta, momentum, p->N, p->ties_prefix_c,
                                           p->ties_prefix_f, p->ties_fail, o.outer_lr, o.momentum, p->err_d);
    }
    CUDA_TRY(cudaGetLastError());
    return finish_call(p, st, o.sync);
}

// A host pointer the device may read in place: page-locked memory registered with CUDA.
static bool mapped_host(const void* h, const void** dptr) {
    cudaPointerAttributes at;
    if (cudaPointerGetAttributes(&at, h) != cudaSuccess) {
        (void)cudaGetLastError();
        return false;
    }
    if (at.type != cudaMemoryTypeHost || !at.devicePointer) return false;
    *dptr = at.devicePointer;
    return true;
}

int isoloco_outer_step_host(isoloco_plan_t p, float* theta_h, float* mom_h, const void* const* reps_h,
                            const isoloco_opts_t* opts, void* stream) {
    if (!p) return fail(ISOLOCO_ERR_INVALID, "plan is NULL");
    if (!theta_h || !mom_h || !reps_h) return fail(ISOLOCO_ERR_INVALID, "NULL host buffer");
    for (int k = 0; k < p->K; ++k)
        if (!reps_h[k]) return fail(ISOLOCO_ERR_INVALID, "NULL host replica");
    CUDA_TRY(cudaSetDevice(p->device));
    const size_t eb = p->dtype == ISOLOCO_F32 ? 4 : 2;
    const size_t rep_bytes = round_up((int64_t)(p->N * eb), 256);
    int rc;
    isoloco_opts_t o;
    if ((rc = check_opts(opts, &o))) return rc;
    o.sync = 0;
    if (!p->st_theta)
        if ((rc = dalloc(p, &p->st_theta, p->N)) || (rc = dalloc(p, &p->st_mom, p->N))) return rc;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    // pinned inputs: replicas, theta and B read in place by the reduce (no staging copy)
    std::vector<const void*> dr(p->K);
    const void* th_d = nullptr;
    const void* mom_d = nullptr;
    bool mapped = mapped_host(theta_h, &th_d) && mapped_host(mom_h, &mom_d) && ((uintptr_t)th_d & 15u) == 0 &&
                  ((uintptr_t)mom_d & 15u) == 0;
    for (int k = 0; mapped && k < p->K; ++k) mapped = mapped_host(reps_h[k], &dr[k]);
    if (mapped) {
        if (!p->side_st) {
            CUDA_TRY(cudaStreamCreateWithFlags(&p->side_st, cudaStreamNonBlocking));
            CUDA_TRY(cudaEventCreateWithFlags(&p->ev_reduced, cudaEventDisableTiming));
            CUDA_TRY(cudaEventCreateWithFlags(&p->ev_copied, cudaEventDisableTiming));
        }
        const HostInputs hin{static_cast<const float*>(th_d), static_cast<const float*>(mom_d)};
        if ((rc = run_isoc_step(p, 0, p->st_theta, p->st_mom, dr.data(), &o, st, nullptr, nullptr, nullptr, 0.f,
                                &hin)))
            return rc;
    } else {
        if (!p->st_reps) {
            uint8_t* r = nullptr;
            if ((rc = dalloc(p, &r, (int64_t)rep_bytes * p->K))) return rc;
            p->st_reps = r;
        }
        CUDA_TRY(cudaMemcpyAsync(p->st_theta, theta_h, p->N * 4, cudaMemcpyHostToDevice, st));
        CUDA_TRY(cudaMemcpyAsync(p->st_mom, mom_h, p->N * 4, cudaMemcpyHostToDevice, st));
        for (int k = 0; k < p->K; ++k) {
            void* d = static_cast<uint8_t*>(p->st_reps) + k * rep_bytes;
            CUDA_TRY(cudaMemcpyAsync(d, reps_h[k], p->N * eb, cudaMemcpyHostToDevice, st));
            dr[k] = d;
        }
        if ((rc = run_isoc_step(p, 0, p->st_theta, p->st_mom, dr.data(), &o, st, nullptr, nullptr, nullptr, 0.f)))
            return rc;
    }
    CUDA_TRY(cudaMemcpyAsync(theta_h, p->st_theta, p->N * 4, cudaMemcpyDeviceToHost, st));
    CUDA_TRY(cudaMemcpyAsync(mom_h, p->st_mom, p->N * 4, cudaMemcpyDeviceToHost, st));
    return isoloco_last_status(p, st);
}

int isoloco_last_status(isoloco_plan_t p, void* stream) {
    if (!p) return fail(ISOLOCO_ERR_INVALID, "plan is NULL");
    CUDA_TRY(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)));
    CUDA_TRY(cudaEventSynchronize(p->done_ev));
    const uint32_t e = *p->err_h;
    if (e & kErrTimeout) return fail(ISOLOCO_ERR_TIMEOUT, "a device-side wait timed out");
    if (e & kErrNonFinite) return fail(ISOLOCO_ERR_NONFINITE, "non-finite pseudo-gradient");
    if (e & kErrNotConverged) return fail(ISOLOCO_ERR_NOT_CONVERGED, "polar iteration hit max_iter");
    return ISOLOCO_OK;
}

int isoloco_profile_enable(isoloco_plan_t p, int enable) {
    if (!p) return fail(ISOLOCO_ERR_INVALID, "plan is NULL");
    CUDA_TRY(cudaDeviceSynchronize());
    for (int ph = 0; ph < ISOLOCO_NUM_PHASES; ++ph) {
        for (auto& pr : p->pend[ph]) {
            p->ev_pool.push_back(pr.first);
            p->ev_pool.push_back(pr.second);
        }
        p->pend[ph].clear();
        p->prof_ms[ph] = 0.0;
        p->prof_n[ph] = 0;
    }
    p->prof = enable != 0;
    return ISOLOCO_OK;
}

int isoloco_profile_read(isoloco_plan_t p, void* stream, double* ms, int64_t* launches, int nphases) {
    if (!p) return fail(ISOLOCO_ERR_INVALID, "plan is NULL");
    CUDA_TRY(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)));
    for (int ph = 0; ph < ISOLOCO_NUM_PHASES; ++ph) {
        for (auto& pr : p->pend[ph]) {
            float t = 0.f;
            CUDA_TRY(cudaEventElapsedTime(&t, pr.first, pr.second));
            p->prof_ms[ph] += t;
            p->ev_pool.push_back(pr.first);
            p->ev_pool.push_back(pr.second);
        }
        p->pend[ph].clear();
    }
    for (int ph = 0; ph < nphases && ph < ISOLOCO_NUM_PHASES; ++ph) {
        if (ms) ms[ph] = p->prof_ms[ph];
        if (launches) launches[ph] = p->prof_n[ph];
    }
    return ISOLOCO_OK;
}

int64_t isoloco_plan_launches(isoloco_plan_t p) {
    if (!p) return 0;
    // kernels launched directly, plus those of every run of the polar graph's body
    long long runs[2] = {0, 0};
    if (p->body_launches > 0 && cudaMemcpy(runs, p->loopc, sizeof(runs), cudaMemcpyDeviceToHost) != cudaSuccess)
        runs[1] = 0;
    return p->launches + p->body_launches * static_cast<int64_t>(runs[1]) + (p->aux ? isoloco_plan_launches(p->aux) : 0);
}

int isoloco_read_diag(isoloco_plan_t p, void* stream, float* sigma_bar, int32_t* iters, int32_t* status,
                      float* resid) {
    if (!p) return fail(ISOLOCO_ERR_INVALID, "plan is NULL");
    CUDA_TRY(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)));
    if (p->nmat == 0) return ISOLOCO_OK;
    std::vector<MatState> s(p->nmat);
    CUDA_TRY(cudaMemcpy(s.data(), p->state, sizeof(MatState) * p->nmat, cudaMemcpyDeviceToHost));
    // report in table order of the 2-D tensors
    std::vector<int> order(p->nmat);
    for (int i = 0; i < p->nmat; ++i) order[i] = i;
    std::sort(order.begin(), order.end(), [&](int a, int b) { return p->mat_param[a] < p->mat_param[b]; });
    for (int j = 0; j < p->nmat; ++j) {
        const MatState& m = s[order[j]];
        if (sigma_bar) sigma_bar[j] = m.sigma_bar;
        if (iters) iters[j] = m.iters;
        if (status) status[j] = m.status ? ISOLOCO_ERR_NOT_CONVERGED : ISOLOCO_OK;
        if (resid) resid[j] = m.resid;
    }
    return ISOLOCO_OK;
}

int isoloco_check_guards(isoloco_plan_t p, void* stream) {
    if (!p) return fail(ISOLOCO_ERR_INVALID, "plan is NULL");
    CUDA_TRY(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)));
    std::vector<uint8_t> h;
    for (isoloco_plan* q = p; q; q = q->aux) {
        for (size_t r = 0; r < q->guards.size(); ++r) {
            uint8_t* base = q->guards[r].first;
            const size_t bytes = q->guards[r].second;
            const size_t body = (bytes + kGuardBytes - 1) / kGuardBytes * kGuardBytes;
            const size_t tail = body - bytes + kGuardBytes;
            h.resize(kGuardBytes + tail);
            CUDA_TRY(cudaMemcpy(h.data(), base, kGuardBytes, cudaMemcpyDeviceToHost));
            CUDA_TRY(cudaMemcpy(h.data() + kGuardBytes, base + kGuardBytes + bytes, tail, cudaMemcpyDeviceToHost));
            for (size_t i = 0; i < h.size(); ++i)
                if (h[i] != static_cast<uint8_t>(kGuardByte)) {
                    const bool front = i < kGuardBytes;
                    return fail(ISOLOCO_ERR_GUARD, std::string("workspace region ") + std::to_string(r) + " of " +
                                                       (q == p ? "the plan" : "its auxiliary plan") + ": byte " +
                                                       std::to_string(front ? kGuardBytes - i : i - kGuardBytes + 1) +
                                                       (front ? " before its start" : " past its end") +
                                                       " overwritten");
                }
        }
    }
    return ISOLOCO_OK;
}

int isoloco_debug_touch_guard(isoloco_plan_t p, int region, int after) {
    if (!p) return fail(ISOLOCO_ERR_INVALID, "plan is NULL");
    if (region < 0 || region >= static_cast<int>(p->guards.size()))
        return fail(ISOLOCO_ERR_INVALID, "no such workspace region");
    uint8_t* base = p->guards[region].first;
    uint8_t* at = after ? base + kGuardBytes + p->guards[region].second : base + kGuardBytes - 1;
    CUDA_TRY(cudaMemset(at, 0x5A, 1));  // one guard byte, inside the allocation
    return ISOLOCO_OK;
}

int isoloco_read_singular_values(isoloco_plan_t p, void* stream, int matrix, float* out, int capacity) {
    if (!p) return fail(ISOLOCO_ERR_INVALID, "plan is NULL");
    if (matrix < 0 || matrix >= p->nmat) return fail(ISOLOCO_ERR_INVALID, "matrix index out of range");
    if (!p->sv) return fail(ISOLOCO_ERR_INVALID, "no singular values: run a step with spectrum_kind = 3 first");
    // table order of the 2-D tensors -> plan order
    std::vector<int> order(p->nmat);
    for (int i = 0; i < p->nmat; ++i) order[i] = i;
    std::sort(order.begin(), order.end(), [&](int a, int b) { return p->mat_param[a] < p->mat_param[b]; });
    const int mi = order[matrix];
    const int n = p->mats_h[mi].n;
    if (!out || capacity < n) return fail(ISOLOCO_ERR_INVALID, "output buffer smaller than min(rows, cols)");
    CUDA_TRY(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)));
    CUDA_TRY(cudaMemcpy(out, p->sv + p->sv_off_h[mi], sizeof(float) * n, cudaMemcpyDeviceToHost));
    return n;
}

int isoloco_debug_wait_timeout(int64_t limit_ns, int64_t* elapsed_ns, void* stream) {
    if (limit_ns < 1000000 || limit_ns > 1000000000) return fail(ISOLOCO_ERR_INVALID, "limit_ns outside 1 ms .. 1 s");
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    uint32_t* err = nullptr;
    unsigned long long* el = nullptr;
    if (cudaMalloc(&err, 4) != cudaSuccess || cudaMalloc(&el, 8) != cudaSuccess) {
        cudaFree(err);
        return fail(ISOLOCO_ERR_OOM, "debug_wait_timeout scratch allocation failed");
    }
    uint32_t herr = 0;
    unsigned long long hel = 0;
    cudaError_t e = cudaMemsetAsync(err, 0, 4, st);
    if (e == cudaSuccess) {
        k_debug_wait<<<1, 32, 0, st>>>(err, static_cast<uint64_t>(limit_ns), el);
        e = cudaGetLastError();
    }
    if (e == cudaSuccess) e = cudaMemcpyAsync(&herr, err, 4, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaMemcpyAsync(&hel, el, 8, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    cudaFree(err);
    cudaFree(el);
    if (e != cudaSuccess) return fail(ISOLOCO_ERR_CUDA, std::string("debug_wait_timeout: ") + cudaGetErrorString(e));
    if (elapsed_ns) *elapsed_ns = static_cast<int64_t>(hel);
    if (herr & kErrTimeout) return fail(ISOLOCO_ERR_TIMEOUT, "debug_wait_timeout: the wait gave up");
    return ISOLOCO_OK;
}

int isoloco_debug_gemm(int a_mn, int b_mn, int precision, int batch, int M, int N, int K, const float* A,
                       const float* B, float* D, void* stream) {
    if (precision < 0 || precision > 3) return fail(ISOLOCO_ERR_INVALID, "bad debug_gemm precision");
    if (batch <= 0 || M <= 0 || N <= 0 || K <= 0 || !A || !B || !D)
        return fail(ISOLOCO_ERR_INVALID, "bad debug_gemm arguments");
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const int a_rows = a_mn ? K : M, a_cols = a_mn ? M : K;
    const int b_rows = b_mn ? K : N, b_cols = b_mn ? N : K;
    const int lda = (int)round_up(a_cols, 8), ldb = (int)round_up(b_cols, 8);
    const int64_t asz = (int64_t)batch * a_rows * lda, bsz = (int64_t)batch * b_rows * ldb;
    __nv_bfloat16 *ah = nullptr, *al = nullptr, *bh = nullptr, *bl = nullptr;
    CUtensorMap* maps_d = nullptr;
    MatState* dummy_state = nullptr;
    uint32_t* err = nullptr;
    auto cleanup = [&]() {
        cudaFree(ah); cudaFree(al); cudaFree(bh); cudaFree(bl); cudaFree(maps_d); cudaFree(dummy_state); cudaFree(err);
    };
    if (cudaMalloc(&ah, asz * 2) || cudaMalloc(&al, asz * 2) || cudaMalloc(&bh, bsz * 2) || cudaMalloc(&bl, bsz * 2) ||
        cudaMalloc(&maps_d, 4 * sizeof(CUtensorMap)) || cudaMalloc(&err, 8)) {
        cleanup();
        return fail(ISOLOCO_ERR_OOM, "debug_gemm scratch allocation failed");
    }
    cudaMemsetAsync(ah, 0, asz * 2, st); cudaMemsetAsync(al, 0, asz * 2, st);
    cudaMemsetAsync(bh, 0, bsz * 2, st); cudaMemsetAsync(bl, 0, bsz * 2, st);
    cudaMemsetAsync(err, 0, 8, st);  // err word and the tile counter
    const int f16 = precision > 0 ? 1 : 0;
    k_split_planes<<<1024, 256, 0, st>>>(A, (int64_t)batch * a_rows * a_cols, a_rows, a_cols, lda, ah, al, f16);
    k_split_planes<<<1024, 256, 0, st>>>(B, (int64_t)batch * b_rows * b_cols, b_rows, b_cols, ldb, bh, bl, f16);
    CUtensorMap maps[4];
    const int ra = a_mn ? kRoleMN : kRoleKA, rb = b_mn ? kRoleMN : kRoleKB;
    if (!make_map(&maps[0], ah, a_cols, a_rows, batch, lda, ra) || !make_map(&maps[1], al, a_cols, a_rows, batch, lda, ra) ||
        !make_map(&maps[2], bh, b_cols, b_rows, batch, ldb, rb) || !make_map(&maps[3], bl, b_cols, b_rows, batch, ldb, rb)) {
        cleanup();
        return fail(ISOLOCO_ERR_CUDA, "cuTensorMapEncodeTiled failed");
    }
    cudaMemcpyAsync(maps_d, maps, sizeof(maps), cudaMemcpyHostToDevice, st);
    GemmParams gp;
    memset(&gp, 0, sizeof(gp));
    gp.epi = kEpiF32;
    gp.gate = kGateNone;
    gp.in_f16 = f16;
    gp.a_split = (precision == 0 || precision == 1 || precision == 3) ? 1 : 0;
    gp.b_split = (precision == 0 || precision == 2 || precision == 3) ? 1 : 0;
    gp.err = err;
    GemmGroup& g = gp.g[0];
    g.a_hi = maps_d; g.a_lo = maps_d + 1; g.b_hi = maps_d + 2; g.b_lo = maps_d + 3;
    g.a_mn = a_mn != 0 ? 1 : 0;
    g.b_mn = b_mn != 0 ? 1 : 0;
    g.a_split = gp.a_split;
    g.b_split = gp.b_split;
    set_group_common(g, M, N, K, batch, 1, 0);
    g.cta_begin = 0;
    g.out_f32 = D;
    g.f32_batch_stride = (int64_t)M * N;
    g.f32_split_stride = 0;
    g.ld_f32 = N;
    gp.num_groups = 1;
    gp.total_tiles = batch * g.tiles_m * g.tiles_n;
    gp.counter = reinterpret_cast<int*>(err) + 1;
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    cudaError_t e = launch_gemm(gp, sms, st);
    uint32_t herr = 0;
    if (e == cudaSuccess) e = cudaMemcpyAsync(&herr, err, 4, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    cleanup();
    if (e != cudaSuccess) return fail(ISOLOCO_ERR_CUDA, std::string("debug_gemm: ") + cudaGetErrorString(e));
    if (herr & kErrTimeout) return fail(ISOLOCO_ERR_TIMEOUT, "debug_gemm: device wait timed out");
    return ISOLOCO_OK;
}

}  // extern "C"

// ================================================================== GEMM without allocation
// Scratch of isoloco_debug_gemm_noalloc: one array per device, shared by every call.
//   [0, 4)     error word      \  zeroed by every call before its launches
//   [4, 8)     tile counter    /
//   [256, 768) the four tensor maps (A hi, A lo, B hi, B lo), written by every call
//   [1024, ..) A hi, A lo, B hi, B lo planes, each starting on a 256-byte boundary and
//              fully written by the split kernel before the GEMM reads them
namespace {
constexpr int64_t kNoAllocScratchBytes = int64_t(16) << 20;  // 16 MiB
constexpr int64_t kNoAllocMapsOffset = 256;
constexpr int64_t kNoAllocPlanesOffset = 1024;
constexpr int kNoAllocMaxDevices = 64;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_noalloc_mutex;
unsigned char* g_noalloc_ptr[kNoAllocMaxDevices] = {};

// Address of the scratch array in the current device's context.  In host code the name
// g_noalloc_scratch stands for a host-side shadow, not a device address, so kernels are
// given this looked-up pointer instead.  The first call on a device (that device
// current) does the lookup; later calls reuse it.
int noalloc_scratch(unsigned char** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return fail(ISOLOCO_ERR_CUDA, std::string("cudaGetDevice: ") + cudaGetErrorString(e));
    if (dev < 0 || dev >= kNoAllocMaxDevices) return fail(ISOLOCO_ERR_INVALID, "device ordinal beyond 63");
    std::lock_guard<std::mutex> lock(g_noalloc_mutex);
    if (!g_noalloc_ptr[dev]) {
        void* ptr = nullptr;
        e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
        if (e != cudaSuccess || !ptr)
            return fail(ISOLOCO_ERR_CUDA, std::string("cudaGetSymbolAddress(scratch): ") + cudaGetErrorString(e));
        g_noalloc_ptr[dev] = static_cast<unsigned char*>(ptr);
    }
    *out = g_noalloc_ptr[dev];
    return ISOLOCO_OK;
}
}  // namespace

extern "C" {

int isoloco_debug_gemm_noalloc(int a_mn, int b_mn, int precision, int batch, int M, int N, int K, const float* A,
                               const float* B, float* D, void* stream) {
    if (precision < 0 || precision > 3) return fail(ISOLOCO_ERR_INVALID, "bad debug_gemm_noalloc precision");
    if (batch <= 0 || M <= 0 || N <= 0 || K <= 0 || !A || !B || !D)
        return fail(ISOLOCO_ERR_INVALID, "bad debug_gemm_noalloc arguments");
    const int a_rows = a_mn ? K : M, a_cols = a_mn ? M : K;
    const int b_rows = b_mn ? K : N, b_cols = b_mn ? N : K;
    const int lda = (int)round_up(a_cols, 8), ldb = (int)round_up(b_cols, 8);
    const int64_t asz = (int64_t)batch * a_rows * lda, bsz = (int64_t)batch * b_rows * ldb;
    const int64_t a_bytes = round_up(asz * 2, 256), b_bytes = round_up(bsz * 2, 256);
    const int64_t need = kNoAllocPlanesOffset + 2 * a_bytes + 2 * b_bytes;
    if (need > kNoAllocScratchBytes) {
        char msg[200];
        snprintf(msg, sizeof(msg),
                 "debug_gemm_noalloc: these operands need %lld bytes of scratch; the static scratch holds %lld",
                 (long long)need, (long long)kNoAllocScratchBytes);
        return fail(ISOLOCO_ERR_INVALID, msg);
    }
    unsigned char* base = nullptr;
    int rc = noalloc_scratch(&base);
    if (rc != ISOLOCO_OK) return rc;
    uint32_t* err = reinterpret_cast<uint32_t*>(base);
    CUtensorMap* maps_d = reinterpret_cast<CUtensorMap*>(base + kNoAllocMapsOffset);
    __nv_bfloat16* ah = reinterpret_cast<__nv_bfloat16*>(base + kNoAllocPlanesOffset);
    __nv_bfloat16* al = reinterpret_cast<__nv_bfloat16*>(base + kNoAllocPlanesOffset + a_bytes);
    __nv_bfloat16* bh = reinterpret_cast<__nv_bfloat16*>(base + kNoAllocPlanesOffset + 2 * a_bytes);
    __nv_bfloat16* bl = reinterpret_cast<__nv_bfloat16*>(base + kNoAllocPlanesOffset + 2 * a_bytes + b_bytes);

    cudaStream_t st = static_cast<cudaStream_t>(stream);
    CUtensorMap maps[4];
    const int ra = a_mn ? kRoleMN : kRoleKA, rb = b_mn ? kRoleMN : kRoleKB;
    if (!make_map(&maps[0], ah, a_cols, a_rows, batch, lda, ra) || !make_map(&maps[1], al, a_cols, a_rows, batch, lda, ra) ||
        !make_map(&maps[2], bh, b_cols, b_rows, batch, ldb, rb) || !make_map(&maps[3], bl, b_cols, b_rows, batch, ldb, rb))
        return fail(ISOLOCO_ERR_CUDA, "cuTensorMapEncodeTiled failed");
    CUDA_TRY(cudaMemsetAsync(err, 0, 8, st));  // error word and tile counter
    CUDA_TRY(cudaMemcpyAsync(maps_d, maps, sizeof(maps), cudaMemcpyHostToDevice, st));
    const int f16 = precision > 0 ? 1 : 0;
    k_split_planes<<<1024, 256, 0, st>>>(A, (int64_t)batch * a_rows * a_cols, a_rows, a_cols, lda, ah, al, f16);
    k_split_planes<<<1024, 256, 0, st>>>(B, (int64_t)batch * b_rows * b_cols, b_rows, b_cols, ldb, bh, bl, f16);
    CUDA_TRY(cudaGetLastError());
    GemmParams gp;
    memset(&gp, 0, sizeof(gp));
    gp.epi = kEpiF32;
    gp.gate = kGateNone;
    gp.in_f16 = f16;
    gp.a_split = (precision == 0 || precision == 1 || precision == 3) ? 1 : 0;
    gp.b_split = (precision == 0 || precision == 2 || precision == 3) ? 1 : 0;
    gp.err = err;
    GemmGroup& g = gp.g[0];
    g.a_hi = maps_d; g.a_lo = maps_d + 1; g.b_hi = maps_d + 2; g.b_lo = maps_d + 3;
    g.a_mn = a_mn != 0 ? 1 : 0;
    g.b_mn = b_mn != 0 ? 1 : 0;
    g.a_split = gp.a_split;
    g.b_split = gp.b_split;
    set_group_common(g, M, N, K, batch, 1, 0);
    g.cta_begin = 0;
    g.out_f32 = D;
    g.f32_batch_stride = (int64_t)M * N;
    g.f32_split_stride = 0;
    g.ld_f32 = N;
    gp.num_groups = 1;
    gp.total_tiles = batch * g.tiles_m * g.tiles_n;
    gp.counter = reinterpret_cast<int*>(err) + 1;
    int dev = 0, sms = 148;
    CUDA_TRY(cudaGetDevice(&dev));
    CUDA_TRY(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
    CUDA_TRY(launch_gemm(gp, sms, st));
    uint32_t herr = 0;
    CUDA_TRY(cudaMemcpyAsync(&herr, err, 4, cudaMemcpyDeviceToHost, st));
    CUDA_TRY(cudaStreamSynchronize(st));
    if (herr & kErrTimeout) return fail(ISOLOCO_ERR_TIMEOUT, "debug_gemm_noalloc: device wait timed out");
    return ISOLOCO_OK;
}

}  // extern "C"
