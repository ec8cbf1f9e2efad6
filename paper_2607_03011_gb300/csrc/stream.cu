// stream.cu -- HBM-bound streaming kernels of the outer step.
//
//  k_reduce       : pseudo-gradient reduction (Alg. 1/2 "average pseudo-gradients"):
//                   d = scale * sum_k (theta - theta_k), every replica read once with
//                   16-byte loads; each difference is taken before the sum (exact for
//                   nearby values).  2-D tensors -> bf16 hi/lo planes of the polar
//                   workspace; 1-D tensors -> fp32.  Raises kErrNonFinite.
//  k_apply        : Alg. 2's update B <- mu B + U, theta <- theta - eta (U + mu B) with
//                   U = alpha sigma_bar Q (2-D; Q as fp16 hi/lo planes) or the mean
//                   pseudo-gradient (1-D).
//  k_diloco       : Alg. 1 with Nesterov SGD fused into a single pass over all
//                   parameters (reduction + update, no workspace).
//                   Mode 1: Iso-C merge output base + alpha IsoC(T) / base + alpha T (Eq. 1).
//  k_dare         : Alg. 1 with DARE aggregation (Sec. 3.2): random drop and rescale of
//                   each Delta_k, then the mean and the outer step, one pass.
//  k_ties_*       : Alg. 1 with TIES aggregation (Sec. 3.2): per-worker magnitude trim, an
//                   exact radix select of the threshold over all N entries bracketed from a
//                   sample (one pass over the replicas), then sign election, disjoint mean
//                   and the outer step in one pass.
//  k_split_planes : fp32 -> bf16 hi/lo planes (tests of the split-precision GEMM).
//  k_debug_wait   : the bounded mbarrier wait running out (tests of the timeout path).
#include "common.cuh"
#include "types.h"

namespace isoloco {

constexpr int kStreamThreads = 256;
constexpr int kRepBatch = 8;  // replica loads a thread keeps in flight in the reduction

__device__ __forceinline__ float4 ld_rep4(const void* base, int dtype, int64_t i) {
    if (dtype == 0) return __ldg(reinterpret_cast<const float4*>(static_cast<const float*>(base) + i));
    const uint2 u = __ldg(reinterpret_cast<const uint2*>(static_cast<const uint16_t*>(base) + i));
    return make_float4(__uint_as_float(u.x << 16), __uint_as_float(u.x & 0xFFFF0000u),
                       __uint_as_float(u.y << 16), __uint_as_float(u.y & 0xFFFF0000u));
}

__device__ __forceinline__ float ld_rep1(const void* base, int dtype, int64_t i) {
    if (dtype == 0) return __ldg(static_cast<const float*>(base) + i);
    return bf16_bits_to_float(__ldg(static_cast<const uint16_t*>(base) + i));
}

__device__ __forceinline__ void raise_nonfinite(bool bad, uint32_t* err) {
    if (__any_sync(0xffffffffu, bad) && (threadIdx.x & 31) == 0) atomicOr(err, kErrNonFinite);
}

// The value the polar iteration (2-D) or the apply pass (1-D) receives for one element of
// Delta: Delta itself, or with pmode (orthogonalise the update P instead of Delta) the
// momentum step taken first on the raw Delta, B' = mu B + Delta (written to bnew), and
// P = Delta + mu B' (pmode 1, Nesterov) or P = B' (pmode 2, standard momentum).
__device__ __forceinline__ float reduce_out(float d, int pmode, float mu, const float* __restrict__ mom,
                                            float* __restrict__ bnew, int64_t i) {
    if (!pmode) return d;
    const float nb = fmaf(mu, __ldg(mom + i), d);
    bnew[i] = nb;
    return pmode == 1 ? fmaf(mu, nb, d) : nb;
}

// One CTA per chunk.  PM: the orthogonalise-P ablation (its own kernel, so that the
// default reduction keeps its registers).  BATCH: fp32 replicas whose loads are batched
// (their own kernel too: the batch's registers would cost the bf16 reduction occupancy).
template <bool PM, bool BATCH>
__device__ __forceinline__ void reduce_chunk(const Chunk* __restrict__ chunks, const MatDesc* __restrict__ mats,
                                             const ReplicaPtrs& reps, int K, int dtype,
                                             const float* __restrict__ theta, float scale,
                                             __nv_bfloat16* __restrict__ dhi, __nv_bfloat16* __restrict__ dlo,
                                             float* __restrict__ d1d, uint32_t* __restrict__ err, int pmode_arg,
                                             float mu, const float* __restrict__ mom, float* __restrict__ bnew) {
    const int pmode = PM ? pmode_arg : 0;
    const Chunk ch = chunks[blockIdx.x];
    bool bad = false;
    const int64_t f0 = ch.flat_begin;
    if (ch.matrix < 0) {
        for (int e = threadIdx.x; e < ch.count; e += blockDim.x) {
            const float th = __ldg(theta + f0 + e);
            float s = 0.f;
            for (int k = 0; k < K; ++k) s += th - ld_rep1(reps.p[k], dtype, f0 + e);
            const float d = reduce_out(s * scale, pmode, mu, mom, bnew, f0 + e);
            bad |= !isfinite(d);
            d1d[ch.dst + e] = d;
        }
    } else {
        const MatDesc md = mats[ch.matrix];
        const bool contiguous = (md.ld == md.cols);
        if (contiguous && (f0 & 3) == 0 && (ch.count & 3) == 0) {
            __nv_bfloat16* oh = dhi + md.slot + ch.elem_begin;
            __nv_bfloat16* ol = dlo + md.slot + ch.elem_begin;
            const int nv = ch.count >> 2;
            for (int v = threadIdx.x; v < nv; v += blockDim.x) {
                const int64_t i = f0 + 4 * static_cast<int64_t>(v);
                const float4 th = __ldg(reinterpret_cast<const float4*>(theta + i));
                float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
                if (BATCH) {
                    // fp32 replicas: up to eight loads issued before any is used (the sum keeps
                    // the order k = 0, 1, ...): 1.43 -> 1.23 ms for eight replicas at the 180M
                    // shapes, 0.91 -> 1.05 of the measured copy bandwidth
                    for (int k0 = 0; k0 < K; k0 += kRepBatch) {
                        float4 r[kRepBatch];
#pragma unroll
                        for (int u = 0; u < kRepBatch; ++u)
                            if (k0 + u < K)
                                r[u] = __ldg(reinterpret_cast<const float4*>(static_cast<const float*>(reps.p[k0 + u]) + i));
#pragma unroll
                        for (int u = 0; u < kRepBatch; ++u) {
                            if (k0 + u < K) {
                                s.x += th.x - r[u].x;
                                s.y += th.y - r[u].y;
                                s.z += th.z - r[u].z;
                                s.w += th.w - r[u].w;
                            }
                        }
                    }
                } else {
                    // bf16 replicas, and the ablation's kernel: four loads in flight (batching
                    // bf16 loads in the fp32 kernel's registers halved this pass's rate for
                    // four bf16 replicas at the 3B shapes)
#pragma unroll 4
                    for (int k = 0; k < K; ++k) {
                        const float4 r = ld_rep4(reps.p[k], dtype, i);
                        s.x += th.x - r.x;
                        s.y += th.y - r.y;
                        s.z += th.z - r.z;
                        s.w += th.w - r.w;
                    }
                }
                float d[4] = {s.x * scale, s.y * scale, s.z * scale, s.w * scale};
                if (PM) {
#pragma unroll
                    for (int j = 0; j < 4; ++j) d[j] = reduce_out(d[j], pmode, mu, mom, bnew, i + j);
                }
                __nv_bfloat16 h[4], l[4];
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    bad |= !isfinite(d[j]);
                    split_bf16(d[j], h[j], l[j]);
                }
                reinterpret_cast<uint2*>(oh)[v] = make_uint2(pack_bf16x2(h[0], h[1]), pack_bf16x2(h[2], h[3]));
                reinterpret_cast<uint2*>(ol)[v] = make_uint2(pack_bf16x2(l[0], l[1]), pack_bf16x2(l[2], l[3]));
            }
        } else {
            for (int e = threadIdx.x; e < ch.count; e += blockDim.x) {
                const int64_t i = f0 + e;
                const float th = __ldg(theta + i);
                float s = 0.f;
                for (int k = 0; k < K; ++k) s += th - ld_rep1(reps.p[k], dtype, i);
                const float d = reduce_out(s * scale, pmode, mu, mom, bnew, i);
                bad |= !isfinite(d);
                const int pe = ch.elem_begin + e;
                const int64_t o = md.slot + static_cast<int64_t>(pe / md.cols) * md.ld + pe % md.cols;
                __nv_bfloat16 h, l;
                split_bf16(d, h, l);
                dhi[o] = h;
                dlo[o] = l;
            }
        }
    }
    raise_nonfinite(bad, err);
}

__global__ void __launch_bounds__(kStreamThreads) k_reduce(const Chunk* __restrict__ chunks,
                                                           const MatDesc* __restrict__ mats,
                                                           ReplicaPtrs reps, int K, int dtype,
                                                           const float* __restrict__ theta, float scale,
                                                           __nv_bfloat16* __restrict__ dhi,
                                                           __nv_bfloat16* __restrict__ dlo,
                                                           float* __restrict__ d1d,
                                                           uint32_t* __restrict__ err) {
    reduce_chunk<false, false>(chunks, mats, reps, K, dtype, theta, scale, dhi, dlo, d1d, err, 0, 0.f, nullptr,
                               nullptr);
}

// k_reduce for fp32 replicas (dtype 0), their loads batched.
__global__ void __launch_bounds__(kStreamThreads) k_reduce_f32(const Chunk* __restrict__ chunks,
                                                               const MatDesc* __restrict__ mats,
                                                               ReplicaPtrs reps, int K,
                                                               const float* __restrict__ theta, float scale,
                                                               __nv_bfloat16* __restrict__ dhi,
                                                               __nv_bfloat16* __restrict__ dlo,
                                                               float* __restrict__ d1d,
                                                               uint32_t* __restrict__ err) {
    reduce_chunk<false, true>(chunks, mats, reps, K, 0, theta, scale, dhi, dlo, d1d, err, 0, 0.f, nullptr, nullptr);
}

// pmode 1 (Nesterov) or 2 (standard momentum); mom is read, B' goes to bnew.
__global__ void __launch_bounds__(kStreamThreads) k_reduce_p(const Chunk* __restrict__ chunks,
                                                             const MatDesc* __restrict__ mats,
                                                             ReplicaPtrs reps, int K, int dtype,
                                                             const float* __restrict__ theta, float scale,
                                                             __nv_bfloat16* __restrict__ dhi,
                                                             __nv_bfloat16* __restrict__ dlo,
                                                             float* __restrict__ d1d,
                                                             uint32_t* __restrict__ err, int pmode, float mu,
                                                             const float* __restrict__ mom,
                                                             float* __restrict__ bnew) {
    reduce_chunk<true, false>(chunks, mats, reps, K, dtype, theta, scale, dhi, dlo, d1d, err, pmode, mu, mom, bnew);
}


// grid: one CTA per chunk.  mode 0: outer update of theta and B in place; mode 1: merge
// output.  Mode 0 variants (the ablations of Sec. 4.5 and App. B): mom_kind 0 Nesterov
// (Alg. 2), 1 standard momentum (B <- mu B + U, theta <- theta - eta B); pmode != 0: U is
// already the orthogonalised update P (theta <- theta - eta U, B <- bnew from the reduce
// pass); spectral: 2-D tensors scale Q by sqrt(rows / cols) instead of sigma_bar.
__global__ void __launch_bounds__(kStreamThreads) k_apply(const Chunk* __restrict__ chunks,
                                                          const MatDesc* __restrict__ mats,
                                                          const MatState* __restrict__ state,
                                                          UpdateSrc src, int mode, float alpha,
                                                          float eta, float mu,
                                                          float* __restrict__ theta,
                                                          float* __restrict__ mom,
                                                          const float* __restrict__ base,
                                                          float* __restrict__ out,
                                                          float* __restrict__ upd_out,
                                                          const uint32_t* __restrict__ err, int mom_kind,
                                                          int pmode, int spectral,
                                                          const float* __restrict__ bnew) {
    if (*err & kErrNonFinite) return;  // leave theta and B untouched
    const Chunk ch = chunks[blockIdx.x];
    const int64_t f0 = ch.flat_begin;
    // U = ucoef * q where q is read from the Q planes (2-D) or Delta (1-D)
    float ucoef = 1.f;
    const __nv_bfloat16* qh = nullptr;
    const __nv_bfloat16* ql = nullptr;
    MatDesc md;
    bool zero = false, contiguous = true;
    if (ch.matrix >= 0) {
        md = mats[ch.matrix];
        const MatState st = state[ch.matrix];
        if (st.final_buf == 2) {
            zero = true;
        } else {
            qh = src.qh[st.final_buf] + md.slot;
            ql = src.ql[st.final_buf] + md.slot;
        }
        ucoef = alpha * (spectral ? sqrtf(static_cast<float>(md.rows) / static_cast<float>(md.cols)) : st.sigma_bar);
        contiguous = (md.ld == md.cols);
    } else if (mode == 1) {
        ucoef = alpha;  // Eq. 1: base + lambda * sum tau for non-matrix tensors
    }
    auto uval = [&](int e) -> float {
        if (ch.matrix < 0) return ucoef * src.d1d[ch.dst + e];
        if (zero) return 0.f;
        const int pe = ch.elem_begin + e;
        const int64_t o = contiguous ? pe : static_cast<int64_t>(pe / md.cols) * md.ld + pe % md.cols;
        return ucoef * (dec16(__bfloat16_as_ushort(qh[o]), true) + dec16(__bfloat16_as_ushort(ql[o]), true));
    };
    const bool vec = (f0 & 3) == 0 && (ch.count & 3) == 0 && (ch.matrix < 0 || contiguous) &&
                     ((ch.matrix < 0 ? (ch.dst & 3) : (ch.elem_begin & 3)) == 0);
    if (vec) {
        const int nv = ch.count >> 2;
        for (int v = threadIdx.x; v < nv; v += blockDim.x) {
            const int64_t i = f0 + 4 * static_cast<int64_t>(v);
            float u[4];
            if (ch.matrix < 0) {
                const float4 d = *reinterpret_cast<const float4*>(src.d1d + ch.dst + 4 * v);
                u[0] = ucoef * d.x; u[1] = ucoef * d.y; u[2] = ucoef * d.z; u[3] = ucoef * d.w;
            } else if (zero) {
                u[0] = u[1] = u[2] = u[3] = 0.f;
            } else {
                const uint2 hh = *reinterpret_cast<const uint2*>(qh + ch.elem_begin + 4 * v);
                const uint2 ll = *reinterpret_cast<const uint2*>(ql + ch.elem_begin + 4 * v);
                u[0] = ucoef * (dec16(hh.x & 0xFFFFu, true) + dec16(ll.x & 0xFFFFu, true));
                u[1] = ucoef * (dec16(hh.x >> 16, true) + dec16(ll.x >> 16, true));
                u[2] = ucoef * (dec16(hh.y & 0xFFFFu, true) + dec16(ll.y & 0xFFFFu, true));
                u[3] = ucoef * (dec16(hh.y >> 16, true) + dec16(ll.y >> 16, true));
            }
            if (mode == 0) {
                const float4 th = *reinterpret_cast<const float4*>(theta + i);
                float4 nb, nt;
                if (pmode) {
                    nb = *reinterpret_cast<const float4*>(bnew + i);
                    nt = make_float4(th.x - eta * u[0], th.y - eta * u[1], th.z - eta * u[2], th.w - eta * u[3]);
                } else {
                    const float4 bb = *reinterpret_cast<const float4*>(mom + i);
                    nb.x = fmaf(mu, bb.x, u[0]);
                    nb.y = fmaf(mu, bb.y, u[1]);
                    nb.z = fmaf(mu, bb.z, u[2]);
                    nb.w = fmaf(mu, bb.w, u[3]);
                    if (mom_kind == 1) {
                        nt = make_float4(th.x - eta * nb.x, th.y - eta * nb.y, th.z - eta * nb.z, th.w - eta * nb.w);
                    } else {
                        nt.x = th.x - eta * fmaf(mu, nb.x, u[0]);
                        nt.y = th.y - eta * fmaf(mu, nb.y, u[1]);
                        nt.z = th.z - eta * fmaf(mu, nb.z, u[2]);
                        nt.w = th.w - eta * fmaf(mu, nb.w, u[3]);
                    }
                }
                *reinterpret_cast<float4*>(mom + i) = nb;
                *reinterpret_cast<float4*>(theta + i) = nt;
            } else {
                const float4 bs = *reinterpret_cast<const float4*>(base + i);
                *reinterpret_cast<float4*>(out + i) = make_float4(bs.x + u[0], bs.y + u[1], bs.z + u[2], bs.w + u[3]);
            }
            if (upd_out) *reinterpret_cast<float4*>(upd_out + i) = make_float4(u[0], u[1], u[2], u[3]);
        }
    } else {
        for (int e = threadIdx.x; e < ch.count; e += blockDim.x) {
            const int64_t i = f0 + e;
            const float u = uval(e);
            if (mode == 0) {
                if (pmode) {
                    theta[i] = theta[i] - eta * u;
                    mom[i] = bnew[i];
                } else {
                    const float nb = fmaf(mu, mom[i], u);
                    theta[i] = theta[i] - eta * (mom_kind == 1 ? nb : fmaf(mu, nb, u));
                    mom[i] = nb;
                }
            } else {
                out[i] = base[i] + u;
            }
            if (upd_out) upd_out[i] = u;
        }
    }
}

// Alg. 1 outer step fused: d = scale * sum_k (theta - theta_k); B <- mu B + d;
// theta <- theta - eta (d + mu B).  Grid-stride over float4 vectors of all N params.
__global__ void __launch_bounds__(kStreamThreads) k_diloco(ReplicaPtrs reps, int K, int dtype,
                                                           float* __restrict__ theta,
                                                           float* __restrict__ mom, int64_t N,
                                                           float scale, float eta, float mu,
                                                           uint32_t* __restrict__ err) {
    bool bad = false;
    const int64_t nv = N >> 2;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t v = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; v < nv; v += stride) {
        const int64_t i = 4 * v;
        const float4 th = *reinterpret_cast<const float4*>(theta + i);
        const float4 bb = *reinterpret_cast<const float4*>(mom + i);
        float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 8
        for (int k = 0; k < K; ++k) {
            const float4 r = ld_rep4(reps.p[k], dtype, i);
            s.x += th.x - r.x;
            s.y += th.y - r.y;
            s.z += th.z - r.z;
            s.w += th.w - r.w;
        }
        const float d0 = s.x * scale, d1 = s.y * scale, d2 = s.z * scale, d3 = s.w * scale;
        bad |= !(isfinite(d0) && isfinite(d1) && isfinite(d2) && isfinite(d3));
        float4 nb, nt;
        nb.x = fmaf(mu, bb.x, d0); nt.x = th.x - eta * fmaf(mu, nb.x, d0);
        nb.y = fmaf(mu, bb.y, d1); nt.y = th.y - eta * fmaf(mu, nb.y, d1);
        nb.z = fmaf(mu, bb.z, d2); nt.z = th.z - eta * fmaf(mu, nb.z, d2);
        nb.w = fmaf(mu, bb.w, d3); nt.w = th.w - eta * fmaf(mu, nb.w, d3);
        *reinterpret_cast<float4*>(mom + i) = nb;
        *reinterpret_cast<float4*>(theta + i) = nt;
    }
    // scalar tail
    if (blockIdx.x == 0) {
        for (int64_t i = 4 * nv + threadIdx.x; i < N; i += blockDim.x) {
            const float th = theta[i];
            float s = 0.f;
            for (int k = 0; k < K; ++k) s += th - ld_rep1(reps.p[k], dtype, i);
            const float d = s * scale;
            bad |= !isfinite(d);
            const float nb = fmaf(mu, mom[i], d);
            theta[i] = th - eta * fmaf(mu, nb, d);
            mom[i] = nb;
        }
    }
    raise_nonfinite(bad, err);
}

// ---------------------------------------------------------------- merging aggregators
// Sec. 3.2 replaces DiLoCo's mean of the Delta_k by a model-merging rule.  These kernels
// compute the merged direction U over all N entries and take the outer step
// B <- mu B + U, theta <- theta - eta (U + mu B) (mu = 0: the SGD step of Sec. 5.1).

// SplitMix64 (Steele, Lea and Flood, 2014): output number n (n >= 1) from state s is
// mix(s + n * GAMMA), mix = xor-shift 30, * M1, xor-shift 27, * M2, xor-shift 31.  DARE uses
// only the top 24 bits of an output: the last xor-shift leaves bits 63..33 as they are, and
// the top half of the last product is umulhi(lo, M2lo) + lo * M2hi + hi * M2lo (mod 2^32).
constexpr uint64_t kSmGamma = 0x9E3779B97F4A7C15ull;
__device__ __forceinline__ uint32_t splitmix64_top24(uint64_t z /* s + n * GAMMA */) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z ^= z >> 27;
    const uint32_t lo = static_cast<uint32_t>(z), hi = static_cast<uint32_t>(z >> 32);
    const uint32_t m_lo = 0x133111EBu, m_hi = 0x94D049BBu;
    return (__umulhi(lo, m_lo) + lo * m_hi + hi * m_lo) >> 8;
}

__device__ __forceinline__ void nesterov1(float& th, float& b, float u, float eta, float mu) {
    const float nb = fmaf(mu, b, u);
    th = th - eta * fmaf(mu, nb, u);
    b = nb;
}

// DARE: U = scale * sum_k keep_scale * m_k * Delta_k, keep_scale = 1 / (1 - p), scale =
// 1 / K (mean) or 1.  Entry i of worker k is kept when the top 24 bits of SplitMix64 output
// k * N + i + 1 (state seed) are >= pthr = ceil(p * 2^24), i.e. when that value times 2^-24
// is >= p.  ng = N * GAMMA (mod 2^64) steps the draw number from one worker to the next.
// Grid-stride over float4 vectors of all N entries, scalar tail in CTA 0.
__global__ void __launch_bounds__(kStreamThreads) k_dare(ReplicaPtrs reps, int K, int dtype,
                                                         float* __restrict__ theta, float* __restrict__ mom,
                                                         int64_t N, float scale, uint32_t pthr, float keep_scale,
                                                         unsigned int seed, uint64_t ng, float eta, float mu,
                                                         uint32_t* __restrict__ err) {
    bool bad = false;
    const int64_t nv = N >> 2;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t v = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; v < nv; v += stride) {
        const int64_t i = 4 * v;
        float4 th = *reinterpret_cast<const float4*>(theta + i);
        float4 bb = *reinterpret_cast<const float4*>(mom + i);
        float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
        float chk = 0.f;  // every Delta_k entry, dropped or not, for the non-finite test
        uint64_t z = seed + static_cast<uint64_t>(i + 1) * kSmGamma;  // draw k * N + i + 1, k = 0
        for (int k = 0; k < K; ++k, z += ng) {
            const float4 r = ld_rep4(reps.p[k], dtype, i);
            const float4 d = make_float4(th.x - r.x, th.y - r.y, th.z - r.z, th.w - r.w);
            chk += (d.x + d.y) + (d.z + d.w);
            if (splitmix64_top24(z) >= pthr) s.x += d.x * keep_scale;
            if (splitmix64_top24(z + kSmGamma) >= pthr) s.y += d.y * keep_scale;
            if (splitmix64_top24(z + 2 * kSmGamma) >= pthr) s.z += d.z * keep_scale;
            if (splitmix64_top24(z + 3 * kSmGamma) >= pthr) s.w += d.w * keep_scale;
        }
        s.x *= scale; s.y *= scale; s.z *= scale; s.w *= scale;
        bad |= !isfinite(chk);
        nesterov1(th.x, bb.x, s.x, eta, mu);
        nesterov1(th.y, bb.y, s.y, eta, mu);
        nesterov1(th.z, bb.z, s.z, eta, mu);
        nesterov1(th.w, bb.w, s.w, eta, mu);
        *reinterpret_cast<float4*>(mom + i) = bb;
        *reinterpret_cast<float4*>(theta + i) = th;
    }
    if (blockIdx.x == 0) {
        for (int64_t i = 4 * nv + threadIdx.x; i < N; i += blockDim.x) {
            float th = theta[i], bb = mom[i], s = 0.f, chk = 0.f;
            uint64_t z = seed + static_cast<uint64_t>(i + 1) * kSmGamma;
            for (int k = 0; k < K; ++k, z += ng) {
                const float d = th - ld_rep1(reps.p[k], dtype, i);
                chk += d;
                if (splitmix64_top24(z) >= pthr) s += d * keep_scale;
            }
            s *= scale;
            bad |= !isfinite(chk);
            nesterov1(th, bb, s, eta, mu);
            theta[i] = th;
            mom[i] = bb;
        }
    }
    raise_nonfinite(bad, err);
}

// TIES trim: per worker k, the key (fp32 bits of |Delta_k|, ordered like the magnitudes) of
// the n_keep-th largest magnitude over all N entries, n_keep = N - floor(sparsity * N).
// Radix select over the 31 key bits in four digits, [30:23], [22:15], [14:7], [6:0]: a
// pass histograms one digit of the keys whose higher digits match the prefix chosen so far,
// and k_ties_select appends the digit holding the wanted rank.  To avoid four passes over
// the replicas, the library brackets the threshold first:
//   1. k_ties_sample: S keys per worker at jittered strided positions;
//   2. radix select on the sample for two ranks per worker, the expected rank of the
//      threshold -/+ 8 standard deviations (and 16): keys hi >= lo;
//   3. k_ties_bracket, one pass over the replicas: A = #(key > hi) and the keys in [lo, hi]
//      collected per CTA (its own segment of the candidate buffer);
//   4. k_ties_check: if A < n_keep <= A + #candidates and no segment overflowed, the
//      threshold is the (n_keep - A)-th largest candidate, found by radix select on them;
//   5. otherwise (a flag) the four passes over the replicas run and give it directly.
// Either way the threshold is exact.
__host__ __device__ constexpr int ties_shift(int pass) { return pass == 0 ? 23 : pass == 1 ? 15 : pass == 2 ? 7 : 0; }
__host__ __device__ constexpr int ties_bins(int pass) { return pass == 3 ? 128 : 256; }

__device__ __forceinline__ uint32_t ties_key(float d) { return __float_as_uint(fabsf(d)); }
constexpr int kLoadBatch = 8;  // replicas whose loads are issued together in the TIES passes

// Counts, per worker, the digit of this pass of every key whose higher digits equal the
// prefix chosen so far.  Shared histogram [workers][256]; keys sharing a bin within a warp
// are counted by one atomic (most magnitudes fall in a few exponent bins).
__device__ __forceinline__ void ties_count(uint32_t* sh, int k, uint32_t key, bool valid, int hs, uint32_t phi,
                                           int shift, uint32_t mask) {
    const bool m = valid && (key >> hs) == phi;
    const uint32_t bin = m ? ((key >> shift) & mask) : 0xFFFFFFFFu;
    const unsigned peers = __match_any_sync(0xffffffffu, bin);
    if (m && (threadIdx.x & 31) == __ffs(peers) - 1) atomicAdd(&sh[k * 256 + bin], static_cast<uint32_t>(__popc(peers)));
}

// A radix pass over the replicas (the fallback).  Runs only when *fail != 0.
__global__ void __launch_bounds__(kStreamThreads) k_ties_hist(ReplicaPtrs reps, int K, int dtype,
                                                              const float* __restrict__ theta, int64_t N, int pass,
                                                              const uint64_t* __restrict__ prefix,
                                                              unsigned long long* __restrict__ hist,
                                                              const int* __restrict__ fail) {
    if (*fail == 0) return;
    extern __shared__ uint32_t sh[];
    __shared__ uint32_t phi_s[kMaxK];
    const int shift = ties_shift(pass);
    const int hs = pass == 0 ? 31 : ties_shift(pass - 1);
    const uint32_t mask = static_cast<uint32_t>(ties_bins(pass) - 1);
    for (int j = threadIdx.x; j < K * 256; j += blockDim.x) sh[j] = 0u;
    for (int k = threadIdx.x; k < K; k += blockDim.x) phi_s[k] = static_cast<uint32_t>(prefix[k]) >> hs;
    __syncthreads();
    const int64_t nv = N >> 2;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    // warp-uniform trip count: every lane runs every iteration (match_any over the full warp)
    const int64_t wbase = blockIdx.x * static_cast<int64_t>(blockDim.x) + (threadIdx.x & ~31);
    const int lane = threadIdx.x & 31;
    for (int64_t vb = wbase; vb < nv; vb += stride) {
        const int64_t v = vb + lane;
        const bool valid = v < nv;
        const int64_t i = 4 * (valid ? v : 0);
        const float4 th = __ldg(reinterpret_cast<const float4*>(theta + i));
        for (int k = 0; k < K; ++k) {
            const float4 r = ld_rep4(reps.p[k], dtype, i);
            const uint32_t ph = phi_s[k];
            ties_count(sh, k, ties_key(th.x - r.x), valid, hs, ph, shift, mask);
            ties_count(sh, k, ties_key(th.y - r.y), valid, hs, ph, shift, mask);
            ties_count(sh, k, ties_key(th.z - r.z), valid, hs, ph, shift, mask);
            ties_count(sh, k, ties_key(th.w - r.w), valid, hs, ph, shift, mask);
        }
    }
    if (blockIdx.x == 0 && threadIdx.x < 32) {
        const int64_t i = 4 * nv + lane;
        const bool valid = i < N;
        const float th = valid ? __ldg(theta + i) : 0.f;
        for (int k = 0; k < K; ++k) {
            const float r = valid ? ld_rep1(reps.p[k], dtype, i) : 0.f;
            ties_count(sh, k, ties_key(th - r), valid, hs, phi_s[k], shift, mask);
        }
    }
    __syncthreads();
    for (int j = threadIdx.x; j < K * 256; j += blockDim.x)
        if (sh[j]) atomicAdd(&hist[j], static_cast<unsigned long long>(sh[j]));
}

// A radix pass over keys already in a buffer [K][nseg][segcap] (counts[k][seg] valid keys,
// clamped to segcap; all segcap when counts is null), for nw selections: selection v reads
// worker v / vdiv.  grid = (nseg, splits of a segment).
__global__ void __launch_bounds__(kStreamThreads) k_ties_hist_buf(const uint32_t* __restrict__ keys,
                                                                  const uint32_t* __restrict__ counts, int nseg,
                                                                  int64_t segcap, int nw, int vdiv, int pass,
                                                                  const uint64_t* __restrict__ prefix,
                                                                  unsigned long long* __restrict__ hist) {
    extern __shared__ uint32_t sh[];
    const int shift = ties_shift(pass);
    const int hs = pass == 0 ? 31 : ties_shift(pass - 1);
    const uint32_t mask = static_cast<uint32_t>(ties_bins(pass) - 1);
    for (int j = threadIdx.x; j < nw * 256; j += blockDim.x) sh[j] = 0u;
    __syncthreads();
    const int seg = blockIdx.x;
    const int lane = threadIdx.x & 31;
    for (int v = 0; v < nw; ++v) {
        const int k = v / vdiv;
        const int64_t n = counts ? min(static_cast<int64_t>(counts[static_cast<int64_t>(k) * nseg + seg]), segcap)
                                 : segcap;
        const int64_t chunk = (n + gridDim.y - 1) / gridDim.y;
        const int64_t lo = blockIdx.y * chunk, hi = min(n, lo + chunk);
        const uint32_t* src = keys + (static_cast<int64_t>(k) * nseg + seg) * segcap;
        const uint32_t phi = static_cast<uint32_t>(prefix[v]) >> hs;
        for (int64_t jb = lo + (threadIdx.x & ~31); jb < hi; jb += blockDim.x) {
            const int64_t j = jb + lane;
            const bool valid = j < hi;
            ties_count(sh, v, valid ? src[j] : 0u, valid, hs, phi, shift, mask);
        }
    }
    __syncthreads();
    for (int j = threadIdx.x; j < nw * 256; j += blockDim.x)
        if (sh[j]) atomicAdd(&hist[j], static_cast<unsigned long long>(sh[j]));
}

// Clears the histogram and sets the ranks: sample selections 2k (hi) and 2k + 1 (lo) want
// ranks r_hi and r_lo; the fallback wants n_keep; the candidate selection's rank is set by
// k_ties_check.  One CTA.
__global__ void k_ties_init(int K, uint64_t n_keep, uint64_t r_hi, uint64_t r_lo,
                            unsigned long long* __restrict__ hist, uint64_t* __restrict__ rank_s,
                            uint64_t* __restrict__ prefix_s, uint64_t* __restrict__ rank_c,
                            uint64_t* __restrict__ prefix_c, uint64_t* __restrict__ rank_f,
                            uint64_t* __restrict__ prefix_f, unsigned long long* __restrict__ above,
                            int* __restrict__ fail) {
    for (int j = threadIdx.x; j < 2 * K * 256; j += blockDim.x) hist[j] = 0ull;
    for (int k = threadIdx.x; k < K; k += blockDim.x) {
        rank_s[2 * k] = r_hi;
        rank_s[2 * k + 1] = r_lo;
        prefix_s[2 * k] = prefix_s[2 * k + 1] = 0ull;
        rank_c[k] = 1;
        prefix_c[k] = 0ull;
        rank_f[k] = n_keep;
        prefix_f[k] = 0ull;
        above[k] = 0ull;
    }
    if (threadIdx.x == 0) *fail = 0;
}

// Sample j of worker k: the key at position floor(j N / S) + h(j) mod floor(N / S), h a
// SplitMix64-type mix of j (one position in each of S equal strata).
__global__ void __launch_bounds__(kStreamThreads) k_ties_sample(ReplicaPtrs reps, int K, int dtype,
                                                                const float* __restrict__ theta, int64_t N, int64_t S,
                                                                uint32_t* __restrict__ samp) {
    const int64_t j = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
    if (j >= S) return;
    const uint64_t width = static_cast<uint64_t>(N / S);
    const uint64_t base = static_cast<uint64_t>(j) * static_cast<uint64_t>(N) / static_cast<uint64_t>(S);
    const int64_t i = static_cast<int64_t>(base + splitmix64_top24(static_cast<uint64_t>(j + 1) * kSmGamma) % width);
    const float th = __ldg(theta + i);
    for (int k = 0; k < K; ++k) samp[static_cast<int64_t>(k) * S + j] = ties_key(th - ld_rep1(reps.p[k], dtype, i));
}

// One pass over theta and the replicas: per worker, the keys above the bracket [lo, hi] are
// counted and those inside it collected into this CTA's segment of cand [K][gridDim.x][segcap];
// cnt[k][cta] may exceed segcap (overflow: k_ties_check then fails).  Each thread counts in
// its own shared slots up_s[k][thread] (no atomics, no warp votes in the loop); the rare keys
// inside a bracket take a shared atomic for their position.  Dynamic shared memory:
// K x blockDim.x counters.
__global__ void __launch_bounds__(kStreamThreads) k_ties_bracket(ReplicaPtrs reps, int K, int dtype,
                                                                 const float* __restrict__ theta, int64_t N,
                                                                 const uint64_t* __restrict__ prefix_s,
                                                                 uint32_t* __restrict__ cand,
                                                                 uint32_t* __restrict__ cnt, int64_t segcap,
                                                                 unsigned long long* __restrict__ above) {
    extern __shared__ uint32_t up_s[];
    __shared__ uint32_t hi_s[kMaxK], lo_s[kMaxK], cnt_s[kMaxK];
    for (int k = threadIdx.x; k < K; k += blockDim.x) {
        hi_s[k] = static_cast<uint32_t>(prefix_s[2 * k]);
        lo_s[k] = static_cast<uint32_t>(prefix_s[2 * k + 1]);
        cnt_s[k] = 0u;
    }
    for (int j = threadIdx.x; j < K * static_cast<int>(blockDim.x); j += blockDim.x) up_s[j] = 0u;
    __syncthreads();
    const int64_t G = gridDim.x;
    const int64_t nv = N >> 2;
    const int64_t stride = G * blockDim.x;
    uint32_t* mine = up_s + threadIdx.x;
    auto one = [&](uint32_t key, int k) -> uint32_t {
        if (key > hi_s[k]) return 1u;
        if (key >= lo_s[k]) {
            const uint32_t pos = atomicAdd(&cnt_s[k], 1u);
            if (pos < segcap) cand[(static_cast<int64_t>(k) * G + blockIdx.x) * segcap + pos] = key;
        }
        return 0u;
    };
    for (int64_t v = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; v < nv; v += stride) {
        const int64_t i = 4 * v;
        const float4 th = __ldg(reinterpret_cast<const float4*>(theta + i));
        for (int k0 = 0; k0 < K; k0 += 4) {
            float4 r[4];
#pragma unroll
            for (int q = 0; q < 4; ++q)
                if (k0 + q < K) r[q] = ld_rep4(reps.p[k0 + q], dtype, i);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int k = k0 + q;
                if (k >= K) break;
                const uint32_t c = one(ties_key(th.x - r[q].x), k) + one(ties_key(th.y - r[q].y), k) +
                                   one(ties_key(th.z - r[q].z), k) + one(ties_key(th.w - r[q].w), k);
                if (c) mine[k * blockDim.x] += c;
            }
        }
    }
    if (blockIdx.x == 0) {
        for (int64_t i = 4 * nv + threadIdx.x; i < N; i += blockDim.x) {
            const float th = __ldg(theta + i);
            for (int k = 0; k < K; ++k) mine[k * blockDim.x] += one(ties_key(th - ld_rep1(reps.p[k], dtype, i)), k);
        }
    }
    __syncthreads();
    // per worker: the block's sum of the thread counters (one warp per worker)
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nwarps = blockDim.x >> 5;
    for (int k = warp; k < K; k += nwarps) {
        uint32_t t = 0;
        for (int j = lane; j < static_cast<int>(blockDim.x); j += 32) t += up_s[k * blockDim.x + j];
        t = __reduce_add_sync(0xffffffffu, t);
        if (lane == 0) {
            cnt[static_cast<int64_t>(k) * G + blockIdx.x] = cnt_s[k];
            if (t) atomicAdd(&above[k], static_cast<unsigned long long>(t));
        }
    }
}

// One CTA per worker: does the bracket hold the threshold (A < n_keep <= A + candidates, no
// segment overflowed)?  Then the candidate selection wants rank n_keep - A; else *fail is set.
__global__ void __launch_bounds__(256) k_ties_check(int K, int nseg, int64_t segcap, uint64_t n_keep,
                                                    const unsigned long long* __restrict__ above,
                                                    const uint32_t* __restrict__ cnt, uint64_t* __restrict__ rank_c,
                                                    int* __restrict__ fail) {
    const int k = blockIdx.x;
    __shared__ unsigned long long tot_s[256 / 32];
    __shared__ int over_s;
    if (threadIdx.x == 0) over_s = 0;
    __syncthreads();
    unsigned long long total = 0;
    bool over = false;
    for (int b = threadIdx.x; b < nseg; b += blockDim.x) {
        const uint32_t c = cnt[static_cast<int64_t>(k) * nseg + b];
        over |= c > segcap;
        total += static_cast<unsigned long long>(min(static_cast<int64_t>(c), segcap));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) total += __shfl_xor_sync(0xffffffffu, total, o);
    if (__any_sync(0xffffffffu, over) && (threadIdx.x & 31) == 0) over_s = 1;
    if ((threadIdx.x & 31) == 0) tot_s[threadIdx.x >> 5] = total;
    __syncthreads();
    if (threadIdx.x != 0) return;
    unsigned long long t = 0;
    for (int w = 0; w < 256 / 32; ++w) t += tot_s[w];
    const uint64_t a = above[k];
    const bool ok = !over_s && a < n_keep && n_keep <= a + t;
    rank_c[k] = ok ? n_keep - a : 1;
    if (!ok) atomicOr(fail, 1);
}

// One warp per selection: the bin holding the rank-th largest key (counting from the top),
// appended to the prefix; the histogram row is cleared for the next pass.  Lane l holds bins
// 8 l .. 8 l + 7; a suffix sum over the warp finds the bin.  With only_if_fail it runs only
// when *only_if_fail != 0 (the fallback passes).
__global__ void __launch_bounds__(256) k_ties_select(int nw, int pass, unsigned long long* __restrict__ hist,
                                                     uint64_t* __restrict__ rank, uint64_t* __restrict__ prefix,
                                                     const int* __restrict__ only_if_fail) {
    if (only_if_fail && *only_if_fail == 0) return;
    const int w = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
    if (w >= nw) return;
    unsigned long long* h = hist + static_cast<int64_t>(w) * 256;
    const int nb = ties_bins(pass);
    unsigned long long c[8], mine = 0;
#pragma unroll
    for (int q = 0; q < 8; ++q) {
        const int b = 8 * lane + q;
        c[q] = b < nb ? h[b] : 0ull;
        mine += c[q];
        h[b] = 0ull;
    }
    // above = keys in the bins of the lanes above this one
    unsigned long long incl = mine;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const unsigned long long t = __shfl_down_sync(0xffffffffu, incl, o);
        if (lane + o < 32) incl += t;
    }
    const unsigned long long above = incl - mine;
    const uint64_t r = rank[w];
    // the lane whose bins hold rank r: above < r <= above + mine
    const bool here = above < r && r <= above + mine;
    const unsigned who = __ballot_sync(0xffffffffu, here);
    if (!here) {
        if (who == 0 && lane == 0) {  // not found (a count mismatch): keep the old behaviour, digit 0
            rank[w] = r;
        }
        return;
    }
    unsigned long long rr = r - above;
    int digit = 8 * lane;
#pragma unroll
    for (int q = 7; q >= 0; --q) {
        if (rr <= c[q]) {
            digit = 8 * lane + q;
            break;
        }
        rr -= c[q];
    }
    rank[w] = rr;
    prefix[w] |= static_cast<uint64_t>(digit) << ties_shift(pass);
}

// TIES elect and disjoint merge.  Entry kept when its key >= the threshold (ties kept).  P and N
// are the fp32 sums, in worker order, of the kept positive and negative values; the elected
// sign is that of P + N, and U the mean of the kept values of that sign (0 if P + N = 0).
__device__ __forceinline__ float ties_u(float P, float Nn, int cp, int cn) {
    const float S = __fadd_rn(P, Nn);
    return S > 0.f ? __fdiv_rn(P, static_cast<float>(cp)) : S < 0.f ? __fdiv_rn(Nn, static_cast<float>(cn)) : 0.f;
}

__device__ __forceinline__ void ties_acc(float d, uint32_t t, float& P, float& Nn, int& cp, int& cn) {
    if (__float_as_uint(fabsf(d)) >= t) {
        if (d > 0.f) { P = __fadd_rn(P, d); ++cp; }
        if (d < 0.f) { Nn = __fadd_rn(Nn, d); ++cn; }
    }
}

__global__ void __launch_bounds__(kStreamThreads) k_ties_merge(ReplicaPtrs reps, int K, int dtype,
                                                               float* __restrict__ theta, float* __restrict__ mom,
                                                               int64_t N, const uint64_t* __restrict__ thr_c,
                                                               const uint64_t* __restrict__ thr_f,
                                                               const int* __restrict__ fail, float eta, float mu,
                                                               uint32_t* __restrict__ err) {
    __shared__ uint32_t thr_s[kMaxK];
    const uint64_t* thr = *fail ? thr_f : thr_c;  // the bracket's result, or the fallback's
    for (int k = threadIdx.x; k < K; k += blockDim.x) thr_s[k] = static_cast<uint32_t>(thr[k]);
    __syncthreads();
    bool bad = false;
    const int64_t nv = N >> 2;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t v = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; v < nv; v += stride) {
        const int64_t i = 4 * v;
        float4 th = *reinterpret_cast<const float4*>(theta + i);
        float4 bb = *reinterpret_cast<const float4*>(mom + i);
        float P[4] = {0.f, 0.f, 0.f, 0.f}, Nn[4] = {0.f, 0.f, 0.f, 0.f}, T = 0.f;
        int cp[4] = {0, 0, 0, 0}, cn[4] = {0, 0, 0, 0};
        for (int k0 = 0; k0 < K; k0 += kLoadBatch) {
            float4 r[kLoadBatch];
#pragma unroll
            for (int q = 0; q < kLoadBatch; ++q)
                if (k0 + q < K) r[q] = ld_rep4(reps.p[k0 + q], dtype, i);
#pragma unroll
            for (int q = 0; q < kLoadBatch; ++q) {
                if (k0 + q >= K) break;
                const uint32_t t = thr_s[k0 + q];
                const float d[4] = {th.x - r[q].x, th.y - r[q].y, th.z - r[q].z, th.w - r[q].w};
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    T += d[j];
                    ties_acc(d[j], t, P[j], Nn[j], cp[j], cn[j]);
                }
            }
        }
        bad |= !isfinite(T);
        nesterov1(th.x, bb.x, ties_u(P[0], Nn[0], cp[0], cn[0]), eta, mu);
        nesterov1(th.y, bb.y, ties_u(P[1], Nn[1], cp[1], cn[1]), eta, mu);
        nesterov1(th.z, bb.z, ties_u(P[2], Nn[2], cp[2], cn[2]), eta, mu);
        nesterov1(th.w, bb.w, ties_u(P[3], Nn[3], cp[3], cn[3]), eta, mu);
        *reinterpret_cast<float4*>(mom + i) = bb;
        *reinterpret_cast<float4*>(theta + i) = th;
    }
    if (blockIdx.x == 0) {
        for (int64_t i = 4 * nv + threadIdx.x; i < N; i += blockDim.x) {
            float th = theta[i], bb = mom[i], P = 0.f, Nn = 0.f, T = 0.f;
            int cp = 0, cn = 0;
            for (int k = 0; k < K; ++k) {
                const float d = th - ld_rep1(reps.p[k], dtype, i);
                T += d;
                ties_acc(d, thr_s[k], P, Nn, cp, cn);
            }
            bad |= !isfinite(T);
            nesterov1(th, bb, ties_u(P, Nn, cp, cn), eta, mu);
            theta[i] = th;
            mom[i] = bb;
        }
    }
    raise_nonfinite(bad, err);
}

// fp32 [batch][rows][cols] -> bf16 (f16 = 0) or fp16 hi/lo planes with leading dimension ld.
__global__ void k_split_planes(const float* __restrict__ x, int64_t total, int rows, int cols, int ld,
                               __nv_bfloat16* __restrict__ hi, __nv_bfloat16* __restrict__ lo, int f16) {
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < total; i += stride) {
        const int64_t bm = i / cols;
        const int c = static_cast<int>(i - bm * cols);
        const int64_t b = bm / rows;
        const int r = static_cast<int>(bm - b * rows);
        const int64_t o = (b * rows + r) * ld + c;
        uint16_t h, l;
        split16(x[i], f16 != 0, h, l);
        reinterpret_cast<uint16_t*>(hi)[o] = h;
        reinterpret_cast<uint16_t*>(lo)[o] = l;
    }
}

// One thread waits, with the bounded wait of the GEMM's pipeline, on a fresh mbarrier that
// nothing arrives on (its phase 0 never completes) and gives up after limit_ns; it then
// raises kErrTimeout and returns, as a pipelined kernel does.  elapsed[0]: the wait's
// duration (ns).
__global__ void k_debug_wait(uint32_t* __restrict__ err, uint64_t limit_ns, unsigned long long* __restrict__ elapsed) {
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x != 0) return;
    mbar_init(&bar, 1);
    fence_mbar_init();
    const uint64_t t0 = globaltimer_ns();
    const bool ok = mbar_wait(&bar, 0u, limit_ns);
    elapsed[0] = globaltimer_ns() - t0;
    if (!ok) atomicOr(err, kErrTimeout);
}

}  // namespace isoloco
