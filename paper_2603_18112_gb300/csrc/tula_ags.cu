// libtula_ags: the AGS optimizer step (Tula, arXiv 2603.18112) for sm_103a.
//
// Two streaming passes over every parameter tensor, load-balanced by a chunk
// table (each tensor cut into chunks of kChunk elements; tiny tensors are one
// chunk, 100M-element tensors thousands):
//
//   k_reduce  (pass 1)  K-way replica mean (Eq. 1c) written over replica 0,
//                       per-chunk fp64 partials of |gbar|^2, |g_0|^2 [, |w|^2];
//                       the CTA finishing a tensor's last chunk combines that
//                       tensor's partials in a fixed order, and the CTA
//                       finishing the last tensor runs the finalize step:
//                       |G|^2, Delta (Eq. 5), the branch of Algorithm 1, the
//                       per-tensor coefficients, statistics, state, and
//                       UpdateGradScale.  No CTA ever waits on another: the
//                       hand-off is a counter ticket.
//   k_update  (pass 2)  d = c gbar + wd w; m = mu m + d; w = w - lr m, with
//                       |w|^2 taken on the way for the statistics.
//
// Both are HBM-bound streaming kernels (a few flops per 20-70 bytes): 128-bit
// coalesced loads, one persistent wave of CTAs, no tensor cores (nothing here
// is a contraction).  The chunk table, pointers and sizes travel in the kernel
// parameter block (__grid_constant__, up to ~31 KB per launch), so no
// host-to-device copy, allocation or host sync is ever needed and every call
// can be captured in a CUDA graph.  Reduction order depends only on the
// numels: results are bitwise reproducible and independent of the grid size.
#include "tula_ags.h"

#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <memory>
#include <mutex>
#include <vector>

namespace {

constexpr int kThreads = 512;            // threads per CTA
constexpr int kWarps = kThreads / 32;
constexpr int kChunk = 16384;            // elements per chunk (work item)
constexpr int kParamBudget = 31 * 1024;  // kernel parameter bytes per launch (limit 32764)
constexpr int kAcc = 3;                  // partial sums per chunk: |gbar|^2, |g_0|^2, |w|^2
constexpr int kTsum = 4;                 // per-tensor sums (stride)

enum Mode { kModeStep = 0, kModeStats = 1, kModeScale = 2 };

// ----------------------------------------------------------------------------
// Launch tables (kernel parameters)
// ----------------------------------------------------------------------------

template <int NP>
struct Table {
    static constexpr int kMaxT = (kParamBudget - 64) / (NP * 8 + 12);
    int n;    // tensors in this launch
    int t0;   // global index of its first tensor
    int c0;   // global index of its first chunk
    int nc;   // chunks in this launch
    long long numel[kMaxT];
    int cstart[kMaxT + 1];  // first chunk of each tensor, relative to c0; cstart[n] = nc
    const float *ptr[kMaxT][NP];
};

struct Scalars {
    int K, rule, gran, force, refresh, mode, n_total, has_small;
    int pow2K, read_w, pad0, pad1;
    float delta, eps, s_max, static_s, lars_trust, lr, mu, wd, invK, Kf;
    float *scale;
    double *state;
    double *stats;
    unsigned *tctr1;    // per-tensor chunk tickets, pass 1
    unsigned *tctr2;    // per-tensor chunk tickets, pass 2
    unsigned *done;     // [0]: tensors finished in pass 1
    int *flags;         // [0]: branch of the last step (1 = scaled)
    double *partials;   // [chunk][kAcc]
    double *tsum;       // [tensor][kTsum]: |gbar|^2, |g_0|^2, |w|^2
    float *coef;        // [tensor]: c_p
};

// ----------------------------------------------------------------------------
// Device helpers
// ----------------------------------------------------------------------------

__device__ __forceinline__ float4 ld_stream(const float *p) {
    return __ldcs(reinterpret_cast<const float4 *>(p));
}
__device__ __forceinline__ void st_stream(float *p, float4 v) {
    __stcs(reinterpret_cast<float4 *>(p), v);
}
__device__ __forceinline__ void st_keep(float *p, float4 v) {
    *reinterpret_cast<float4 *>(p) = v;
}

// fp32 sum of squares into a running fp32 partial, one FFMA per term
__device__ __forceinline__ float sq4(float acc, float4 v) {
    acc = __fmaf_rn(v.x, v.x, acc);
    acc = __fmaf_rn(v.y, v.y, acc);
    acc = __fmaf_rn(v.z, v.z, acc);
    acc = __fmaf_rn(v.w, v.w, acc);
    return acc;
}

// fp64 sum of exact squares (an fp32 square is exact in fp64), one DFMA per term
__device__ __forceinline__ double dsq4(double acc, float4 v) {
    acc = __fma_rn((double)v.x, (double)v.x, acc);
    acc = __fma_rn((double)v.y, (double)v.y, acc);
    acc = __fma_rn((double)v.z, (double)v.z, acc);
    acc = __fma_rn((double)v.w, (double)v.w, acc);
    return acc;
}

__device__ __forceinline__ float4 add4(float4 a, float4 b) {
    return make_float4(__fadd_rn(a.x, b.x), __fadd_rn(a.y, b.y), __fadd_rn(a.z, b.z),
                       __fadd_rn(a.w, b.w));
}

// Eq. 1c: divide the k-ascending sum by K (exact reciprocal when K is a power of 2)
__device__ __forceinline__ float mean1(float s, const Scalars &sc) {
    return sc.pow2K ? __fmul_rn(s, sc.invK) : __fdiv_rn(s, sc.Kf);
}
__device__ __forceinline__ float4 mean4(float4 s, const Scalars &sc) {
    return make_float4(mean1(s.x, sc), mean1(s.y, sc), mean1(s.z, sc), mean1(s.w, sc));
}

__device__ __forceinline__ double warp_sum(double v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = __dadd_rn(v, __shfl_down_sync(0xffffffffu, v, o));
    return v;
}

// Block sum of NV doubles in a fixed tree; result valid in thread 0.
template <int NV>
__device__ __forceinline__ void block_sum(double (&v)[NV], double (*red)[kWarps]) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int a = 0; a < NV; ++a) {
        double x = warp_sum(v[a]);
        if (lane == 0) red[a][warp] = x;
    }
    __syncthreads();
    if (warp == 0) {
#pragma unroll
        for (int a = 0; a < NV; ++a) {
            double x = lane < kWarps ? red[a][lane] : 0.0;
            v[a] = warp_sum(x);
        }
    }
    __syncthreads();
}

// Per-tensor coefficient c_p (Algorithm 1, Eq. 8, LARS).
__device__ __forceinline__ float coefficient(const Scalars &sc, int scaled, float scale_p,
                                             double sw, double sg) {
    switch (sc.rule) {
    case TULA_RULE_AGS: return scaled ? scale_p : 1.0f;
    case TULA_RULE_STATIC: return scaled ? sc.static_s : 1.0f;
    case TULA_RULE_LARS:
        if (sw > 0.0 && sg > 0.0) return (float)((double)sc.lars_trust * (sqrt(sw) / sqrt(sg)));
        return 1.0f;
    default: return 1.0f;
    }
}

// UpdateGradScale on tensor norms: min(|g_s| / (|g_l| + eps), s_max), fp64, rounded once.
__device__ __forceinline__ float scale_tensor(double s_small, double s_large, const Scalars &sc) {
    double q = sqrt(s_small) / (sqrt(s_large) + (double)sc.eps);
    return (float)fmin(q, (double)sc.s_max);
}

__device__ __forceinline__ int find_tensor(const int *cstart, int n, int c) {
    int lo = 0, hi = n;  // cstart[lo] <= c < cstart[hi]
    while (hi - lo > 1) {
        int mid = (lo + hi) >> 1;
        if (cstart[mid] <= c) lo = mid; else hi = mid;
    }
    return lo;
}

// ----------------------------------------------------------------------------
// Finalize (one CTA, after every tensor's sums are in sc.tsum)
// ----------------------------------------------------------------------------

__device__ void finalize(const Scalars &sc, double (*red)[kWarps]) {
    __shared__ int s_scaled;
    if (sc.mode == kModeStep) {
        double v[1] = {0.0};
        for (int t = threadIdx.x; t < sc.n_total; t += kThreads)
            v[0] = __dadd_rn(v[0], __ldcg(&sc.tsum[(size_t)t * kTsum + 0]));
        block_sum<1>(v, red);
        if (threadIdx.x == 0) {
            const double g2 = v[0];
            const double g2_prev = sc.state[TULA_STATE_G2_PREV];
            const double steps = sc.state[TULA_STATE_STEPS];
            // Eq. 5; no previous step -> +inf (sensitive)
            const double dv = steps == 0.0 ? (double)INFINITY : fabs((g2 - g2_prev) / g2_prev);
            int scaled;
            if (sc.force == TULA_BRANCH_SCALED) scaled = 1;
            else if (sc.force == TULA_BRANCH_UNSCALED) scaled = 0;
            else scaled = dv < (double)sc.delta;  // Algorithm 1: scaled iff Delta < delta
            sc.state[TULA_STATE_G2_PREV] = g2;
            sc.state[TULA_STATE_STEPS] = steps + 1.0;
            sc.state[TULA_STATE_DELTA] = dv;
            sc.state[TULA_STATE_SCALED] = (double)scaled;
            sc.flags[0] = scaled;
            s_scaled = scaled;
        }
        __syncthreads();
        const int scaled = s_scaled;
        const bool per_elem = sc.rule == TULA_RULE_AGS && sc.gran == TULA_SCALE_PER_ELEMENT;
        for (int t = threadIdx.x; t < sc.n_total; t += kThreads) {
            const double sg = __ldcg(&sc.tsum[(size_t)t * kTsum + 0]);
            const double ss = __ldcg(&sc.tsum[(size_t)t * kTsum + 1]);
            const double sw = __ldcg(&sc.tsum[(size_t)t * kTsum + 2]);
            const float scale_p = sc.scale ? sc.scale[t] : 1.0f;
            float c = coefficient(sc, scaled, scale_p, sw, sg);
            sc.coef[t] = c;
            float s_after = sc.scale ? scale_p : 0.0f;
            if (sc.refresh && sc.scale) {
                s_after = scale_tensor(ss, sg, sc);
                sc.scale[t] = s_after;
            }
            if (sc.stats) {
                double *row = sc.stats + (size_t)t * TULA_STATS_LEN;
                row[TULA_STAT_G_SQ] = sg;
                row[TULA_STAT_G0_SQ] = ss;
                row[TULA_STAT_G_NORM] = sqrt(sg);
                row[TULA_STAT_COEF] = per_elem ? (scaled ? (double)NAN : 1.0) : (double)c;
                row[TULA_STAT_SCALE] = (double)s_after;
                if (sc.read_w) {
                    row[TULA_STAT_W_SQ] = sw;
                    row[TULA_STAT_W_NORM] = sqrt(sw);
                    row[TULA_STAT_RATIO] = sg > 0.0 ? sqrt(sw) / sqrt(sg) : 0.0;
                }
            }
        }
    } else if (sc.mode == kModeStats) {
        for (int t = threadIdx.x; t < sc.n_total; t += kThreads) {
            const double sg = __ldcg(&sc.tsum[(size_t)t * kTsum + 0]);
            const double ss = __ldcg(&sc.tsum[(size_t)t * kTsum + 1]);
            const double sw = __ldcg(&sc.tsum[(size_t)t * kTsum + 2]);
            double *row = sc.stats + (size_t)t * TULA_STATS_LEN;
            row[TULA_STAT_W_SQ] = sw;
            row[TULA_STAT_G_SQ] = sg;
            row[TULA_STAT_G0_SQ] = ss;
            row[TULA_STAT_W_NORM] = sqrt(sw);
            row[TULA_STAT_G_NORM] = sqrt(sg);
            row[TULA_STAT_RATIO] = sg > 0.0 ? sqrt(sw) / sqrt(sg) : 0.0;
            row[TULA_STAT_COEF] = 0.0;
            row[TULA_STAT_SCALE] = 0.0;
        }
    } else {  // kModeScale: g_0 = g_large, small = g_small
        for (int t = threadIdx.x; t < sc.n_total; t += kThreads) {
            const double sl = __ldcg(&sc.tsum[(size_t)t * kTsum + 0]);
            const double ss = __ldcg(&sc.tsum[(size_t)t * kTsum + 1]);
            sc.scale[t] = scale_tensor(ss, sl, sc);
        }
    }
    if (threadIdx.x == 0) sc.done[0] = 0u;  // re-arm for the next call
}

// ----------------------------------------------------------------------------
// Pass 1: replica mean + per-tensor squared norms (+ finalize by the last CTA)
// ----------------------------------------------------------------------------
//
// Template: KT = replicas known at compile time (0: runtime K <= 16);
// WM = write the mean over replica 0; RW = also reduce |w|^2;
// SS = g_small is a separate stream (role KS + 1) instead of replica 0;
// PR = precise norms: every exact fp64 square is added in fp64 (relative error
// ~1e-15), for norms that feed a per-tensor coefficient (UpdateGradScale, LARS);
// otherwise each thread sums <= 16 squares in fp32 before one fp64 add (~1e-7),
// which is what the variability metric and the statistics need, at a fraction
// of GB300's FP64 rate.
// Pointer roles per tensor: [0, K) replicas, KS = w, KS + 1 = g_small.

template <int KT>
struct P1 {
    static constexpr int KS = KT > 0 ? KT : TULA_MAX_K;
    static constexpr int NP = KS + 2;
};

template <int KT, bool WM, bool RW, bool SS, bool PR>
__device__ __forceinline__ void reduce_vec(const Table<P1<KT>::NP> &tab, int t, long long begin,
                                           int nv, const Scalars &sc, double &ag, double &as,
                                           double &aw) {
    constexpr int KS = P1<KT>::KS;
    constexpr int NS = (KT > 0 ? KT : 4) + (RW ? 1 : 0) + (SS ? 1 : 0);  // streams read
    constexpr int U = NS >= 4 ? 1 : 4 / NS;  // >= 4 float4 loads per thread in flight
    constexpr int KL = KT > 0 ? KT : TULA_MAX_K;  // load slots
    const int K = KT > 0 ? KT : sc.K;
    const float *g[KL];
#pragma unroll
    for (int k = 0; k < KL; ++k) g[k] = (k < K) ? tab.ptr[t][k] + begin : nullptr;
    const float *wp = RW ? tab.ptr[t][KS] + begin : nullptr;
    const float *sp = SS ? tab.ptr[t][KS + 1] + begin : nullptr;
    float *out = const_cast<float *>(tab.ptr[t][0]) + begin;

#pragma unroll 1
    for (int v0 = threadIdx.x; v0 < nv; v0 += kThreads * U) {
        float4 x[U][KL];
        float4 wv[U], sv[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int v = v0 + u * kThreads;
            if (v < nv) {
#pragma unroll
                for (int k = 0; k < KL; ++k)
                    if (k < K) x[u][k] = ld_stream(g[k] + 4 * (size_t)v);
                if (RW) wv[u] = ld_stream(wp + 4 * (size_t)v);
                if (SS) sv[u] = ld_stream(sp + 4 * (size_t)v);
            }
        }
        float pg = 0.f, ps = 0.f, pw = 0.f;
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int v = v0 + u * kThreads;
            if (v < nv) {
                float4 s = x[u][0];
#pragma unroll
                for (int k = 1; k < KL; ++k)
                    if (k < K) s = add4(s, x[u][k]);
                if (K > 1) {
                    s = mean4(s, sc);
                    if (WM) st_keep(out + 4 * (size_t)v, s);
                    if (PR) as = dsq4(as, x[u][0]); else ps = sq4(ps, x[u][0]);
                }
                if (PR) {
                    ag = dsq4(ag, s);
                    if (SS) as = dsq4(as, sv[u]);
                    if (RW) aw = dsq4(aw, wv[u]);
                } else {
                    pg = sq4(pg, s);
                    if (SS) ps = sq4(ps, sv[u]);
                    if (RW) pw = sq4(pw, wv[u]);
                }
            }
        }
        if (!PR) {
            ag = __dadd_rn(ag, (double)pg);
            if (K > 1 || SS) as = __dadd_rn(as, (double)ps);
            if (RW) aw = __dadd_rn(aw, (double)pw);
        }
    }
}

template <int KT, bool WM, bool RW, bool SS>
__device__ __forceinline__ void reduce_scalar(const Table<P1<KT>::NP> &tab, int t, long long j0,
                                              long long j1, const Scalars &sc, double &ag,
                                              double &as, double &aw) {
    constexpr int KS = P1<KT>::KS;
    constexpr int KL = KT > 0 ? KT : TULA_MAX_K;
    const int K = KT > 0 ? KT : sc.K;
    for (long long j = j0 + threadIdx.x; j < j1; j += kThreads) {
        float x0 = __ldcs(tab.ptr[t][0] + j);
        float s = x0;
#pragma unroll
        for (int k = 1; k < KL; ++k)
            if (k < K) s = __fadd_rn(s, __ldcs(tab.ptr[t][k] + j));
        if (K > 1) {
            s = mean1(s, sc);
            if (WM) const_cast<float *>(tab.ptr[t][0])[j] = s;
            as = __fma_rn((double)x0, (double)x0, as);
        }
        ag = __fma_rn((double)s, (double)s, ag);
        if (SS) {
            const double y = __ldcs(tab.ptr[t][KS + 1] + j);
            as = __fma_rn(y, y, as);
        }
        if (RW) {
            const double y = __ldcs(tab.ptr[t][KS] + j);
            aw = __fma_rn(y, y, aw);
        }
    }
}

template <int KT, bool WM, bool RW, bool SS, bool PR>
__global__ void __launch_bounds__(kThreads, 2)
    k_reduce(const __grid_constant__ Table<P1<KT>::NP> tab, const __grid_constant__ Scalars sc) {
    constexpr int KS = P1<KT>::KS;
    __shared__ double red[kAcc][kWarps];
    __shared__ int s_last;
    const int K = KT > 0 ? KT : sc.K;

    for (int c = blockIdx.x; c < tab.nc; c += gridDim.x) {
        const int t = find_tensor(tab.cstart, tab.n, c);
        const long long n = tab.numel[t];
        const long long begin = (long long)(c - tab.cstart[t]) * kChunk;
        const long long end = min(begin + (long long)kChunk, n);
        double acc[kAcc] = {0.0, 0.0, 0.0};

        if (end > begin) {
            uintptr_t al = 0;
            for (int k = 0; k < K; ++k) al |= reinterpret_cast<uintptr_t>(tab.ptr[t][k]);
            if (RW) al |= reinterpret_cast<uintptr_t>(tab.ptr[t][KS]);
            if (SS) al |= reinterpret_cast<uintptr_t>(tab.ptr[t][KS + 1]);
            const int nv = (al & 15u) == 0 ? (int)((end - begin) >> 2) : 0;
            if (nv > 0)
                reduce_vec<KT, WM, RW, SS, PR>(tab, t, begin, nv, sc, acc[0], acc[1], acc[2]);
            reduce_scalar<KT, WM, RW, SS>(tab, t, begin + 4 * (long long)nv, end, sc, acc[0],
                                          acc[1], acc[2]);
        }
        block_sum<kAcc>(acc, red);

        const int tg = tab.t0 + t;
        const int nch = tab.cstart[t + 1] - tab.cstart[t];
        if (threadIdx.x == 0) {
            double *P = sc.partials + (size_t)(tab.c0 + c) * kAcc;
            P[0] = acc[0];
            P[1] = acc[1];
            P[2] = acc[2];
            __threadfence();
            s_last = atomicAdd(&sc.tctr1[tg], 1u) == (unsigned)(nch - 1);
        }
        __syncthreads();
        if (!s_last) continue;

        // This CTA counted the tensor's last chunk: combine its partials in a
        // fixed order (strided per thread, then the block tree).
        __threadfence();
        double tot[kAcc] = {0.0, 0.0, 0.0};
        const double *P = sc.partials + (size_t)(tab.c0 + tab.cstart[t]) * kAcc;
        for (int i = threadIdx.x; i < nch; i += kThreads) {
#pragma unroll
            for (int a = 0; a < kAcc; ++a) tot[a] = __dadd_rn(tot[a], __ldcg(P + (size_t)i * kAcc + a));
        }
        block_sum<kAcc>(tot, red);
        if (threadIdx.x == 0) {
            double *T = sc.tsum + (size_t)tg * kTsum;
            T[0] = tot[0];
            T[1] = (K > 1 || SS) ? tot[1] : tot[0];  // K = 1: replica 0 is the mean
            T[2] = tot[2];
            sc.tctr1[tg] = 0u;  // re-arm
            __threadfence();
            s_last = atomicAdd(&sc.done[0], 1u) == (unsigned)(sc.n_total - 1);
        }
        __syncthreads();
        if (s_last) {
            __threadfence();
            finalize(sc, red);
        }
        __syncthreads();
    }
}

// Degenerate launch with no chunk at all cannot happen (every tensor has >= 1
// chunk), so the finalize always runs inside k_reduce.

// ----------------------------------------------------------------------------
// Pass 2: scaled momentum-SGD + weight-decay update (Eq. 7b, Algorithm 1)
// ----------------------------------------------------------------------------
// Pointer roles: 0 = gbar, 1 = w, 2 = m, 3 = per-element gradscale.

constexpr int kNP2 = 4;

__device__ __forceinline__ void sgd1(float g, float c, float &w, float &m, const Scalars &sc,
                                     bool has_m) {
    const float gt = __fmul_rn(c, g);
    const float d = __fadd_rn(gt, __fmul_rn(sc.wd, w));
    if (has_m) {
        m = __fadd_rn(__fmul_rn(sc.mu, m), d);
        w = __fsub_rn(w, __fmul_rn(sc.lr, m));
    } else {
        w = __fsub_rn(w, __fmul_rn(sc.lr, d));
    }
}

template <bool HM, bool PE, bool SW>
__global__ void __launch_bounds__(kThreads, 2)
    k_update(const __grid_constant__ Table<kNP2> tab, const __grid_constant__ Scalars sc) {
    constexpr int U = 2;
    __shared__ double red[1][kWarps];
    __shared__ int s_last;
    const int scaled = sc.flags[0];

    for (int c = blockIdx.x; c < tab.nc; c += gridDim.x) {
        const int t = find_tensor(tab.cstart, tab.n, c);
        const int tg = tab.t0 + t;
        const long long n = tab.numel[t];
        const long long begin = (long long)(c - tab.cstart[t]) * kChunk;
        const long long end = min(begin + (long long)kChunk, n);
        const float ct = sc.coef[tg];
        const bool use_se = PE && scaled;
        double aw[1] = {0.0};

        if (end > begin) {
            const float *gp = tab.ptr[t][0] + begin;
            float *wp = const_cast<float *>(tab.ptr[t][1]) + begin;
            float *mp = HM ? const_cast<float *>(tab.ptr[t][2]) + begin : nullptr;
            const float *sp = use_se ? tab.ptr[t][3] + begin : nullptr;
            uintptr_t al = reinterpret_cast<uintptr_t>(gp) | reinterpret_cast<uintptr_t>(wp);
            if (HM) al |= reinterpret_cast<uintptr_t>(mp);
            if (use_se) al |= reinterpret_cast<uintptr_t>(sp);
            const int nv = (al & 15u) == 0 ? (int)((end - begin) >> 2) : 0;
#pragma unroll 1
            for (int v0 = threadIdx.x; v0 < nv; v0 += kThreads * U) {
                float4 gv[U], wv[U], mv[U], sv[U];
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    const int v = v0 + u * kThreads;
                    if (v < nv) {
                        gv[u] = ld_stream(gp + 4 * (size_t)v);
                        wv[u] = ld_stream(wp + 4 * (size_t)v);
                        if (HM) mv[u] = ld_stream(mp + 4 * (size_t)v);
                        if (use_se) sv[u] = ld_stream(sp + 4 * (size_t)v);
                    }
                }
                float pw = 0.f;
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    const int v = v0 + u * kThreads;
                    if (v < nv) {
                        if (SW) pw = sq4(pw, wv[u]);
                        float4 cc = use_se ? sv[u] : make_float4(ct, ct, ct, ct);
                        if (PE && !scaled) cc = make_float4(1.f, 1.f, 1.f, 1.f);
                        float4 w4 = wv[u], m4 = HM ? mv[u] : make_float4(0.f, 0.f, 0.f, 0.f);
                        sgd1(gv[u].x, cc.x, w4.x, m4.x, sc, HM);
                        sgd1(gv[u].y, cc.y, w4.y, m4.y, sc, HM);
                        sgd1(gv[u].z, cc.z, w4.z, m4.z, sc, HM);
                        sgd1(gv[u].w, cc.w, w4.w, m4.w, sc, HM);
                        st_stream(wp + 4 * (size_t)v, w4);
                        if (HM) st_stream(mp + 4 * (size_t)v, m4);
                    }
                }
                if (SW) aw[0] = __dadd_rn(aw[0], (double)pw);
            }
            for (long long j = 4 * (long long)nv + threadIdx.x; j < end - begin; j += kThreads) {
                const float g = __ldcs(gp + j);
                float w = __ldcs(wp + j);
                float m = HM ? __ldcs(mp + j) : 0.f;
                float cj = use_se ? __ldcs(sp + j) : (PE ? 1.f : ct);
                if (SW) aw[0] = __dadd_rn(aw[0], (double)__fmul_rn(w, w));
                sgd1(g, cj, w, m, sc, HM);
                __stcs(wp + j, w);
                if (HM) __stcs(mp + j, m);
            }
        }
        if (!SW) continue;

        block_sum<1>(aw, red);
        const int nch = tab.cstart[t + 1] - tab.cstart[t];
        if (threadIdx.x == 0) {
            sc.partials[(size_t)(tab.c0 + c) * kAcc + 2] = aw[0];
            __threadfence();
            s_last = atomicAdd(&sc.tctr2[tg], 1u) == (unsigned)(nch - 1);
        }
        __syncthreads();
        if (!s_last) continue;
        __threadfence();
        double tot[1] = {0.0};
        const double *P = sc.partials + (size_t)(tab.c0 + tab.cstart[t]) * kAcc + 2;
        for (int i = threadIdx.x; i < nch; i += kThreads)
            tot[0] = __dadd_rn(tot[0], __ldcg(P + (size_t)i * kAcc));
        block_sum<1>(tot, red);
        if (threadIdx.x == 0) {
            const double sw = tot[0];
            const double sg = __ldcg(&sc.tsum[(size_t)tg * kTsum + 0]);
            double *row = sc.stats + (size_t)tg * TULA_STATS_LEN;
            row[TULA_STAT_W_SQ] = sw;
            row[TULA_STAT_W_NORM] = sqrt(sw);
            row[TULA_STAT_RATIO] = sg > 0.0 ? sqrt(sw) / sqrt(sg) : 0.0;
            sc.tctr2[tg] = 0u;
        }
        __syncthreads();
    }
}

// ----------------------------------------------------------------------------
// UpdateGradScale, element-wise (Algorithm 1): s = fminf(|gs / (gl + eps)|, s_max)
// ----------------------------------------------------------------------------
// Pointer roles: 0 = g_small, 1 = g_large, 2 = s_out.

constexpr int kNP3 = 3;

__device__ __forceinline__ float scale1(float gs, float gl, const Scalars &sc) {
    return fminf(fabsf(__fdiv_rn(gs, __fadd_rn(gl, sc.eps))), sc.s_max);
}

__global__ void __launch_bounds__(kThreads, 2)
    k_scale_elem(const __grid_constant__ Table<kNP3> tab, const __grid_constant__ Scalars sc) {
    for (int c = blockIdx.x; c < tab.nc; c += gridDim.x) {
        const int t = find_tensor(tab.cstart, tab.n, c);
        const long long n = tab.numel[t];
        const long long begin = (long long)(c - tab.cstart[t]) * kChunk;
        const long long end = min(begin + (long long)kChunk, n);
        if (end <= begin) continue;
        const float *a = tab.ptr[t][0] + begin;
        const float *b = tab.ptr[t][1] + begin;
        float *o = const_cast<float *>(tab.ptr[t][2]) + begin;
        const uintptr_t al = reinterpret_cast<uintptr_t>(a) | reinterpret_cast<uintptr_t>(b) |
                             reinterpret_cast<uintptr_t>(o);
        const int nv = (al & 15u) == 0 ? (int)((end - begin) >> 2) : 0;
        for (int v = threadIdx.x; v < nv; v += kThreads) {
            const float4 x = ld_stream(a + 4 * (size_t)v), y = ld_stream(b + 4 * (size_t)v);
            st_stream(o + 4 * (size_t)v, make_float4(scale1(x.x, y.x, sc), scale1(x.y, y.y, sc),
                                                     scale1(x.z, y.z, sc), scale1(x.w, y.w, sc)));
        }
        for (long long j = 4 * (long long)nv + threadIdx.x; j < end - begin; j += kThreads)
            o[j] = scale1(__ldcs(a + j), __ldcs(b + j), sc);
    }
}

// ----------------------------------------------------------------------------
// Host side
// ----------------------------------------------------------------------------

std::atomic<uint64_t> g_launches{0};
thread_local int g_last_cuda = 0;

inline long long chunks_of(int64_t n) { return n <= 0 ? 1 : (n + kChunk - 1) / kChunk; }

struct WsLayout {
    size_t tctr1, tctr2, done, flags, partials, tsum, coef, total;
};

WsLayout ws_layout(int n_tensors, long long n_chunks) {
    size_t off = 0;
    auto take = [&](size_t bytes) {
        size_t o = off;
        off = (off + bytes + 255) & ~size_t(255);
        return o;
    };
    WsLayout L;
    L.tctr1 = take(sizeof(unsigned) * (size_t)n_tensors);
    L.tctr2 = take(sizeof(unsigned) * (size_t)n_tensors);
    L.done = take(sizeof(unsigned) * 4);
    L.flags = take(sizeof(int) * 4);
    L.partials = take(sizeof(double) * kAcc * (size_t)n_chunks);
    L.tsum = take(sizeof(double) * kTsum * (size_t)n_tensors);
    L.coef = take(sizeof(float) * (size_t)n_tensors);
    L.total = off;
    return L;
}

bool valid_numels(const int64_t *numels, int n, long long *total_chunks) {
    if (!numels || n < 1) return false;
    long long tot = 0;
    for (int p = 0; p < n; ++p) {
        if (numels[p] < 0) return false;
        tot += chunks_of(numels[p]);
    }
    if (tot >= (1LL << 31)) return false;
    *total_chunks = tot;
    return true;
}

inline bool aligned4(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 3u) == 0; }

// One wave of resident CTAs for `kernel` on the current device (cached).
int resident_ctas(const void *kernel) {
    struct Entry { const void *k; int dev; int ctas; };
    static std::mutex mu;
    static std::vector<Entry> cache;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    {
        std::lock_guard<std::mutex> lock(mu);
        for (const Entry &e : cache)
            if (e.k == kernel && e.dev == dev) return e.ctas;
    }
    int sms = 0, per = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per, kernel, kThreads, 0) != cudaSuccess)
        return 0;
    const int ctas = std::max(1, sms * std::max(per, 1));
    std::lock_guard<std::mutex> lock(mu);
    cache.push_back({kernel, dev, ctas});
    return ctas;
}

// Splits tensors [0, n) into launches that fit one parameter block and
// launches `kernel` once per group.  fill(p, ptrs) writes tensor p's pointers.
template <int NP, typename Kernel, typename Fill>
int launch_groups(Kernel kernel, int n, const int64_t *numels, const Scalars &sc, int grid_override,
                  cudaStream_t stream, Fill fill) {
    using T = Table<NP>;
    std::unique_ptr<T> tab(new T);
    int grid_cap = grid_override > 0 ? grid_override : resident_ctas((const void *)kernel);
    if (grid_cap <= 0) {
        g_last_cuda = (int)cudaGetLastError();
        return TULA_ERR_CUDA;
    }
    long long c_global = 0;
    int p = 0;
    while (p < n) {
        std::memset(tab.get(), 0, sizeof(T));
        tab->t0 = p;
        tab->c0 = (int)c_global;
        int cnt = 0, nc = 0;
        while (p < n && cnt < T::kMaxT) {
            tab->numel[cnt] = numels[p];
            tab->cstart[cnt] = nc;
            fill(p, tab->ptr[cnt]);
            nc += (int)chunks_of(numels[p]);
            ++cnt;
            ++p;
        }
        tab->n = cnt;
        tab->nc = nc;
        tab->cstart[cnt] = nc;
        c_global += nc;
        const int grid = std::min(nc, grid_cap);
        kernel<<<grid, kThreads, 0, stream>>>(*tab, sc);
        g_launches.fetch_add(1, std::memory_order_relaxed);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) {
            g_last_cuda = (int)e;
            return TULA_ERR_CUDA;
        }
    }
    return TULA_OK;
}

Scalars make_scalars(const tula_ags_hparams *hp, int K, int n, void *ws, const WsLayout &L,
                     int mode) {
    Scalars sc;
    std::memset(&sc, 0, sizeof(sc));
    sc.K = K;
    sc.mode = mode;
    sc.n_total = n;
    sc.pow2K = (K & (K - 1)) == 0;
    sc.invK = 1.0f / (float)K;
    sc.Kf = (float)K;
    if (hp) {
        sc.rule = hp->rule;
        sc.gran = hp->granularity;
        sc.force = hp->force_branch;
        sc.refresh = hp->refresh_scale;
        sc.delta = hp->delta;
        sc.eps = hp->eps;
        sc.s_max = hp->s_max;
        sc.static_s = hp->static_s;
        sc.lars_trust = hp->lars_trust;
        sc.scale = hp->scale;
        sc.state = hp->state;
        sc.stats = hp->layer_stats;
    }
    char *b = static_cast<char *>(ws);
    sc.tctr1 = reinterpret_cast<unsigned *>(b + L.tctr1);
    sc.tctr2 = reinterpret_cast<unsigned *>(b + L.tctr2);
    sc.done = reinterpret_cast<unsigned *>(b + L.done);
    sc.flags = reinterpret_cast<int *>(b + L.flags);
    sc.partials = reinterpret_cast<double *>(b + L.partials);
    sc.tsum = reinterpret_cast<double *>(b + L.tsum);
    sc.coef = reinterpret_cast<float *>(b + L.coef);
    return sc;
}

// Pass-1 dispatch over the compile-time replica count.
template <int KT, bool WM, bool RW, bool SS, bool PR, typename Fill>
int run_reduce_k(int n, const int64_t *numels, const Scalars &sc, int grid, cudaStream_t s,
                 Fill fill) {
    return launch_groups<P1<KT>::NP>(k_reduce<KT, WM, RW, SS, PR>, n, numels, sc, grid, s, fill);
}

template <bool WM, bool RW, bool SS, bool PR, typename Fill>
int run_reduce(int K, int n, const int64_t *numels, const Scalars &sc, int grid, cudaStream_t s,
               Fill fill) {
    switch (K) {
    case 1: return run_reduce_k<1, false, RW, SS, PR>(n, numels, sc, grid, s, fill);
    case 2: return run_reduce_k<2, WM, RW, SS, PR>(n, numels, sc, grid, s, fill);
    case 4: return run_reduce_k<4, WM, RW, SS, PR>(n, numels, sc, grid, s, fill);
    case 8: return run_reduce_k<8, WM, RW, SS, PR>(n, numels, sc, grid, s, fill);
    case 16: return run_reduce_k<16, WM, RW, SS, PR>(n, numels, sc, grid, s, fill);
    default: return run_reduce_k<0, WM, RW, SS, PR>(n, numels, sc, grid, s, fill);
    }
}

int check_ws(void *ws, size_t bytes, int n, long long nch) {
    if (!ws) return TULA_ERR_WORKSPACE;
    if (bytes < ws_layout(n, nch).total) return TULA_ERR_WORKSPACE;
    if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return TULA_ERR_WORKSPACE;
    return TULA_OK;
}

void record(void *ev, cudaStream_t s) {
    if (ev) cudaEventRecord(static_cast<cudaEvent_t>(ev), s);
}

}  // namespace

// ============================================================================
// C ABI
// ============================================================================

extern "C" {

void tula_ags_default_hparams(tula_ags_hparams *hp, int K) {
    if (!hp) return;
    std::memset(hp, 0, sizeof(*hp));
    hp->K = K;
    hp->rule = TULA_RULE_AGS;
    hp->granularity = TULA_SCALE_PER_TENSOR;
    hp->force_branch = TULA_BRANCH_AUTO;
    hp->refresh_scale = 0;
    hp->delta = 0.5f;
    hp->eps = 1e-8f;
    hp->s_max = std::sqrt((float)(K > 0 ? K : 1));
    hp->static_s = 1.0f;
    hp->lars_trust = 1.0f;
}

int tula_ags_workspace_size(const int64_t *numels, int n_tensors, int K, size_t *bytes) {
    long long nch = 0;
    if (!bytes || K < 1 || K > TULA_MAX_K || !valid_numels(numels, n_tensors, &nch))
        return TULA_ERR_ARG;
    *bytes = ws_layout(n_tensors, nch).total;
    return TULA_OK;
}

int tula_ags_chunk_elems(void) { return kChunk; }

int tula_ags_plan_chunks(const int64_t *numels, int n_tensors, int64_t *chunk_start_out) {
    long long nch = 0;
    if (!chunk_start_out || !valid_numels(numels, n_tensors, &nch)) return TULA_ERR_ARG;
    int64_t c = 0;
    for (int p = 0; p < n_tensors; ++p) {
        chunk_start_out[p] = c;
        c += chunks_of(numels[p]);
    }
    chunk_start_out[n_tensors] = c;
    return TULA_OK;
}

int tula_ags_step(float *const *param_ptrs, float *const *grad_ptrs, float *const *mom_ptrs,
                  const int64_t *numels, int n_tensors, float lr, float momentum,
                  float weight_decay, const tula_ags_hparams *hp, void *stream) {
    long long nch = 0;
    if (!hp || !param_ptrs || !grad_ptrs || !valid_numels(numels, n_tensors, &nch))
        return TULA_ERR_ARG;
    const int K = hp->K, n = n_tensors;
    if (K < 1 || K > TULA_MAX_K) return TULA_ERR_ARG;
    if (hp->rule < TULA_RULE_AGS || hp->rule > TULA_RULE_STATIC) return TULA_ERR_ARG;
    if (hp->granularity != TULA_SCALE_PER_TENSOR && hp->granularity != TULA_SCALE_PER_ELEMENT)
        return TULA_ERR_ARG;
    if (hp->force_branch < TULA_BRANCH_AUTO || hp->force_branch > TULA_BRANCH_UNSCALED)
        return TULA_ERR_ARG;
    if (!hp->state) return TULA_ERR_ARG;
    const bool per_elem = hp->rule == TULA_RULE_AGS && hp->granularity == TULA_SCALE_PER_ELEMENT;
    if (hp->rule == TULA_RULE_AGS && !per_elem && !hp->scale) return TULA_ERR_ARG;
    if (per_elem && !hp->scale_elem) return TULA_ERR_ARG;
    if (!mom_ptrs && momentum != 0.0f) return TULA_ERR_ARG;
    if (hp->refresh_scale) {
        if (K == 1 || !hp->scale) return TULA_ERR_ARG;
        if (hp->granularity != TULA_SCALE_PER_TENSOR) return TULA_ERR_UNSUPPORTED;
    }
    for (int p = 0; p < n; ++p) {
        if (numels[p] == 0) continue;
        if (!param_ptrs[p] || !aligned4(param_ptrs[p])) return TULA_ERR_ARG;
        if (mom_ptrs && (!mom_ptrs[p] || !aligned4(mom_ptrs[p]))) return TULA_ERR_ARG;
        if (per_elem && (!hp->scale_elem[p] || !aligned4(hp->scale_elem[p]))) return TULA_ERR_ARG;
        for (int k = 0; k < K; ++k) {
            const float *g = grad_ptrs[(size_t)k * n + p];
            if (!g || !aligned4(g)) return TULA_ERR_ARG;
        }
    }
    int rc = check_ws(hp->workspace, hp->workspace_bytes, n, nch);
    if (rc) return rc;

    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const WsLayout L = ws_layout(n, nch);
    Scalars sc = make_scalars(hp, K, n, hp->workspace, L, kModeStep);
    const bool lars = hp->rule == TULA_RULE_LARS;
    sc.read_w = lars ? 1 : 0;
    sc.lr = lr;
    sc.mu = momentum;
    sc.wd = weight_decay;

    auto fill1 = [&](int p, const float **dst) {
        const int KS = (K == 1 || K == 2 || K == 4 || K == 8 || K == 16) ? K : TULA_MAX_K;
        for (int k = 0; k < K; ++k) dst[k] = grad_ptrs[(size_t)k * n + p];
        dst[KS] = param_ptrs[p];
        dst[KS + 1] = nullptr;
    };
    record(hp->trace_events[0], s);
    // Norms feeding a coefficient (LARS, UpdateGradScale) are taken precisely.
    if (lars)
        rc = run_reduce<true, true, false, true>(K, n, numels, sc, hp->grid_ctas, s, fill1);
    else if (hp->refresh_scale)
        rc = run_reduce<true, false, false, true>(K, n, numels, sc, hp->grid_ctas, s, fill1);
    else
        rc = run_reduce<true, false, false, false>(K, n, numels, sc, hp->grid_ctas, s, fill1);
    if (rc) return rc;
    record(hp->trace_events[1], s);

    auto fill2 = [&](int p, const float **dst) {
        dst[0] = grad_ptrs[p];
        dst[1] = param_ptrs[p];
        dst[2] = mom_ptrs ? mom_ptrs[p] : nullptr;
        dst[3] = per_elem ? hp->scale_elem[p] : nullptr;
    };
    const bool hm = mom_ptrs != nullptr;
    const bool sw = hp->layer_stats != nullptr && !lars;
#define TULA_UPD(HM, PE, SW) \
    launch_groups<kNP2>(k_update<HM, PE, SW>, n, numels, sc, hp->grid_ctas, s, fill2)
    if (hm) {
        if (per_elem) rc = sw ? TULA_UPD(true, true, true) : TULA_UPD(true, true, false);
        else rc = sw ? TULA_UPD(true, false, true) : TULA_UPD(true, false, false);
    } else {
        if (per_elem) rc = sw ? TULA_UPD(false, true, true) : TULA_UPD(false, true, false);
        else rc = sw ? TULA_UPD(false, false, true) : TULA_UPD(false, false, false);
    }
#undef TULA_UPD
    if (rc) return rc;
    record(hp->trace_events[2], s);
    return TULA_OK;
}

int tula_layer_stats(const float *const *param_ptrs, const float *const *grad_ptrs, int K,
                     const int64_t *numels, int n_tensors, double *stats_out, void *workspace,
                     size_t workspace_bytes, void *stream) {
    long long nch = 0;
    if (!param_ptrs || !grad_ptrs || !stats_out || !valid_numels(numels, n_tensors, &nch))
        return TULA_ERR_ARG;
    if (K < 1 || K > TULA_MAX_K) return TULA_ERR_ARG;
    const int n = n_tensors;
    for (int p = 0; p < n; ++p) {
        if (numels[p] == 0) continue;
        if (!param_ptrs[p] || !aligned4(param_ptrs[p])) return TULA_ERR_ARG;
        for (int k = 0; k < K; ++k) {
            const float *g = grad_ptrs[(size_t)k * n + p];
            if (!g || !aligned4(g)) return TULA_ERR_ARG;
        }
    }
    int rc = check_ws(workspace, workspace_bytes, n, nch);
    if (rc) return rc;
    const WsLayout L = ws_layout(n, nch);
    Scalars sc = make_scalars(nullptr, K, n, workspace, L, kModeStats);
    sc.stats = stats_out;
    sc.read_w = 1;
    auto fill = [&](int p, const float **dst) {
        const int KS = (K == 1 || K == 2 || K == 4 || K == 8 || K == 16) ? K : TULA_MAX_K;
        for (int k = 0; k < K; ++k) dst[k] = grad_ptrs[(size_t)k * n + p];
        dst[KS] = param_ptrs[p];
        dst[KS + 1] = nullptr;
    };
    return run_reduce<false, true, false, false>(K, n, numels, sc, 0,
                                          static_cast<cudaStream_t>(stream), fill);
}

int tula_ags_update_scale(const float *const *g_small, const float *const *g_large,
                          const int64_t *numels, int n_tensors, const tula_ags_hparams *hp,
                          void *stream) {
    long long nch = 0;
    if (!hp || !g_small || !g_large || !valid_numels(numels, n_tensors, &nch)) return TULA_ERR_ARG;
    const int n = n_tensors;
    const bool per_elem = hp->granularity == TULA_SCALE_PER_ELEMENT;
    if (!per_elem && hp->granularity != TULA_SCALE_PER_TENSOR) return TULA_ERR_ARG;
    if (per_elem ? !hp->scale_elem : !hp->scale) return TULA_ERR_ARG;
    for (int p = 0; p < n; ++p) {
        if (numels[p] == 0) continue;
        if (!g_small[p] || !g_large[p] || !aligned4(g_small[p]) || !aligned4(g_large[p]))
            return TULA_ERR_ARG;
        if (per_elem && (!hp->scale_elem[p] || !aligned4(hp->scale_elem[p]))) return TULA_ERR_ARG;
    }
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (per_elem) {
        Scalars sc;
        std::memset(&sc, 0, sizeof(sc));
        sc.eps = hp->eps;
        sc.s_max = hp->s_max;
        auto fill = [&](int p, const float **dst) {
            dst[0] = g_small[p];
            dst[1] = g_large[p];
            dst[2] = hp->scale_elem[p];
        };
        return launch_groups<kNP3>(k_scale_elem, n, numels, sc, hp->grid_ctas, s, fill);
    }
    int rc = check_ws(hp->workspace, hp->workspace_bytes, n, nch);
    if (rc) return rc;
    const WsLayout L = ws_layout(n, nch);
    Scalars sc = make_scalars(hp, 1, n, hp->workspace, L, kModeScale);
    sc.has_small = 1;
    auto fill = [&](int p, const float **dst) {
        dst[0] = g_large[p];
        dst[1] = nullptr;
        dst[2] = g_small[p];
    };
    return run_reduce_k<1, false, false, true, true>(n, numels, sc, hp->grid_ctas, s, fill);
}

const char *tula_ags_error_string(int code) {
    switch (code) {
    case TULA_OK: return "ok";
    case TULA_ERR_ARG: return "invalid argument";
    case TULA_ERR_WORKSPACE: return "workspace missing, too small or not 256-byte aligned";
    case TULA_ERR_CUDA: return "CUDA launch failed";
    case TULA_ERR_UNSUPPORTED: return "unsupported combination of options";
    case TULA_ERR_SCRATCH_LIMIT:
        return "tensor list needs more than the library's static scratch "
               "(TULA_STATIC_SCRATCH_BYTES); use tula_ags_step with a workspace";
    default: return "unknown status";
    }
}

int tula_ags_last_cuda_error(void) { return g_last_cuda; }

uint64_t tula_ags_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

}  // extern "C"

// ============================================================================
// Allocation-free step: the scratch in a static device array
// ============================================================================
// For callers that cannot allocate device memory (see the header).  The step
// itself is tula_ags_step; only where its scratch lives differs.

namespace {

constexpr size_t kStaticScratchBytes = TULA_STATIC_SCRATCH_BYTES;
constexpr int kMaxDevices = 64;

// One copy per device, alive until the process exits.  In host code this name
// is only a handle: its device address comes from cudaGetSymbolAddress.
static __device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

std::mutex g_static_mu;
void *g_static_ptr[kMaxDevices] = {};

// Device address of g_static_scratch on the current device, looked up once per device.
int static_scratch_address(void **out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) {
        g_last_cuda = (int)e;
        return TULA_ERR_CUDA;
    }
    if (dev < 0 || dev >= kMaxDevices) return TULA_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_static_mu);
    if (!g_static_ptr[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_static_scratch);
        if (e != cudaSuccess || !p) {
            g_last_cuda = (int)e;
            return TULA_ERR_CUDA;
        }
        g_static_ptr[dev] = p;
    }
    *out = g_static_ptr[dev];
    return TULA_OK;
}

}  // namespace

extern "C" int tula_ags_step_static_scratch(float *const *param_ptrs, float *const *grad_ptrs,
                                            float *const *mom_ptrs, const int64_t *numels,
                                            int n_tensors, float lr, float momentum,
                                            float weight_decay, const tula_ags_hparams *hp,
                                            void *stream) {
    long long nch = 0;
    if (!hp || !valid_numels(numels, n_tensors, &nch)) return TULA_ERR_ARG;
    const WsLayout L = ws_layout(n_tensors, nch);
    if (L.total > kStaticScratchBytes) return TULA_ERR_SCRATCH_LIMIT;
    void *scratch = nullptr;
    int rc = static_scratch_address(&scratch);
    if (rc) return rc;
    // The array keeps the last call's contents: zero the tickets, done counter and
    // branch flag (they precede the partial sums) before this call's kernels.
    cudaError_t e = cudaMemsetAsync(scratch, 0, L.partials, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) {
        g_last_cuda = (int)e;
        return TULA_ERR_CUDA;
    }
    tula_ags_hparams local = *hp;
    local.workspace = scratch;
    local.workspace_bytes = kStaticScratchBytes;
    return tula_ags_step(param_ptrs, grad_ptrs, mom_ptrs, numels, n_tensors, lr, momentum,
                         weight_decay, &local, stream);
}
