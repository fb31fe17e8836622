// libtula_ags: the AGS optimizer step (Tula, arXiv 2603.18112) for sm_103a.
//
// Two streaming passes over every parameter tensor, load-balanced by a chunk
// table: each tensor is cut into chunks of kChunk elements (tiny tensors are one
// chunk, 100M-element tensors tens of thousands) and every chunk is one warp's
// work item, so the streaming loops contain no block-wide barrier:
//
//   k_reduce  (pass 1)  K-way replica mean (Eq. 1c) written over replica 0, and
//                       fp64 per-chunk partial sums of |gbar|^2, |g_0|^2 [, |w|^2].
//                       Partials are combined in a fixed order in two levels
//                       (32-chunk groups, then the tensor) by whichever warp takes
//                       the last ticket of a group / of a tensor; that warp also
//                       derives the tensor's statistics, its coefficient when
//                       scaled (the old gradscale, Eq. 8's s, or the LARS ratio)
//                       and, when asked, the refreshed gradscale (UpdateGradScale,
//                       Algorithm 1).  The warp finishing the last tensor forms
//                       |G|^2, Delta (Eq. 5) and the branch of Algorithm 1.
//   k_update  (pass 2)  d = c gbar + wd w; m = mu m + d; w = w - lr m (Eq. 7b with
//                       the wrapped SGD), in reverse chunk order so that it starts
//                       on the mean lines pass 1 left in L2; |w|^2 for statistics.
//
// No warp ever waits on another: hand-offs are counter tickets.  Both kernels
// are HBM-bound (a few flops per 20-70 bytes): 128-bit coalesced loads, one
// wave of resident CTAs, no tensor cores (nothing here is a contraction).  The
// chunk table, pointers and sizes travel in the kernel parameter block
// (__grid_constant__, up to ~31 KB per launch), so no host-to-device copy,
// allocation or host sync is ever needed.  The reduction order depends on the
// numels only: results are bitwise reproducible and independent of the grid.
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

constexpr int kThreads = 512;            // threads per CTA (16 independent warps)
constexpr int kChunk = 4096;             // elements per chunk = one warp's work item
constexpr int kGroup = 32;               // chunks per first-level combine group
constexpr int kParamBudget = 31 * 1024;  // kernel parameter bytes per launch (limit 32764)
constexpr int kAcc = 3;                  // partial sums per chunk: |gbar|^2, |g_0|^2, |w|^2
constexpr int kTsum = 4;                 // per-tensor sums (stride)
constexpr unsigned kFull = 0xffffffffu;

enum Mode { kModeStep = 0, kModeStats = 1, kModeScale = 2 };

// ----------------------------------------------------------------------------
// Launch tables (kernel parameters)
// ----------------------------------------------------------------------------

template <int NP>
struct Table {
    static constexpr int kMaxT = (kParamBudget - 64) / (NP * 8 + 16);
    int n;    // tensors in this launch
    int t0;   // global index of its first tensor
    int c0;   // global index of its first chunk
    int nc;   // chunks in this launch
    int g0;   // global index of its first combine group
    int pad[3];
    long long numel[kMaxT];
    int cstart[kMaxT + 1];  // first chunk of each tensor, relative to c0; cstart[n] = nc
    int gstart[kMaxT + 1];  // first group of each tensor, relative to g0
    const float *ptr[kMaxT][NP];
};

struct Scalars {
    int K, rule, gran, force, refresh, mode, n_total, read_w;
    int pow2K, pad0, pad1, pad2;
    float delta, eps, s_max, static_s, lars_trust, lr, mu, wd, invK, Kf;
    float *scale;
    double *state;
    double *stats;
    unsigned *gctr1, *gctr2;  // per-group chunk tickets, pass 1 / pass 2
    unsigned *tctr1, *tctr2;  // per-tensor group tickets, pass 1 / pass 2
    unsigned *done;           // [0]: tensors finished in pass 1
    int *flags;               // [0]: branch of the last step (1 = scaled)
    double *partials;         // [chunk][kAcc]
    double *gpart;            // [group][kAcc]
    double *tsum;             // [tensor][kTsum]: |gbar|^2, |g_0|^2, |w|^2
    float *cand;              // [tensor]: c_p of the scaled branch (AGS: the old gradscale)
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

// Warp sum in a fixed tree (lane 0's result), broadcast to every lane.
__device__ __forceinline__ double warp_sum(double v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = __dadd_rn(v, __shfl_down_sync(kFull, v, o));
    return __shfl_sync(kFull, v, 0);
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

// Where a chunk sits: its tensor, its range and the global indices of its
// tensor's first chunk and first group.
struct ChunkPos {
    int t, tg, c_in_t, nch, ngr;
    long long begin, end, cfirst, gfirst;
};

template <int NP>
__device__ __forceinline__ ChunkPos locate(const Table<NP> &tab, int c) {
    ChunkPos q;
    q.t = find_tensor(tab.cstart, tab.n, c);
    q.tg = tab.t0 + q.t;
    q.c_in_t = c - tab.cstart[q.t];
    q.nch = tab.cstart[q.t + 1] - tab.cstart[q.t];
    q.ngr = tab.gstart[q.t + 1] - tab.gstart[q.t];
    q.begin = (long long)q.c_in_t * kChunk;
    q.end = min(q.begin + (long long)kChunk, tab.numel[q.t]);
    q.cfirst = (long long)tab.c0 + tab.cstart[q.t];
    q.gfirst = (long long)tab.g0 + tab.gstart[q.t];
    return q;
}

// Hand-off of one chunk's partial sums (every lane holds acc[]).  Lane 0 stores
// them and takes a ticket of the chunk's 32-chunk group; the warp holding the
// group's last ticket adds the group's partials (lane i <- chunk i, then a
// fixed tree) and takes a ticket of the tensor; the warp holding the tensor's
// last ticket adds the group sums (lane-strided in order, then a fixed tree).
// Returns true, with the tensor's sums in tot[] (every lane), on that warp only.
// Counters are re-armed to zero by the warp that took their last ticket.
template <int NA>
__device__ __forceinline__ bool hand_off(const double (&acc)[NA], int slot, const ChunkPos &q,
                                         double *partials, double *gpart, unsigned *gctr,
                                         unsigned *tctr, double (&tot)[NA]) {
    const int lane = threadIdx.x & 31;
    const int grp = q.c_in_t / kGroup;
    const int gsize = min(kGroup, q.nch - grp * kGroup);
    const long long cg = q.cfirst + q.c_in_t;
    const long long gg = q.gfirst + grp;
    int last = 0;
    if (lane == 0) {
#pragma unroll
        for (int a = 0; a < NA; ++a) partials[cg * kAcc + slot + a] = acc[a];
        __threadfence();
        last = atomicAdd(&gctr[gg], 1u) == (unsigned)(gsize - 1);
    }
    if (!__shfl_sync(kFull, last, 0)) return false;
    __threadfence();
    double g[NA];
    const long long c0 = q.cfirst + (long long)grp * kGroup;
#pragma unroll
    for (int a = 0; a < NA; ++a) {
        g[a] = lane < gsize ? __ldcg(&partials[(c0 + lane) * kAcc + slot + a]) : 0.0;
        g[a] = warp_sum(g[a]);
    }
    if (q.ngr == 1) {  // a single group is the whole tensor
        if (lane == 0) gctr[gg] = 0u;
#pragma unroll
        for (int a = 0; a < NA; ++a) tot[a] = g[a];
        return true;
    }
    last = 0;
    if (lane == 0) {
#pragma unroll
        for (int a = 0; a < NA; ++a) gpart[gg * kAcc + slot + a] = g[a];
        gctr[gg] = 0u;
        __threadfence();
        last = atomicAdd(&tctr[q.tg], 1u) == (unsigned)(q.ngr - 1);
    }
    if (!__shfl_sync(kFull, last, 0)) return false;
    __threadfence();
#pragma unroll
    for (int a = 0; a < NA; ++a) tot[a] = 0.0;
    for (int i = lane; i < q.ngr; i += 32) {
#pragma unroll
        for (int a = 0; a < NA; ++a)
            tot[a] = __dadd_rn(tot[a], __ldcg(&gpart[(q.gfirst + i) * kAcc + slot + a]));
    }
#pragma unroll
    for (int a = 0; a < NA; ++a) tot[a] = warp_sum(tot[a]);
    if (lane == 0) tctr[q.tg] = 0u;
    return true;
}

// ----------------------------------------------------------------------------
// Per-tensor results of pass 1 (lane 0 of the warp that finished the tensor)
// ----------------------------------------------------------------------------

__device__ void tensor_done(const Scalars &sc, int tg, double sg, double ss, double sw) {
    double *T = sc.tsum + (size_t)tg * kTsum;
    T[0] = sg;
    T[1] = ss;
    T[2] = sw;
    double *row = sc.stats ? sc.stats + (size_t)tg * TULA_STATS_LEN : nullptr;
    if (sc.mode == kModeScale) {
        sc.scale[tg] = scale_tensor(ss, sg, sc);  // g_0 = g_large, small = g_small
        return;
    }
    if (sc.mode == kModeStats) {
        row[TULA_STAT_W_SQ] = sw;
        row[TULA_STAT_G_SQ] = sg;
        row[TULA_STAT_G0_SQ] = ss;
        row[TULA_STAT_W_NORM] = sqrt(sw);
        row[TULA_STAT_G_NORM] = sqrt(sg);
        row[TULA_STAT_RATIO] = sg > 0.0 ? sqrt(sw) / sqrt(sg) : 0.0;
        row[TULA_STAT_COEF] = 0.0;
        row[TULA_STAT_SCALE] = 0.0;
        return;
    }
    // kModeStep: the coefficient this tensor gets when the step is scaled (Algorithm 1,
    // Eq. 8) or always (LARS), before UpdateGradScale may overwrite gradscale.
    const float old = sc.scale ? sc.scale[tg] : 1.0f;
    float cand;
    switch (sc.rule) {
    case TULA_RULE_AGS: cand = old; break;
    case TULA_RULE_STATIC: cand = sc.static_s; break;
    case TULA_RULE_LARS:
        cand = (sw > 0.0 && sg > 0.0) ? (float)((double)sc.lars_trust * (sqrt(sw) / sqrt(sg)))
                                      : 1.0f;
        break;
    default: cand = 1.0f;
    }
    sc.cand[tg] = cand;
    float s_after = sc.scale ? old : 0.0f;
    if (sc.refresh && sc.scale) {
        s_after = scale_tensor(ss, sg, sc);
        sc.scale[tg] = s_after;
    }
    if (row) {
        row[TULA_STAT_G_SQ] = sg;
        row[TULA_STAT_G0_SQ] = ss;
        row[TULA_STAT_G_NORM] = sqrt(sg);
        row[TULA_STAT_SCALE] = (double)s_after;
        if (sc.read_w) {
            row[TULA_STAT_W_SQ] = sw;
            row[TULA_STAT_W_NORM] = sqrt(sw);
            row[TULA_STAT_RATIO] = sg > 0.0 ? sqrt(sw) / sqrt(sg) : 0.0;
        }
    }
}

// |G|^2, Delta (Eq. 5) and the branch of Algorithm 1 (one warp, after every
// tensor's sums are in sc.tsum).
__device__ void finalize_step(const Scalars &sc) {
    const int lane = threadIdx.x & 31;
    double v = 0.0;
    for (int t = lane; t < sc.n_total; t += 32)
        v = __dadd_rn(v, __ldcg(&sc.tsum[(size_t)t * kTsum + 0]));
    const double g2 = warp_sum(v);
    if (lane != 0) return;
    const double g2_prev = sc.state[TULA_STATE_G2_PREV];
    const double steps = sc.state[TULA_STATE_STEPS];
    // no previous step -> +inf (sensitive)
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
    sc.done[0] = 0u;  // re-arm for the next call
}

// ----------------------------------------------------------------------------
// Pass 1: replica mean + per-tensor squared norms
// ----------------------------------------------------------------------------
//
// Template: KT = replicas known at compile time (0: runtime K <= 16);
// WM = write the mean over replica 0; RW = also reduce |w|^2;
// SS = g_small is a separate stream (role KS + 1) instead of replica 0;
// PR = precise norms: every exact fp64 square is added in fp64 (relative error
// ~1e-15), for norms that feed a per-tensor coefficient (UpdateGradScale, LARS);
// otherwise each lane sums <= 16 squares in fp32 before one fp64 add (~1e-7),
// which is what the variability metric and the statistics need, at a fraction
// of GB300's FP64 rate.
// Pointer roles per tensor: [0, K) replicas, KS = w, KS + 1 = g_small.

template <int KT>
struct P1 {
    static constexpr int KS = KT > 0 ? KT : TULA_MAX_K;
    static constexpr int NP = KS + 2;
};

template <int KT, bool WM, bool RW, bool SS, bool PR>
__device__ __forceinline__ void reduce_vec(const float *const *ptr, long long begin, int nv,
                                           const Scalars &sc, double &ag, double &as,
                                           double &aw) {
    constexpr int KS = P1<KT>::KS;
    constexpr int NS = (KT > 0 ? KT : 4) + (RW ? 1 : 0) + (SS ? 1 : 0);  // streams read
    constexpr int U = NS >= 4 ? 1 : 4 / NS;  // >= 4 float4 loads per lane in flight
    constexpr int KL = KT > 0 ? KT : TULA_MAX_K;  // load slots
    const int lane = threadIdx.x & 31;
    const int K = KT > 0 ? KT : sc.K;
    const float *g[KL];
#pragma unroll
    for (int k = 0; k < KL; ++k) g[k] = (KT > 0 && k < K) ? ptr[k] + begin : nullptr;
    const float *wp = RW ? ptr[KS] + begin : nullptr;
    const float *sp = SS ? ptr[KS + 1] + begin : nullptr;
    float *out = const_cast<float *>(ptr[0]) + begin;

    if constexpr (KT == 0) {
        // K not known at compile time: replicas 1..K-1 in groups of four, k ascending.
#pragma unroll 1
        for (int v = lane; v < nv; v += 32) {
            const float4 x0 = ld_stream(ptr[0] + begin + 4 * (size_t)v);
            float4 s = x0;
            for (int k0 = 1; k0 < K; k0 += 4) {
                float4 y[4];
#pragma unroll
                for (int j = 0; j < 4; ++j)
                    if (k0 + j < K) y[j] = ld_stream(ptr[k0 + j] + begin + 4 * (size_t)v);
#pragma unroll
                for (int j = 0; j < 4; ++j)
                    if (k0 + j < K) s = add4(s, y[j]);
            }
            s = mean4(s, sc);
            if (WM) st_keep(out + 4 * (size_t)v, s);
            float4 wv = RW ? ld_stream(wp + 4 * (size_t)v) : s;
            float4 sv = SS ? ld_stream(sp + 4 * (size_t)v) : s;
            if (PR) {
                as = dsq4(as, x0);
                ag = dsq4(ag, s);
                if (SS) as = dsq4(as, sv);
                if (RW) aw = dsq4(aw, wv);
            } else {
                as = __dadd_rn(as, (double)sq4(0.f, x0));
                ag = __dadd_rn(ag, (double)sq4(0.f, s));
                if (SS) as = __dadd_rn(as, (double)sq4(0.f, sv));
                if (RW) aw = __dadd_rn(aw, (double)sq4(0.f, wv));
            }
        }
        return;
    }

#pragma unroll 1
    for (int v0 = lane; v0 < nv; v0 += 32 * U) {
        float4 x[U][KL];
        float4 wv[U], sv[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int v = v0 + u * 32;
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
            const int v = v0 + u * 32;
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
__device__ __forceinline__ void reduce_scalar(const float *const *ptr, long long j0, long long j1,
                                              const Scalars &sc, double &ag, double &as,
                                              double &aw) {
    constexpr int KS = P1<KT>::KS;
    constexpr int KL = KT > 0 ? KT : TULA_MAX_K;
    const int K = KT > 0 ? KT : sc.K;
    for (long long j = j0 + (threadIdx.x & 31); j < j1; j += 32) {
        float x0 = __ldcs(ptr[0] + j);
        float s = x0;
#pragma unroll
        for (int k = 1; k < KL; ++k)
            if (k < K) s = __fadd_rn(s, __ldcs(ptr[k] + j));
        if (K > 1) {
            s = mean1(s, sc);
            if (WM) const_cast<float *>(ptr[0])[j] = s;
            as = __fma_rn((double)x0, (double)x0, as);
        }
        ag = __fma_rn((double)s, (double)s, ag);
        if (SS) {
            const double y = __ldcs(ptr[KS + 1] + j);
            as = __fma_rn(y, y, as);
        }
        if (RW) {
            const double y = __ldcs(ptr[KS] + j);
            aw = __fma_rn(y, y, aw);
        }
    }
}

template <int KT, bool WM, bool RW, bool SS, bool PR>
__global__ void __launch_bounds__(kThreads, 2)
    k_reduce(const __grid_constant__ Table<P1<KT>::NP> tab, const __grid_constant__ Scalars sc) {
    constexpr int KS = P1<KT>::KS;
    const int K = KT > 0 ? KT : sc.K;
    const int warp = (int)((blockIdx.x * (unsigned)kThreads + threadIdx.x) >> 5);
    const int nwarps = (int)((gridDim.x * (unsigned)kThreads) >> 5);

    for (int c = warp; c < tab.nc; c += nwarps) {
        const ChunkPos q = locate(tab, c);
        const float *const *ptr = tab.ptr[q.t];
        double acc[kAcc] = {0.0, 0.0, 0.0};
        if (q.end > q.begin) {
            uintptr_t al = 0;
            for (int k = 0; k < K; ++k) al |= reinterpret_cast<uintptr_t>(ptr[k]);
            if (RW) al |= reinterpret_cast<uintptr_t>(ptr[KS]);
            if (SS) al |= reinterpret_cast<uintptr_t>(ptr[KS + 1]);
            const int nv = (al & 15u) == 0 ? (int)((q.end - q.begin) >> 2) : 0;
            if (nv > 0)
                reduce_vec<KT, WM, RW, SS, PR>(ptr, q.begin, nv, sc, acc[0], acc[1], acc[2]);
            reduce_scalar<KT, WM, RW, SS>(ptr, q.begin + 4 * (long long)nv, q.end, sc, acc[0],
                                          acc[1], acc[2]);
        }
#pragma unroll
        for (int a = 0; a < kAcc; ++a) acc[a] = warp_sum(acc[a]);
        double tot[kAcc];
        if (!hand_off<kAcc>(acc, 0, q, sc.partials, sc.gpart, sc.gctr1, sc.tctr1, tot)) continue;
        // This warp finished tensor q.tg.
        if ((threadIdx.x & 31) == 0) {
            const double ss = (K > 1 || SS) ? tot[1] : tot[0];  // K = 1: replica 0 is the mean
            tensor_done(sc, q.tg, tot[0], ss, tot[2]);
        }
        if (sc.mode != kModeStep) continue;
        int last = 0;
        if ((threadIdx.x & 31) == 0) {
            __threadfence();
            last = atomicAdd(&sc.done[0], 1u) == (unsigned)(sc.n_total - 1);
        }
        if (__shfl_sync(kFull, last, 0)) {
            __threadfence();
            finalize_step(sc);
        }
    }
}

// ----------------------------------------------------------------------------
// Pass 2: scaled momentum-SGD + weight-decay update (Eq. 7b, Algorithm 1)
// ----------------------------------------------------------------------------
// Pointer roles: 0 = gbar, 1 = w, 2 = m, 3 = per-element gradscale.
// Chunks run in reverse order: the mean pass 1 wrote last is still in L2.

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
    const int lane = threadIdx.x & 31;
    const int warp = (int)((blockIdx.x * (unsigned)kThreads + threadIdx.x) >> 5);
    const int nwarps = (int)((gridDim.x * (unsigned)kThreads) >> 5);
    const int scaled = sc.flags[0];
    const bool gated = sc.rule == TULA_RULE_AGS || sc.rule == TULA_RULE_STATIC;
    const bool use_se = PE && scaled;

    for (int i = warp; i < tab.nc; i += nwarps) {
        const int c = tab.nc - 1 - i;
        const ChunkPos q = locate(tab, c);
        const float cand = sc.cand[q.tg];
        const float ct = gated ? (scaled ? cand : 1.0f) : cand;
        if (sc.stats && q.c_in_t == 0 && lane == 0)
            sc.stats[(size_t)q.tg * TULA_STATS_LEN + TULA_STAT_COEF] =
                PE ? (scaled ? (double)NAN : 1.0) : (double)ct;
        double aw[1] = {0.0};

        if (q.end > q.begin) {
            const float *const *ptr = tab.ptr[q.t];
            const float *gp = ptr[0] + q.begin;
            float *wp = const_cast<float *>(ptr[1]) + q.begin;
            float *mp = HM ? const_cast<float *>(ptr[2]) + q.begin : nullptr;
            const float *sp = use_se ? ptr[3] + q.begin : nullptr;
            uintptr_t al = reinterpret_cast<uintptr_t>(gp) | reinterpret_cast<uintptr_t>(wp);
            if (HM) al |= reinterpret_cast<uintptr_t>(mp);
            if (use_se) al |= reinterpret_cast<uintptr_t>(sp);
            const int nv = (al & 15u) == 0 ? (int)((q.end - q.begin) >> 2) : 0;
#pragma unroll 1
            for (int v0 = lane; v0 < nv; v0 += 32 * U) {
                float4 gv[U], wv[U], mv[U], sv[U];
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    const int v = v0 + u * 32;
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
                    const int v = v0 + u * 32;
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
            const long long n = q.end - q.begin;
            for (long long j = 4 * (long long)nv + lane; j < n; j += 32) {
                const float g = __ldcs(gp + j);
                float w = __ldcs(wp + j);
                float m = HM ? __ldcs(mp + j) : 0.f;
                float cj = use_se ? __ldcs(sp + j) : (PE ? 1.f : ct);
                if (SW) aw[0] = __fma_rn((double)w, (double)w, aw[0]);
                sgd1(g, cj, w, m, sc, HM);
                __stcs(wp + j, w);
                if (HM) __stcs(mp + j, m);
            }
        }
        if (!SW) continue;
        aw[0] = warp_sum(aw[0]);
        double tot[1];
        if (!hand_off<1>(aw, 2, q, sc.partials, sc.gpart, sc.gctr2, sc.tctr2, tot)) continue;
        if (lane == 0) {
            const double sw = tot[0];
            const double sg = __ldcg(&sc.tsum[(size_t)q.tg * kTsum + 0]);
            double *row = sc.stats + (size_t)q.tg * TULA_STATS_LEN;
            row[TULA_STAT_W_SQ] = sw;
            row[TULA_STAT_W_NORM] = sqrt(sw);
            row[TULA_STAT_RATIO] = sg > 0.0 ? sqrt(sw) / sqrt(sg) : 0.0;
        }
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
    const int lane = threadIdx.x & 31;
    const int warp = (int)((blockIdx.x * (unsigned)kThreads + threadIdx.x) >> 5);
    const int nwarps = (int)((gridDim.x * (unsigned)kThreads) >> 5);
    for (int c = warp; c < tab.nc; c += nwarps) {
        const ChunkPos q = locate(tab, c);
        if (q.end <= q.begin) continue;
        const float *const *ptr = tab.ptr[q.t];
        const float *a = ptr[0] + q.begin;
        const float *b = ptr[1] + q.begin;
        float *o = const_cast<float *>(ptr[2]) + q.begin;
        const uintptr_t al = reinterpret_cast<uintptr_t>(a) | reinterpret_cast<uintptr_t>(b) |
                             reinterpret_cast<uintptr_t>(o);
        const int nv = (al & 15u) == 0 ? (int)((q.end - q.begin) >> 2) : 0;
        for (int v = lane; v < nv; v += 32) {
            const float4 x = ld_stream(a + 4 * (size_t)v), y = ld_stream(b + 4 * (size_t)v);
            st_stream(o + 4 * (size_t)v, make_float4(scale1(x.x, y.x, sc), scale1(x.y, y.y, sc),
                                                     scale1(x.z, y.z, sc), scale1(x.w, y.w, sc)));
        }
        const long long n = q.end - q.begin;
        for (long long j = 4 * (long long)nv + lane; j < n; j += 32)
            o[j] = scale1(__ldcs(a + j), __ldcs(b + j), sc);
    }
}

// ----------------------------------------------------------------------------
// Host side
// ----------------------------------------------------------------------------

std::atomic<uint64_t> g_launches{0};
thread_local int g_last_cuda = 0;

inline long long chunks_of(int64_t n) { return n <= 0 ? 1 : (n + kChunk - 1) / kChunk; }
inline long long groups_of(long long nch) { return (nch + kGroup - 1) / kGroup; }

struct Plan {
    long long chunks = 0, groups = 0;
};

// Workspace layout.  Every counter and flag precedes `partials`, so zeroing
// [0, partials) clears all of them.
struct WsLayout {
    size_t gctr1, gctr2, tctr1, tctr2, done, flags, partials, gpart, tsum, cand, total;
};

WsLayout ws_layout(int n_tensors, const Plan &pl) {
    size_t off = 0;
    auto take = [&](size_t bytes) {
        size_t o = off;
        off = (off + bytes + 255) & ~size_t(255);
        return o;
    };
    WsLayout L;
    L.gctr1 = take(sizeof(unsigned) * (size_t)pl.groups);
    L.gctr2 = take(sizeof(unsigned) * (size_t)pl.groups);
    L.tctr1 = take(sizeof(unsigned) * (size_t)n_tensors);
    L.tctr2 = take(sizeof(unsigned) * (size_t)n_tensors);
    L.done = take(sizeof(unsigned) * 4);
    L.flags = take(sizeof(int) * 4);
    L.partials = take(sizeof(double) * kAcc * (size_t)pl.chunks);
    L.gpart = take(sizeof(double) * kAcc * (size_t)pl.groups);
    L.tsum = take(sizeof(double) * kTsum * (size_t)n_tensors);
    L.cand = take(sizeof(float) * (size_t)n_tensors);
    L.total = off;
    return L;
}

bool valid_numels(const int64_t *numels, int n, Plan *pl) {
    if (!numels || n < 1) return false;
    Plan p;
    for (int i = 0; i < n; ++i) {
        if (numels[i] < 0) return false;
        const long long c = chunks_of(numels[i]);
        p.chunks += c;
        p.groups += groups_of(c);
        if (p.chunks >= (1LL << 31)) return false;
    }
    *pl = p;
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

// Splits tensors [0, n) into parameter blocks and launches `kernel` once per
// block (in reverse block order when `reverse`).  fill(p, ptrs) writes tensor
// p's pointers.
template <int NP, typename Kernel, typename Fill>
int launch_groups(Kernel kernel, int n, const int64_t *numels, const Scalars &sc, int grid_override,
                  cudaStream_t stream, Fill fill, bool reverse = false) {
    using T = Table<NP>;
    int grid_cap = grid_override > 0 ? grid_override : resident_ctas((const void *)kernel);
    if (grid_cap <= 0) {
        g_last_cuda = (int)cudaGetLastError();
        return TULA_ERR_CUDA;
    }
    std::vector<std::unique_ptr<T>> tabs;
    long long c_global = 0, g_global = 0;
    int p = 0;
    while (p < n) {
        std::unique_ptr<T> tab(new T);
        std::memset(tab.get(), 0, sizeof(T));
        tab->t0 = p;
        tab->c0 = (int)c_global;
        tab->g0 = (int)g_global;
        int cnt = 0, nc = 0, ng = 0;
        while (p < n && cnt < T::kMaxT) {
            tab->numel[cnt] = numels[p];
            tab->cstart[cnt] = nc;
            tab->gstart[cnt] = ng;
            fill(p, tab->ptr[cnt]);
            const long long c = chunks_of(numels[p]);
            nc += (int)c;
            ng += (int)groups_of(c);
            ++cnt;
            ++p;
        }
        tab->n = cnt;
        tab->nc = nc;
        tab->cstart[cnt] = nc;
        tab->gstart[cnt] = ng;
        c_global += nc;
        g_global += ng;
        tabs.push_back(std::move(tab));
    }
    if (reverse) std::reverse(tabs.begin(), tabs.end());
    for (const auto &tab : tabs) {
        const int need = (tab->nc + kThreads / 32 - 1) / (kThreads / 32);  // one warp per chunk
        const int grid = std::max(1, std::min(need, grid_cap));
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
    sc.gctr1 = reinterpret_cast<unsigned *>(b + L.gctr1);
    sc.gctr2 = reinterpret_cast<unsigned *>(b + L.gctr2);
    sc.tctr1 = reinterpret_cast<unsigned *>(b + L.tctr1);
    sc.tctr2 = reinterpret_cast<unsigned *>(b + L.tctr2);
    sc.done = reinterpret_cast<unsigned *>(b + L.done);
    sc.flags = reinterpret_cast<int *>(b + L.flags);
    sc.partials = reinterpret_cast<double *>(b + L.partials);
    sc.gpart = reinterpret_cast<double *>(b + L.gpart);
    sc.tsum = reinterpret_cast<double *>(b + L.tsum);
    sc.cand = reinterpret_cast<float *>(b + L.cand);
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

int check_ws(void *ws, size_t bytes, int n, const Plan &pl) {
    if (!ws) return TULA_ERR_WORKSPACE;
    if (bytes < ws_layout(n, pl).total) return TULA_ERR_WORKSPACE;
    if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return TULA_ERR_WORKSPACE;
    return TULA_OK;
}

void record(void *ev, cudaStream_t s) {
    if (ev) cudaEventRecord(static_cast<cudaEvent_t>(ev), s);
}

inline int replica_slot(int K) {
    return (K == 1 || K == 2 || K == 4 || K == 8 || K == 16) ? K : TULA_MAX_K;
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
    Plan pl;
    if (!bytes || K < 1 || K > TULA_MAX_K || !valid_numels(numels, n_tensors, &pl))
        return TULA_ERR_ARG;
    *bytes = ws_layout(n_tensors, pl).total;
    return TULA_OK;
}

int tula_ags_chunk_elems(void) { return kChunk; }

int tula_ags_plan_chunks(const int64_t *numels, int n_tensors, int64_t *chunk_start_out) {
    Plan pl;
    if (!chunk_start_out || !valid_numels(numels, n_tensors, &pl)) return TULA_ERR_ARG;
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
    Plan pl;
    if (!hp || !param_ptrs || !grad_ptrs || !valid_numels(numels, n_tensors, &pl))
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
    int rc = check_ws(hp->workspace, hp->workspace_bytes, n, pl);
    if (rc) return rc;

    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const WsLayout L = ws_layout(n, pl);
    Scalars sc = make_scalars(hp, K, n, hp->workspace, L, kModeStep);
    const bool lars = hp->rule == TULA_RULE_LARS;
    sc.read_w = lars ? 1 : 0;
    sc.lr = lr;
    sc.mu = momentum;
    sc.wd = weight_decay;

    const int KS = replica_slot(K);
    auto fill1 = [&](int p, const float **dst) {
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
    launch_groups<kNP2>(k_update<HM, PE, SW>, n, numels, sc, hp->grid_ctas, s, fill2, true)
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
    Plan pl;
    if (!param_ptrs || !grad_ptrs || !stats_out || !valid_numels(numels, n_tensors, &pl))
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
    int rc = check_ws(workspace, workspace_bytes, n, pl);
    if (rc) return rc;
    const WsLayout L = ws_layout(n, pl);
    Scalars sc = make_scalars(nullptr, K, n, workspace, L, kModeStats);
    sc.stats = stats_out;
    sc.read_w = 1;
    const int KS = replica_slot(K);
    auto fill = [&](int p, const float **dst) {
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
    Plan pl;
    if (!hp || !g_small || !g_large || !valid_numels(numels, n_tensors, &pl)) return TULA_ERR_ARG;
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
    int rc = check_ws(hp->workspace, hp->workspace_bytes, n, pl);
    if (rc) return rc;
    const WsLayout L = ws_layout(n, pl);
    Scalars sc = make_scalars(hp, 1, n, hp->workspace, L, kModeScale);
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
    Plan pl;
    if (!hp || !valid_numels(numels, n_tensors, &pl)) return TULA_ERR_ARG;
    const WsLayout L = ws_layout(n_tensors, pl);
    if (L.total > kStaticScratchBytes) return TULA_ERR_SCRATCH_LIMIT;
    void *scratch = nullptr;
    int rc = static_scratch_address(&scratch);
    if (rc) return rc;
    // The array keeps the last call's contents: zero the tickets, counters and
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
