// libtula_ags: the AGS optimizer step (Tula, arXiv 2603.18112) for sm_103a.
//
// Per step, four kernels on the caller's stream, chained by programmatic
// dependent launch so that each one's launch and prologue overlap the tail of
// the one before:
//
//   k_reduce   (pass 1)  K-way replica mean (Eq. 1c) written over replica 0; each
//                        tile's sums of |gbar|^2, |g_0|^2 [, |w|^2] are added
//                        exactly into per-tensor accumulators (and |gbar|^2 into
//                        the step's |G|^2 accumulator) by L2 atomics.
//   k_finish             per tensor, the norms rounded from its accumulators, its
//                        statistics, its coefficient when scaled (the old
//                        gradscale, Eq. 8's s, or the LARS ratio) and, when
//                        asked, the refreshed gradscale (UpdateGradScale,
//                        Algorithm 1); one more warp forms |G|^2, Delta (Eq. 5)
//                        and the branch of Algorithm 1.
//   k_update   (pass 2)  d = c gbar + wd w; m = mu m + d; w = w - lr m (Eq. 7b with
//                        the wrapped SGD); |w|^2 per tile for the statistics,
//   k_finish             then rounded per tensor.
//
// The streaming passes: each tensor is cut into tiles of T elements (T fixed
// per pass by how many tensors it streams, so that one tile of every stream
// fills one shared-memory stage: 36 KB in pass 1, 24 KB in pass 2).  One
// persistent CTA per SM; small launches deal tiles round-robin, larger ones
// claim them from a global counter (SMs stream at unequal rates).  The producer
// warp moves tiles from HBM into the stage ring with TMA bulk copies
// (cp.async.bulk ... mbarrier::complete_tx), one copy per stream issued by one
// lane each; consumer warps, each owning whole stages, compute from shared
// memory and release the stage through an mbarrier.  Tile partials are fp32
// sums within a tile (float-float pairs per lane in the precise mode for norms
// that feed a coefficient), range-checked per tile, and leave the tile only as
// exact integer additions into the accumulators.
//
// Every mbarrier wait is bounded; a wait that runs out sets an error word in
// the workspace (tula_ags_workspace_error) and the CTA drains its copies in
// flight and returns.  The streaming kernels are HBM-bound (a few flops per
// 20-70 bytes); nothing here is a contraction, so no tensor cores.  The tile
// table, pointers and sizes travel in the kernel parameter block
// (__grid_constant__, up to ~31 KB per launch): no host-to-device copy,
// allocation or host sync is ever needed.  Integer addition does not depend on
// the order in which tiles land, so results are bitwise reproducible and
// independent of the grid and of which CTA took which tile.
#include "tula_ags.h"

#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <memory>
#include <mutex>
#include <new>
#include <type_traits>
#include <utility>
#include <vector>

namespace {

// A stage ring: kStages shared-memory stages of kStageBytes each (one tile of
// every stream), one producer warp and kConsumers consumer warps.  A consumer
// must own whole stages: the tile it waits for on a stage is then always the
// one after its own previous tile there, so a parity wait never sees a phase
// two ahead.
template <int StageKB, int Stages, int Consumers>
struct Ring {
    static constexpr int kStageBytes = StageKB * 1024;
    static constexpr int kStages = Stages;
    static constexpr int kConsumers = Consumers;
    static constexpr int kThreads = 32 * (1 + Consumers);
    static constexpr int kSmemBytes = Stages * kStageBytes + 2 * Stages * 8 + Stages * 4;
    static_assert(Stages % Consumers == 0, "consumers own whole stages");
    static_assert(kSmemBytes <= 227 * 1024, "one CTA per SM");
    // Elements per tile when `streams` tensors share one stage (multiple of 128).
    __host__ __device__ static constexpr int tile_elems(int streams) {
        return (kStageBytes / (4 * streams)) / 128 * 128;
    }
};
// Pass 1 streams K (+1, +2) tensors through 36 KB stages.  Six consumer warps, two per
// scheduler: the precise norms spend ~13 dependent FP32 instructions per element and norm, and
// the default ones add their tile sums into the accumulators at the end of each batch; with
// three warps the reduction ran 0.8 % slower alone (the same step time).
using Ring1 = Ring<36, 6, 6>;
// Pass 1 when it also reads w (LARS, tula_layer_stats) streams through five 45 KB stages with
// five consumers: the larger tiles (1280 elements for K = 8 and w) make every bulk copy 5 KB
// instead of 4 KB, and the LARS step ran 2.5 % faster (ResNet-50, 248.1 -> 241.9 us); without
// w (8 streams) the same ring measured 0.5 % slower.
using Ring1W = Ring<45, 5, 5>;
template <bool RW>
using Ring1Of = std::conditional_t<RW, Ring1W, Ring1>;
// Pass 2 does ~11 flops per element over 3-4 streams: with three consumer warps they, not HBM,
// set its pace, so it runs four.
using Ring2 = Ring<24, 8, 4>;
constexpr int kDynTiles = 64;            // tiles per CTA from which a launch claims its tiles
constexpr unsigned kClaim = 4;           // tiles per claim
constexpr unsigned kClaimTail = 16;      // single-tile claims for the last kClaimTail per CTA
constexpr int kPend = 4;                // tiles whose warp reductions run together
constexpr int kFinWarps = 4;            // k_finish: one warp per tensor, 4 per CTA
constexpr int kParamBudget = 31 * 1024; // kernel parameter bytes per launch (limit 32764)
constexpr int kAcc = 3;                 // partial sums per pass-1 tile: |gbar|^2, |g_0|^2, |w|^2
constexpr int kPrecCols = 1;            // float4 columns per step of the precise path's tile loop
constexpr int kTsum = 4;                // per-tensor sums (stride)
constexpr unsigned kFull = 0xffffffffu;
constexpr uint32_t kSpinLimit = 1u << 19;  // bound on every mbarrier wait (~2 s on GB300)

enum Mode { kModeStep = 0, kModeStats = 1, kModeScale = 2, kModeUpdate = 3 };


// ----------------------------------------------------------------------------
// Launch tables (kernel parameters)
// ----------------------------------------------------------------------------

template <int NP>
struct Table {
    static constexpr int kMaxT = (kParamBudget - 64) / (NP * 8 + 12);
    int n;      // tensors in this launch
    int t0;     // global index of its first tensor
    int c0;     // global index of its first tile
    int nc;     // tiles in this launch
    int chunk;  // elements per tile
    int first;  // 1 for the first launch of the pass (in issue order)
    int pad[2];
    long long numel[kMaxT];
    int cstart[kMaxT + 1];  // first tile of each tensor, relative to c0; cstart[n] = nc
    const float *ptr[kMaxT][NP];
};

struct Scalars {
    int K, rule, gran, force, refresh, mode, n_total, read_w;
    int pow2K, evict_first, fin2, pad2;  // evict_first: TMA loads ask L2 to drop their lines first;
                                         // fin2: a finish kernel follows the update
    float delta, eps, s_max, static_s, lars_trust, lr, mu, wd, invK, Kf;
    float *scale;
    double *state;
    double *stats;
    int *flags;                // [0]: branch of the last step (1 = scaled)
    unsigned *err;             // [0]: bounded waits that ran out (sticky until read)
    unsigned long long *acc1;  // [tensor][kAcc][kTCopies][kAccWords]: |gbar|^2, |g_0|^2, |w|^2
    unsigned long long *gacc;  // [kGCopies][kAccWords]: |G|^2 = every tensor's |gbar|^2
    unsigned long long *acc2;  // [tensor][kTCopies][kAccWords]: |w|^2, pass 2
    double *tsum;              // [tensor][kTsum]: |gbar|^2, |g_0|^2, |w|^2
    float *cand;               // [tensor]: c_p of the scaled branch (AGS: the old gradscale)
    unsigned *tiles;           // [2 * pass]: next tile to claim, [2 * pass + 1]: CTAs finished
    const unsigned long long *g2ext;  // a sharded step's |G|^2: the ranks' shares summed (or NULL)
};

// ----------------------------------------------------------------------------
// Device helpers: memory, arithmetic
// ----------------------------------------------------------------------------

__device__ __forceinline__ void st_stream(float *p, float4 v) {
    __stcs(reinterpret_cast<float4 *>(p), v);
}
__device__ __forceinline__ void st_keep(float *p, float4 v) {
    *reinterpret_cast<float4 *>(p) = v;
}
// 16-byte load from shared memory (a shared-window address).
__device__ __forceinline__ float4 lds4(uint32_t addr) {
    float4 v;
    asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "r"(addr));
    return v;
}

// fp32 sum of squares into a running fp32 partial, one FFMA per term
__device__ __forceinline__ float sq4(float acc, float4 v) {
    acc = __fmaf_rn(v.x, v.x, acc);
    acc = __fmaf_rn(v.y, v.y, acc);
    acc = __fmaf_rn(v.z, v.z, acc);
    acc = __fmaf_rn(v.w, v.w, acc);
    return acc;
}

__device__ __forceinline__ float4 add4(float4 a, float4 b) {
    return make_float4(__fadd_rn(a.x, b.x), __fadd_rn(a.y, b.y), __fadd_rn(a.z, b.z),
                       __fadd_rn(a.w, b.w));
}

// Eq. 1c: divide the k-ascending sum by K (exact reciprocal when K is a power of 2)
template <int KT>
__device__ __forceinline__ float mean1(float s, const Scalars &sc) {
    if constexpr (KT > 0 && (KT & (KT - 1)) == 0) {
        return __fmul_rn(s, 1.0f / (float)KT);
    } else if constexpr (KT > 0) {
        return __fdiv_rn(s, (float)KT);
    } else {
        return sc.pow2K ? __fmul_rn(s, sc.invK) : __fdiv_rn(s, sc.Kf);
    }
}
template <int KT>
__device__ __forceinline__ float4 mean4(float4 s, const Scalars &sc) {
    return make_float4(mean1<KT>(s.x, sc), mean1<KT>(s.y, sc), mean1<KT>(s.z, sc),
                       mean1<KT>(s.w, sc));
}


// Fixed-tree warp sum of R values at once (lane 0 gets the sums); the R chains
// are independent, so their shuffle and fp64 add latencies overlap.
template <int R>
__device__ __forceinline__ void warp_sums(double (&v)[R]) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        double t[R];
#pragma unroll
        for (int r = 0; r < R; ++r) t[r] = __shfl_down_sync(kFull, v[r], o);
#pragma unroll
        for (int r = 0; r < R; ++r) v[r] = __dadd_rn(v[r], t[r]);
    }
}

template <int R>
__device__ __forceinline__ void warp_sums(float (&v)[R]) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        float t[R];
#pragma unroll
        for (int r = 0; r < R; ++r) t[r] = __shfl_down_sync(kFull, v[r], o);
#pragma unroll
        for (int r = 0; r < R; ++r) v[r] = __fadd_rn(v[r], t[r]);
    }
}

// Warp reduce-scatter of R values per lane (R a power of two, <= 32): each of log2(R) halving
// steps sends half of a lane's values to the lane `off` away and keeps the sums of the other
// half; the remaining steps add the one value left across the lanes still sharing it.
// Afterwards every lane holds the warp total of value `index` (bits of the lane id reversed):
// with R = 16, lanes 2i and 2i + 1 hold the same one.  16 + 1 shuffles for R = 16 instead of
// the 5 R of a tree per value, so the owners of R sums can store them at once.  The order of
// the additions is fixed (results do not depend on timing), and the two lanes that end with
// the same sum add the same two terms.
__device__ __forceinline__ float add_rn(float a, float b) { return __fadd_rn(a, b); }
__device__ __forceinline__ double add_rn(double a, double b) { return __dadd_rn(a, b); }
template <int R, typename T>
__device__ __forceinline__ T warp_reduce_scatter(T (&v)[R], int &index) {
    static_assert(R >= 1 && R <= 32 && (R & (R - 1)) == 0, "R: a power of two <= 32");
    const int lane = threadIdx.x & 31;
    int idx = 0, off = 16;
#pragma unroll
    for (int h = R / 2; h >= 1; h >>= 1, off >>= 1) {
        const bool up = (lane & off) != 0;
#pragma unroll
        for (int j = 0; j < h; ++j) {
            const T send = up ? v[j] : v[j + h];
            const T keep = up ? v[j + h] : v[j];
            v[j] = add_rn(keep, __shfl_xor_sync(kFull, send, off));
        }
        if (up) idx += h;
    }
#pragma unroll
    for (; off >= 1; off >>= 1) v[0] = add_rn(v[0], __shfl_xor_sync(kFull, v[0], off));
    index = idx;
    return v[0];
}

// Float-float numbers (hi, lo as a float2, value hi + lo, |lo| <= ulp(hi) / 2)
// carry the precise path's per-lane sums: they hold ~48 significant bits and
// add on the FP32 pipes, where an fp64 add costs ~64x more on this part.
// Knuth's TwoSum: s + e == a + b exactly.
__device__ __forceinline__ float2 two_sum(float a, float b) {
    const float s = __fadd_rn(a, b);
    const float bb = __fsub_rn(s, a);
    const float e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
    return make_float2(s, e);
}
// a + b for float-float a, b: TwoSum of the high parts, the low parts added to
// the error, then Dekker's Fast2Sum to renormalise.  All terms here are sums of
// squares (no cancellation): relative error below 2^-46 per addition.
__device__ __forceinline__ float2 ff_add(float2 a, float2 b) {
    const float2 s = two_sum(a.x, b.x);
    const float e = __fadd_rn(s.y, __fadd_rn(a.y, b.y));
    const float hi = __fadd_rn(s.x, e);
    return make_float2(hi, __fsub_rn(e, __fsub_rn(hi, s.x)));
}
__device__ __forceinline__ double ff_to_double(float2 v) {
    return __dadd_rn((double)v.x, (double)v.y);
}

// Precise sums of squares on the FP32 pipes.  x*x == p + e exactly, with
// p = fl(x*x) and e = fma(x, x, -p), unless p overflows or e underflows.  p
// joins the running high part by TwoSum, both error terms join the low part,
// and Fast2Sum renormalises the pair, so each addition errs by at most ~2u^2 of
// the running sum (u = 2^-24) with no fp64 instruction; one pair per float4
// component keeps four independent chains in flight.  The streaming loop has no
// range test (a branch there would cost more than the arithmetic): an overflow
// shows as a non-finite pair, and an underflowed e errs by at most 2^-149, so a
// lane sum of at least 2^-77 is as good as exact; dw_lane_ok tests both once
// per tile, and the tile is redone in fp64 when a lane fails.
struct Dw4 {
    float hi[4], lo[4];
};
__device__ __forceinline__ void dw_zero(Dw4 &a) {
#pragma unroll
    for (int c = 0; c < 4; ++c) a.hi[c] = a.lo[c] = 0.f;
}
__device__ __forceinline__ void dw_sq(float &hi, float &lo, float x) {
    const float p = __fmul_rn(x, x);
    const float e = __fmaf_rn(x, x, -p);
    const float2 t = two_sum(hi, p);
    const float l = __fadd_rn(lo, __fadd_rn(t.y, e));
    hi = __fadd_rn(t.x, l);
    lo = __fsub_rn(l, __fsub_rn(hi, t.x));
}
__device__ __forceinline__ void dw_sq4(Dw4 &a, float4 v) {
    dw_sq(a.hi[0], a.lo[0], v.x);
    dw_sq(a.hi[1], a.lo[1], v.y);
    dw_sq(a.hi[2], a.lo[2], v.z);
    dw_sq(a.hi[3], a.lo[3], v.w);
}
// The four pairs added in a fixed tree.
__device__ __forceinline__ float2 dw_pair(const Dw4 &a) {
    const float2 c01 = ff_add(make_float2(a.hi[0], a.lo[0]), make_float2(a.hi[1], a.lo[1]));
    const float2 c23 = ff_add(make_float2(a.hi[2], a.lo[2]), make_float2(a.hi[3], a.lo[3]));
    return ff_add(c01, c23);
}
__device__ __forceinline__ bool dw_lane_ok(float2 v) {
    return v.x >= 0x1p-77f && v.x <= 3.0e38f;  // false for 0, tiny sums, inf and NaN
}

// Exact powers of two (k within the normal range of the type).
__device__ __forceinline__ float pow2f(int k) { return __int_as_float((k + 127) << 23); }

// Range of a tile's fp32 sums of squares, decided for the whole warp from the largest lane
// sum v (>= 0, or NaN): 0 when every lane sum is safe as it stands, else the exponent e of a
// power-of-two scaling 2^e to apply to the elements before squaring them again.
//  * max in [2^-100, 2^120]: nothing overflows (32 lanes add to < 2^125), and squares or partial
//    sums that fell below fp32's normal range err by at most 2^-150 each, < 2^-38 of the tile
//    sum: kept.
//  * max above 2^120, inf or NaN: a square or a sum reached fp32's top.  Scaled by 2^-72 every
//    finite element is below 2^56, its square below 2^112, a lane's sum of up to 288 squares
//    below 2^121 and the tile's below 2^126; what the scaling pushes below 2^-149 has a square
//    under 2^-254 of the tile sum.  Inf and NaN stay inf and NaN.
//  * max below 2^-100 (zero included): every element is below 2^-50 in magnitude (a sum of
//    squares is at least its largest term), so 2^100 x is exact, below 2^50, and its square is a
//    normal number unless x is 0.
constexpr int kScaleUp = 100, kScaleDown = -72;
// Two-bit codes of those exponents, for the partial sums a batch of tiles carries.
__device__ __forceinline__ unsigned scale_code(int e) { return e == 0 ? 0u : (e > 0 ? 1u : 2u); }
__device__ __forceinline__ int scale_exp(unsigned code) {
    return code == 0u ? 0 : (code == 1u ? kScaleUp : kScaleDown);
}
__device__ __forceinline__ bool sq_in_range(float v) {
    return v >= 0x1p-100f && v <= 0x1p120f;  // false for NaN
}
__device__ __forceinline__ int sq_range_exp(float v) {
    const unsigned m = __reduce_max_sync(kFull, __float_as_uint(v));
    if (m > __float_as_uint(0x1p120f)) return kScaleDown;
    if (m < __float_as_uint(0x1p-100f)) return kScaleUp;
    return 0;
}
__device__ __forceinline__ float4 mul4(float4 v, float f) {
    return make_float4(__fmul_rn(v.x, f), __fmul_rn(v.y, f), __fmul_rn(v.z, f), __fmul_rn(v.w, f));
}

// ----------------------------------------------------------------------------
// Exact accumulation of the squared norms
// ----------------------------------------------------------------------------
//
// The partial sums of squares (one per tile and norm, all >= 0) are added up exactly, in
// integers: an accumulator is a fixed-point number of kAccDigits 32-bit digits, digit i of
// weight 2^(32 i + kAccBase), each held in the low half of a 64-bit word whose high half
// collects carries.  A partial m * 2^E (m an fp32 or fp64 significand) touches two or three
// consecutive words, each by an atomic add that nothing waits for (red.global.add.u64).
// Integer addition is associative, so the sum does not depend on the order the tiles land in:
// norms are bitwise reproducible for any grid and any claim order, and they are the exact sums
// of the tile partials, rounded once to fp64 when read (acc_to_double).
//
// Range: the partials are fp32 tile sums scaled by 2^k (k in {0, -200, 144}, sq_range_exp) or
// fp64 sums of exact squares of fp32 numbers, so their bits lie within 2^-352 .. 2^273; a tensor
// of up to 2^31 tiles, or all tensors together, stays below 2^305; 21 digits from 2^-352 cover
// 2^-352 .. 2^320.  Each word takes at most two adds (< 2^32 each) per tile, so its high half
// cannot overflow for fewer than 2^31 tiles.  A partial that is inf or NaN (an inf or NaN
// element) sets a flag in the last word instead: the norm is then inf, or NaN.
//
// Copies: the tiles of one tensor land close together in time, and every tile of a step adds
// into |G|^2, so one word would take an atomic every few ns, about what an L2 slice can do for
// one address.  Each accumulator therefore has copies, picked by the CTA, that the reading warp
// adds up (exact; all copies together still take fewer than 2^32 adds per word).
constexpr int kAccDigits = 21;
constexpr int kAccWords = 24;             // digits, two spare words, the flags
constexpr int kAccFlags = kAccWords - 1;  // bit 0: an inf partial, bit 1: a NaN partial
constexpr int kAccBase = -352;
constexpr int kTCopies = 2;               // copies of each per-tensor accumulator
constexpr int kGCopies = 8;               // copies of the |G|^2 accumulator
static_assert(kAccDigits <= kAccFlags && kAccWords <= 32, "one word per lane");
static_assert((kTCopies & (kTCopies - 1)) == 0 && (kGCopies & (kGCopies - 1)) == 0, "powers of 2");

// Adds m * 2^E (m < 2^53, kAccBase <= E, E + 53 <= 2^32 weight of the top digit) to A.
__device__ __forceinline__ void acc_add(unsigned long long *A, unsigned long long m, int E) {
    if (m == 0ull) return;
    const int s = E - kAccBase;
    const int i = s >> 5, r = s & 31;
    const unsigned long long lo = m << r;
    const unsigned long long hi = r ? (m >> (64 - r)) : 0ull;
    if (lo & 0xffffffffull) atomicAdd(A + i, lo & 0xffffffffull);
    if (lo >> 32) atomicAdd(A + i + 1, lo >> 32);
    if (hi) atomicAdd(A + i + 2, hi);
}
// Adds f * 2^k for an fp32 f >= 0 (or inf, NaN).
__device__ __forceinline__ void acc_add_f32(unsigned long long *A, float f, int k) {
    const unsigned u = __float_as_uint(f);
    const unsigned e = (u >> 23) & 0xffu;
    if (e == 0xffu) {
        atomicOr(A + kAccFlags, (u & 0x7fffffu) ? 2ull : 1ull);
        return;
    }
    const unsigned long long m = e ? ((u & 0x7fffffu) | 0x800000u) : (u & 0x7fffffu);
    acc_add(A, m, (e ? (int)e : 1) - 150 + k);
}
// Adds an fp64 d >= 0 (or inf, NaN).
__device__ __forceinline__ void acc_add_f64(unsigned long long *A, double d) {
    const unsigned long long u = (unsigned long long)__double_as_longlong(d);
    const unsigned e = (unsigned)(u >> 52) & 0x7ffu;
    const unsigned long long f = u & 0xfffffffffffffull;
    if (e == 0x7ffu) {
        atomicOr(A + kAccFlags, f ? 2ull : 1ull);
        return;
    }
    acc_add(A, e ? (f | (1ull << 52)) : f, (e ? (int)e : 1) - 1075);
}

// The values of R accumulators rounded to the nearest double (ties to even), by the whole
// warp: lane i passes word i of each (any value for lanes >= kAccWords).  Carries first move up
// one word (each high half, < 2^32, into the next digit), which leaves at most one carry per
// digit; those ripple through runs of all-ones digits, found for all 32 digits at once with two
// votes and one integer addition (the carry-lookahead of an adder).  Then the top three digits
// give the 53-bit significand, its round bit and, with every digit below, its sticky bit.  The
// R conversions go stage by stage together, so their shuffle and vote latencies overlap.
template <int R>
__device__ __forceinline__ void acc_to_double(const unsigned long long (&wi)[R], double (&out)[R]) {
    const int lane = threadIdx.x & 31;
    unsigned long long flags[R], v[R];
    unsigned d[R], nz[R];
#pragma unroll
    for (int r = 0; r < R; ++r) flags[r] = __shfl_sync(kFull, wi[r], kAccFlags);
#pragma unroll
    for (int r = 0; r < R; ++r) {
        const unsigned long long w = lane < kAccDigits ? wi[r] : 0ull;
        const unsigned long long up = __shfl_up_sync(kFull, w >> 32, 1);
        v[r] = (w & 0xffffffffull) + (lane > 0 ? up : 0ull);  // < 2^33
    }
#pragma unroll
    for (int r = 0; r < R; ++r) {
        const unsigned G = __ballot_sync(kFull, (v[r] >> 32) != 0ull);
        const unsigned P = __ballot_sync(kFull, (v[r] & 0xffffffffull) == 0xffffffffull);
        const unsigned carries = ((G | P) + G) ^ (G | P) ^ G;  // bit i: a carry into digit i
        d[r] = (unsigned)(v[r] + ((carries >> lane) & 1u));
    }
#pragma unroll
    for (int r = 0; r < R; ++r) nz[r] = __ballot_sync(kFull, d[r] != 0u);
#pragma unroll
    for (int r = 0; r < R; ++r) {
        const int top = nz[r] ? 31 - __clz(nz[r]) : 0;
        const unsigned d0 = __shfl_sync(kFull, d[r], top);
        const unsigned d1 = __shfl_sync(kFull, d[r], top > 0 ? top - 1 : 0);
        const unsigned d2 = __shfl_sync(kFull, d[r], top > 1 ? top - 2 : 0);
        if (flags[r] & 2ull) {
            out[r] = __longlong_as_double(0x7ff8000000000000ll);  // NaN
        } else if (flags[r] & 1ull) {
            out[r] = __longlong_as_double(0x7ff0000000000000ll);  // +inf
        } else if (nz[r] == 0u) {
            out[r] = 0.0;
        } else {
            const unsigned m1 = top > 0 ? d1 : 0u, m2 = top > 1 ? d2 : 0u;
            const bool below = top > 2 && (nz[r] & ((1u << (top - 2)) - 1u)) != 0u;
            const int L = 32 - __clz(d0);  // bit length of the top digit
            const int z = 32 - L;          // shift that puts its leading 1 at bit 63
            const unsigned long long hi = ((unsigned long long)d0 << 32) | m1;
            const unsigned long long T = (hi << z) | (z ? ((unsigned long long)m2 >> (32 - z)) : 0ull);
            const bool rest = (m2 & (0xffffffffu >> z)) != 0u;  // bits of m2 below T
            unsigned long long mant = T >> 11;
            const bool round = (T >> 10) & 1ull;
            const bool sticky = (T & 0x3ffull) != 0ull || rest || below;
            int ex = 32 * top + kAccBase + L - 1;  // weight of the leading bit
            if (round && (sticky || (mant & 1ull))) {
                if (++mant == (1ull << 53)) {
                    mant >>= 1;
                    ++ex;
                }
            }
            out[r] = __longlong_as_double(
                (long long)(((unsigned long long)(ex + 1023) << 52) | (mant & 0xfffffffffffffull)));
        }
    }
}

// ----------------------------------------------------------------------------
// Device helpers: programmatic dependent launch, mbarrier, TMA (inline PTX)
// ----------------------------------------------------------------------------

// Wait for the grids this one depends on to complete and their memory to be
// visible, then let the next grid in the stream begin launching.
__device__ __forceinline__ void grid_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void grid_launch_dependents() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

__device__ __forceinline__ uint32_t smem_addr(const void *p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count)
                 : "memory");
}
__device__ __forceinline__ void mbar_fence_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive_tx(uint64_t *bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)),
                 "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_test(uint64_t *bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_addr(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}
// Waits for the phase of `bar` with this parity to complete; gives up after
// kSpinLimit tries (returns false).  try_wait suspends the thread in hardware
// until the phase completes or a short time limit passes; only a wait that is
// already far too long backs off with a sleep.
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity) {
    for (uint32_t i = 0; i < kSpinLimit; ++i) {
        if (mbar_test(bar, parity)) return true;
        if (i >= (1u << 16)) __nanosleep(256);
    }
    return false;
}
// One TMA bulk copy global -> shared, completing `bytes` of `bar`'s transaction count.
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void *src, uint32_t bytes,
                                         uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
            "r"(dst),
        "l"(src), "r"(bytes), "r"(smem_addr(bar))
        : "memory");
}
// The same with an L2 cache policy for the source lines.
__device__ __forceinline__ void bulk_g2s_hint(uint32_t dst, const void *src, uint32_t bytes,
                                              uint64_t *bar, uint64_t policy) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1], %2, [%3], %4;" ::"r"(dst),
        "l"(src), "r"(bytes), "r"(smem_addr(bar)), "l"(policy)
        : "memory");
}
// L2 policy: these lines are the first to go.
__device__ __forceinline__ uint64_t policy_evict_first() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}


__device__ __forceinline__ void report_timeout(const Scalars &sc) {
    atomicOr(sc.err, 1u);
}

// ----------------------------------------------------------------------------
// Tile table lookups
// ----------------------------------------------------------------------------

__device__ __forceinline__ int find_tensor(const int *cstart, int n, int c) {
    int lo = 0, hi = n;  // cstart[lo] <= c < cstart[hi]
    while (hi - lo > 1) {
        int mid = (lo + hi) >> 1;
        if (cstart[mid] <= c) lo = mid; else hi = mid;
    }
    return lo;
}

// Follows the tensor index along a monotone sequence of tiles (one CTA's tiles,
// ascending or descending): O(1) per tile instead of a search.
struct Walker {
    int t = -1;
    template <int NP>
    __device__ __forceinline__ int to(const Table<NP> &tab, int c) {
        if (t < 0) return t = find_tensor(tab.cstart, tab.n, c);
        while (c >= tab.cstart[t + 1]) ++t;
        while (c < tab.cstart[t]) --t;
        return t;
    }
};

// A tile: its tensor, its element range.
struct TilePos {
    int t, tg, c_in_t;
    long long begin, end;
};

template <int NP>
__device__ __forceinline__ TilePos locate(const Table<NP> &tab, int c, int t, int chunk) {
    TilePos q;
    q.t = t;
    q.tg = tab.t0 + t;
    q.c_in_t = c - tab.cstart[t];
    q.begin = (long long)q.c_in_t * chunk;
    q.end = min(q.begin + (long long)chunk, tab.numel[t]);
    return q;
}

// Float4 a tile moves by TMA: its 16-byte body when every stream of the tensor
// is 16-byte aligned (lane i < ns holds stream i's pointer), else none.
__device__ __forceinline__ int tile_vecs(const float *mine, int ns, const TilePos &q) {
    if (q.end <= q.begin) return 0;
    const unsigned low = (threadIdx.x & 31) < ns ? (unsigned)(reinterpret_cast<uintptr_t>(mine) & 15u)
                                                 : 0u;
    return __reduce_or_sync(kFull, low) == 0u ? (int)((q.end - q.begin) >> 2) : 0;
}

// The tensor of the previous tile, kept while the next tile stays in it: its
// index, its streams' alignment and the lane's stream pointer, so a tile in
// the same tensor needs no table look-up.
struct TensorCache {
    Walker walk;
    int t = -1;
    long long numel = 0;
    const float *mine = nullptr;
    bool aligned = false;
    int nv = 0;  // float4 moved by TMA for the last tile asked for
    template <int NP>
    __device__ __forceinline__ TilePos at(const Table<NP> &tab, int c, int chunk, int role, int ns) {
        const int tn = walk.to(tab, c);
        if (tn != t) {
            t = tn;
            numel = tab.numel[t];
            mine = (threadIdx.x & 31) < ns ? tab.ptr[t][role] : nullptr;
            const unsigned low =
                (threadIdx.x & 31) < ns ? (unsigned)(reinterpret_cast<uintptr_t>(mine) & 15u) : 0u;
            aligned = __reduce_or_sync(kFull, low) == 0u;
        }
        TilePos q;
        q.t = t;
        q.tg = tab.t0 + t;
        q.c_in_t = c - tab.cstart[t];
        q.begin = (long long)q.c_in_t * chunk;
        q.end = min(q.begin + (long long)chunk, numel);
        nv = (aligned && q.end > q.begin) ? (int)((q.end - q.begin) >> 2) : 0;
        return q;
    }
};

// ----------------------------------------------------------------------------
// The producer: TMA bulk copies of each tile's streams into the stage ring
// ----------------------------------------------------------------------------
//
// Two ways to deal a launch's tiles to its persistent CTAs:
//  * round-robin (tile blockIdx.x + j * gridDim.x), for launches of fewer than
//    kDynTiles tiles per CTA: nothing to claim, nothing to wait for;
//  * claimed, for larger launches: the producer warp of each CTA takes kClaim
//    consecutive tiles at a time from a global counter (ctr[0]), with one
//    claim in flight while it issues the range before (see produce()).  SMs
//    do not stream at equal rates (on
//    large launches the last CTA of a round-robin deal finished 15-30% after
//    the median), so claiming lets the faster SMs take more tiles and the
//    launch end with the memory system rather than with its slowest SM.  The
//    last CTA to finish puts both counters (ctr[0], ctr[1]) back to zero.
// Where a tile is processed never changes its result: each tile's partial sums
// are added exactly, in integers, into its tensor's accumulators.  The j-th
// tile of a CTA goes to stage j % kStages and is consumed by consumer warp
// j % kConsumers; its launch tile index is left in stage_tile[stage] before the
// stage's full barrier is armed (the barrier's release/acquire orders it), and
// -1 there tells a consumer that no tile is left.  Lane i < ns of the producer
// fetches stream i's pointer (role roles[i]) and issues that stream's copy to
// offset i * chunk floats of the stage.  Both passes walk the tiles in the same
// order (measured: walking pass 2 backwards, to start on the mean pass 1 wrote
// last, was 1 % slower per step).

__device__ __forceinline__ unsigned claim_tiles(unsigned *ctr, unsigned n) {
    return atomicAdd(ctr, n);
}

// Round-robin tiles of this CTA (0 when the launch claims its tiles).
__device__ __forceinline__ int static_tiles(int nc) {
    const int g = (int)gridDim.x, b = (int)blockIdx.x;
    if (nc >= kDynTiles * g) return 0;
    return b < nc ? (nc - b + g - 1) / g : 0;
}
__device__ __forceinline__ bool claims_tiles(int nc) { return nc >= kDynTiles * (int)gridDim.x; }
__device__ __forceinline__ int static_tile(int j) { return (int)blockIdx.x + j * (int)gridDim.x; }

template <typename R, int NP, int NS>
__device__ __forceinline__ void produce(const Table<NP> &tab, const Scalars &sc,
                                        const int (&roles)[NS], int ns, int chunk,
                                        int js, unsigned *ctr, uint32_t ring,
                                        uint64_t *full, uint64_t *empty, int *stage_tile) {
    const int lane = threadIdx.x & 31;
    const int role = lane < ns ? roles[lane] : 0;
    const unsigned nc = (unsigned)tab.nc;
    const bool claim = claims_tiles(tab.nc);
    const bool hint = sc.evict_first != 0;
    const uint64_t policy = policy_evict_first();
    TensorCache tc;
    // Claiming (lane 0): tiles [cur, cur_end) are being issued, [nxt, nxt_end) come next and
    // one claim is in flight.  The first two ranges of each CTA are dealt, not claimed (152
    // CTAs claiming at once would queue on the counter at the start); claimed ranges begin
    // after them.  Near the end, claims shrink to one tile so that CTAs do not hold tiles
    // others could have taken.
    const unsigned G = gridDim.x, b = blockIdx.x;
    const unsigned base = 2u * G * kClaim;
    unsigned cur = b * kClaim, cur_end = cur + kClaim;
    unsigned nxt = (G + b) * kClaim, nxt_end = nxt + kClaim;
    unsigned pend = 0u, pend_k = kClaim;
    if (claim && lane == 0) pend = claim_tiles(ctr, kClaim);
    int issued = 0, ending = 0;
    for (int j = 0; ending < R::kConsumers; ++j) {
        const int s = j % R::kStages;
        unsigned i = nc;  // past the end: an end marker
        if (j < js) {
            i = blockIdx.x + (unsigned)j * gridDim.x;
        } else if (claim) {
            if (lane == 0) {
                if (cur == cur_end) {
                    cur = nxt;
                    cur_end = nxt_end;
                    if (nxt < nc) {  // the counter only grows: no more claims once past the end
                        nxt = base + pend;
                        nxt_end = nxt + pend_k;
                        if (nxt < nc) {
                            pend_k = nxt + kClaimTail * G >= nc ? 1u : kClaim;
                            pend = claim_tiles(ctr, pend_k);
                        }
                    }
                }
                i = cur++;
            }
            i = __shfl_sync(kFull, i, 0);
        }
        if (j >= R::kStages) {
            int w = 1;
            if (lane == 0) w = mbar_wait(&empty[s], (uint32_t)((j / R::kStages - 1) & 1));
            if (!__shfl_sync(kFull, w, 0)) {
                if (lane == 0) report_timeout(sc);
                break;
            }
        }
        if (i >= nc) {  // one end marker per consumer warp
            if (lane == 0) {
                stage_tile[s] = -1;
                mbar_arrive_tx(&full[s], 0u);
            }
            ++ending;
            issued = j + 1;
            continue;
        }
        const int c = (int)i;
        const TilePos q = tc.at(tab, c, chunk, role, ns);
        const uint32_t bytes = 16u * (uint32_t)tc.nv;
        if (lane == 0) {
            stage_tile[s] = c;
            mbar_arrive_tx(&full[s], bytes * (uint32_t)ns);
        }
        __syncwarp();
        if (bytes && lane < ns) {
            const uint32_t dst = ring + (uint32_t)s * R::kStageBytes + (uint32_t)(lane * chunk * 4);
            if (hint) bulk_g2s_hint(dst, tc.mine + q.begin, bytes, &full[s], policy);
            else bulk_g2s(dst, tc.mine + q.begin, bytes, &full[s]);
        }
        issued = j + 1;
    }
    // Drain: never leave the CTA with a copy still writing into its shared memory.
    if (lane == 0) {
        for (int s = 0; s < R::kStages && s < issued; ++s) {
            const int jl = s + ((issued - 1 - s) / R::kStages) * R::kStages;  // last tile on stage s
            if (!mbar_wait(&full[s], (uint32_t)((jl / R::kStages) & 1))) report_timeout(sc);
        }
        // Every claim of this CTA is performed before it counts itself finished;
        // the last CTA re-arms the counters for the next launch.
        if (claim) {
            __threadfence();
            if (atomicAdd(ctr + 1, 1u) == gridDim.x - 1u) {
                atomicExch(ctr, 0u);
                atomicExch(ctr + 1, 0u);
            }
        }
    }
}

// Shared prologue of the streaming kernels: barrier init.
template <typename R>
__device__ __forceinline__ void ring_setup(unsigned char *smem, uint64_t *&full, uint64_t *&empty,
                                           int *&stage_tile) {
    full = reinterpret_cast<uint64_t *>(smem + R::kStages * R::kStageBytes);
    empty = full + R::kStages;
    stage_tile = reinterpret_cast<int *>(empty + R::kStages);
    if (threadIdx.x == 0) {
        for (int s = 0; s < R::kStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_fence_init();
    }
    __syncthreads();
}

// A consumer's wait for its j-th tile: the launch tile index, -1 when no tile
// is left, -2 when the wait ran out (reported).  Called by the whole warp; the
// result is the same in every lane (a lane whose bounded wait ran out makes
// the warp stop), so the warp stays converged for its shuffles and votes.
template <typename R>
__device__ __forceinline__ int next_tile(const Scalars &sc, int j, uint64_t *full,
                                         const int *stage_tile) {
    const int s = j % R::kStages;
    if (!__all_sync(kFull, mbar_wait(&full[s], (uint32_t)((j / R::kStages) & 1)))) {
        if ((threadIdx.x & 31) == 0) report_timeout(sc);
        return -2;
    }
    return *reinterpret_cast<const volatile int *>(stage_tile + s);
}

// ----------------------------------------------------------------------------
// Pass 1: replica mean + per-tile squared norms
// ----------------------------------------------------------------------------
//
// Template: KT = replicas known at compile time (0: runtime K <= 16);
// WM = write the mean over replica 0; RW = also reduce |w|^2;
// SS = g_small is a separate stream instead of replica 0;
// PR = precise norms: every square is split exactly into two fp32 parts and
// added as a float-float pair (Dw4), each lane's pairs go to fp64 once per tile,
// and the tile's lanes are added in an fp64 tree (relative error ~1e-14), for
// norms that feed a per-tensor coefficient (UpdateGradScale, LARS).  Otherwise the tile's sum
// stays in fp32: each lane adds <= 16 squares per group of 4 columns, then the
// group sums, then a 5-level tree across lanes, a relative error below 71 ulp
// (4e-6) of the tile's sum; tiles are added exactly into the tensor's
// accumulator.  That is what the
// variability metric and the statistics need, and it keeps GB300's slow FP64
// pipe out of the streaming loop.  One warp vote per tile (sq_range_exp) keeps
// it valid over the whole fp32 range: a tile whose fp32 sums would overflow or
// lose precision to underflow is summed again from shared memory with its
// elements scaled by an exact power of two, and the scaling is undone in fp64.
// Pointer roles per tensor: [0, K) replicas, KS = w, KS + 1 = g_small.
// Stage streams: replicas 0..K-1, then w (RW), then g_small (SS).

template <int KT>
struct P1 {
    static constexpr int KS = KT > 0 ? KT : TULA_MAX_K;
    static constexpr int NP = KS + 2;
};

// One float4 column of a tile: mean, squares.  x0 = replica 0, s = sum.
template <int KT, bool WM, bool RW, bool SS, bool PR>
__device__ __forceinline__ void column1(float4 x0, float4 s, float4 wv, float4 sv, float *out,
                                        const Scalars &sc, int K, Dw4 &ag, Dw4 &as, Dw4 &aw,
                                        float &pg, float &ps, float &pw) {
    if (K > 1) {
        s = mean4<KT>(s, sc);
        if (WM) st_keep(out, s);
    }
    if (PR) {
        dw_sq4(ag, s);
        if (K > 1) dw_sq4(as, x0);
        if (SS) dw_sq4(as, sv);
        if (RW) dw_sq4(aw, wv);
    } else {
        pg = sq4(pg, s);
        if (K > 1) ps = sq4(ps, x0);
        if (SS) ps = sq4(ps, sv);
        if (RW) pw = sq4(pw, wv);
    }
}

// A tile's shared-memory columns again, every square exact in fp64 and added
// in fp64: the precise path's fallback when a lane's float-float sum is not
// finite or too small to hold its error (dw_lane_ok).  Out of line, so that
// the streaming loop keeps its shape.
struct D3 {
    double g, s, w;
};
template <int KT, bool RW, bool SS>
__device__ __noinline__ D3 tile_cols_fp64(uint32_t stage, int chunk, int nv, const Scalars &sc) {
    const int lane = threadIdx.x & 31;
    const int K = KT > 0 ? KT : sc.K;
    const uint32_t sw_s = stage + (uint32_t)(K * chunk * 4);
    const uint32_t ss_s = stage + (uint32_t)((K + (RW ? 1 : 0)) * chunk * 4);
    D3 r = {0.0, 0.0, 0.0};
    for (int v = lane; v < nv; v += 32) {
        const float4 x0 = lds4(stage + (uint32_t)(16 * v));
        float4 s = x0;
        for (int k = 1; k < K; ++k) s = add4(s, lds4(stage + (uint32_t)((k * chunk + 4 * v) * 4)));
        if (K > 1) s = mean4<KT>(s, sc);
        const float gs[4] = {s.x, s.y, s.z, s.w};
        const float g0[4] = {x0.x, x0.y, x0.z, x0.w};
        float4 wv = make_float4(0.f, 0.f, 0.f, 0.f), sv = wv;
        if (RW) wv = lds4(sw_s + (uint32_t)(16 * v));
        if (SS) sv = lds4(ss_s + (uint32_t)(16 * v));
        const float ws[4] = {wv.x, wv.y, wv.z, wv.w};
        const float ss[4] = {sv.x, sv.y, sv.z, sv.w};
        for (int c = 0; c < 4; ++c) {
            r.g = __fma_rn((double)gs[c], (double)gs[c], r.g);
            if (K > 1) r.s = __fma_rn((double)g0[c], (double)g0[c], r.s);
            if (SS) r.s = __fma_rn((double)ss[c], (double)ss[c], r.s);
            if (RW) r.w = __fma_rn((double)ws[c], (double)ws[c], r.w);
        }
    }
    return r;
}

// A tile's shared-memory columns again in fp32, every element multiplied by an exact power of
// two first (sq_range_exp): the default path's fallback when a tile's fp32 sums of squares
// would overflow or lose their precision to underflow.  Returns this lane's sums of the scaled
// squares.  Out of line, so that the streaming loop keeps its shape.
struct F3 {
    float g, s, w;
};
template <int KT, bool RW, bool SS>
__device__ __noinline__ F3 tile_cols_scaled(uint32_t stage, int chunk, int nv, const Scalars &sc,
                                            float fg, float fs, float fw) {
    const int lane = threadIdx.x & 31;
    const int K = KT > 0 ? KT : sc.K;
    const uint32_t sw_s = stage + (uint32_t)(K * chunk * 4);
    const uint32_t ss_s = stage + (uint32_t)((K + (RW ? 1 : 0)) * chunk * 4);
    F3 r = {0.f, 0.f, 0.f};
    for (int v = lane; v < nv; v += 32) {
        const float4 x0 = lds4(stage + (uint32_t)(16 * v));
        float4 s = x0;
        for (int k = 1; k < K; ++k) s = add4(s, lds4(stage + (uint32_t)((k * chunk + 4 * v) * 4)));
        if (K > 1) s = mean4<KT>(s, sc);
        r.g = sq4(r.g, mul4(s, fg));
        if (K > 1) r.s = sq4(r.s, mul4(x0, fs));
        if (SS) r.s = sq4(r.s, mul4(lds4(ss_s + (uint32_t)(16 * v)), fs));
        if (RW) r.w = sq4(r.w, mul4(lds4(sw_s + (uint32_t)(16 * v)), fw));
    }
    return r;
}

// Per-lane partial sums of one tile (not yet reduced across the warp).  Precise mode (PR):
// accd holds the lane's fp64 sums.  Default mode: accf holds the lane's fp32 sums over the
// tile's shared-memory columns, scaled by 2^(2 acce) (acce is the same in every lane), and accd
// the lane's exact fp64 sums over the elements loaded directly (tail, misaligned tensor).
template <int KT, bool WM, bool RW, bool SS, bool PR>
__device__ __forceinline__ void reduce_tile(uint32_t stage, int chunk, const float *const *ptr,
                                            const TilePos &q, int nv, const Scalars &sc,
                                            double (&accd)[kAcc], float (&accf)[kAcc],
                                            int (&acce)[kAcc], unsigned &ecode, bool &tail) {
    constexpr int KS = P1<KT>::KS;
    const int lane = threadIdx.x & 31;
    const int K = KT > 0 ? KT : sc.K;
    const uint32_t sw_s = stage + (uint32_t)(K * chunk * 4);
    const uint32_t ss_s = stage + (uint32_t)((K + (RW ? 1 : 0)) * chunk * 4);
    float *out = const_cast<float *>(ptr[0]) + q.begin;
    Dw4 ag, as, aw;                       // precise (PR) sums of the shared-memory columns
    dw_zero(ag);
    dw_zero(as);
    dw_zero(aw);
    double rg = 0.0, rs = 0.0, rw = 0.0;  // exact fp64 sums of the elements loaded directly
    const int ncols = nv;                 // the shared-memory columns (nv is reused below)
    tail = false;                         // the tile has elements loaded one by one
    ecode = 0u;                           // scale_code of acce[a] in bits 2a, 2a + 1
    float fg = 0.f, fs = 0.f, fw = 0.f;   // fp32 sums (not PR)

    if constexpr (KT > 0) {
        constexpr int CH = Ring1Of<RW>::tile_elems(KT + (RW ? 1 : 0) + (SS ? 1 : 0));
        constexpr int COLS = CH / 128;  // float4 columns per lane of a full tile
        if (nv == CH / 4) {
            // Full tile: every lane has COLS columns; all loads of a column issue together.
            // The loop over groups of G columns stays rolled: unrolled over the tile (and
            // again for each of the kPend tiles), the body outgrows the instruction cache.
            // The precise path's float-float arithmetic takes kPrecCols columns per group.
            constexpr int G = PR ? kPrecCols : 4;
#pragma unroll 1
            for (int c0 = 0; c0 < COLS; c0 += G) {
                float pg = 0.f, ps = 0.f, pw = 0.f;
#pragma unroll
                for (int u = 0; u < G; ++u) {
                    if (c0 + u < COLS) {
                        const int v = lane + 32 * (c0 + u);
                        float4 x[KT];
#pragma unroll
                        for (int k = 0; k < KT; ++k)
                            x[k] = lds4(stage + (uint32_t)((k * CH + 4 * v) * 4));
                        const float4 wv = RW ? lds4(sw_s + (uint32_t)(16 * v)) : x[0];
                        const float4 sv = SS ? lds4(ss_s + (uint32_t)(16 * v)) : x[0];
                        float4 s = x[0];
#pragma unroll
                        for (int k = 1; k < KT; ++k) s = add4(s, x[k]);
                        column1<KT, WM, RW, SS, PR>(x[0], s, wv, sv, out + 4 * v, sc, K, ag, as,
                                                    aw, pg, ps, pw);
                    }
                }
                if (!PR) {
                    fg = __fadd_rn(fg, pg);
                    if (K > 1 || SS) fs = __fadd_rn(fs, ps);
                    if (RW) fw = __fadd_rn(fw, pw);
                }
            }
            nv = -1;  // done
        }
    }
    if (nv >= 0) {
        // Ragged tile, or K known only at run time.
        for (int v0 = lane; v0 < nv; v0 += 32 * 4) {
            float pg = 0.f, ps = 0.f, pw = 0.f;
            for (int u = 0; u < 4; ++u) {
                const int v = v0 + 32 * u;
                if (v >= nv) break;
                const float4 x0 = lds4(stage + (uint32_t)(16 * v));
                float4 s = x0;
                for (int k = 1; k < K; ++k)
                    s = add4(s, lds4(stage + (uint32_t)((k * chunk + 4 * v) * 4)));
                const float4 wv = RW ? lds4(sw_s + (uint32_t)(16 * v)) : x0;
                const float4 sv = SS ? lds4(ss_s + (uint32_t)(16 * v)) : x0;
                column1<KT, WM, RW, SS, PR>(x0, s, wv, sv, out + 4 * v, sc, K, ag, as, aw, pg, ps,
                                            pw);
            }
            if (!PR) {
                fg = __fadd_rn(fg, pg);
                if (K > 1 || SS) fs = __fadd_rn(fs, ps);
                if (RW) fw = __fadd_rn(fw, pw);
            }
        }
        // Tail (< 4 elements) or a misaligned tensor: plain loads from global memory, exact
        // squares in fp64 (this is where replica 0 is overwritten, so there is no second look).
        tail = q.begin + 4 * (long long)nv < q.end;  // the same in every lane
        for (long long j = q.begin + 4 * (long long)nv + lane; j < q.end; j += 32) {
            const float x0 = __ldcs(ptr[0] + j);
            float s = x0;
            for (int k = 1; k < K; ++k) s = __fadd_rn(s, __ldcs(ptr[k] + j));
            if (K > 1) {
                s = mean1<KT>(s, sc);
                if (WM) const_cast<float *>(ptr[0])[j] = s;
            }
            const float y_s = SS ? __ldcs(ptr[KS + 1] + j) : 0.f;
            const float y_w = RW ? __ldcs(ptr[KS] + j) : 0.f;
            if (K > 1) rs = __fma_rn((double)x0, (double)x0, rs);
            rg = __fma_rn((double)s, (double)s, rg);
            if (SS) rs = __fma_rn((double)y_s, (double)y_s, rs);
            if (RW) rw = __fma_rn((double)y_w, (double)y_w, rw);
        }
    }
    if (PR) {
        // The warp is converged again here (the loops above end in every lane).
        const float2 pg = dw_pair(ag), ps = dw_pair(as), pw = dw_pair(aw);
        const bool bad = lane < ncols && !(dw_lane_ok(pg) && (!(K > 1 || SS) || dw_lane_ok(ps)) &&
                                           (!RW || dw_lane_ok(pw)));
        double cg, cs, cw;
        if (__any_sync(kFull, bad)) {
            const D3 f = tile_cols_fp64<KT, RW, SS>(stage, chunk, ncols, sc);
            cg = f.g;
            cs = f.s;
            cw = f.w;
        } else {
            cg = ff_to_double(pg);
            cs = ff_to_double(ps);
            cw = ff_to_double(pw);
        }
        accd[0] = __dadd_rn(cg, rg);
        accd[1] = (K > 1 || SS) ? __dadd_rn(cs, rs) : accd[0];  // K = 1: replica 0 is the mean
        accd[2] = RW ? __dadd_rn(cw, rw) : 0.0;
    } else {
        // The warp is converged again here; ncols is the same in every lane.
        int eg = 0, es = 0, ew = 0;
        // One vote per tile; the warp maxima only when some lane is out of range.  A lane
        // without columns (lane >= ncols) has nothing to check.
        const bool lane_ok = lane >= ncols || (sq_in_range(fg) && (!(K > 1 || SS) || sq_in_range(fs)) &&
                                               (!RW || sq_in_range(fw)));
        if (ncols > 0 && !__all_sync(kFull, lane_ok)) {
            eg = sq_range_exp(fg);
            if (K > 1 || SS) es = sq_range_exp(fs);
            if (RW) ew = sq_range_exp(fw);
            if (eg | es | ew) {
                const F3 r = tile_cols_scaled<KT, RW, SS>(stage, chunk, ncols, sc, pow2f(eg),
                                                          pow2f(es), pow2f(ew));
                if (eg) fg = r.g;
                if (es) fs = r.s;
                if (ew) fw = r.w;
                const bool own = K > 1 || SS;
                ecode = scale_code(eg) | scale_code(own ? es : eg) << 2 | scale_code(ew) << 4;
            }
        }
        const bool own_s = K > 1 || SS;  // K = 1: replica 0 is the mean
        accf[0] = fg;
        acce[0] = eg;
        accd[0] = rg;
        accf[1] = own_s ? fs : fg;
        acce[1] = own_s ? es : eg;
        accd[1] = own_s ? rs : rg;
        accf[2] = fw;
        acce[2] = ew;
        accd[2] = rw;
    }
}

static_assert(kPend == 4, "the owner lanes below pick one of four tiles");

// This CTA's copies of the accumulators: tensor tg's pass-1 norm a, |G|^2, tensor tg's |w|^2
// in pass 2.
__device__ __forceinline__ unsigned long long *acc1_of(const Scalars &sc, int tg, int a) {
    return sc.acc1 + (((size_t)tg * kAcc + a) * kTCopies + (blockIdx.x & (kTCopies - 1))) * kAccWords;
}
__device__ __forceinline__ unsigned long long *gacc_of(const Scalars &sc) {
    return sc.gacc + (size_t)(blockIdx.x & (kGCopies - 1)) * kAccWords;
}
__device__ __forceinline__ unsigned long long *acc2_of(const Scalars &sc, int tg) {
    return sc.acc2 + ((size_t)tg * kTCopies + (blockIdx.x & (kTCopies - 1))) * kAccWords;
}

// A default-mode tile with elements loaded one by one (the last tile of a tensor whose size is
// not a multiple of 4, or a misaligned tensor): its sums are reduced across the warp at once,
// fp32 part and fp64 part, and lane 0 adds both into the tensor's accumulators.
__device__ __noinline__ void add_tile_now(const Scalars &sc, int tg, const float (&accf)[kAcc],
                                          const int (&acce)[kAcc], const double (&accd)[kAcc]) {
    float f[kAcc];
    double d[kAcc];
#pragma unroll
    for (int a = 0; a < kAcc; ++a) {
        f[a] = accf[a];
        d[a] = accd[a];
    }
    warp_sums<kAcc>(f);
    warp_sums<kAcc>(d);
    if ((threadIdx.x & 31) == 0) {
#pragma unroll
        for (int a = 0; a < kAcc; ++a) {
            acc_add_f32(acc1_of(sc, tg, a), f[a], -2 * acce[a]);
            acc_add_f64(acc1_of(sc, tg, a), d[a]);
        }
        if (sc.mode == kModeStep) {
            acc_add_f32(gacc_of(sc), f[0], -2 * acce[0]);
            acc_add_f64(gacc_of(sc), d[0]);
        }
    }
}

template <int KT, bool WM, bool RW, bool SS, bool PR>
__global__ void __launch_bounds__(Ring1Of<RW>::kThreads, 1)
    k_reduce(const __grid_constant__ Table<P1<KT>::NP> tab, const __grid_constant__ Scalars sc) {
    constexpr int KS = P1<KT>::KS;
    constexpr int NSMAX = KS + 2;
    extern __shared__ __align__(128) unsigned char smem[];
    // In a step that does not read w, the first launch of the pass starts at
    // once.  It can only have been started early by the previous step's pass-2
    // finish (the update triggers its successor only when that finish
    // follows), and that finish starts it after its own wait, i.e. once the
    // previous update has completed (and, before it, the pass-1 finish that
    // re-armed the pass-1 accumulators): nothing still running then reads the
    // replicas or the pass-1 accumulators this kernel adds into, and nothing
    // writes what it loads.  The running finish reads the per-tensor sums the
    // next pass-1 finish writes, so this kernel does not complete before it
    // (one wait per CTA at the end).  Otherwise the whole CTA waits first.
    grid_launch_dependents();
    const bool early = !RW && !SS && sc.mode == kModeStep && tab.first;
    if (!early) grid_wait();
    uint64_t *full, *empty;
    int *stage_tile;
    using R1 = Ring1Of<RW>;
    ring_setup<R1>(smem, full, empty, stage_tile);
    const int js = static_tiles(tab.nc);
    const uint32_t ring = smem_addr(smem);
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int K = KT > 0 ? KT : sc.K;
    const int chunk = tab.chunk;
    int roles[NSMAX];
    int ns = 0;
    for (int k = 0; k < K; ++k) roles[ns++] = k;
    if (RW) roles[ns++] = KS;
    if (SS) roles[ns++] = KS + 1;
    if (warp == 0) {
        produce<R1, P1<KT>::NP, NSMAX>(tab, sc, roles, ns, chunk, js, sc.tiles, ring, full,
                                          empty, stage_tile);
        return;
    }
    const int my_role = lane < ns ? roles[lane] : 0;

    const int cw = warp - 1;
    TensorCache tc;
    bool stop = false;
    const bool step_g2 = sc.mode == kModeStep;  // |gbar|^2 also goes into |G|^2
    // The partial sums of a batch of kPend tiles are reduced across the warp together
    // (reduce-scatter, kRS values with padding) and added into the accumulators by the lanes
    // that own them.
    constexpr int kRS = 16;
    static_assert(kPend * kAcc <= kRS, "one reduce-scatter per batch");
    for (int jb = cw; !stop; jb += R1::kConsumers * kPend) {
        // PR: the lanes' fp64 sums.  Default: fp32 sums of the shared-memory columns, scaled by
        // 2^(2e) with e coded in two bits per value in `ecode` (same in every lane); a tile with
        // elements loaded one by one (fp64, rare) is stored at once instead (store_tile_now).
        double pendd[PR ? kRS : 1];
        float pendf[PR ? 1 : kRS];
        unsigned ecode = 0u;
        int ptensor[kPend];  // global index of each pending tile's tensor, -1: none
#pragma unroll
        for (int i = 0; i < kRS; ++i) {
            if constexpr (PR) pendd[i] = 0.0;
            else pendf[i] = 0.f;
        }
#pragma unroll
        for (int p = 0; p < kPend; ++p) {
            const int j = jb + p * R1::kConsumers;
            ptensor[p] = -1;
            if (stop) continue;
            // A round-robin tile is located before its wait, a claimed one after.
            int c = j < js ? static_tile(j) : -1;
            TilePos q;
            if (c >= 0) q = tc.at(tab, c, chunk, my_role, ns);
            const int got = next_tile<R1>(sc, j, full, stage_tile);
            if (got < 0) {
                stop = true;
                continue;
            }
            if (c < 0) {
                c = got;
                q = tc.at(tab, c, chunk, my_role, ns);
            }
            const int s = j % R1::kStages;
            const float *const *ptr = tab.ptr[q.t];
            double accd[kAcc];
            float accf[kAcc];
            int acce[kAcc];
            unsigned tcode;
            bool tile_tail;
            reduce_tile<KT, WM, RW, SS, PR>(ring + (uint32_t)s * R1::kStageBytes, chunk, ptr, q,
                                            tc.nv, sc, accd, accf, acce, tcode, tile_tail);
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[s]);
            if constexpr (PR) {
                ptensor[p] = q.tg;
#pragma unroll
                for (int a = 0; a < kAcc; ++a) pendd[p * kAcc + a] = accd[a];
            } else if (tile_tail) {
                add_tile_now(sc, q.tg, accf, acce, accd);
            } else {
                ptensor[p] = q.tg;
#pragma unroll
                for (int a = 0; a < kAcc; ++a) pendf[p * kAcc + a] = accf[a];
                ecode |= tcode << (2 * kAcc * p);
            }
        }
        int idx;
        double vd = 0.0;
        float vf = 0.f;
        if constexpr (PR) vd = warp_reduce_scatter<kRS>(pendd, idx);
        else vf = warp_reduce_scatter<kRS>(pendf, idx);
        // lanes 2i hold value i = p * kAcc + a of the batch
        if ((lane & 1) == 0 && idx < kPend * kAcc) {
            const int p = idx / kAcc, a = idx - p * kAcc;
            const int tg = p == 0 ? ptensor[0] : p == 1 ? ptensor[1] : p == 2 ? ptensor[2] : ptensor[3];
            if (tg >= 0) {
                unsigned long long *A = acc1_of(sc, tg, a);
                if constexpr (PR) {
                    acc_add_f64(A, vd);
                    if (a == 0 && step_g2) acc_add_f64(gacc_of(sc), vd);
                } else {
                    const int k = -2 * scale_exp((ecode >> (2 * idx)) & 3u);
                    acc_add_f32(A, vf, k);
                    if (a == 0 && step_g2) acc_add_f32(gacc_of(sc), vf, k);
                }
            }
        }
        if (stop) break;
    }
    if (early && threadIdx.x == 32) grid_wait();  // see the top of the kernel
}

// ----------------------------------------------------------------------------
// k_finish: per-tensor results from the exact accumulators
// ----------------------------------------------------------------------------
//
// One warp per tensor reads its accumulators (one word per lane), rounds them to fp64
// (acc_to_double), puts them back to zero for the next call and finishes the tensor: after
// pass 1 its statistics and coefficient (tensor_done), after pass 2 |w|^2 for the statistics.
// After pass 1 of a step, one more warp forms |G|^2 from the global accumulator, then Delta
// (Eq. 5) and the branch of Algorithm 1 (finalize_step).  No warp waits for another.

// The square roots of three norms (lanes 0-2 in one fp64 sequence) and the two ratios of a
// tensor (lanes 0 and 1): UpdateGradScale's |g_s| / (|g_l| + eps) and |w| / |gbar| (LARS, the
// statistics).  GB300's FP64 pipe is slow, so the lanes share its latency instead of queueing
// behind it.  Called by the whole warp; every lane gets every result.
struct Norms {
    double ng, ns, nw, q_scale, q_w;
};
__device__ __forceinline__ Norms tensor_norms(const Scalars &sc, double sg, double ss, double sw) {
    const int lane = threadIdx.x & 31;
    const double r = sqrt(lane == 0 ? sg : (lane == 1 ? ss : sw));
    Norms o;
    o.ng = __shfl_sync(kFull, r, 0);
    o.ns = __shfl_sync(kFull, r, 1);
    o.nw = __shfl_sync(kFull, r, 2);
    const double q = (lane == 0 ? o.ns : o.nw) / (lane == 0 ? o.ng + (double)sc.eps : o.ng);
    o.q_scale = __shfl_sync(kFull, q, 0);
    o.q_w = __shfl_sync(kFull, q, 1);
    return o;
}

// The statistics row of a tensor from its squared norms (sw: |w|^2 before the update).
__device__ __forceinline__ void stats_row(double *row, double sg, double ss, double sw,
                                          const Norms &o) {
    row[TULA_STAT_W_SQ] = sw;
    row[TULA_STAT_G_SQ] = sg;
    row[TULA_STAT_G0_SQ] = ss;
    row[TULA_STAT_W_NORM] = o.nw;
    row[TULA_STAT_G_NORM] = o.ng;
    row[TULA_STAT_RATIO] = sg > 0.0 ? o.q_w : 0.0;
}

// Per-tensor results after pass 1, by the whole warp holding the tensor's norms.
// tula_layer_stats and tula_ags_update_scale: everything here.  A step: what the update needs
// (the coefficient c_p) and the norms, kept in tsum with the old gradscale; the square roots,
// the statistics and UpdateGradScale follow the update (tensor_after_update), off the path
// between the passes, except for LARS, whose coefficient is a ratio of norms.
__device__ void tensor_done(const Scalars &sc, int tg, double sg, double ss, double sw, float old) {
    const int lane = threadIdx.x & 31;
    if (sc.mode == kModeScale || sc.mode == kModeStats || sc.rule == TULA_RULE_LARS) {
        const Norms o = tensor_norms(sc, sg, ss, sw);
        if (lane != 0) return;
        if (sc.mode == kModeScale) {
            // UpdateGradScale, g_0 = g_large, small = g_small: min(|g_s| / (|g_l| + eps), s_max)
            sc.scale[tg] = (float)fmin(o.q_scale, (double)sc.s_max);
            return;
        }
        if (sc.mode == kModeStats) {
            double *row = sc.stats + (size_t)tg * TULA_STATS_LEN;
            stats_row(row, sg, ss, sw, o);
            row[TULA_STAT_COEF] = 0.0;
            row[TULA_STAT_SCALE] = 0.0;
            return;
        }
        // LARS (Sec. V-B): c_p = trust * |w| / |gbar|, every step (1 when either norm is 0)
        sc.cand[tg] = (sw > 0.0 && sg > 0.0) ? (float)((double)sc.lars_trust * o.q_w) : 1.0f;
    } else if (lane == 0) {
        // the coefficient this tensor gets when the step is scaled (Algorithm 1, Eq. 8), before
        // UpdateGradScale may overwrite gradscale
        sc.cand[tg] = sc.rule == TULA_RULE_AGS ? old
                      : (sc.rule == TULA_RULE_STATIC ? sc.static_s : 1.0f);
    }
    if (lane != 0) return;
    double *T = sc.tsum + (size_t)tg * kTsum;
    T[0] = sg;
    T[1] = ss;
    T[2] = sw;
    T[3] = (double)old;
}

// After the update of a step: the statistics row and UpdateGradScale of tensor t, from the
// pass-1 norms kept in tsum and, when the update took it, |w|^2 from pass 2 (sw2).
__device__ void tensor_after_update(const Scalars &sc, int t, double sw2, bool have_sw2) {
    const int lane = threadIdx.x & 31;
    const double *T = sc.tsum + (size_t)t * kTsum;
    const double sg = T[0], ss = T[1], sw = have_sw2 ? sw2 : T[2];
    const float old = (float)T[3];
    const Norms o = tensor_norms(sc, sg, ss, sw);
    if (lane != 0) return;
    float s_after = sc.scale ? old : 0.0f;
    if (sc.refresh && sc.scale) {
        // UpdateGradScale with g_small = replica 0 and g_large = the mean
        s_after = (float)fmin(o.q_scale, (double)sc.s_max);
        sc.scale[t] = s_after;
    }
    if (sc.stats) {
        double *row = sc.stats + (size_t)t * TULA_STATS_LEN;
        if (have_sw2 || sc.read_w) {
            stats_row(row, sg, ss, sw, o);
        } else {
            row[TULA_STAT_G_SQ] = sg;
            row[TULA_STAT_G0_SQ] = ss;
            row[TULA_STAT_G_NORM] = o.ng;
        }
        row[TULA_STAT_SCALE] = (double)s_after;
    }
}

// Delta (Eq. 5): this step's |G|^2 against the last step's, +inf at the first step (no previous
// norm; the step is then unscaled, the sensitive phase).
__device__ __forceinline__ double variability(double g2, double g2_prev, double steps) {
    return steps == 0.0 ? (double)INFINITY : fabs((g2 - g2_prev) / g2_prev);
}
// The branch of Algorithm 1: scaled iff Delta < delta, unless forced.
__device__ __forceinline__ int branch_of(const Scalars &sc, double dv) {
    if (sc.force == TULA_BRANCH_SCALED) return 1;
    if (sc.force == TULA_BRANCH_UNSCALED) return 0;
    return dv < (double)sc.delta;
}
// The step record from this step's |G|^2 (one lane).
__device__ void finalize_step(const Scalars &sc, double g2, double g2_prev, double steps) {
    const double dv = variability(g2, g2_prev, steps);
    const int scaled = branch_of(sc, dv);
    sc.state[TULA_STATE_G2_PREV] = g2;
    sc.state[TULA_STATE_STEPS] = steps + 1.0;
    sc.state[TULA_STATE_DELTA] = dv;
    sc.state[TULA_STATE_SCALED] = (double)scaled;
    sc.flags[0] = scaled;
}

// This lane's word of the sum of R accumulators' Copies copies each (A[r] the first copy of
// accumulator r): digits and carries added, the flags or-ed.  Every load is issued before the
// first sum (one round trip); with `rearm`, the copies are put back to zero.
template <int R, int Copies>
__device__ __forceinline__ void acc_words(unsigned long long *const (&A)[R], bool rearm,
                                          unsigned long long (&w)[R]) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int r = 0; r < R; ++r) w[r] = 0ull;
    if (lane >= kAccWords) return;
    unsigned long long x[R][Copies];
#pragma unroll
    for (int r = 0; r < R; ++r)
#pragma unroll
        for (int c = 0; c < Copies; ++c) x[r][c] = __ldcg(A[r] + c * kAccWords + lane);
#pragma unroll
    for (int r = 0; r < R; ++r)
#pragma unroll
        for (int c = 0; c < Copies; ++c) w[r] = lane == kAccFlags ? (w[r] | x[r][c]) : (w[r] + x[r][c]);
    if (rearm) {
#pragma unroll
        for (int r = 0; r < R; ++r)
#pragma unroll
            for (int c = 0; c < Copies; ++c) A[r][c * kAccWords + lane] = 0ull;
    }
}
// One accumulator's value (its copies summed), rounded to fp64 by the whole warp.
template <int Copies>
__device__ __forceinline__ double acc_read(unsigned long long *A, bool rearm) {
    unsigned long long *const a[1] = {A};
    unsigned long long w[1];
    acc_words<1, Copies>(a, rearm, w);
    double v[1];
    acc_to_double<1>(w, v);
    return v[0];
}

// A sharded step's share of |G|^2 (TULA_G2_SHARE_WORDS words): words 0 .. kAccDigits - 1 are the
// digits of the global accumulator with its copies added, word kAccDigits counts inf partials
// and the next one NaN partials, the rest are 0.  Every word adds as an integer, so the ranks'
// shares combine by any integer sum, in any order, to the share of the whole step.
static_assert(kAccDigits + 2 <= kAccWords && TULA_G2_SHARE_WORDS == kAccWords, "share layout");
__device__ __forceinline__ double share_to_double(const unsigned long long *share) {
    const int lane = threadIdx.x & 31;
    unsigned long long w = lane < kAccWords ? __ldcg(share + lane) : 0ull;
    const unsigned long long n_inf = __shfl_sync(kFull, w, kAccDigits);
    const unsigned long long n_nan = __shfl_sync(kFull, w, kAccDigits + 1);
    if (lane == kAccFlags) w = (n_nan ? 2ull : 0ull) | (n_inf ? 1ull : 0ull);
    else if (lane >= kAccDigits) w = 0ull;
    unsigned long long wi[1] = {w};
    double v[1];
    acc_to_double<1>(wi, v);
    return v[0];
}

// Pass 1 of a sharded step, after the reduction: this rank's share of |G|^2 out of the global
// accumulator, which is re-armed.  One warp.
__global__ void __launch_bounds__(32) k_share(const __grid_constant__ Scalars sc,
                                              unsigned long long *share) {
    grid_wait();
    const int lane = threadIdx.x & 31;
    unsigned long long *const a[1] = {sc.gacc};
    unsigned long long w[1];
    acc_words<1, kGCopies>(a, true, w);
    const unsigned long long flags = __shfl_sync(kFull, w[0], kAccFlags);
    if (lane < kAccDigits) share[lane] = w[0];
    else if (lane == kAccDigits) share[lane] = (flags & 1ull) ? 1ull : 0ull;
    else if (lane == kAccDigits + 1) share[lane] = (flags & 2ull) ? 1ull : 0ull;
    else if (lane < kAccWords) share[lane] = 0ull;
}

// NA = kAcc: after pass 1 (the pass-1 norms; in a step also the branch, which the update then
// reads).  NA = 1: after the update of a step (its statistics and UpdateGradScale, with |w|^2
// from pass 2 when the update took it).
template <int NA>
__global__ void __launch_bounds__(32 * kFinWarps) k_finish(const __grid_constant__ Scalars sc) {
    constexpr bool P1 = NA == kAcc;  // pass-1 accumulators
    const int lane = threadIdx.x & 31;
    const int t = (int)blockIdx.x * kFinWarps + (int)(threadIdx.x >> 5);
    const int n = sc.n_total;
    const bool step = P1 && sc.mode == kModeStep;
    const bool active = t < n + (step ? 1 : 0);
    // This kernel is launched early and waits here for the kernel before it; the old gradscale
    // and the step record are read after the wait, together with the accumulators (no round
    // trip is added, and no kernel of an earlier call can still be writing them).
    grid_wait();
    // Inside a step the successor (the update, or the next step's reduction) may start now;
    // after tula_layer_stats or tula_ags_update_scale it starts when this kernel has completed
    // (a step's reduction that starts early adds into the accumulators this kernel reads).
    if (sc.mode == kModeStep || NA == 1) grid_launch_dependents();
    if (!active) return;
    const float scale_old = (t < n && step && sc.scale) ? sc.scale[t] : 1.0f;
    const double g2_prev = step ? sc.state[TULA_STATE_G2_PREV] : 0.0;
    const double steps = step ? sc.state[TULA_STATE_STEPS] : 0.0;
    if (t == n) {  // the record and the branch
        double g2;
        if (sc.g2ext) {
            g2 = share_to_double(sc.g2ext);
        } else {
            g2 = acc_read<kGCopies>(sc.gacc, true);
        }
        if (lane == 0) finalize_step(sc, g2, g2_prev, steps);
        return;
    }
    unsigned long long *A1 = sc.acc1 + (size_t)t * kAcc * kTCopies * kAccWords;
    unsigned long long *A2 = sc.acc2 + (size_t)t * kTCopies * kAccWords;
    if constexpr (NA == kAcc) {
        unsigned long long *const a[kAcc] = {A1, A1 + kTCopies * kAccWords,
                                             A1 + 2 * kTCopies * kAccWords};
        unsigned long long w[kAcc];
        acc_words<kAcc, kTCopies>(a, true, w);
        double v[kAcc];
        acc_to_double<kAcc>(w, v);
        tensor_done(sc, t, v[0], v[1], v[2], scale_old);
    } else {
        const bool have_sw2 = sc.stats && !sc.read_w;  // the update's |w|^2 (k_update<..., SW>)
        const double sw2 = have_sw2 ? acc_read<kTCopies>(A2, true) : 0.0;
        tensor_after_update(sc, t, sw2, have_sw2);
    }
}

// ----------------------------------------------------------------------------
// Pass 2: scaled momentum-SGD + weight-decay update (Eq. 7b, Algorithm 1)
// ----------------------------------------------------------------------------
// Pointer roles: 0 = gbar, 1 = w, 2 = m, 3 = per-element gradscale.
// Stage streams: gbar, w, then m (HM), then the per-element scale (PE, scaled).

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

// One float4 column of the update; returns the squares of w (before the update).
template <bool HM>
__device__ __forceinline__ float update4(float4 g4, float4 w4, float4 m4, float4 cc, float *wp,
                                         float *mp, const Scalars &sc, float pw) {
    pw = sq4(pw, w4);
    sgd1(g4.x, cc.x, w4.x, m4.x, sc, HM);
    sgd1(g4.y, cc.y, w4.y, m4.y, sc, HM);
    sgd1(g4.z, cc.z, w4.z, m4.z, sc, HM);
    sgd1(g4.w, cc.w, w4.w, m4.w, sc, HM);
    st_stream(wp, w4);
    if (HM) st_stream(mp, m4);
    return pw;
}

// |w|^2 of a tile's shared-memory w columns in fp32, every element multiplied by the power of
// two f first (sq_range_exp): the statistics' fallback when the tile's fp32 sums would overflow
// or lose their precision to underflow.  Out of line, like tile_cols_scaled.
__device__ __noinline__ float w_cols_scaled(uint32_t w_stage, int nv, float f) {
    float a = 0.f;
    for (int v = threadIdx.x & 31; v < nv; v += 32) a = sq4(a, mul4(lds4(w_stage + (uint32_t)(16 * v)), f));
    return a;
}

// A tile of the update with elements loaded one by one: its |w|^2 (fp32 part scaled by 2^(2e),
// fp64 part) reduced across the warp at once and added into the accumulator A by lane 0.
__device__ __noinline__ void add_w_tile_now(unsigned long long *A, float aw, int e, double awt) {
    float f[1] = {aw};
    double d[1] = {awt};
    warp_sums<1>(f);
    warp_sums<1>(d);
    if ((threadIdx.x & 31) == 0) {
        acc_add_f32(A, f[0], -2 * e);
        acc_add_f64(A, d[0]);
    }
}

template <bool HM, bool PE, bool SW>
__global__ void __launch_bounds__(Ring2::kThreads, 1)
    k_update(const __grid_constant__ Table<kNP2> tab, const __grid_constant__ Scalars sc) {
    extern __shared__ __align__(128) unsigned char smem[];
    // The first launch of the pass follows the pass-1 finish, which starts it
    // once the reduction kernel has completed (the finish's own wait).  gbar, w
    // and m are then final, so the producer streams tiles in while the finish
    // still runs; the branch and the coefficients the consumers apply are the
    // finish's output, so every consumer waits for its completion first.  The
    // whole CTA waits per element (the producer's stream count depends on the
    // branch) and in later launches of the pass (which share the tile counter
    // with the launch before).
    // Successors may start early only when the pass-2 finish follows (it waits
    // for this kernel); the next step's reduction, when it follows directly,
    // must start after this kernel has completed (see k_reduce).
    if (sc.fin2) grid_launch_dependents();
    const bool early = !PE && tab.first;
    if (!early) grid_wait();
    uint64_t *full, *empty;
    int *stage_tile;
    ring_setup<Ring2>(smem, full, empty, stage_tile);
    const int js = static_tiles(tab.nc);
    const uint32_t ring = smem_addr(smem);
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int chunk = tab.chunk;
    int roles[4] = {0, 1, 2, 3};
    if (!HM) roles[2] = 3;
    if (warp == 0) {
        const bool se = PE && sc.flags[0];
        produce<Ring2, kNP2, 4>(tab, sc, roles, 2 + (HM ? 1 : 0) + (se ? 1 : 0), chunk, js,
                                sc.tiles + 2, ring, full, empty, stage_tile);
        return;
    }
    if (early) grid_wait();
    const int scaled = sc.flags[0];
    const bool gated = sc.rule == TULA_RULE_AGS || sc.rule == TULA_RULE_STATIC;
    const bool use_se = PE && scaled;
    const int ns = 2 + (HM ? 1 : 0) + (use_se ? 1 : 0);
    const int my_role = lane < ns ? roles[lane] : 0;
    constexpr int CH = Ring2::tile_elems(2 + (HM ? 1 : 0) + (PE ? 1 : 0));
    constexpr int COLS = CH / 128;
    const uint32_t w_off = (uint32_t)(CH * 4);
    const uint32_t m_off = (uint32_t)(2 * CH * 4);
    const uint32_t se_off = (uint32_t)((HM ? 3 : 2) * CH * 4);

    TensorCache tc;
    const int cw = warp - 1;
    int cand_t = -1;
    float cand = 0.f;
    bool stop = false;
    for (int jb = cw; !stop; jb += Ring2::kConsumers * kPend) {
        // fp32 |w|^2 of the tiles' shared-memory columns, scaled by 2^(2e) (e coded in `ecode`);
        // a tile with elements loaded one by one (fp64, rare) is stored at once instead.
        float pend[kPend];
        unsigned ecode = 0u;
        int ptensor[kPend];  // global index of each pending tile's tensor, -1: none
#pragma unroll
        for (int p = 0; p < kPend; ++p) {
            const int j = jb + p * Ring2::kConsumers;
            ptensor[p] = -1;
            pend[p] = 0.f;
            if (stop) continue;
            int c = j < js ? static_tile(j) : -1;
            TilePos q;
            if (c >= 0) q = tc.at(tab, c, chunk, my_role, ns);
            const int got = next_tile<Ring2>(sc, j, full, stage_tile);
            if (got < 0) {
                stop = true;
                continue;
            }
            if (c < 0) {
                c = got;
                q = tc.at(tab, c, chunk, my_role, ns);
            }
            const int s = j % Ring2::kStages;
            const float *const *ptr = tab.ptr[q.t];
            const int nv = tc.nv;
            if (q.tg != cand_t) {  // c_p changes only with the tensor
                cand = sc.cand[q.tg];
                cand_t = q.tg;
            }
            const float ct = gated ? (scaled ? cand : 1.0f) : cand;
            if (sc.stats && q.c_in_t == 0 && lane == 0)
                sc.stats[(size_t)q.tg * TULA_STATS_LEN + TULA_STAT_COEF] =
                    PE ? (scaled ? (double)NAN : 1.0) : (double)ct;
            const uint32_t stage = ring + (uint32_t)s * Ring2::kStageBytes;
            float *wp = const_cast<float *>(ptr[1]) + q.begin;
            float *mp = HM ? const_cast<float *>(ptr[2]) + q.begin : nullptr;
            const float4 cdef = PE ? make_float4(1.f, 1.f, 1.f, 1.f) : make_float4(ct, ct, ct, ct);
            float aw = 0.f;    // fp32 |w|^2 of the tile's columns (statistics only)
            double awt = 0.0;  // exact fp64 |w|^2 of its tail
            if (nv == CH / 4) {
                // Two columns per step of a rolled loop (unrolled over the tile, the body
                // outgrew the instruction cache: 82.5 -> 75.5 us per ResNet-50 update pass).
#pragma unroll 1
                for (int c0 = 0; c0 < COLS; c0 += 2) {
                    float pw = 0.f;
#pragma unroll
                    for (int u = 0; u < 2; ++u) {
                        if (c0 + u < COLS) {
                            const int v = lane + 32 * (c0 + u);
                            const float4 g4 = lds4(stage + (uint32_t)(16 * v));
                            const float4 w4 = lds4(stage + w_off + (uint32_t)(16 * v));
                            const float4 m4 = HM ? lds4(stage + m_off + (uint32_t)(16 * v)) : g4;
                            const float4 cc =
                                use_se ? lds4(stage + se_off + (uint32_t)(16 * v)) : cdef;
                            pw = update4<HM>(g4, w4, m4, cc, wp + 4 * v, mp + 4 * v, sc, pw);
                        }
                    }
                    if (SW) aw = __fadd_rn(aw, pw);
                }
            } else {
                for (int v0 = lane; v0 < nv; v0 += 32 * 4) {
                    float pw = 0.f;
                    for (int u = 0; u < 4; ++u) {
                        const int v = v0 + 32 * u;
                        if (v >= nv) break;
                        const float4 g4 = lds4(stage + (uint32_t)(16 * v));
                        const float4 w4 = lds4(stage + w_off + (uint32_t)(16 * v));
                        const float4 m4 = HM ? lds4(stage + m_off + (uint32_t)(16 * v)) : g4;
                        const float4 cc = use_se ? lds4(stage + se_off + (uint32_t)(16 * v)) : cdef;
                        pw = update4<HM>(g4, w4, m4, cc, wp + 4 * v, mp + 4 * v, sc, pw);
                    }
                    if (SW) aw = __fadd_rn(aw, pw);
                }
            }
            // The warp is converged again; nv is the same in every lane.  The stage still holds
            // the tile's w before the update.
            int ew = 0;
            if (SW && nv > 0 && !__all_sync(kFull, lane >= nv || sq_in_range(aw))) {
                ew = sq_range_exp(aw);
                if (ew) aw = w_cols_scaled(stage + w_off, nv, pow2f(ew));
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[s]);
            const long long n = q.end - q.begin;
            const bool tile_tail = 4 * (long long)nv < n;  // the same in every lane
            for (long long jj = 4 * (long long)nv + lane; jj < n; jj += 32) {
                const float g = __ldcs(ptr[0] + q.begin + jj);
                float w = wp[jj];
                float m = HM ? mp[jj] : 0.f;
                const float cj = use_se ? __ldcs(ptr[3] + q.begin + jj) : (PE ? 1.f : ct);
                if (SW) awt = __fma_rn((double)w, (double)w, awt);
                sgd1(g, cj, w, m, sc, HM);
                wp[jj] = w;
                if (HM) mp[jj] = m;
            }
            if (SW) {
                if (tile_tail) {
                    add_w_tile_now(acc2_of(sc, q.tg), aw, ew, awt);
                } else {
                    ptensor[p] = q.tg;
                    pend[p] = aw;
                    if (ew) ecode |= scale_code(ew) << (2 * p);
                }
            }
        }
        if (SW) {
            // reduce-scatter: lanes 8p hold tile p's total
            int idx;
            const float f = warp_reduce_scatter<kPend>(pend, idx);
            if ((lane & 7) == 0) {
                const int tg = idx == 0 ? ptensor[0] : idx == 1 ? ptensor[1] : idx == 2 ? ptensor[2] : ptensor[3];
                if (tg >= 0)
                    acc_add_f32(acc2_of(sc, tg), f,
                                -2 * scale_exp((ecode >> (2 * idx)) & 3u));
            }
        }
        if (stop) break;
    }
}

// ----------------------------------------------------------------------------
// UpdateGradScale, element-wise (Algorithm 1): s = fminf(|gs / (gl + eps)|, s_max)
// ----------------------------------------------------------------------------
// A once-per-epoch call: plain 128-bit loads, one warp per tile.
// Pointer roles: 0 = g_small, 1 = g_large, 2 = s_out.

constexpr int kNP3 = 3;

__device__ __forceinline__ float scale1(float gs, float gl, const Scalars &sc) {
    return fminf(fabsf(__fdiv_rn(gs, __fadd_rn(gl, sc.eps))), sc.s_max);
}

// The bounded wait itself, on an mbarrier that nothing ever arrives on: the
// wait runs out and the kernel reports it in the error word, the way every
// streaming kernel reports a stage that never fills.  (Failure detection is
// checked with this, not with a real fault.)
__global__ void __launch_bounds__(32) k_wait_check(unsigned *err) {
    __shared__ uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        mbar_fence_init();
    }
    __syncwarp();
    if (threadIdx.x == 0 && !mbar_wait(&bar, 0u)) atomicOr(err, 1u);
}

constexpr int kScaleThreads = 128;

__global__ void __launch_bounds__(kScaleThreads)
    k_scale_elem(const __grid_constant__ Table<kNP3> tab, const __grid_constant__ Scalars sc) {
    grid_wait();  // no early start for the successor: it may overwrite what this kernel reads
    const int lane = threadIdx.x & 31;
    const int warp = (int)((blockIdx.x * (unsigned)kScaleThreads + threadIdx.x) >> 5);
    const int nwarps = (int)((gridDim.x * (unsigned)kScaleThreads) >> 5);
    Walker walk;
    for (int c = warp; c < tab.nc; c += nwarps) {
        const TilePos q = locate(tab, c, walk.to(tab, c), tab.chunk);
        const float *const *ptr = tab.ptr[q.t];
        const int nv = tile_vecs(lane < 3 ? ptr[lane] : nullptr, 3, q);
        const float *a = ptr[0] + q.begin;
        const float *b = ptr[1] + q.begin;
        float *o = const_cast<float *>(ptr[2]) + q.begin;
        // Four float4 columns of each input per lane per step: eight 16-byte loads in flight
        // per lane, which a plain-load streaming kernel needs to cover HBM latency.
        for (int v0 = lane; v0 < nv; v0 += 4 * 32) {
            float4 x[4], y[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int v = v0 + 32 * u;
                if (v < nv) {
                    x[u] = __ldcs(reinterpret_cast<const float4 *>(a) + v);
                    y[u] = __ldcs(reinterpret_cast<const float4 *>(b) + v);
                }
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int v = v0 + 32 * u;
                if (v < nv)
                    st_stream(o + 4 * v, make_float4(scale1(x[u].x, y[u].x, sc), scale1(x[u].y, y[u].y, sc),
                                                     scale1(x[u].z, y[u].z, sc), scale1(x[u].w, y[u].w, sc)));
            }
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

inline long long tiles_of(int64_t n, int chunk) { return n <= 0 ? 1 : (n + chunk - 1) / chunk; }

inline int replica_slot(int K) {
    return (K == 1 || K == 2 || K == 4 || K == 8 || K == 16) ? K : TULA_MAX_K;
}

// Tile sizes: the smallest a pass can use for K replicas sizes the workspace.
inline int chunk1(int K, bool rw, bool ss) {
    const int streams = K + (rw ? 1 : 0) + (ss ? 1 : 0);
    return rw ? Ring1W::tile_elems(streams) : Ring1::tile_elems(streams);
}
inline int chunk2(bool hm, bool pe) { return Ring2::tile_elems(2 + (hm ? 1 : 0) + (pe ? 1 : 0)); }
// No pass-1 tile is smaller: K (+1 with g_small) streams in 36 KB, or K + 1 in 45 KB.
inline int chunk1_min(int K) { return Ring1::tile_elems(K + 1 + (K == 1 ? 1 : 0)); }
inline int chunk2_min() { return chunk2(true, true); }

struct Plan {
    long long c1 = 0, c2 = 0;  // tiles of each pass (at the smallest tile sizes)
};

// Workspace layout.  Every counter, flag and accumulator precedes `tsum`, so zeroing
// [0, tsum) clears all of them; the error word is the only one no call clears.
struct WsLayout {
    size_t flags, err, tiles, acc1, gacc, acc2, tsum, cand, total;
};

WsLayout ws_layout(int n_tensors, const Plan &) {
    size_t off = 0;
    auto take = [&](size_t bytes) {
        size_t o = off;
        off = (off + bytes + 255) & ~size_t(255);
        return o;
    };
    const size_t acc = sizeof(unsigned long long) * kAccWords;
    WsLayout L;
    L.flags = take(sizeof(int) * 4);
    L.err = take(sizeof(unsigned) * 4);
    L.tiles = take(sizeof(unsigned) * 4);
    L.acc1 = take(acc * kAcc * kTCopies * (size_t)n_tensors);
    L.gacc = take(acc * kGCopies);
    L.acc2 = take(acc * kTCopies * (size_t)n_tensors);
    L.tsum = take(sizeof(double) * kTsum * (size_t)n_tensors);
    L.cand = take(sizeof(float) * (size_t)n_tensors);
    L.total = off;
    return L;
}

// The tile index of either pass must fit an int, which also keeps every accumulator word's
// carries within its high half (at most two adds below 2^32 per tile).
bool valid_numels(const int64_t *numels, int n, int K, Plan *pl) {
    if (!numels || n < 1 || K < 1 || K > TULA_MAX_K) return false;
    const int t1 = chunk1_min(K), t2 = chunk2_min();
    Plan p;
    for (int i = 0; i < n; ++i) {
        if (numels[i] < 0) return false;
        p.c1 += tiles_of(numels[i], t1);
        p.c2 += tiles_of(numels[i], t2);
        if (p.c1 >= (1LL << 31) || p.c2 >= (1LL << 31)) return false;
    }
    *pl = p;
    return true;
}

inline bool aligned4(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 3u) == 0; }

// One wave of resident CTAs of `kernel` on the current device (cached); sets
// the kernel's dynamic shared memory limit on first use.
int resident_ctas(const void *kernel, int threads, int smem) {
    struct Entry { const void *k; int dev; int ctas; };
    static std::mutex mu;
    static std::vector<Entry> cache;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    std::lock_guard<std::mutex> lock(mu);
    for (const Entry &e : cache)
        if (e.k == kernel && e.dev == dev) return e.ctas;
    if (smem > 48 * 1024 &&
        cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) !=
            cudaSuccess)
        return 0;
    int sms = 0, per = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per, kernel, threads, smem) != cudaSuccess)
        return 0;
    const int ctas = std::max(1, sms * std::max(per, 1));
    cache.push_back({kernel, dev, ctas});
    return ctas;
}

// L2 capacity of the current device in bytes (cached; 0 if unknown).
long long l2_bytes() {
    static std::mutex mu;
    static std::vector<std::pair<int, long long>> cache;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    std::lock_guard<std::mutex> lock(mu);
    for (const auto &e : cache)
        if (e.first == dev) return e.second;
    int v = 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrL2CacheSize, dev) != cudaSuccess) v = 0;
    cache.emplace_back(dev, (long long)v);
    return v;
}

// Launch with programmatic stream serialization: the kernel may begin while
// the previous kernel in the stream finishes; its griddepcontrol.wait orders
// every memory access after that kernel's completion.
template <typename... KArgs, typename... Args>
int launch_pdl(void (*kernel)(KArgs...), int grid, int threads, int smem, cudaStream_t s,
               Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3((unsigned)threads);
    cfg.dynamicSmemBytes = (size_t)smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
    g_launches.fetch_add(1, std::memory_order_relaxed);
    if (e == cudaSuccess) e = cudaGetLastError();
    if (e != cudaSuccess) {
        g_last_cuda = (int)e;
        return TULA_ERR_CUDA;
    }
    return TULA_OK;
}

// The launch tables of a plan (tula_ags_plan_create): for each kernel instantiation and tile
// size, its parameter blocks, built by the first call that launches them and reused by every
// later one (they hold only sizes and pointers, which a plan fixes).
struct TableCache {
    struct Entry {
        const void *kernel;
        int chunk;
        std::vector<std::shared_ptr<const void>> blocks;
    };
    std::vector<Entry> entries;
    const std::vector<std::shared_ptr<const void>> *find(const void *kernel, int chunk) const {
        for (const Entry &e : entries)
            if (e.kernel == kernel && e.chunk == chunk) return &e.blocks;
        return nullptr;
    }
};

// Splits tensors [0, n) into parameter blocks of tiles of `chunk` elements and
// launches `kernel` once per block.
// fill(p, ptrs) writes tensor p's pointers.  With a cache, the blocks are taken from it, or
// built once and kept there.
template <int NP, typename Kernel, typename Fill>
int launch_streaming(Kernel kernel, int n, const int64_t *numels, int chunk, int threads,
                     int smem, const Scalars &sc, int grid_override, cudaStream_t stream,
                     Fill fill, TableCache *cache = nullptr) {
    using T = Table<NP>;
    const int grid_cap = resident_ctas((const void *)kernel, threads, smem);
    if (grid_cap <= 0) {
        g_last_cuda = (int)cudaGetLastError();
        return TULA_ERR_CUDA;
    }
    const std::vector<std::shared_ptr<const void>> *blocks =
        cache ? cache->find((const void *)kernel, chunk) : nullptr;
    std::vector<std::shared_ptr<const void>> built;
    if (!blocks) {
        try {
            long long c_global = 0;
            int p = 0;
            while (p < n) {
                std::shared_ptr<T> tab = std::make_shared<T>();
                std::memset(tab.get(), 0, sizeof(T));
                tab->t0 = p;
                tab->c0 = (int)c_global;
                tab->chunk = chunk;
                tab->first = p == 0 ? 1 : 0;
                int cnt = 0, nc = 0;
                while (p < n && cnt < T::kMaxT) {
                    tab->numel[cnt] = numels[p];
                    tab->cstart[cnt] = nc;
                    fill(p, tab->ptr[cnt]);
                    nc += (int)tiles_of(numels[p], chunk);
                    ++cnt;
                    ++p;
                }
                tab->n = cnt;
                tab->nc = nc;
                tab->cstart[cnt] = nc;
                c_global += nc;
                built.push_back(std::move(tab));
            }
            if (cache) {
                cache->entries.push_back({(const void *)kernel, chunk, std::move(built)});
                blocks = &cache->entries.back().blocks;
            }
        } catch (const std::bad_alloc &) {
            return TULA_ERR_NO_MEMORY;
        }
        if (!blocks) blocks = &built;
    }
    for (const auto &b : *blocks) {
        const T &tab = *static_cast<const T *>(b.get());
        int grid = grid_override > 0 ? grid_override : grid_cap;
        grid = std::max(1, std::min(grid, tab.nc));
        const int rc = launch_pdl(kernel, grid, threads, smem, stream, tab, sc);
        if (rc) return rc;
    }
    return TULA_OK;
}

// k_finish over all tensors: NA accumulators per tensor (+ the branch after pass 1 of a step).
template <int NA>
int launch_finish(int n, const Scalars &sc, cudaStream_t s) {
    const bool record = NA == kAcc && sc.mode == kModeStep;  // + the branch's warp
    const int warps = n + (record ? 1 : 0);
    return launch_pdl(k_finish<NA>, (warps + kFinWarps - 1) / kFinWarps, 32 * kFinWarps, 0, s, sc);
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
    sc.flags = reinterpret_cast<int *>(b + L.flags);
    sc.err = reinterpret_cast<unsigned *>(b + L.err);
    sc.tiles = reinterpret_cast<unsigned *>(b + L.tiles);
    sc.acc1 = reinterpret_cast<unsigned long long *>(b + L.acc1);
    sc.gacc = reinterpret_cast<unsigned long long *>(b + L.gacc);
    sc.acc2 = reinterpret_cast<unsigned long long *>(b + L.acc2);
    sc.tsum = reinterpret_cast<double *>(b + L.tsum);
    sc.cand = reinterpret_cast<float *>(b + L.cand);
    return sc;
}

void record(void *ev, cudaStream_t s) {
    if (ev) cudaEventRecord(static_cast<cudaEvent_t>(ev), s);
}

// Pass 1 (+ its finish) dispatched over the compile-time replica count.
template <int KT, bool WM, bool RW, bool SS, bool PR, typename Fill>
int run_reduce_k(int K, int n, const int64_t *numels, const Scalars &sc, int grid, cudaStream_t s,
                 Fill fill, void *mid_event, bool finish, TableCache *cache) {
    const int chunk = chunk1(K, RW, SS);
    int rc = launch_streaming<P1<KT>::NP>(k_reduce<KT, WM, RW, SS, PR>, n, numels, chunk,
                                          Ring1Of<RW>::kThreads, Ring1Of<RW>::kSmemBytes, sc,
                                          grid, s, fill, cache);
    if (rc) return rc;
    record(mid_event, s);
    return finish ? launch_finish<kAcc>(n, sc, s) : TULA_OK;
}

template <bool WM, bool RW, bool SS, bool PR, typename Fill>
int run_reduce(int K, int n, const int64_t *numels, const Scalars &sc, int grid, cudaStream_t s,
               Fill fill, void *mid_event = nullptr, bool finish = true,
               TableCache *cache = nullptr) {
    switch (K) {
    case 1: return run_reduce_k<1, false, RW, SS, PR>(K, n, numels, sc, grid, s, fill, mid_event, finish, cache);
    case 2: return run_reduce_k<2, WM, RW, SS, PR>(K, n, numels, sc, grid, s, fill, mid_event, finish, cache);
    case 4: return run_reduce_k<4, WM, RW, SS, PR>(K, n, numels, sc, grid, s, fill, mid_event, finish, cache);
    case 8: return run_reduce_k<8, WM, RW, SS, PR>(K, n, numels, sc, grid, s, fill, mid_event, finish, cache);
    case 16: return run_reduce_k<16, WM, RW, SS, PR>(K, n, numels, sc, grid, s, fill, mid_event, finish, cache);
    default: return run_reduce_k<0, WM, RW, SS, PR>(K, n, numels, sc, grid, s, fill, mid_event, finish, cache);
    }
}

int check_ws(void *ws, size_t bytes, int n, const Plan &pl) {
    if (!ws) return TULA_ERR_WORKSPACE;
    if (bytes < ws_layout(n, pl).total) return TULA_ERR_WORKSPACE;
    if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return TULA_ERR_WORKSPACE;
    return TULA_OK;
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
    if (!bytes || !valid_numels(numels, n_tensors, K, &pl)) return TULA_ERR_ARG;
    *bytes = ws_layout(n_tensors, pl).total;
    return TULA_OK;
}

int tula_ags_chunk_elems(int pass, int streams) {
    if (streams < 1 || streams > TULA_MAX_K + 2) return TULA_ERR_ARG;
    if (pass == 1) return Ring1::tile_elems(streams);
    if (pass == 2 && streams <= 4) return Ring2::tile_elems(streams);
    if (pass == 3) return Ring1W::tile_elems(streams);
    return TULA_ERR_ARG;
}

int tula_ags_plan_chunks(const int64_t *numels, int n_tensors, int chunk_elems,
                         int64_t *chunk_start_out) {
    Plan pl;
    if (!chunk_start_out || chunk_elems < 1 || !valid_numels(numels, n_tensors, 1, &pl))
        return TULA_ERR_ARG;
    int64_t c = 0;
    for (int p = 0; p < n_tensors; ++p) {
        chunk_start_out[p] = c;
        c += tiles_of(numels[p], chunk_elems);
    }
    chunk_start_out[n_tensors] = c;
    return TULA_OK;
}

int tula_ags_check_wait_timeout(void *workspace, size_t workspace_bytes, void *stream) {
    const WsLayout L = ws_layout(1, Plan{});
    if (!workspace || workspace_bytes < L.err + sizeof(unsigned)) return TULA_ERR_WORKSPACE;
    if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return TULA_ERR_WORKSPACE;
    unsigned *err = reinterpret_cast<unsigned *>(static_cast<char *>(workspace) + L.err);
    k_wait_check<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(err);
    g_launches.fetch_add(1, std::memory_order_relaxed);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) {
        g_last_cuda = (int)e;
        return TULA_ERR_CUDA;
    }
    return TULA_OK;
}

int tula_ags_workspace_error(const void *workspace, size_t workspace_bytes,
                             const int64_t *numels, int n_tensors, int K, int *error_out) {
    Plan pl;
    if (!workspace || !error_out || !valid_numels(numels, n_tensors, K, &pl)) return TULA_ERR_ARG;
    const WsLayout L = ws_layout(n_tensors, pl);
    if (workspace_bytes < L.total) return TULA_ERR_WORKSPACE;
    unsigned v = 0;
    unsigned *dev = reinterpret_cast<unsigned *>(static_cast<char *>(const_cast<void *>(workspace)) +
                                                 L.err);
    cudaError_t e = cudaMemcpy(&v, dev, sizeof(v), cudaMemcpyDeviceToHost);
    if (e == cudaSuccess && v) e = cudaMemset(dev, 0, sizeof(v));
    if (e != cudaSuccess) {
        g_last_cuda = (int)e;
        return TULA_ERR_CUDA;
    }
    *error_out = (int)v;
    return TULA_OK;
}

}  // extern "C"

namespace {

// Every host-side check of a step's arguments except the workspace: TULA_OK or the status
// tula_ags_step returns.  Nothing is enqueued before it passes.
// The options of a step (hp apart from its workspace, and the momentum) against the buffers the
// step has: momentum buffers (has_mom) and per-element gradscales (has_se).
int check_step_options(const tula_ags_hparams *hp, float momentum, bool has_mom, bool has_se) {
    if (!hp || hp->K < 1 || hp->K > TULA_MAX_K) return TULA_ERR_ARG;
    if (hp->rule < TULA_RULE_AGS || hp->rule > TULA_RULE_STATIC) return TULA_ERR_ARG;
    if (hp->granularity != TULA_SCALE_PER_TENSOR && hp->granularity != TULA_SCALE_PER_ELEMENT)
        return TULA_ERR_ARG;
    if (hp->force_branch < TULA_BRANCH_AUTO || hp->force_branch > TULA_BRANCH_UNSCALED)
        return TULA_ERR_ARG;
    if (!hp->state) return TULA_ERR_ARG;
    const bool per_elem = hp->rule == TULA_RULE_AGS && hp->granularity == TULA_SCALE_PER_ELEMENT;
    if (hp->rule == TULA_RULE_AGS && !per_elem && !hp->scale) return TULA_ERR_ARG;
    if (per_elem && !has_se) return TULA_ERR_ARG;
    if (!has_mom && momentum != 0.0f) return TULA_ERR_ARG;
    if (hp->refresh_scale) {
        if (hp->K == 1 || !hp->scale) return TULA_ERR_ARG;
        if (hp->granularity != TULA_SCALE_PER_TENSOR) return TULA_ERR_UNSUPPORTED;
    }
    return TULA_OK;
}

// The tensors of a step: their sizes, and every pointer of a non-empty tensor non-NULL and
// 4-byte aligned (scale_elem: the per-element gradscales, or NULL when the step has none).
int check_step_tensors(float *const *param_ptrs, float *const *grad_ptrs, float *const *mom_ptrs,
                       float *const *scale_elem, const int64_t *numels, int n, int K, Plan *pl) {
    if (!param_ptrs || !grad_ptrs || !valid_numels(numels, n, K, pl)) return TULA_ERR_ARG;
    for (int p = 0; p < n; ++p) {
        if (numels[p] == 0) continue;
        if (!param_ptrs[p] || !aligned4(param_ptrs[p])) return TULA_ERR_ARG;
        if (mom_ptrs && (!mom_ptrs[p] || !aligned4(mom_ptrs[p]))) return TULA_ERR_ARG;
        if (scale_elem && (!scale_elem[p] || !aligned4(scale_elem[p]))) return TULA_ERR_ARG;
        for (int k = 0; k < K; ++k) {
            const float *g = grad_ptrs[(size_t)k * n + p];
            if (!g || !aligned4(g)) return TULA_ERR_ARG;
        }
    }
    return TULA_OK;
}

int check_step_args(float *const *param_ptrs, float *const *grad_ptrs, float *const *mom_ptrs,
                    const int64_t *numels, int n_tensors, float momentum,
                    const tula_ags_hparams *hp, Plan *pl) {
    int rc = check_step_options(hp, momentum, mom_ptrs != nullptr, hp && hp->scale_elem);
    if (rc) return rc;
    const bool per_elem = hp->rule == TULA_RULE_AGS && hp->granularity == TULA_SCALE_PER_ELEMENT;
    return check_step_tensors(param_ptrs, grad_ptrs, mom_ptrs, per_elem ? hp->scale_elem : nullptr,
                              numels, n_tensors, hp->K, pl);
}

// Which part of a step run_step launches: all of it, or one half of a sharded step (pass 1 up to
// this rank's share of |G|^2; then, from the ranks' shares summed, the rest).
enum StepPart { kPartWhole = 0, kPartReduce = 1, kPartUpdate = 2 };

// The step's launches, once its arguments (check_step_args) and its scratch `ws` (the caller's
// workspace or the static array) have been accepted.
int run_step(float *const *param_ptrs, float *const *grad_ptrs, float *const *mom_ptrs,
             const int64_t *numels, int n, float lr, float momentum, float weight_decay,
             const tula_ags_hparams *hp, void *ws, const Plan &pl, void *stream,
             StepPart part = kPartWhole, unsigned long long *share_out = nullptr,
             const unsigned long long *g2_in = nullptr, TableCache *cache = nullptr) {
    const int K = hp->K;
    const bool per_elem = hp->rule == TULA_RULE_AGS && hp->granularity == TULA_SCALE_PER_ELEMENT;
    int rc = TULA_OK;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const WsLayout L = ws_layout(n, pl);
    Scalars sc = make_scalars(hp, K, n, ws, L, kModeStep);
    const bool lars = hp->rule == TULA_RULE_LARS;
    sc.read_w = lars ? 1 : 0;
    // When the mean fits in L2, every bulk load is marked to leave L2 first, so
    // that the lines the step writes (the mean, w, m), which the update and the
    // next step read again, stay there instead (ResNet-18 K = 4: 103 -> 79 us per
    // step).  For larger models the mark only costs bandwidth.
    long long n_total = 0;
    for (int p = 0; p < n; ++p) n_total += numels[p];
    sc.evict_first = (K > 1 && 4 * n_total <= l2_bytes()) ? 1 : 0;
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
    if (part == kPartUpdate) {
        // the ranks' shares summed give |G|^2; the local accumulators the tensors' norms
        sc.g2ext = g2_in;
        record(hp->trace_events[1], s);
        rc = launch_finish<kAcc>(n, sc, s);
        sc.g2ext = nullptr;
    } else {
        const bool fin = part == kPartWhole;
        // Norms feeding a coefficient (LARS, UpdateGradScale) are taken precisely.
        if (lars)
            rc = run_reduce<true, true, false, true>(K, n, numels, sc, hp->grid_ctas, s, fill1,
                                                     hp->trace_events[1], fin, cache);
        else if (hp->refresh_scale)
            rc = run_reduce<true, false, false, true>(K, n, numels, sc, hp->grid_ctas, s, fill1,
                                                      hp->trace_events[1], fin, cache);
        else
            rc = run_reduce<true, false, false, false>(K, n, numels, sc, hp->grid_ctas, s, fill1,
                                                       hp->trace_events[1], fin, cache);
        if (rc == TULA_OK && part == kPartReduce)
            return launch_pdl(k_share, 1, 32, 0, s, sc, share_out);
    }
    if (rc) return rc;
    record(hp->trace_events[2], s);

    auto fill2 = [&](int p, const float **dst) {
        dst[0] = grad_ptrs[p];
        dst[1] = param_ptrs[p];
        dst[2] = mom_ptrs ? mom_ptrs[p] : nullptr;
        dst[3] = per_elem ? hp->scale_elem[p] : nullptr;
    };
    const bool hm = mom_ptrs != nullptr;
    const bool sw = hp->layer_stats != nullptr && !lars;  // the update takes |w|^2
    // The statistics and UpdateGradScale are finished after the update (k_finish<1>).
    sc.fin2 = (hp->layer_stats != nullptr || hp->refresh_scale) ? 1 : 0;
    const int c2 = chunk2(hm, per_elem);
    sc.mode = kModeUpdate;
#define TULA_UPD(HM, PE, SW)                                                                \
    launch_streaming<kNP2>(k_update<HM, PE, SW>, n, numels, c2, Ring2::kThreads,             \
                           Ring2::kSmemBytes, sc, hp->grid_ctas, s, fill2, cache)
    if (hm) {
        if (per_elem) rc = sw ? TULA_UPD(true, true, true) : TULA_UPD(true, true, false);
        else rc = sw ? TULA_UPD(true, false, true) : TULA_UPD(true, false, false);
    } else {
        if (per_elem) rc = sw ? TULA_UPD(false, true, true) : TULA_UPD(false, true, false);
        else rc = sw ? TULA_UPD(false, false, true) : TULA_UPD(false, false, false);
    }
#undef TULA_UPD
    if (rc) return rc;
    record(hp->trace_events[3], s);
    if (sc.fin2) rc = launch_finish<1>(n, sc, s);
    if (rc) return rc;
    record(hp->trace_events[4], s);
    return TULA_OK;
}

}  // namespace

// A plan (tula_ags_plan_create): the step's sizes and pointer arrays, checked once, on one
// device, and the launch tables built from them by the first step of each kernel variant.
struct tula_ags_plan {
    int n = 0, K = 0, device = 0;
    Plan tiles;
    std::vector<int64_t> numels;
    std::vector<float *> params, grads, moms, scale_elem;
    TableCache tables;
};

extern "C" {

int tula_ags_step(float *const *param_ptrs, float *const *grad_ptrs, float *const *mom_ptrs,
                  const int64_t *numels, int n_tensors, float lr, float momentum,
                  float weight_decay, const tula_ags_hparams *hp, void *stream) {
    Plan pl;
    int rc = check_step_args(param_ptrs, grad_ptrs, mom_ptrs, numels, n_tensors, momentum, hp, &pl);
    if (rc) return rc;
    rc = check_ws(hp->workspace, hp->workspace_bytes, n_tensors, pl);
    if (rc) return rc;
    return run_step(param_ptrs, grad_ptrs, mom_ptrs, numels, n_tensors, lr, momentum,
                    weight_decay, hp, hp->workspace, pl, stream);
}

int tula_ags_plan_create(float *const *param_ptrs, float *const *grad_ptrs,
                         float *const *mom_ptrs, const int64_t *numels, int n_tensors,
                         const tula_ags_hparams *hp, tula_ags_plan **plan_out) {
    if (!plan_out) return TULA_ERR_ARG;
    *plan_out = nullptr;
    if (!hp || hp->K < 1 || hp->K > TULA_MAX_K) return TULA_ERR_ARG;
    Plan pl;
    int rc = check_step_tensors(param_ptrs, grad_ptrs, mom_ptrs, hp->scale_elem, numels,
                                n_tensors, hp->K, &pl);
    if (rc) return rc;
    int dev = 0;
    const cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) {
        g_last_cuda = (int)e;
        return TULA_ERR_CUDA;
    }
    try {
        std::unique_ptr<tula_ags_plan> P(new tula_ags_plan);
        const size_t n = (size_t)n_tensors, K = (size_t)hp->K;
        P->n = n_tensors;
        P->K = hp->K;
        P->device = dev;
        P->tiles = pl;
        P->numels.assign(numels, numels + n);
        P->params.assign(param_ptrs, param_ptrs + n);
        P->grads.assign(grad_ptrs, grad_ptrs + K * n);
        if (mom_ptrs) P->moms.assign(mom_ptrs, mom_ptrs + n);
        if (hp->scale_elem) P->scale_elem.assign(hp->scale_elem, hp->scale_elem + n);
        *plan_out = P.release();
    } catch (const std::bad_alloc &) {
        return TULA_ERR_NO_MEMORY;
    }
    return TULA_OK;
}

int tula_ags_plan_step(tula_ags_plan *plan, float lr, float momentum, float weight_decay,
                       const tula_ags_hparams *hp, void *stream) {
    if (!plan || !hp || hp->K != plan->K) return TULA_ERR_ARG;
    int rc = check_step_options(hp, momentum, !plan->moms.empty(), !plan->scale_elem.empty());
    if (rc) return rc;
    rc = check_ws(hp->workspace, hp->workspace_bytes, plan->n, plan->tiles);
    if (rc) return rc;
    int dev = 0;
    const cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) {
        g_last_cuda = (int)e;
        return TULA_ERR_CUDA;
    }
    if (dev != plan->device) return TULA_ERR_ARG;
    tula_ags_hparams h = *hp;
    h.scale_elem = plan->scale_elem.empty() ? nullptr : plan->scale_elem.data();
    return run_step(plan->params.data(), plan->grads.data(),
                    plan->moms.empty() ? nullptr : plan->moms.data(), plan->numels.data(),
                    plan->n, lr, momentum, weight_decay, &h, h.workspace, plan->tiles, stream,
                    kPartWhole, nullptr, nullptr, &plan->tables);
}

int tula_ags_plan_destroy(tula_ags_plan *plan) {
    delete plan;
    return TULA_OK;
}

int tula_ags_shard_reduce(float *const *param_ptrs, float *const *grad_ptrs,
                          float *const *mom_ptrs, const int64_t *numels, int n_tensors,
                          float momentum, const tula_ags_hparams *hp, uint64_t *g2_share,
                          void *stream) {
    Plan pl;
    int rc = check_step_args(param_ptrs, grad_ptrs, mom_ptrs, numels, n_tensors, momentum, hp, &pl);
    if (rc) return rc;
    if (!g2_share || (reinterpret_cast<uintptr_t>(g2_share) & 7u)) return TULA_ERR_ARG;
    rc = check_ws(hp->workspace, hp->workspace_bytes, n_tensors, pl);
    if (rc) return rc;
    return run_step(param_ptrs, grad_ptrs, mom_ptrs, numels, n_tensors, 0.f, momentum, 0.f, hp,
                    hp->workspace, pl, stream, kPartReduce,
                    reinterpret_cast<unsigned long long *>(g2_share), nullptr);
}

int tula_ags_shard_update(float *const *param_ptrs, float *const *grad_ptrs,
                          float *const *mom_ptrs, const int64_t *numels, int n_tensors, float lr,
                          float momentum, float weight_decay, const tula_ags_hparams *hp,
                          const uint64_t *g2_total, void *stream) {
    Plan pl;
    int rc = check_step_args(param_ptrs, grad_ptrs, mom_ptrs, numels, n_tensors, momentum, hp, &pl);
    if (rc) return rc;
    if (!g2_total || (reinterpret_cast<uintptr_t>(g2_total) & 7u)) return TULA_ERR_ARG;
    rc = check_ws(hp->workspace, hp->workspace_bytes, n_tensors, pl);
    if (rc) return rc;
    return run_step(param_ptrs, grad_ptrs, mom_ptrs, numels, n_tensors, lr, momentum,
                    weight_decay, hp, hp->workspace, pl, stream, kPartUpdate, nullptr,
                    reinterpret_cast<const unsigned long long *>(g2_total));
}

int tula_layer_stats(const float *const *param_ptrs, const float *const *grad_ptrs, int K,
                     const int64_t *numels, int n_tensors, double *stats_out, void *workspace,
                     size_t workspace_bytes, void *stream) {
    Plan pl;
    if (!param_ptrs || !grad_ptrs || !stats_out || !valid_numels(numels, n_tensors, K, &pl))
        return TULA_ERR_ARG;
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
    if (!hp || !g_small || !g_large || !valid_numels(numels, n_tensors, 1, &pl))
        return TULA_ERR_ARG;
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
        return launch_streaming<kNP3>(k_scale_elem, n, numels, 4096, kScaleThreads, 0, sc,
                                      hp->grid_ctas, s,
                                      fill);
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
    return run_reduce_k<1, false, false, true, true>(1, n, numels, sc, hp->grid_ctas, s, fill,
                                                     nullptr, true, nullptr);
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
    case TULA_ERR_NO_MEMORY: return "host memory allocation failed";
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
// itself is tula_ags_step's; only where its scratch lives differs.

namespace {

constexpr size_t kStaticScratchBytes = TULA_STATIC_SCRATCH_BYTES;

// One copy per device, alive until the process exits.  In host code this name
// is only a handle: its device address comes from cudaGetSymbolAddress.
static __device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

// Device address of g_static_scratch in the current device's context.  Looked up on every call
// (a host-side table lookup once the module is loaded): a cached address would go stale when the
// context is destroyed and re-created (cudaDeviceReset).
int static_scratch_address(void **out) {
    void *p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_static_scratch);
    if (e != cudaSuccess || !p) {
        g_last_cuda = (int)e;
        return TULA_ERR_CUDA;
    }
    *out = p;
    return TULA_OK;
}

// The static array's error word (its layout's `err` section does not depend on the tensors).
int static_scratch_error_word(unsigned **out) {
    void *base = nullptr;
    const int rc = static_scratch_address(&base);
    if (rc) return rc;
    *out = reinterpret_cast<unsigned *>(static_cast<char *>(base) + ws_layout(1, Plan{}).err);
    return TULA_OK;
}

}  // namespace

extern "C" int tula_ags_step_static_scratch(float *const *param_ptrs, float *const *grad_ptrs,
                                            float *const *mom_ptrs, const int64_t *numels,
                                            int n_tensors, float lr, float momentum,
                                            float weight_decay, const tula_ags_hparams *hp,
                                            void *stream) {
    Plan pl;
    int rc = check_step_args(param_ptrs, grad_ptrs, mom_ptrs, numels, n_tensors, momentum, hp, &pl);
    if (rc) return rc;
    const WsLayout L = ws_layout(n_tensors, pl);
    if (L.total > kStaticScratchBytes) return TULA_ERR_SCRATCH_LIMIT;
    void *scratch = nullptr;
    rc = static_scratch_address(&scratch);
    if (rc) return rc;
    // The array keeps the last call's contents: zero the branch flag, the tile counters and the
    // accumulators (they precede the per-tensor sums) before this call's kernels.  The error
    // word between them is left alone, so that a wait that ran out stays reported until
    // tula_ags_static_scratch_error reads it.
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    char *b = static_cast<char *>(scratch);
    cudaError_t e = cudaMemsetAsync(b, 0, L.err, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(b + L.tiles, 0, L.tsum - L.tiles, s);
    if (e != cudaSuccess) {
        g_last_cuda = (int)e;
        return TULA_ERR_CUDA;
    }
    return run_step(param_ptrs, grad_ptrs, mom_ptrs, numels, n_tensors, lr, momentum,
                    weight_decay, hp, scratch, pl, stream);
}

extern "C" int tula_ags_static_scratch_error(void *stream, int *error_out) {
    if (!error_out) return TULA_ERR_ARG;
    unsigned *word = nullptr;
    int rc = static_scratch_error_word(&word);
    if (rc) return rc;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    unsigned v = 0;
    cudaError_t e = cudaMemcpyAsync(&v, word, sizeof(v), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e == cudaSuccess && v) e = cudaMemsetAsync(word, 0, sizeof(v), s);
    if (e == cudaSuccess && v) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) {
        g_last_cuda = (int)e;
        return TULA_ERR_CUDA;
    }
    *error_out = (int)v;
    return TULA_OK;
}

extern "C" int tula_ags_static_scratch_check_wait_timeout(void *stream) {
    unsigned *word = nullptr;
    const int rc = static_scratch_error_word(&word);
    if (rc) return rc;
    k_wait_check<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(word);
    g_launches.fetch_add(1, std::memory_order_relaxed);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) {
        g_last_cuda = (int)e;
        return TULA_ERR_CUDA;
    }
    return TULA_OK;
}
