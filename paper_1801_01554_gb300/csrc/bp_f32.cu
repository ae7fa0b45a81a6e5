// float32 back-propagation step on CUDA cores (FFMA).
//
// One training step over a group of B patterns runs in two phases:
//
//   pattern phase (case-parallel, Section 4.1): every CTA copies all the
//     weights into its shared memory with one bulk copy (they fit for the
//     NETtalk-sized nets of Section 6.3; larger nets read them from L2), while
//     its first input and target rows arrive, then runs the whole net on its
//     share of the patterns: forward pass (Section 3), output delta (t-o)o(1-o)
//     with the summed squared error, hidden deltas (W^T delta) h(1-h) for every
//     hidden layer and none for the inputs (Section 6.1).  Weights are kept as
//     padded rows [W | b | 0..] and activations with a trailing 1, so a row
//     product is a unit's net input with its bias; the forward pass sums each
//     dot product as a binary tree across a lane group (Section 10.3).
//     Activation and delta rows go to global scratch in column blocks
//     ([cap][32] activations, [cap][8] deltas).
//
//   weight phase (Section 5's "bundle" of weights processed over the whole
//     group of cases): one CTA per 8 x 32 tile of [W_l | b_l] streams the
//     group's deltas and activations through shared memory, two contiguous
//     bulk copies per chunk of 512 patterns,
//     sums delta[p,j] a[p,i] over all patterns with 4 x 4 register blocks per
//     lane and a warp butterfly (Sections 3, 4.1), then either accumulates into
//     G (bp_backward) or applies the momentum update of Section 6.2.1 at once
//     (training), so the pooled change never goes to memory.
//
// A training launch is a persistent cooperative kernel that loops over any
// number of groups with a grid barrier between the phases; every wait in the
// barrier is bounded and latches kFlagTimeout instead of hanging.  Groups of at
// most 4 patterns run on one CTA instead (k_train_small), with the weights
// resident in its shared memory for the whole launch.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdio>

#include "bp_internal.h"

namespace bp {
namespace {

constexpr int kThreads = 512;
constexpr int kWarps = kThreads / 32;
constexpr int kTU = 8;            // weight-tile rows (output units) of the whole-tile weight phase
constexpr int kTUW = 16;          // weight-tile rows of the balanced weight phase (large groups)
constexpr int kDB = 8;            // delta columns per scratch block
constexpr int kTJ = 32;           // weight-tile columns (inputs; the bias is the last input)
constexpr int kPC = 512;          // patterns per staged chunk of the weight phase
static_assert(kPC % (kWarps * 4) == 0, "each warp takes whole groups of 4 rows of a chunk");
// a chunk buffer of a TU-row tile: the [kPC][kTJ] activation block, then TU / kDB delta blocks
template <int TU>
__host__ __device__ constexpr int chunk_floats() { return kPC * (kTJ + TU); }
constexpr int kWarpRows = kPC / kWarps;   // rows of a chunk per warp
// chunk buffers in flight: the CTA syncs once per chunk, so the chunk is as
// large as two buffers allow (256 x 3 and 128 x 6 measured slower)
constexpr int kNBuf = 2;
constexpr int kWidePG = 32;       // patterns per pass of the whole-row-per-lane forward
// weight-phase buffers (each chunk: the [kPC][kTJ] activation block, 128-byte
// swizzled, then the [kPC][kTU] delta block), plus room to align them to 1 KB
constexpr size_t kGradFloats = kNBuf * chunk_floats<kTU>() + 256;
constexpr size_t kGradFloatsW = kNBuf * chunk_floats<kTUW>() + 256;   // balanced weight phase

constexpr unsigned long long kWaitNs = 2000000000ull;   // 2 s per wait
constexpr unsigned kWaitIters = 1u << 26;

// ------------------------------------------------------------ small helpers
// Logistic: CUDA's expf and the fast reciprocal divide (2 ulp, far inside the
// float32 bar; for 1 + e^-x beyond 2^126 the quotient is 0, the logistic's value).
__device__ __forceinline__ float sigmoid_f(float x) { return __fdividef(1.0f, 1.0f + expf(-x)); }

// Checked build (-DBP_CHECK): phases test that their shared-memory regions fit
// the launch's dynamic shared memory and that their rows and tile origins lie
// inside their buffers; a failed test latches kFlagBounds (bp_check reports it)
// and the phase skips its accesses.  Without BP_CHECK the tests compile away.
extern __shared__ __align__(128) float g_dyn_smem[];   // every kernel's dynamic shared memory
__device__ __forceinline__ const float* pattern_smem_base() { return g_dyn_smem; }
__device__ __forceinline__ unsigned dyn_smem_floats() {
    unsigned b;
    asm("mov.u32 %0, %%dynamic_smem_size;" : "=r"(b));
    return b / 4;
}
__device__ __forceinline__ bool bounds_ok(bool ok, int* flags) {
#ifdef BP_CHECK
    if (!ok) {
        atomicOr(flags, kFlagBounds);
        return false;
    }
#else
    (void)ok;
    (void)flags;
#endif
    return true;
}

// Table-lookup logistic (Section 4.3, Figure 3): the logistic at 256 equally
// spaced points over [-15, 15], built in shared memory by each CTA that runs a
// forward pass with the table mode on.  Inputs outside the range take the end
// values; inside, x is remapped to [0, 255], the integer part picks the entry
// and the fractional part interpolates linearly to the next one.  NaN stays NaN.
constexpr int kSigPoints = 256;
__shared__ float s_sigtab[kSigPoints];

__device__ void sigmoid_table_init(const F32View& v) {
    if (v.sig_table)
        for (int k = threadIdx.x; k < kSigPoints; k += blockDim.x)
            s_sigtab[k] = sigmoid_f(-15.f + (30.f * (float)k) / (float)(kSigPoints - 1));
}

__device__ __forceinline__ float sigmoid_tab(float x) {
    if (x != x) return x;
    const float xc = fminf(fmaxf(x, -15.f), 15.f);
    const float x1 = (xc + 15.f) * ((float)(kSigPoints - 1) / 30.f);
    const int i = min((int)x1, kSigPoints - 2);   // x1 >= 0: truncation is the floor
    const float f = x1 - (float)i;
    const float t0 = s_sigtab[i];
    return fmaf(f, s_sigtab[i + 1] - t0, t0);
}

__device__ __forceinline__ unsigned ld_acquire(const unsigned* p) {
    unsigned v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ unsigned long long global_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}

// Grid barrier for a cooperative launch.  bar[1] counts arrivals over every
// launch on the net; bar[0] holds its value at the end of the previous launch.
// Barrier k of a launch completes when the count reaches bar[0] + k * grid:
// thread 0 of each CTA adds its arrival with a fire-and-forget release
// reduction and then polls the count (no CTA has to relay a release).  The
// wait is bounded; on a timeout the error word latches kFlagTimeout and the
// function returns false in every thread of the CTA (the caller must then
// return).  Counts compare modulo 2^32.
__device__ __forceinline__ bool count_reached(unsigned v, unsigned target) {
    return (int)(v - target) >= 0;
}
__device__ bool grid_barrier(unsigned* bar, unsigned target, int* flags, unsigned long long limit_ns) {
    __syncthreads();
    int ok = 1;
    if (threadIdx.x == 0) {
        // the release is cumulative: with the CTA barrier above it also orders
        // every thread's earlier writes before the arrival (no separate fence)
        asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(bar + 1), "r"(1u) : "memory");
        const unsigned long long t0 = global_ns();
        unsigned it = 0;
        while (!count_reached(ld_acquire(bar + 1), target)) {
            ++it;
            if (it > kWaitIters || ((it & 63u) == 0 && global_ns() - t0 > limit_ns)) {
                atomicOr(flags, kFlagTimeout);
                ok = 0;
                break;
            }
        }
    }
    return __syncthreads_and(ok) != 0;
}

// Limit of the grid barrier's wait: 2 s, or in the checked build the limit a
// test set on the net (bp_debug_wait_test), so that a test can make a wait run
// out in about a millisecond.
__device__ __forceinline__ unsigned long long wait_limit_ns(const F32View& v) {
#ifdef BP_CHECK
    return v.wait_ns != 0 ? v.wait_ns : kWaitNs;
#else
    (void)v;
    return kWaitNs;
#endif
}

__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

// Sum held in thread 0 (deterministic order).
__device__ float block_sum(float x) {
    __shared__ float red[kWarps];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    x = warp_sum(x);
    __syncthreads();
    if (lane == 0) red[warp] = x;
    __syncthreads();
    float r = 0.f;
    if (threadIdx.x == 0) {
        for (int w = 0; w < kWarps; ++w) r += red[w];
    }
    return r;
}

// ------------------------------------------------------------ weights in shared memory
__device__ __forceinline__ void mbar_init1(uint64_t* bar) {
    if (threadIdx.x == 0) {
        asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(bar)) : "memory");
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();
}

__device__ __forceinline__ bool mbar_try(uint64_t* bar, unsigned parity) {
    unsigned done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return done != 0;
}

// Waits (bounded) for the phase with the given parity of an mbarrier; on a
// timeout latches kFlagTimeout and returns false.  The copy it waited for may
// then still be in flight: the caller issues no more copies and drains
// (mbar_drain) every copy it issued before the CTA may return.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, unsigned parity, int* flags,
                                          unsigned long long limit_ns = kWaitNs) {
    const unsigned long long t0 = global_ns();
    for (unsigned it = 0;; ++it) {
        if (mbar_try(bar, parity)) return true;
        if ((it & 255u) == 255u && global_ns() - t0 > limit_ns) {
            atomicOr(flags, kFlagTimeout);
            return false;
        }
    }
}

// Second bounded wait for a copy whose first wait ran out, so that its bulk
// writes land before the CTA exits (shared memory of an exited CTA may belong
// to the next CTA on that SM).  The error is already latched.
__device__ __forceinline__ void mbar_drain(uint64_t* bar, unsigned parity, unsigned long long limit_ns = kWaitNs) {
    const unsigned long long t0 = global_ns();
    while (!mbar_try(bar, parity) && global_ns() - t0 < limit_ns) {
    }
}

__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }
__device__ __forceinline__ void cp_async4(float* dst, const float* src) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}

// Starts the copy of theta[0, P) into shared memory Ws: one bulk copy on the
// mbarrier for the 16-byte aligned part (thread 0), and 4-byte cp.async copies
// for the tail of at most 3 floats by the last threads (no thread stalls on a
// load here; the tail belongs to the issuing thread's next cp.async group,
// which stage_weights_wait waits for).
__device__ void stage_weights_issue(const float* theta, long long P, float* Ws, uint64_t* bar) {
    const long long P16 = P & ~3LL;
    if (threadIdx.x == 0 && P16 > 0) {
        asm volatile("fence.proxy.async.global;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        const unsigned bytes = (unsigned)(P16 * 4);
        asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
                     "r"(bytes)
                     : "memory");
        asm volatile(
            "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
                "r"(smem_u32(Ws)),
            "l"(theta), "r"(bytes), "r"(smem_u32(bar))
            : "memory");
    }
    const long long k = P16 + (kThreads - 1 - (int)threadIdx.x);
    if (k < P) cp_async4(Ws + k, theta + k);
}

// Bounded wait for a copy started by stage_weights_issue (every thread; the
// tail needs a CTA barrier after this).  The thread's cp.async groups are
// waited for too (the tail's, and any rows issued since).  Returns false in a
// thread whose wait ran out; callers make that CTA-uniform with
// __syncthreads_or and then call stage_weights_drain before returning.
// A copy in flight: its mbarrier (none if bar is null), the parity of the
// phase it completes, and its length.  Passed by value, so that nothing of it
// lives in local memory.
struct WeightCopy {
    uint64_t* bar;
    unsigned parity;
    long long P;
};
__device__ __forceinline__ bool stage_weights_wait(const WeightCopy& w, int* flags) {
    bool ok = true;
    if (w.bar != nullptr && (w.P & ~3LL) > 0) ok = mbar_wait(w.bar, w.parity, flags);
    cp_async_commit();
    cp_async_wait<0>();
    return ok;
}

// The mbarrier phase parity after a copy started by stage_weights_issue.
__device__ __forceinline__ unsigned after_copy(unsigned parity, long long P) {
    return (P & ~3LL) > 0 ? parity ^ 1u : parity;
}

// After a weight copy whose wait ran out in some thread: thread 0 waits for
// that copy again (bounded) so that no bulk write is still landing when the CTA
// returns.  Every thread calls it.
__device__ void stage_weights_drain(const WeightCopy& w) {
    if (threadIdx.x == 0 && w.bar != nullptr && (w.P & ~3LL) > 0) mbar_drain(w.bar, w.parity);
    __syncthreads();
}

// Copies the weights into shared memory and waits for them; false (in every
// thread) if the copy timed out, in which case it has been drained and the
// caller must return.
__device__ bool stage_weights(const float* theta, long long P, float* Ws, uint64_t* bar,
                              unsigned& phase, int* flags) {
    stage_weights_issue(theta, P, Ws, bar);
    const WeightCopy wc{bar, phase, P};
    phase = after_copy(phase, P);
    if (__syncthreads_or(!stage_weights_wait(wc, flags))) {
        stage_weights_drain(wc);
        return false;
    }
    return true;
}

// ------------------------------------------------------------ pattern phase

// Shared memory: the weights (WS) at the bottom, the pattern buffers above
// them; the weight phase reuses the bottom kGradFloats floats for its tiles.
template <bool WS>
__device__ __forceinline__ float* pattern_base(const F32View& v, float* smem) {
    return WS ? smem + v.wsm : smem;
}

// Pattern buffers (PatLayout, computed on the host): the activation rows keep
// the true unit's 1 in column n_l and zeros after it, so that a padded weight
// row times an activation row is the unit's net input with its bias.
//
// Row loops below give each pattern kThreads / PG threads (a compile-time
// split: pattern = thread / TP, column = thread % TP), so no thread divides.

// Issues the copies of the input rows (into the layer-0 activation rows) and
// target rows of patterns [p0, p0 + np), and writes the true unit's 1 and the
// zero pads of every activation and delta row; rows past np are zeroed.  One
// cp.async group; the caller waits for it before use.
template <int PG>
__device__ void load_rows(const F32View& v, const PatLayout& q, const float* X, const float* T,
                          int p0, int np, float* smem) {
    constexpr int TP = kThreads / PG;
    const int p = threadIdx.x / TP, c0 = threadIdx.x % TP;
    const bool live = p < np;
    const int n0 = v.n[0], nL = v.n[v.L];
    if (X != nullptr) {
        float* dst = smem + q.sa[0] + p * v.apitch[0];
        const float* src = X + (size_t)(p0 + p) * n0;
        for (int i = c0; i < n0; i += TP) {
            if (live) cp_async4(dst + i, src + i);
            else dst[i] = 0.f;
        }
    }
    if (T != nullptr) {
        float* dst = smem + q.st + p * nL;
        const float* src = T + (size_t)(p0 + p) * nL;
        for (int k = c0; k < nL; k += TP) {
            if (live) cp_async4(dst + k, src + k);
            else dst[k] = 0.f;
        }
    }
    cp_async_commit();
    // pads: at most 4 columns per row (apitch - n in [1, 4], dpitch - n in [0, 3])
    if (c0 < 4) {
        for (int l = 0; l <= v.L; ++l) {
            const int col = v.n[l] + c0;
            if (col < v.apitch[l]) smem[q.sa[l] + p * v.apitch[l] + col] = (c0 == 0) ? 1.f : 0.f;
            if (l >= 1 && col < v.dpitch[l]) smem[q.sd[l] + p * v.dpitch[l] + col] = 0.f;
        }
    }
}

// Butterfly reduce-scatter of V per-lane values over aligned groups of V lanes:
// afterwards lane k of a group holds in v[0] the group's sum of value k mod V.
// A binary-tree sum (Section 10.3), V - 1 shuffles for V sums.
template <int V>
__device__ __forceinline__ void reduce_scatter(float (&v)[V], int lane) {
#pragma unroll
    for (int half = V / 2; half >= 1; half >>= 1) {
        const bool up = (lane & half) != 0;
#pragma unroll
        for (int k = 0; k < half; ++k) {
            const float send = up ? v[k] : v[k + half];
            const float keep = up ? v[k + half] : v[k];
            v[k] = keep + __shfl_xor_sync(0xffffffffu, send, half);
        }
    }
}

__device__ __forceinline__ float4 ld4(const float* p) { return *reinterpret_cast<const float4*>(p); }

// Units per lane group of the forward pass for a group size: every unit's
// weights are read once per CTA, every activation row once per lane group.
template <int PG>
__host__ __device__ constexpr int fwd_units() { return PG >= 8 ? 4 : 8 / PG; }

// Forward through one layer for PG patterns held in shared memory:
// out[p][j] = sigma(sum_i W[j][i] in[p][i]) over the kp columns of the padded
// rows (the bias column meets the activation row's 1).  A group of S lanes
// (V = U * PG, 2V or 4V up to 32; within one warp) owns U units and sums V
// dot products over interleaved float4 columns, then reduces them across its
// lanes: a reduce-scatter inside each V-lane block, then butterflies across
// blocks.
template <int PG>
__device__ void forward_layer(const float* W, int kp, int n_out, const float* s_in, float* s_out,
                              int kp_out, bool table) {
    constexpr int U = fwd_units<PG>();
    constexpr int V = U * PG;
    static_assert(V <= 32, "a lane group holds at most 32 sums");
    const int G = (n_out + U - 1) / U;
    int S = 32;
    while (S > V && G * S > kThreads) S >>= 1;
    const int gpp = kThreads / S;
    const int tid = threadIdx.x, lane = tid & 31;
    const int s = tid & (S - 1), g0 = tid / S;
    const int K4 = kp >> 2;
    for (int gb = 0; gb < G; gb += gpp) {   // uniform trip count: every lane shuffles
        const int g = gb + g0;
        const int j0 = g * U;
        float acc[V];
#pragma unroll
        for (int k = 0; k < V; ++k) acc[k] = 0.f;
        if (g < G) {
            const float* wr[U];
#pragma unroll
            for (int u = 0; u < U; ++u) wr[u] = W + (size_t)min(j0 + u, n_out - 1) * kp;
            for (int k = s; k < K4; k += S) {
                float4 a[PG];
#pragma unroll
                for (int p = 0; p < PG; ++p) a[p] = ld4(s_in + p * kp + 4 * k);
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    const float4 w = ld4(wr[u] + 4 * k);
#pragma unroll
                    for (int p = 0; p < PG; ++p) {
                        float t = acc[u * PG + p];
                        t = fmaf(w.x, a[p].x, t);
                        t = fmaf(w.y, a[p].y, t);
                        t = fmaf(w.z, a[p].z, t);
                        t = fmaf(w.w, a[p].w, t);
                        acc[u * PG + p] = t;
                    }
                }
            }
        }
        reduce_scatter<V>(acc, lane);
        float r = acc[0];
        for (int o = V; o < S; o <<= 1) r += __shfl_xor_sync(0xffffffffu, r, o);
        if (s < V && g < G) {
            const int u = s / PG, p = s % PG;
            const int j = j0 + u;
            if (j < n_out) s_out[p * kp_out + j] = table ? sigmoid_tab(r) : sigmoid_f(r);
        }
    }
}

// Forward through one layer for groups of 32 patterns (PG a multiple of 32):
// lane p of a warp owns pattern p of its warp's group and sums that pattern's
// dot products over whole rows for U units at a time, with no cross-lane
// reduction.  The warps of a group split the units; every lane of a warp reads
// the same weight float4 (a broadcast), so each activation float4 feeds 4 U
// FMAs.  The activation rows are read at stride kp: kp / 4 odd keeps the 32
// lanes' float4 reads at the minimum of four wavefronts (f32_plan checks it).
template <int PG, int U>
__device__ void forward_layer_lanes(const float* W, int kp, int n_out, const float* s_in, float* s_out,
                                    int kp_out, bool table) {
    static_assert(PG % 32 == 0, "whole warps of patterns");
    constexpr int kGroups = PG / 32;
    constexpr int kWarpsPerGroup = kWarps / kGroups;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int p = (warp / kWarpsPerGroup) * 32 + lane, wi = warp % kWarpsPerGroup;
    const int K4 = kp >> 2;
    const float* a = s_in + p * kp;
    for (int j0 = wi * U; j0 < n_out; j0 += kWarpsPerGroup * U) {
        int wo[U];   // row offsets (rows past the layer repeat its last row)
#pragma unroll
        for (int u = 0; u < U; ++u) wo[u] = min(j0 + u, n_out - 1) * kp;
        float acc[U];
#pragma unroll
        for (int u = 0; u < U; ++u) acc[u] = 0.f;
        for (int k = 0; k < K4; ++k) {
            const float4 x = ld4(a + 4 * k);
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const float4 w = ld4(W + wo[u] + 4 * k);
                float t = acc[u];
                t = fmaf(w.x, x.x, t);
                t = fmaf(w.y, x.y, t);
                t = fmaf(w.z, x.z, t);
                t = fmaf(w.w, x.w, t);
                acc[u] = t;
            }
        }
#pragma unroll
        for (int u = 0; u < U; ++u)
            if (j0 + u < n_out) s_out[p * kp_out + j0 + u] = table ? sigmoid_tab(acc[u]) : sigmoid_f(acc[u]);
    }
}

// Forward through one layer for groups of 32 patterns, register-blocked: lane
// l holds patterns l % 16 and l % 16 + 16 of its warp's group and units
// j0 + 4 (l / 16) .. + 3 of the warp's 8, so every activation float4 feeds 16
// FMAs and every weight float4 8.  A warp's loads per float4 step are two
// activation reads of 16 rows each and four weight reads of 2 rows each (4
// rows apart), for 32 FMAs per lane.  With kp / 4 odd (f32_plan checks it) the
// 16 rows fall on 8 distinct 16-byte bank groups twice (two wavefronts, the
// minimum for 256 bytes) and the two weight rows, kp float4 apart, on
// different bank groups (one wavefront each).
template <int PG>
__device__ void forward_layer_blocked(const float* W, int kp, int n_out, const float* s_in, float* s_out,
                                      int kp_out, bool table) {
    static_assert(PG % 32 == 0, "whole warps of patterns");
    constexpr int kGroups = PG / 32;
    constexpr int kWarpsPerGroup = kWarps / kGroups;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int p0 = (warp / kWarpsPerGroup) * 32 + (lane & 15), wi = warp % kWarpsPerGroup;
    const int K4 = kp >> 2;
    const float* a0 = s_in + p0 * kp;
    const float* a1 = a0 + 16 * kp;
    for (int jb = wi * 8; jb < n_out; jb += kWarpsPerGroup * 8) {
        const int j0 = jb + 4 * (lane >> 4);
        const float* w0 = W + min(j0, n_out - 1) * kp;   // rows past the layer repeat its last row
        const float* w1 = W + min(j0 + 1, n_out - 1) * kp;
        const float* w2 = W + min(j0 + 2, n_out - 1) * kp;
        const float* w3 = W + min(j0 + 3, n_out - 1) * kp;
        float c0[4] = {0.f, 0.f, 0.f, 0.f}, c1[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 2
        for (int k = 0; k < K4; ++k) {
            const float4 x0 = ld4(a0 + 4 * k), x1 = ld4(a1 + 4 * k);
            const float4 w[4] = {ld4(w0 + 4 * k), ld4(w1 + 4 * k), ld4(w2 + 4 * k), ld4(w3 + 4 * k)};
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                float t0 = c0[u], t1 = c1[u];
                t0 = fmaf(w[u].x, x0.x, t0);
                t1 = fmaf(w[u].x, x1.x, t1);
                t0 = fmaf(w[u].y, x0.y, t0);
                t1 = fmaf(w[u].y, x1.y, t1);
                t0 = fmaf(w[u].z, x0.z, t0);
                t1 = fmaf(w[u].z, x1.z, t1);
                t0 = fmaf(w[u].w, x0.w, t0);
                t1 = fmaf(w[u].w, x1.w, t1);
                c0[u] = t0;
                c1[u] = t1;
            }
        }
        float* o0 = s_out + p0 * kp_out + j0;
        float* o1 = o0 + 16 * kp_out;
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            if (j0 + u < n_out) {
                o0[u] = table ? sigmoid_tab(c0[u]) : sigmoid_f(c0[u]);
                o1[u] = table ? sigmoid_tab(c1[u]) : sigmoid_f(c1[u]);
            }
        }
    }
}

// Forward through one layer for PG patterns held in shared memory: the
// lane-group form below for small groups, whole rows per lane from 32 up.
template <int PG>
__device__ __forceinline__ void forward_any(const float* W, int kp, int n_out, const float* s_in, float* s_out,
                                            int kp_out, bool table) {
    if constexpr (PG >= 32) {
        if (n_out >= 4 * kWarps / (PG / 32))
            forward_layer_blocked<PG>(W, kp, n_out, s_in, s_out, kp_out, table);
        else
            forward_layer_lanes<PG, 2>(W, kp, n_out, s_in, s_out, kp_out, table);
    } else {
        forward_layer<PG>(W, kp, n_out, s_in, s_out, kp_out, table);
    }
}

// Hidden deltas of layer l for PG patterns: d_l[p][i] = (sum_j W_{l+1}[j][i]
// d_{l+1}[p][j]) a_l[p][i] (1 - a_l[p][i]), one thread per (pattern, unit)
// summing over the next layer's units in order.  dnt holds d_{l+1}
// pattern-minor ([nn][PG]).  Writes d_l as rows (dl, pitch dpl) and, if dlt is
// not null, pattern-minor (dlt).
template <int PG>
__device__ void hidden_delta(const float* Wn, int kpn, int n, int nn, const float* dnt,
                             const float* al, int apl, float* dl, int dpl, float* dlt) {
    for (int e = threadIdx.x; e < PG * n; e += kThreads) {
        const int p = e / n, i = e - p * n;
        float acc = 0.f;
#pragma unroll 4
        for (int j = 0; j < nn; ++j) acc = fmaf(dnt[j * PG + p], Wn[(size_t)j * kpn + i], acc);
        const float a = al[p * apl + i];
        const float d = acc * a * (1.f - a);
        dl[p * dpl + i] = d;
        if (dlt != nullptr) dlt[i * PG + p] = d;
    }
}

// Hidden deltas for groups of 32 patterns (PG a multiple of 32): lane p owns
// pattern p of its warp's group and sums over the next layer's units for U of
// this layer's units at a time.  The next layer's deltas are read
// pattern-minor (consecutive lanes, no bank conflict), the weight row pieces
// W_{l+1}[j][i0 .. i0 + U) as broadcasts.
template <int PG, int U>
__device__ void hidden_delta_lanes(const float* Wn, int kpn, int n, int nn, const float* dnt, const float* al,
                                   int apl, float* dl, int dpl, float* dlt) {
    static_assert(PG % 32 == 0 && U % 4 == 0, "whole warps of patterns, float4 pieces of rows");
    constexpr int kGroups = PG / 32;
    constexpr int kWarpsPerGroup = kWarps / kGroups;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int p = (warp / kWarpsPerGroup) * 32 + lane, wi = warp % kWarpsPerGroup;
    for (int i0 = wi * U; i0 < n; i0 += kWarpsPerGroup * U) {
        float acc[U];
#pragma unroll
        for (int u = 0; u < U; ++u) acc[u] = 0.f;
        if (i0 + U <= kpn) {   // the row piece lies inside the padded row
            for (int j = 0; j < nn; ++j) {
                const float d = dnt[j * PG + p];
                const float* wrow = Wn + (size_t)j * kpn + i0;
#pragma unroll
                for (int q = 0; q < U / 4; ++q) {
                    const float4 w = ld4(wrow + 4 * q);
                    acc[4 * q] = fmaf(d, w.x, acc[4 * q]);
                    acc[4 * q + 1] = fmaf(d, w.y, acc[4 * q + 1]);
                    acc[4 * q + 2] = fmaf(d, w.z, acc[4 * q + 2]);
                    acc[4 * q + 3] = fmaf(d, w.w, acc[4 * q + 3]);
                }
            }
        } else {
            for (int j = 0; j < nn; ++j) {
                const float d = dnt[j * PG + p];
#pragma unroll
                for (int u = 0; u < U; ++u)
                    if (i0 + u < n) acc[u] = fmaf(d, Wn[(size_t)j * kpn + i0 + u], acc[u]);
            }
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int i = i0 + u;
            if (i < n) {
                const float a = al[p * apl + i];
                const float dv = acc[u] * a * (1.f - a);
                dl[p * dpl + i] = dv;
                if (dlt != nullptr) dlt[i * PG + p] = dv;
            }
        }
    }
}

// Scratch addresses (see F32View): float4 chunk k (columns 4k .. 4k + 3) of
// pattern p's activations of layer l, and of its deltas.
__device__ __forceinline__ float4* act_chunk(const F32View& v, int l, long long p, int k) {
    return reinterpret_cast<float4*>(v.A + v.aoff[l] + (long long)(k >> 3) * v.cap * 32 + p * 32) +
           ((k & 7) ^ (int)(p & 7));
}
__device__ __forceinline__ float4* delta_chunk(const F32View& v, int l, long long p, int k) {
    return reinterpret_cast<float4*>(v.D + v.doff[l] + (long long)(k >> 1) * v.cap * 8 + p * 8) +
           ((k & 1) ^ (int)((p >> 2) & 1));
}

// Writes np rows (pitch floats apart in shared memory) of layer l's
// activations (or deltas) to the blocked scratch layout; chunks past the row
// pitch are written as zeros so that every block column is defined.
template <int PG, bool DELTA>
__device__ __forceinline__ void rows_to_scratch(const F32View& v, int l, const float* src, int pitch,
                                                int p0, int np) {
    constexpr int TP = kThreads / PG;
    const int p = threadIdx.x / TP, c0 = threadIdx.x % TP;
    if (p < np) {
        const int q4 = pitch >> 2, nk = DELTA ? 2 * v.dtb[l] : 8 * v.acb[l];
        for (int k = c0; k < nk; k += TP) {
            const float4 x = k < q4 ? reinterpret_cast<const float4*>(src + p * pitch)[k]
                                    : make_float4(0.f, 0.f, 0.f, 0.f);
            *(DELTA ? delta_chunk(v, l, p0 + p, k) : act_chunk(v, l, p0 + p, k)) = x;
        }
    }
}

// Runs the pattern phase for this CTA's share of the group's B patterns
// (patterns [blockIdx.x*B/gridDim.x, (blockIdx.x+1)*B/gridDim.x), PG at a time).
//   Wb: the weights in the padded layout (shared memory copy or global theta)
//   q: the pattern buffers' layout, relative to smem
//   do_fwd: forward pass from X (else the activations are reloaded from scratch)
//   do_bwd: deltas against T, written to scratch
//   Y: if not null, the outputs are copied there ([B, n_L] packed)
// Returns this CTA's summed squared error (valid in thread 0) and whether the
// weight copy arrived.
//   wc: if wc.bar is not null, a weight copy into shared memory is still in
//       flight; it is waited for after the first rows have been issued, so
//       that the two loads overlap
//   to_scratch: write the activation and delta rows to scratch (A, D)
//   rows_issued: the first pass's rows were already issued (load_rows)
//   whole: this CTA takes all B patterns (diagnostic mode) instead of its share
// ok is false (in every thread) if the weight copy timed out: it has then been
// drained and the phase did nothing, so the caller returns.
struct PhaseResult {
    float sse;
    bool ok;
};
template <int PG>
__device__ PhaseResult pattern_phase(const F32View& v, const PatLayout& q, const float* Wb,
                                     const float* __restrict__ X, const float* __restrict__ T, int B,
                                     bool do_fwd, bool do_bwd, float* __restrict__ Y, float* smem,
                                     WeightCopy wc = WeightCopy{nullptr, 0u, 0}, bool to_scratch = true,
                                     bool rows_issued = false, bool whole = false) {
    constexpr int TP = kThreads / PG;
    const int L = v.L;
    const int tid = threadIdx.x;
    const int pr = tid / TP, c0 = tid % TP;   // row-loop split
    const int nL = v.n[L];
    float sse = 0.f;
    const int q_lo = whole ? 0 : (int)((long long)B * blockIdx.x / gridDim.x);
    const int q_hi = whole ? B : (int)((long long)B * (blockIdx.x + 1) / gridDim.x);
    if (!bounds_ok((size_t)(smem - pattern_smem_base()) + q.total <= dyn_smem_floats() &&
                       ((!to_scratch && do_fwd) || B <= v.cap),
                   v.flags)) {
        if (wc.bar != nullptr && __syncthreads_or(!stage_weights_wait(wc, v.flags))) {
            stage_weights_drain(wc);
            return PhaseResult{0.f, false};
        }
        return PhaseResult{block_sum(0.f), true};
    }
    for (int p0 = q_lo; p0 < q_hi; p0 += PG) {
        const int np = min(PG, q_hi - p0);
        if (!(rows_issued && p0 == q_lo))
            load_rows<PG>(v, q, do_fwd ? X : nullptr, do_bwd ? T : nullptr, p0, np, smem);
        if (!do_fwd) {
            // activations of the last forward, reloaded from scratch
            for (int l = 1; l <= L; ++l) {
                const int ap = v.apitch[l], q4 = ap >> 2;
                float4* dst = reinterpret_cast<float4*>(smem + q.sa[l] + pr * ap);
                for (int c = c0; c < q4; c += TP)
                    dst[c] = (pr < np) ? __ldcg(act_chunk(v, l, p0 + pr, c)) : make_float4(0.f, 0.f, 0.f, 0.f);
            }
        }
        bool w_ok = true;
        const WeightCopy waited = wc;
        if (wc.bar != nullptr) {
            w_ok = stage_weights_wait(wc, v.flags);
            wc.bar = nullptr;
        }
        cp_async_wait<0>();
        if (__syncthreads_or(!w_ok)) {
            // the weight copy did not arrive in time: let it land, do nothing more
            stage_weights_drain(waited);
            return PhaseResult{0.f, false};
        }
        if (do_fwd) {
            // the input rows go to scratch first, so that their stores drain during the forward pass
            if (to_scratch) rows_to_scratch<PG, false>(v, 0, smem + q.sa[0], v.apitch[0], p0, np);
            for (int l = 1; l <= L; ++l) {
                forward_any<PG>(Wb + v.woff[l], v.kp[l], v.n[l], smem + q.sa[l - 1], smem + q.sa[l],
                                v.apitch[l], v.sig_table != 0);
                __syncthreads();
            }
            // activation rows, bias column and pads included
            for (int l = 1; l <= L && to_scratch; ++l)
                rows_to_scratch<PG, false>(v, l, smem + q.sa[l], v.apitch[l], p0, np);
            if (Y != nullptr && pr < np) {
                for (int k = c0; k < nL; k += TP)
                    Y[(size_t)(p0 + pr) * nL + k] = smem[q.sa[L] + pr * v.apitch[L] + k];
            }
        }
        if (do_bwd) {
            // output delta and error sum (Section 3, fn. 5)
            const int apL = v.apitch[L], dpL = v.dpitch[L];
            float* dlt = (L >= 2) ? smem + q.sdt[L] : nullptr;
            for (int k = c0; k < nL; k += TP) {
                float d = 0.f;
                if (pr < np) {
                    const float o = smem[q.sa[L] + pr * apL + k];
                    const float err = smem[q.st + pr * nL + k] - o;
                    sse = fmaf(err, err, sse);
                    d = err * o * (1.f - o);
                }
                smem[q.sd[L] + pr * dpL + k] = d;
                if (dlt != nullptr) dlt[k * PG + pr] = d;
            }
            __syncthreads();
            // hidden deltas, output side first; no delta for the input layer
            for (int l = L - 1; l >= 1; --l) {
                if constexpr (PG >= 32)
                    hidden_delta_lanes<PG, 8>(Wb + v.woff[l + 1], v.kp[l + 1], v.n[l], v.n[l + 1],
                                              smem + q.sdt[l + 1], smem + q.sa[l], v.apitch[l], smem + q.sd[l],
                                              v.dpitch[l], l >= 2 ? smem + q.sdt[l] : nullptr);
                else
                    hidden_delta<PG>(Wb + v.woff[l + 1], v.kp[l + 1], v.n[l], v.n[l + 1], smem + q.sdt[l + 1],
                                     smem + q.sa[l], v.apitch[l], smem + q.sd[l], v.dpitch[l],
                                     l >= 2 ? smem + q.sdt[l] : nullptr);
                __syncthreads();
            }
            for (int l = 1; l <= L && to_scratch; ++l)
                rows_to_scratch<PG, true>(v, l, smem + q.sd[l], v.dpitch[l], p0, np);
        }
        __syncthreads();
    }
    if (wc.bar != nullptr && __syncthreads_or(!stage_weights_wait(wc, v.flags))) {   // no patterns here
        stage_weights_drain(wc);
        return PhaseResult{0.f, false};
    }
    // the weight phase reads the activation and delta rows through TMA
    asm volatile("fence.proxy.async.global;" ::: "memory");
    return PhaseResult{block_sum(sse), true};
}

// ------------------------------------------------------------ weight phase
// Fault guard of Section 8: a total weight change outside (-guard, guard), or
// not a number, is set to zero and counted (off while guard <= 0).
__device__ __forceinline__ float guard_change(const F32View& v, float g) {
    if (v.guard > 0.f && !(fabsf(g) <= v.guard)) {
        atomicAdd(v.faults, 1u);
        return 0.f;
    }
    return g;
}

// The same test without an atomic per change: zeroes and counts into n_bad.
__device__ __forceinline__ float guard_count(float guard, float g, unsigned& n_bad) {
    const bool bad = guard > 0.f && !(fabsf(g) <= guard);
    n_bad += bad ? 1u : 0u;
    return bad ? 0.f : g;
}


__device__ __forceinline__ void bulk_load(float* smem_dst, const float* src, unsigned bytes, uint64_t* bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
                     "r"(smem_u32(smem_dst)),
                 "l"(src), "r"(bytes), "r"(smem_u32(bar))
                 : "memory");
}

// Weight-phase pipeline state of a CTA: kNBuf chunk buffers, each filled by
// bulk copies that complete on its own "full" mbarrier, and released by the
// 16 warps on its own "empty" mbarrier (one arrival per warp) before thread 0
// refills it; `parity` and `eparity` hold one phase bit per buffer and persist
// across tiles and groups.
struct ChunkPipe {
    uint64_t* bar;
    unsigned parity;
    uint64_t* ebar;      // per buffer: all warps done with it (thread 0 waits)
    unsigned eparity;    // thread 0's
};

// Issues chunk c of a TU-row tile (patterns [c * kPC, c * kPC + rows)) into
// buffer c % kNBuf: the [rows][kTJ] activation block cb of layer l - 1, then
// the TU / kDB delta blocks of the tile's units (blocks tb * TU / kDB ..) of
// layer l, each one contiguous bulk copy from the blocked scratch.  Thread 0 only.
//   lost: arm the barrier for the chunk's bytes but issue no copy (the checked
//   build's test hook: a copy that never comes, with nothing in flight)
template <int TU>
__device__ __forceinline__ void issue_chunk(const F32View& v, ChunkPipe& pipe, float* wbuf, int l,
                                            int tb, int cb, int c, int rows, bool lost = false) {
    const int b = c % kNBuf;
    float* buf = wbuf + b * chunk_floats<TU>();
    const unsigned abytes = (unsigned)rows * kTJ * 4, dbytes = (unsigned)rows * kDB * 4;
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(pipe.bar + b)),
                 "r"(abytes + (TU / kDB) * dbytes)
                 : "memory");
    if (lost) return;
    const long long p0 = (long long)c * kPC;
    bulk_load(buf, v.A + v.aoff[l - 1] + (long long)cb * v.cap * kTJ + p0 * kTJ, abytes, pipe.bar + b);
#pragma unroll
    for (int h = 0; h < TU / kDB; ++h)
        bulk_load(buf + kPC * kTJ + h * kPC * kDB,
                  v.D + v.doff[l] + ((long long)tb * (TU / kDB) + h) * v.cap * kDB + p0 * kDB, dbytes,
                  pipe.bar + b);
}

// Tile t of the weight phase (TU rows): its layer l, block row tb (units
// TU tb ..) and block column cb (inputs 32 cb ..).
struct Tile {
    int l, tb, cb;
};
template <int TU>
__device__ __forceinline__ const int* tile_starts(const F32View& v) {
    return TU == kTU ? v.tile0 : v.tile0w;
}
template <int TU>
__device__ __forceinline__ Tile tile_at(const F32View& v, int t) {
    const int* t0 = tile_starts<TU>(v);
    int l = 1;
    while (t >= t0[l + 1]) ++l;
    const int lt = t - t0[l];
    const int tb = lt / v.tcols[l];
    return Tile{l, tb, lt - tb * v.tcols[l]};
}

// The weight phase's chunk buffers: the bottom of shared memory, aligned to 1 KB.
__device__ __forceinline__ float* chunk_buffers(float* smem) {
    return reinterpret_cast<float*>((reinterpret_cast<uintptr_t>(smem) + 1023) & ~(uintptr_t)1023);
}
template <int TU>
__device__ __forceinline__ bool chunk_buffers_fit(const F32View& v, int B, const float* wbuf) {
    return (size_t)(wbuf - pattern_smem_base()) + kNBuf * chunk_floats<TU>() <= dyn_smem_floats() && B <= v.cap;
}

// Thread 0: the first kNBuf chunk copies of chunks [c0, c1) of a tile.  The
// proxy fences order the buffers' earlier generic-proxy reads and the scratch
// rows' generic-proxy writes before the bulk copies.
template <int TU>
__device__ __forceinline__ void issue_tile_start(const F32View& v, ChunkPipe& pipe, float* wbuf,
                                                 const Tile& tl, int B, int c0, int c1) {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    asm volatile("fence.proxy.async.global;" ::: "memory");
    bool lose_first = false;
#ifdef BP_CHECK
    lose_first = v.debug_stall != 0;   // test hook: the first chunk's copy never comes
#endif
    for (int c = c0; c < c1 && c < c0 + kNBuf; ++c)
        issue_chunk<TU>(v, pipe, wbuf, tl.l, tl.tb, tl.cb, c, min(kPC, B - c * kPC), lose_first && c == c0);
}

// Balanced weight phase for large groups: on tiles of kTUW rows (twice the
// FMAs per staged byte of the whole-tile form's 8), when these tiles are fewer
// than the CTAs and the group streams at least kSplitMinChunks chunks, the
// tiles' chunks, taken in order (tile by tile) as one sequence of
// ntiles x nchunks, are cut into gridDim.x equal runs, one per CTA.  A run is
// shorter than a tile's chunks, so it covers at most two tiles; the CTA writes
// its sums for each to wpart[CTA][0 or 1], and after a grid barrier
// weight_fixup adds each tile's pieces in CTA order and applies the update.
// Only for the training update (fused), and only with a wpart buffer.
constexpr int kSplitMinChunks = 24;   // measured: 16 chunks slower (the extra barrier), 32 faster
__device__ __forceinline__ bool balanced_split(const F32View& v, int B, bool fused) {
    return fused && v.wpart != nullptr && v.tile0w[v.L + 1] < (int)gridDim.x &&
           (B + kPC - 1) / kPC >= kSplitMinChunks;
}
// First flat chunk index of CTA b's run (b = gridDim.x: the end).
__device__ __forceinline__ long long run_start(long long F, int b) { return F * b / gridDim.x; }

// One weight-phase update: accumulate the change g into G (fused == false), or
// apply lr/momentum (Section 6.2.1) after the fault guard, folding in a pending
// G first when fold_g.
__device__ __forceinline__ void apply_change(const F32View& v, long long idx, float g, float v_old, float g_old,
                                             bool fused, bool fold_g) {
    if (!fused) {
        v.G[idx] = g_old + g;
    } else {
        if (fold_g) {
            g += g_old;
            v.G[idx] = 0.f;
        }
        g = guard_change(v, g);
        const float vel = v.lr * v.grad_scale * g + v.momentum * v_old;
        v.V[idx] = vel;
        v.theta[idx] += vel;
    }
}

// Pooled change of every weight (and bias: the last input column is the true
// unit's 1) over the B patterns of the group, then either accumulate into G
// (fused == false) or apply the update directly.  One CTA per 8 x 32 tile;
// the tile's delta and activation blocks stream through shared memory in
// chunks of kPC patterns, one bulk copy each from the blocked scratch, kNBuf
// chunks in flight.  Every warp computes the whole tile over its sixteenth of
// each chunk's patterns (kPC / 16 consecutive rows): lane l owns column quad
// l % 8 and pattern lane l / 8, holds all 8 units x its 4 columns (32 sums),
// and takes rows 4 i + l / 8 of the warp's share.  A pattern then costs two 16-byte
// delta loads shared by the 8 lanes of a pattern lane and one 16-byte
// activation load for 32 FMAs, which keeps the loop off the shared-memory
// bandwidth limit.  The blocks' row chunks are stored permuted by pattern (see
// F32View), so the lanes' reads are conflict-free.  There is no CTA-wide sync
// per chunk: each warp releases a buffer on its empty barrier and thread 0
// refills it once all have, so warps may run up to a chunk apart (a CTA sync
// per chunk measured 1-2% slower).  The sums meet first across the 4 pattern
// lanes (butterfly), then across the 16 warps in shared memory in warp order:
// the result does not depend on timing.
//
// SPLIT: the balanced form (balanced_split(v, B, fused) must hold): this
// CTA's run of the chunk sequence, sums to wpart (a separate instantiation, so
// that the whole-tile form keeps its registers).
//
// Returns false (in every thread) if a wait ran out: thread 0 then issues no
// more copies and has waited for (or drained) every copy it issued, no weight
// was written for the tile, and the caller must return.
template <bool SPLIT>
__device__ bool weight_phase(const F32View& v, int B, bool fused, bool fold_g, float* smem,
                             ChunkPipe& pipe) {
    constexpr int TU = SPLIT ? kTUW : kTU;   // tile rows
    const int tid = threadIdx.x;
    const int lane = tid & 31, warp = tid >> 5;
    const int cq = lane & 7, pl = lane >> 3;
    float* wbuf = chunk_buffers(smem);
    const int L = v.L;
    const int ntiles = tile_starts<TU>(v)[L + 1];
    const int nchunks = (B + kPC - 1) / kPC;
    if (!bounds_ok(chunk_buffers_fit<TU>(v, B, wbuf), v.flags)) return true;
    // this CTA's work: whole tiles blockIdx.x + k gridDim.x, or (balanced) the
    // one or two tile pieces of its run [f_lo, f_hi) of the flat chunk sequence
    long long f_lo = 0, f_hi = 0;
    int t_begin = blockIdx.x, t_end = ntiles, t_step = gridDim.x;
    if constexpr (SPLIT) {
        const long long F = (long long)ntiles * nchunks;
        f_lo = run_start(F, blockIdx.x);
        f_hi = run_start(F, blockIdx.x + 1);
        t_begin = (int)(f_lo / nchunks);
        t_end = f_hi > f_lo ? (int)((f_hi - 1) / nchunks) + 1 : t_begin;
        t_step = 1;
        if (!bounds_ok(t_end - t_begin <= 2, v.flags)) return true;
    }
    for (int t = t_begin; t < t_end; t += t_step) {
        int c0 = 0, c1 = nchunks;
        if constexpr (SPLIT) {
            const long long t0 = (long long)t * nchunks;
            c0 = (int)(max(f_lo, t0) - t0);
            c1 = (int)(min(f_hi, t0 + nchunks) - t0);
        }
        const Tile tl = tile_at<TU>(v, t);
        const int l = tl.l, tb = tl.tb, cb = tl.cb;
        const int n_in = v.n[l - 1], n_out = v.n[l];
        const int u0 = tb * TU, j0 = cb * kTJ;
        // the tile's blocks exist in the scratch layout
        if (!bounds_ok((tb + 1) * (TU / kDB) <= v.dtb[l] && cb < v.acb[l - 1], v.flags)) return true;
        // the buffers' previous contents (weights, pattern rows, the last tile's
        // sums) were read through the generic proxy by every thread before this sync
        __syncthreads();
        if (tid == 0) issue_tile_start<TU>(v, pipe, wbuf, tl, B, c0, c1);
        // the output of threads 0..TU * 32 - 1 (unit tid / 32, column tid % 32)
        // and its current weight state, loaded now so that their latency hides
        // behind the chunks (a piece of a balanced phase only writes its sums)
        const int uu = u0 + (tid >> 5), ii = j0 + (tid & 31);
        const bool mine = tid < TU * kTJ && uu < n_out && ii <= n_in;
        const long long idx = v.woff[l] + (long long)uu * v.kp[l] + ii;   // ii == n_in: bias
        float v_old = 0.f, g_old = 0.f;
        if (mine && !SPLIT) {
            if (fused) v_old = __ldcg(v.V + idx);
            if (!fused || fold_g) g_old = __ldcg(v.G + idx);
        }
        float acc[TU * 4];   // unit u, column q of this lane's quad at u * 4 + q
#pragma unroll
        for (int q = 0; q < TU * 4; ++q) acc[q] = 0.f;
        bool all_got = true;   // this thread's waits all arrived
        bool stop = false;     // thread 0: a wait ran out, no more copies
        for (int c = c0; c < c1; ++c) {
            const int b = c % kNBuf;
            const unsigned par = (pipe.parity >> b) & 1u;
            const bool got = mbar_wait(pipe.bar + b, par, v.flags, wait_limit_ns(v));
            pipe.parity ^= 1u << b;
            all_got = all_got && got;
            if (tid == 0 && !got) {
                mbar_drain(pipe.bar + b, par, wait_limit_ns(v));   // let the late copy land
                stop = true;
            }
            float* As = wbuf + b * chunk_floats<TU>();
            float* Ds = As + kPC * kTJ;   // TU / kDB delta blocks of [kPC][kDB]
            const int pc = B - c * kPC;
            if (got && warp * kWarpRows < pc) {   // warp-uniform: the warp has live rows
                if (pc < kPC) {
                    // this warp's rows past the group may hold stale scratch rows
                    const int r0 = max(pc, warp * kWarpRows), r1 = (warp + 1) * kWarpRows;
#pragma unroll
                    for (int h = 0; h < TU / kDB; ++h)
                        for (int e = lane; e < (r1 - r0) * kDB; e += 32) Ds[h * kPC * kDB + r0 * kDB + e] = 0.f;
                    for (int e = lane; e < (r1 - r0) * kTJ; e += 32) As[r0 * kTJ + e] = 0.f;
                    __syncwarp();
                }
                // (the 16-row form unrolls less: its 64 sums leave fewer registers)
#pragma unroll(TU == kTU ? kWarpRows / 4 : 2)
                for (int i = 0; i < kWarpRows / 4; ++i) {
                    const int p = warp * kWarpRows + 4 * i + pl;   // row of the chunk
                    const int dsw = (p >> 2) & 1;
                    const float4 a = *reinterpret_cast<const float4*>(As + p * kTJ + ((cq ^ (p & 7)) << 2));
                    const float av[4] = {a.x, a.y, a.z, a.w};
#pragma unroll
                    for (int h = 0; h < TU / kDB; ++h) {   // one delta block (8 units) at a time
                        const float* Dh = Ds + h * kPC * kDB + p * kDB;
                        const float4 d0 = *reinterpret_cast<const float4*>(Dh + (dsw << 2));
                        const float4 d1 = *reinterpret_cast<const float4*>(Dh + ((1 ^ dsw) << 2));
                        const float dv[8] = {d0.x, d0.y, d0.z, d0.w, d1.x, d1.y, d1.z, d1.w};
#pragma unroll
                        for (int u = 0; u < 8; ++u)
#pragma unroll
                            for (int q = 0; q < 4; ++q)
                                acc[(h * 8 + u) * 4 + q] = fmaf(dv[u], av[q], acc[(h * 8 + u) * 4 + q]);
                    }
                }
            }
            // this warp is done with buffer b; thread 0 refills it once all warps are
            __syncwarp();
            if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(pipe.ebar + b)) : "memory");
            if (tid == 0) {
                const unsigned epar = (pipe.eparity >> b) & 1u;
                pipe.eparity ^= 1u << b;
                if (!stop && c + kNBuf < c1) {
                    if (mbar_wait(pipe.ebar + b, epar, v.flags, wait_limit_ns(v))) {
                        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                        issue_chunk<TU>(v, pipe, wbuf, l, tb, cb, c + kNBuf, min(kPC, B - (c + kNBuf) * kPC));
                    } else {
                        stop = true;
                    }
                }
            }
        }
        // a wait ran out: thread 0 has waited for (or drained) every copy it issued
        if (__syncthreads_or(!all_got || stop)) return false;
        // sum over the 4 pattern lanes (lane bits 4, 3), halving the values at
        // each level: afterwards the lane holds values 0 .. TU - 1 of units
        // ub .. ub + TU / 4 - 1, ub = TU / 2 bit4 + TU / 4 bit3 (each sum is
        // (lane 0 + lane 2) + (lane 1 + lane 3) of the pattern lanes)
#pragma unroll
        for (int q = 0; q < TU * 2; ++q) {
            const bool up = (lane & 16) != 0;
            const float send = up ? acc[q] : acc[q + TU * 2];
            const float keep = up ? acc[q + TU * 2] : acc[q];
            acc[q] = keep + __shfl_xor_sync(0xffffffffu, send, 16);
        }
#pragma unroll
        for (int q = 0; q < TU; ++q) {
            const bool up = (lane & 8) != 0;
            const float send = up ? acc[q] : acc[q + TU];
            const float keep = up ? acc[q + TU] : acc[q];
            acc[q] = keep + __shfl_xor_sync(0xffffffffu, send, 8);
        }
        // every warp's sums of the tile to shared memory ([warp][unit * 32 + column]);
        // the chunk buffers are free now
        float* red = wbuf;
        const int ub = ((lane >> 4) & 1) * (TU / 2) + ((lane >> 3) & 1) * (TU / 4);
        __syncthreads();
#pragma unroll
        for (int i = 0; i < TU / 4; ++i)
            *reinterpret_cast<float4*>(red + warp * (TU * kTJ) + (ub + i) * kTJ + 4 * cq) =
                make_float4(acc[4 * i], acc[4 * i + 1], acc[4 * i + 2], acc[4 * i + 3]);
        __syncthreads();
        if (tid < TU * kTJ) {
            float g = 0.f;
#pragma unroll
            for (int w = 0; w < kWarps; ++w) g += red[w * (TU * kTJ) + tid];
            if constexpr (SPLIT) {
                v.wpart[((size_t)blockIdx.x * 2 + (t - t_begin)) * (kTUW * kTJ) + tid] = g;
            } else {
                if (mine) apply_change(v, idx, g, v_old, g_old, fused, fold_g);
                // the next group's bulk copy reads theta through the async proxy
                asm volatile("fence.proxy.async.global;" ::: "memory");
            }
        }
    }
    return true;
}

// Second step of a balanced weight phase (after a grid barrier): CTA t adds
// the pieces of tile t in CTA order (the same order on every run) and applies
// the update.  The CTA holding flat chunk f is the largest b with
// floor(F b / grid) <= f, that is ((f + 1) grid - 1) / F; between the first
// and the last CTA of a tile, CTAs with empty runs (when there are fewer
// chunks than CTAs) hold nothing; piece k of a CTA belongs to its k-th tile.
__device__ void weight_fixup(const F32View& v, int B, bool fold_g) {
    const int t = blockIdx.x, tid = threadIdx.x;
    const int ntiles = v.tile0w[v.L + 1];
    if (t >= ntiles || tid >= kTUW * kTJ) return;
    const int nchunks = (B + kPC - 1) / kPC;
    const long long F = (long long)ntiles * nchunks, grid = gridDim.x;
    const long long t0 = (long long)t * nchunks;
    const int b_first = (int)(((t0 + 1) * grid - 1) / F), b_last = (int)(((t0 + nchunks) * grid - 1) / F);
    float g = 0.f;
    for (int b = b_first; b <= b_last; ++b) {
        const long long start = run_start(F, b);
        if (run_start(F, b + 1) == start) continue;   // an empty run (fewer chunks than CTAs)
        const int k = t - (int)(start / nchunks);
        if (bounds_ok(k >= 0 && k <= 1, v.flags)) g += __ldcg(v.wpart + ((size_t)b * 2 + k) * (kTUW * kTJ) + tid);
    }
    const Tile tl = tile_at<kTUW>(v, t);
    const int l = tl.l;
    const int uu = tl.tb * kTUW + (tid >> 5), ii = tl.cb * kTJ + (tid & 31);
    if (uu < v.n[l] && ii <= v.n[l - 1]) {
        const long long idx = v.woff[l] + (long long)uu * v.kp[l] + ii;
        apply_change(v, idx, g, __ldcg(v.V + idx), fold_g ? __ldcg(v.G + idx) : 0.f, true, fold_g);
    }
    // the next group's bulk copy reads theta through the async proxy
    asm volatile("fence.proxy.async.global;" ::: "memory");
}

// Initialises the weight-phase mbarriers (static shared memory, 2 kNBuf: the
// full barriers, then the empty ones) of a launch.
__device__ void pipe_init(ChunkPipe& pipe, uint64_t* bars) {
    if (threadIdx.x == 0) {
        for (int b = 0; b < kNBuf; ++b)
            asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(bars + b)) : "memory");
        for (int b = 0; b < kNBuf; ++b)
            asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bars + kNBuf + b)), "n"(kWarps) : "memory");
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();
    pipe.bar = bars;
    pipe.parity = 0;
    pipe.ebar = bars + kNBuf;
    pipe.eparity = 0;
}

// Error sum of the group by the first warp of the last CTA: lane-strided
// partial sums then a fixed butterfly (the same order on every run).
__device__ void reduce_sse(const F32View& v, int nparts, float* sse_out) {
    if (blockIdx.x == gridDim.x - 1 && threadIdx.x < 32) {
        float s = 0.f;
        for (int c = threadIdx.x; c < nparts; c += 32) s += __ldcg(v.sse_part + c);
        s = warp_sum(s);
        if (threadIdx.x == 0) {
            if (sse_out != nullptr) *sse_out = s;
            if (!isfinite(s)) atomicOr(v.flags, kFlagNonfinite);
        }
    }
}

// ------------------------------------------------------------ kernels
// WS: the weights are copied into shared memory (else read from global memory).
template <int PG, bool WS>
__global__ void __launch_bounds__(kThreads, 1)
    k_forward(const __grid_constant__ F32View v, const __grid_constant__ PatLayout q, const float* X, int B, float* Y) {
    extern __shared__ __align__(128) float smem[];
    __shared__ __align__(8) uint64_t s_bar;
    unsigned phase = 0;
    sigmoid_table_init(v);
    __syncthreads();
    if (WS) {
        mbar_init1(&s_bar);
        if (!bounds_ok((unsigned)v.wsm <= dyn_smem_floats(), v.flags)) return;
        if (!stage_weights(v.theta, v.P, smem, &s_bar, phase, v.flags)) return;
        pattern_phase<PG>(v, q, smem, X, nullptr, B, true, false, Y, pattern_base<true>(v, smem));
    } else {
        pattern_phase<PG>(v, q, v.theta, X, nullptr, B, true, false, Y, pattern_base<false>(v, smem));
    }
}

template <int PG, bool WS>
__global__ void __launch_bounds__(kThreads, 1)
    k_deltas(const __grid_constant__ F32View v, const __grid_constant__ PatLayout q, const float* T, int B) {
    extern __shared__ __align__(128) float smem[];
    __shared__ __align__(8) uint64_t s_bar;
    unsigned phase = 0;
    float e;
    if (WS) {
        mbar_init1(&s_bar);
        if (!bounds_ok((unsigned)v.wsm <= dyn_smem_floats(), v.flags)) return;
        if (!stage_weights(v.theta, v.P, smem, &s_bar, phase, v.flags)) return;
        e = pattern_phase<PG>(v, q, smem, nullptr, T, B, false, true, nullptr, pattern_base<true>(v, smem)).sse;
    } else {
        e = pattern_phase<PG>(v, q, v.theta, nullptr, T, B, false, true, nullptr, pattern_base<false>(v, smem)).sse;
    }
    if (threadIdx.x == 0) v.sse_part[blockIdx.x] = e;
}

// Diagnostic mode (Section 8): every CTA runs the forward pass and the error of
// all B patterns with the same weights, independently of the others, and
// reports its summed squared error and the SM it ran on.
template <int PG, bool WS>
__global__ void __launch_bounds__(kThreads, 1)
    k_diagnose(const __grid_constant__ F32View v, const __grid_constant__ PatLayout q, const float* X, const float* T,
               int B, float* sse_out, int* sm_out) {
    extern __shared__ __align__(128) float smem[];
    __shared__ __align__(8) uint64_t s_bar;
    unsigned phase = 0;
    sigmoid_table_init(v);
    mbar_init1(&s_bar);
    if (WS && !bounds_ok((unsigned)v.wsm <= dyn_smem_floats(), v.flags)) return;
    float e;
    if (WS) {
        if (!stage_weights(v.theta, v.P, smem, &s_bar, phase, v.flags)) return;
        e = pattern_phase<PG>(v, q, smem, X, T, B, true, true, nullptr, pattern_base<true>(v, smem),
                              WeightCopy{nullptr, 0u, 0}, false, false, true).sse;
    } else {
        e = pattern_phase<PG>(v, q, v.theta, X, T, B, true, true, nullptr, pattern_base<false>(v, smem),
                              WeightCopy{nullptr, 0u, 0}, false, false, true).sse;
    }
    if (threadIdx.x == 0) {
        unsigned sm;
        asm volatile("mov.u32 %0, %%smid;" : "=r"(sm));
        sse_out[blockIdx.x] = e;
        sm_out[blockIdx.x] = (int)sm;
    }
}

__global__ void __launch_bounds__(kThreads, 1)
    k_accumulate(const __grid_constant__ F32View v, int B, int nparts, float* sse_out) {
    extern __shared__ __align__(128) float smem[];
    __shared__ __align__(8) uint64_t s_cbar[2 * kNBuf];
    ChunkPipe pipe;
    pipe_init(pipe, s_cbar);
    reduce_sse(v, nparts, sse_out);
    weight_phase<false>(v, B, false, false, smem, pipe);   // on a timeout it has drained its copies
}

__global__ void __launch_bounds__(256) k_update(const __grid_constant__ F32View v, long long n) {
    const float a = v.lr * v.grad_scale, m = v.momentum;
    for (long long k = blockIdx.x * 256LL + threadIdx.x; k < n; k += (long long)gridDim.x * 256) {
        const float vel = a * guard_change(v, v.G[k]) + m * v.V[k];
        v.V[k] = vel;
        v.theta[k] += vel;
        v.G[k] = 0.f;
    }
}

// SPLIT: groups that qualify (balanced_split) run the balanced weight phase;
// a separate instantiation, chosen on the host for large minibatches, so that
// the kernels of smaller groups carry none of its registers.
template <int PG, bool WS, bool SPLIT>
__global__ void __launch_bounds__(kThreads, 1)
    k_train(const __grid_constant__ F32View v, const __grid_constant__ PatLayout q, const float* X, const float* T,
            int n_patterns, int minibatch, int n_steps, float* sse_out, int fold_g) {
    extern __shared__ __align__(128) float smem[];
    __shared__ __align__(8) uint64_t s_bar;
    __shared__ __align__(8) uint64_t s_cbar[2 * kNBuf];
    // A latched timeout means an earlier launch left the barrier half-way; do
    // nothing until bp_check() has cleared the latch and reset the barrier.
    if (__ldcg(v.flags) & kFlagTimeout) return;
    unsigned phase = 0;
    sigmoid_table_init(v);
    mbar_init1(&s_bar);
    ChunkPipe pipe;
    pipe_init(pipe, s_cbar);
    // arrival count at the end of the previous launch; barrier k waits for
    // base + k * grid arrivals
    unsigned target = __ldcg(v.bar);
    const int n0 = v.n[0], nL = v.n[v.L];
    float* pat = pattern_base<WS>(v, smem);
    if (WS && !bounds_ok((unsigned)v.wsm <= dyn_smem_floats(), v.flags)) return;
    for (int s = 0; s < n_steps; ++s) {
        const long long p0 = (long long)s * minibatch;
        const int B = (int)min((long long)minibatch, (long long)n_patterns - p0);
        const float* Xs = X + p0 * n0;
        const float* Ts = T + p0 * nL;
        float e;
        if (WS) {
            stage_weights_issue(v.theta, v.P, smem, &s_bar);
            const WeightCopy wc{&s_bar, phase, v.P};
            phase = after_copy(phase, v.P);
            const PhaseResult r = pattern_phase<PG>(v, q, smem, Xs, Ts, B, true, true, nullptr, pat, wc);
            if (!r.ok) return;   // the copy was drained; the error is latched
            e = r.sse;
        } else {
            e = pattern_phase<PG>(v, q, v.theta, Xs, Ts, B, true, true, nullptr, pat).sse;
        }
        if (threadIdx.x == 0) v.sse_part[blockIdx.x] = e;
        if (!grid_barrier(v.bar, target += gridDim.x, v.flags, wait_limit_ns(v))) return;
        reduce_sse(v, gridDim.x, sse_out != nullptr ? sse_out + s : nullptr);
        bool balanced = false;
        if constexpr (SPLIT) balanced = balanced_split(v, B, true);
        if (balanced) {
            if (!weight_phase<true>(v, B, true, fold_g != 0 && s == 0, smem, pipe)) return;
            if (!grid_barrier(v.bar, target += gridDim.x, v.flags, wait_limit_ns(v))) return;
            weight_fixup(v, B, fold_g != 0 && s == 0);
        } else {
            if (!weight_phase<false>(v, B, true, fold_g != 0 && s == 0, smem, pipe)) return;
        }
        if (s + 1 < n_steps) {
            if (!grid_barrier(v.bar, target += gridDim.x, v.flags, wait_limit_ns(v))) return;
        }
    }
    // every CTA has passed a barrier, so every CTA has read bar[0]: publish the
    // count for the next launch
    if (blockIdx.x == 0 && threadIdx.x == 0) v.bar[0] = target;
}

// Online and small-group training on one CTA: Section 3's update after every
// group of B <= PG patterns (B = 1 is the per-pattern update).  The weights
// stay in shared memory and the weight changes in registers for the whole
// launch, so a group costs no grid barrier and no weight copy, and the next
// group's rows load while this group's update runs (two pattern buffers).
//
// Update slots: layer l's padded rows are split into float4 columns c = t % K4
// (K4 = kp_l / 4) and rows j = t / K4 + R * r (R = kThreads / K4 rows per
// pass); a thread's slots m in [m0[l], m0[l + 1]) hold the passes r of layer l,
// so each thread keeps one column of inputs per layer and its changes stay in
// fixed registers.
struct SmallPlan {
    int m0[BP_MAX_SIZES + 1];
};

// GUARD: the fault guard is on (a separate instantiation, so that the update
// loop carries no test when it is off).
// (The pattern layout and plan are by-value parameters here: as grid constants
// they cost this kernel register spills at 16 update slots.)
template <int PG, int NV4, bool GUARD>
__global__ void __launch_bounds__(kThreads, 1)
    k_train_small(const __grid_constant__ F32View v, const PatLayout q, const SmallPlan sp,
                  const float* X, const float* T, int n_patterns, int minibatch, int n_steps,
                  float* sse_out) {
    extern __shared__ __align__(128) float smem[];
    __shared__ __align__(8) uint64_t s_bar;
    const int tid = threadIdx.x;
    unsigned phase = 0;
    sigmoid_table_init(v);
    mbar_init1(&s_bar);
    float* pat[2] = {smem + v.wsm, smem + v.wsm + q.total};
    const int n0 = v.n[0], nL = v.n[v.L];
    if (!bounds_ok((unsigned)v.wsm + 2u * (unsigned)q.total <= dyn_smem_floats() && minibatch <= PG,
                   v.flags))
        return;
    // slot m of this thread: layer lm, row jm (or -1), float4 column cm
    float4 vel[NV4];
#pragma unroll
    for (int m = 0; m < NV4; ++m) {
        int l = 1;
        while (l < v.L && m >= sp.m0[l + 1]) ++l;
        const int K4 = v.kp[l] >> 2, R = kThreads / K4;
        const int j = tid / K4 + R * (m - sp.m0[l]), c = tid % K4;
        const bool live = m < sp.m0[v.L + 1] && tid / K4 < R && j < v.n[l];
        vel[m] = live ? reinterpret_cast<const float4*>(v.V + v.woff[l] + (long long)j * v.kp[l])[c]
                      : make_float4(0.f, 0.f, 0.f, 0.f);
    }
    if (!stage_weights(v.theta, v.P, smem, &s_bar, phase, v.flags)) return;
    const float a_lr = v.lr * v.grad_scale, mom = v.momentum, guard = v.guard;
    if (n_steps > 0)
        load_rows<PG>(v, q, X, T, 0, (int)min((long long)minibatch, (long long)n_patterns), pat[0]);
    for (int s = 0; s < n_steps; ++s) {
        const long long p0 = (long long)s * minibatch;
        const int B = (int)min((long long)minibatch, (long long)n_patterns - p0);
        float* ps = pat[s & 1];
        const float e = pattern_phase<PG>(v, q, smem, X + p0 * n0, T + p0 * nL, B, true, true, nullptr,
                                          ps, WeightCopy{nullptr, 0u, 0}, false, true).sse;
        if (tid == 0) {
            if (sse_out != nullptr) sse_out[s] = e;
            if (!isfinite(e)) atomicOr(v.flags, kFlagNonfinite);
        }
        if (s + 1 < n_steps) {
            const long long pn = p0 + minibatch;
            load_rows<PG>(v, q, X + pn * n0, T + pn * nL, 0,
                          (int)min((long long)minibatch, (long long)n_patterns - pn), pat[(s + 1) & 1]);
        }
        // momentum update of every weight from this group's deltas and inputs
        int l = 0, K4 = 1, c = 0, j0 = 0, R = 1;
        unsigned n_bad = 0;
        float4 a[PG];
#pragma unroll
        for (int m = 0; m < NV4; ++m) {
            if (m >= sp.m0[v.L + 1]) break;
            if (l < v.L && m == sp.m0[l + 1]) {   // next layer: its input column
                ++l;
                K4 = v.kp[l] >> 2;
                R = kThreads / K4;
                c = tid % K4;
                j0 = tid / K4;
#pragma unroll
                for (int p = 0; p < PG; ++p) a[p] = ld4(ps + q.sa[l - 1] + p * v.apitch[l - 1] + 4 * c);
            }
            const int j = j0 + R * (m - sp.m0[l]);
            if (j0 < R && j < v.n[l]) {
                float4 g = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                for (int p = 0; p < PG; ++p) {
                    const float d = ps[q.sd[l] + p * v.dpitch[l] + j];
                    g.x = fmaf(d, a[p].x, g.x);
                    g.y = fmaf(d, a[p].y, g.y);
                    g.z = fmaf(d, a[p].z, g.z);
                    g.w = fmaf(d, a[p].w, g.w);
                }
                float4* wp = reinterpret_cast<float4*>(smem + v.woff[l] + (long long)j * v.kp[l]) + c;
                float4 w = *wp;
                if (GUARD) {
                    g.x = guard_count(guard, g.x, n_bad);
                    g.y = guard_count(guard, g.y, n_bad);
                    g.z = guard_count(guard, g.z, n_bad);
                    g.w = guard_count(guard, g.w, n_bad);
                }
                float4& u = vel[m];
                u.x = a_lr * g.x + mom * u.x;
                u.y = a_lr * g.y + mom * u.y;
                u.z = a_lr * g.z + mom * u.z;
                u.w = a_lr * g.w + mom * u.w;
                w.x += u.x;
                w.y += u.y;
                w.z += u.z;
                w.w += u.w;
                *wp = w;
            }
        }
        if (GUARD && n_bad != 0) atomicAdd(v.faults, n_bad);
        __syncthreads();
    }
    // weights and weight changes back to global memory
    for (long long k = tid; k < (v.P >> 2); k += kThreads)
        reinterpret_cast<float4*>(v.theta)[k] = reinterpret_cast<const float4*>(smem)[k];
#pragma unroll
    for (int m = 0; m < NV4; ++m) {
        int l = 1;
        while (l < v.L && m >= sp.m0[l + 1]) ++l;
        const int K4 = v.kp[l] >> 2, R = kThreads / K4;
        const int j = tid / K4 + R * (m - sp.m0[l]), c = tid % K4;
        if (m < sp.m0[v.L + 1] && tid / K4 < R && j < v.n[l])
            reinterpret_cast<float4*>(v.V + v.woff[l] + (long long)j * v.kp[l])[c] = vel[m];
    }
}

// Packed <-> padded parameter layouts, one padded element per thread.
__device__ __forceinline__ bool padded_source(const F32View& v, long long k, long long& src) {
    int l = 1;
    while (l < v.L && k >= v.woff[l + 1]) ++l;
    const long long r = k - v.woff[l];
    const int j = (int)(r / v.kp[l]), i = (int)(r - (long long)j * v.kp[l]);
    const int ni = v.n[l - 1];
    if (i < ni) src = v.pw[l] + (long long)j * ni + i;
    else if (i == ni) src = v.pb[l] + j;
    else return false;
    return true;
}

__global__ void __launch_bounds__(256) k_pad(const __grid_constant__ F32View v, const float* packed,
                                             float* padded) {
    for (long long k = blockIdx.x * 256LL + threadIdx.x; k < v.P; k += (long long)gridDim.x * 256) {
        long long src;
        padded[k] = padded_source(v, k, src) ? packed[src] : 0.f;
    }
}

__global__ void __launch_bounds__(256) k_unpad(const __grid_constant__ F32View v, const float* padded,
                                               float* packed) {
    for (long long k = blockIdx.x * 256LL + threadIdx.x; k < v.P; k += (long long)gridDim.x * 256) {
        long long src;
        if (padded_source(v, k, src)) packed[src] = padded[k];
    }
}

template <int PG, bool WS>
cudaError_t set_smem_attr_ws(size_t bytes) {
    cudaError_t e;
    if ((e = cudaFuncSetAttribute(k_diagnose<PG, WS>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)bytes)) != cudaSuccess)
        return e;
    if ((e = cudaFuncSetAttribute(k_forward<PG, WS>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)bytes)) != cudaSuccess)
        return e;
    if ((e = cudaFuncSetAttribute(k_deltas<PG, WS>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)bytes)) != cudaSuccess)
        return e;
    if constexpr (PG >= 8) {
        if ((e = cudaFuncSetAttribute(k_train<PG, WS, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)bytes)) != cudaSuccess)
            return e;
    }
    return cudaFuncSetAttribute(k_train<PG, WS, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)bytes);
}

template <int PG>
cudaError_t set_smem_attr(size_t bytes) {
    cudaError_t e = set_smem_attr_ws<PG, true>(bytes);
    if (e != cudaSuccess) return e;
    return set_smem_attr_ws<PG, false>(bytes);
}

}  // namespace

// ------------------------------------------------------------ host side
// Dynamic shared memory a CTA may use: the opt-in limit (227 KB on sm_103a)
// minus room for the kernels' static shared arrays.
constexpr size_t kStaticSmemReserve = 2048;
constexpr size_t kSmemLimit = 227 * 1024 - kStaticSmemReserve;

long long f32_layout(F32View& v, const int* n, int L, int cap) {
    v.L = L;
    v.cap = cap;
    long long pos = 0, a = 0, d = 0;
    int tiles = 0, tiles_w = 0;
    for (int l = 0; l <= L; ++l) v.n[l] = n[l];
    v.tile0[0] = v.tile0[1] = 0;
    v.tile0w[0] = v.tile0w[1] = 0;
    for (int l = 0; l <= L; ++l) {
        v.apitch[l] = (n[l] + 1 + 3) & ~3;
        v.acb[l] = (n[l] + 1 + kTJ - 1) / kTJ;
        v.aoff[l] = a;
        a += (long long)cap * v.acb[l] * kTJ;
    }
    long long pp = 0;
    for (int l = 1; l <= L; ++l) {
        v.kp[l] = v.apitch[l - 1];
        v.woff[l] = pos;
        pos += (long long)n[l] * v.kp[l];
        v.pw[l] = pp;
        pp += (long long)n[l] * n[l - 1];
        v.pb[l] = pp;
        pp += n[l];
        v.dpitch[l] = (n[l] + 3) & ~3;
        // an even number of delta blocks, so that a kTUW-row tile always has its two
        v.dtb[l] = ((n[l] + kDB - 1) / kDB + 1) & ~1;
        v.doff[l] = d;
        d += (long long)cap * v.dtb[l] * kDB;
        const int rows = (n[l] + kTU - 1) / kTU, cols = (n[l - 1] + 1 + kTJ - 1) / kTJ;
        v.tcols[l] = cols;
        v.tile0[l] = tiles;
        tiles += rows * cols;
        v.tile0[l + 1] = tiles;
        v.tile0w[l] = tiles_w;
        tiles_w += ((n[l] + kTUW - 1) / kTUW) * cols;
        v.tile0w[l + 1] = tiles_w;
    }
    v.P = pos;   // a multiple of 4: every kp is
    v.Pp = pp;
    v.wsm = (int)pos;
    v.a_floats = a;
    v.d_floats = d;
    return a + d;
}

// Pattern buffers of a CTA for a group size (see PatLayout).
static PatLayout pat_layout(const int* n, int L, int pg) {
    PatLayout q{};
    int off = 0;
    for (int l = 0; l <= L; ++l) { q.sa[l] = off; off += pg * ((n[l] + 1 + 3) & ~3); }
    for (int l = 1; l <= L; ++l) { q.sd[l] = off; off += pg * ((n[l] + 3) & ~3); }
    for (int l = 2; l <= L; ++l) { q.sdt[l] = off; off += (pg * n[l] + 3) & ~3; }
    q.st = off;
    off += (pg * n[L] + 3) & ~3;
    q.total = off;
    return q;
}

static size_t pattern_floats(const int* n, int L, int pg) { return (size_t)pat_layout(n, L, pg).total; }

void f32_pad_host(const F32View& v, const float* packed, float* padded) {
    for (long long k = 0; k < v.P; ++k) padded[k] = 0.f;
    for (int l = 1; l <= v.L; ++l) {
        const int ni = v.n[l - 1];
        for (int j = 0; j < v.n[l]; ++j) {
            float* row = padded + v.woff[l] + (long long)j * v.kp[l];
            for (int i = 0; i < ni; ++i) row[i] = packed[v.pw[l] + (long long)j * ni + i];
            row[ni] = packed[v.pb[l] + j];
        }
    }
}

void f32_unpad_host(const F32View& v, const float* padded, float* packed) {
    for (int l = 1; l <= v.L; ++l) {
        const int ni = v.n[l - 1];
        for (int j = 0; j < v.n[l]; ++j) {
            const float* row = padded + v.woff[l] + (long long)j * v.kp[l];
            for (int i = 0; i < ni; ++i) packed[v.pw[l] + (long long)j * ni + i] = row[i];
            packed[v.pb[l] + j] = row[ni];
        }
    }
}

// Without the weights in shared memory: the pattern buffers and the
// weight-phase tiles share the same bytes.
size_t f32_smem_bytes(const int* n, int L, int pg) {
    const size_t pat = pattern_floats(n, L, pg);
    return (pat > (size_t)kGradFloats ? pat : (size_t)kGradFloats) * sizeof(float);
}

int f32_max_pg(const int* n, int L) {
    int best = 0;
    for (int pg = 1; pg <= 8; pg *= 2)
        if (f32_smem_bytes(n, L, pg) <= kSmemLimit) best = pg;
    return best;
}

// Whether passes of kWidePG patterns (the whole-row-per-lane forward) suit the
// net: every activation row pitch / 4 odd (conflict-free lane reads) and the
// weights and pattern buffers together in shared memory.
static bool wide_pg_ok(const F32View& v) {
    for (int l = 0; l < v.L; ++l)
        if (((v.apitch[l] >> 2) & 1) == 0) return false;
    const size_t need = (size_t)v.wsm + pattern_floats(v.n, v.L, kWidePG);
    return need * sizeof(float) <= kSmemLimit;
}

template <int PG, bool GUARD>
cudaError_t set_small_attr_g(size_t bytes) {
    cudaError_t e = cudaFuncSetAttribute(k_train_small<PG, 4, GUARD>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    if (e != cudaSuccess) return e;
    return cudaFuncSetAttribute(k_train_small<PG, 16, GUARD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)bytes);
}

template <int PG>
cudaError_t set_small_attr(size_t bytes) {
    cudaError_t e = set_small_attr_g<PG, false>(bytes);
    if (e != cudaSuccess) return e;
    return set_small_attr_g<PG, true>(bytes);
}

cudaError_t f32_setup(int device) {
    int optin = 0;
    cudaError_t e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, device);
    if (e != cudaSuccess) return e;
    if ((size_t)optin < kSmemLimit + kStaticSmemReserve) return cudaErrorInvalidConfiguration;
    if ((e = set_smem_attr<1>(kSmemLimit)) != cudaSuccess) return e;
    if ((e = set_smem_attr<2>(kSmemLimit)) != cudaSuccess) return e;
    if ((e = set_smem_attr<4>(kSmemLimit)) != cudaSuccess) return e;
    if ((e = set_smem_attr<8>(kSmemLimit)) != cudaSuccess) return e;
    if ((e = set_smem_attr<kWidePG>(kSmemLimit)) != cudaSuccess) return e;
    if ((e = set_small_attr<1>(kSmemLimit)) != cudaSuccess) return e;
    if ((e = set_small_attr<2>(kSmemLimit)) != cudaSuccess) return e;
    if ((e = set_small_attr<4>(kSmemLimit)) != cudaSuccess) return e;
    return cudaFuncSetAttribute(k_accumulate, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)(kGradFloats * sizeof(float)));
}

F32Plan f32_plan(const F32View& v, int batch, int num_sms) {
    F32Plan p;
    const int maxpg = f32_max_pg(v.n, v.L);
    const int want = (batch + num_sms - 1) / num_sms;
    int pg = 1;
    while (pg < want && pg < maxpg) pg *= 2;
    // more than 16 patterns per CTA: passes of kWidePG, when the net suits them
    // (at 9-16 a half-empty pass of 32 is slower than two passes of 8)
    if (want > 16 && pg == 8 && wide_pg_ok(v)) pg = kWidePG;
    p.pg = pg;
    p.grid = num_sms;
    // weights in shared memory when they fit below the pattern buffers
    const size_t pat = pattern_floats(v.n, v.L, pg);
    p.w_in_smem = (((size_t)v.wsm + pat) * sizeof(float) <= kSmemLimit) ? 1 : 0;
    size_t need = p.w_in_smem ? (size_t)v.wsm + pat : pat;
    // the balanced weight phase (and its larger chunk buffers) when the
    // minibatch qualifies; the kernel still decides per group (a ragged last
    // group may not)
    p.split = (v.wpart != nullptr && v.tile0w[v.L + 1] < num_sms && (batch + kPC - 1) / kPC >= kSplitMinChunks &&
               pg >= 8 && (size_t)kGradFloatsW * sizeof(float) <= kSmemLimit)
                  ? 1
                  : 0;
    const size_t grad = p.split ? kGradFloatsW : kGradFloats;
    if (need < grad) need = grad;
    p.smem = need * sizeof(float);
    p.q = pat_layout(v.n, v.L, pg);
    return p;
}

cudaError_t f32_forward(const F32View& v, const float* X, int batch, float* Y, const F32Plan& plan,
                        cudaStream_t s) {
#define BP_FWD(PG)                                                                        \
    (plan.w_in_smem ? (k_forward<PG, true><<<plan.grid, kThreads, plan.smem, s>>>(v, plan.q, X, batch, Y)) \
                    : (k_forward<PG, false><<<plan.grid, kThreads, plan.smem, s>>>(v, plan.q, X, batch, Y)))
    switch (plan.pg) {
        case 1: BP_FWD(1); break;
        case 2: BP_FWD(2); break;
        case 4: BP_FWD(4); break;
        case 8: BP_FWD(8); break;
        default: BP_FWD(kWidePG); break;
    }
#undef BP_FWD
    return cudaGetLastError();
}

cudaError_t f32_backward(const F32View& v, const float* /*X*/, const float* T, int batch,
                         float* sse_out, const F32Plan& plan, cudaStream_t s) {
#define BP_DEL(PG)                                                                      \
    (plan.w_in_smem ? (k_deltas<PG, true><<<plan.grid, kThreads, plan.smem, s>>>(v, plan.q, T, batch)) \
                    : (k_deltas<PG, false><<<plan.grid, kThreads, plan.smem, s>>>(v, plan.q, T, batch)))
    switch (plan.pg) {
        case 1: BP_DEL(1); break;
        case 2: BP_DEL(2); break;
        case 4: BP_DEL(4); break;
        case 8: BP_DEL(8); break;
        default: BP_DEL(kWidePG); break;
    }
#undef BP_DEL
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const int tiles = v.tile0[v.L + 1];
    const int ggrid = tiles < plan.grid ? tiles : plan.grid;
    k_accumulate<<<ggrid, kThreads, kGradFloats * sizeof(float), s>>>(v, batch, plan.grid, sse_out);
    return cudaGetLastError();
}

static int elementwise_blocks(long long n) {
    long long blocks = (n + 255) / 256;
    if (blocks > 4096) blocks = 4096;
    if (blocks < 1) blocks = 1;
    return (int)blocks;
}

cudaError_t f32_pad_device(const F32View& v, const float* packed, float* padded, cudaStream_t s) {
    k_pad<<<elementwise_blocks(v.P), 256, 0, s>>>(v, packed, padded);
    return cudaGetLastError();
}

cudaError_t f32_unpad_device(const F32View& v, const float* padded, float* packed, cudaStream_t s) {
    k_unpad<<<elementwise_blocks(v.P), 256, 0, s>>>(v, padded, packed);
    return cudaGetLastError();
}

cudaError_t f32_update(const F32View& v, long long n_params, cudaStream_t s) {
    long long blocks = (n_params + 255) / 256;
    if (blocks > 4096) blocks = 4096;
    if (blocks < 1) blocks = 1;
    k_update<<<(int)blocks, 256, 0, s>>>(v, n_params);
    return cudaGetLastError();
}

cudaError_t f32_train(const F32View& v, const float* X, const float* T, int n_patterns,
                      int minibatch, int n_steps, float* sse_out, bool fold_g,
                      const F32Plan& plan, cudaStream_t s) {
    int fold = fold_g ? 1 : 0;
    F32View vv = v;
    PatLayout q = plan.q;
    void* args[] = {(void*)&vv, (void*)&q, (void*)&X, (void*)&T, (void*)&n_patterns, (void*)&minibatch,
                    (void*)&n_steps, (void*)&sse_out, (void*)&fold};
    const void* fn;
    const bool ws = plan.w_in_smem != 0;
    const bool split = plan.split != 0;
    switch (plan.pg) {
        case 1: fn = ws ? (const void*)k_train<1, true, false> : (const void*)k_train<1, false, false>; break;
        case 2: fn = ws ? (const void*)k_train<2, true, false> : (const void*)k_train<2, false, false>; break;
        case 4: fn = ws ? (const void*)k_train<4, true, false> : (const void*)k_train<4, false, false>; break;
        case 8:
            fn = split ? (ws ? (const void*)k_train<8, true, true> : (const void*)k_train<8, false, true>)
                       : (ws ? (const void*)k_train<8, true, false> : (const void*)k_train<8, false, false>);
            break;
        default:
            fn = split ? (ws ? (const void*)k_train<kWidePG, true, true> : (const void*)k_train<kWidePG, false, true>)
                       : (ws ? (const void*)k_train<kWidePG, true, false>
                             : (const void*)k_train<kWidePG, false, false>);
            break;
    }
    return cudaLaunchCooperativeKernel(fn, dim3(plan.grid), dim3(kThreads), args, plan.smem, s);
}

// ------------------------------------------------------------ one-CTA groups
// Groups of at most kSmallMaxB patterns run on one CTA when the padded weights
// and the pattern buffers fit in its shared memory and the weight changes fit
// in its registers (16 float4 per thread).
constexpr int kSmallMaxB = 4;

// Update slots per thread: layer l takes ceil(n_l / (kThreads / (kp_l / 4))) passes.
static SmallPlan small_plan(const F32View& v) {
    SmallPlan sp{};
    int m = 0;
    for (int l = 1; l <= v.L; ++l) {
        sp.m0[l] = m;
        const int K4 = v.kp[l] / 4;
        const int R = K4 <= kThreads ? kThreads / K4 : 0;
        m += R > 0 ? (v.n[l] + R - 1) / R : 1 << 20;
    }
    sp.m0[v.L + 1] = m;
    return sp;
}

bool f32_small_ok(const F32View& v, int minibatch) {
    if (minibatch > kSmallMaxB) return false;
    const int pg = minibatch <= 1 ? 1 : minibatch <= 2 ? 2 : 4;
    if (small_plan(v).m0[v.L + 1] > 16) return false;
    const size_t bytes = ((size_t)v.wsm + 2 * (size_t)pat_layout(v.n, v.L, pg).total) * sizeof(float);
    return bytes <= kSmemLimit;
}

cudaError_t f32_train_small(const F32View& v, const float* X, const float* T, int n_patterns,
                            int minibatch, int n_steps, float* sse_out, cudaStream_t s) {
    if (!f32_small_ok(v, minibatch)) return cudaErrorInvalidValue;
    const int pg = minibatch <= 1 ? 1 : minibatch <= 2 ? 2 : 4;
    const PatLayout q = pat_layout(v.n, v.L, pg);
    const SmallPlan sp = small_plan(v);
    const size_t bytes = ((size_t)v.wsm + 2 * (size_t)q.total) * sizeof(float);
    const bool big = sp.m0[v.L + 1] > 4;
#define BP_SMALL(PG, NV)                                                                           \
    (v.guard > 0.f                                                                                  \
         ? k_train_small<PG, NV, true><<<1, kThreads, bytes, s>>>(v, q, sp, X, T, n_patterns, minibatch, \
                                                                  n_steps, sse_out)                 \
         : k_train_small<PG, NV, false><<<1, kThreads, bytes, s>>>(v, q, sp, X, T, n_patterns,          \
                                                                   minibatch, n_steps, sse_out))
    switch (pg) {
        case 1: if (big) BP_SMALL(1, 16); else BP_SMALL(1, 4); break;
        case 2: if (big) BP_SMALL(2, 16); else BP_SMALL(2, 4); break;
        default: if (big) BP_SMALL(4, 16); else BP_SMALL(4, 4); break;
    }
#undef BP_SMALL
    return cudaGetLastError();
}

// ------------------------------------------------------------ diagnostic mode
cudaError_t f32_diagnose(const F32View& v, const float* X, const float* T, int batch, float* d_sse,
                         int* d_sm, int num_sms, cudaStream_t s) {
    // every CTA takes all `batch` patterns: plan as if each had that many
    const F32Plan plan = f32_plan(v, (int)std::min<long long>((long long)batch * num_sms, 1 << 30), num_sms);
#define BP_DIAG(PG)                                                                          \
    (plan.w_in_smem                                                                          \
         ? (k_diagnose<PG, true><<<num_sms, kThreads, plan.smem, s>>>(v, plan.q, X, T, batch, d_sse, d_sm)) \
         : (k_diagnose<PG, false><<<num_sms, kThreads, plan.smem, s>>>(v, plan.q, X, T, batch, d_sse, d_sm)))
    switch (plan.pg) {
        case 1: BP_DIAG(1); break;
        case 2: BP_DIAG(2); break;
        case 4: BP_DIAG(4); break;
        case 8: BP_DIAG(8); break;
        default: BP_DIAG(kWidePG); break;
    }
#undef BP_DIAG
    return cudaGetLastError();
}

}  // namespace bp
