// float32 back-propagation step on CUDA cores (FFMA), for nets whose per-pattern
// activations fit in shared memory (the NETtalk-sized nets of Section 6.3).
//
// One training step over a group of B patterns runs in two phases:
//
//   pattern phase (case-parallel, Section 4.1): each CTA takes groups of PG
//     patterns and runs the whole net on them -- forward pass (Section 3),
//     output delta (t-o)o(1-o) with the summed squared error, hidden deltas
//     (W^T delta) h(1-h) for every hidden layer and none for the inputs
//     (Section 6.1).  Activations and deltas live in shared memory; weights
//     stream from L2.  Dot products are summed as a binary tree across the
//     warp (Section 10.3).
//
//   weight phase (one CTA per 8 x 32 tile of weights, Section 5's "bundle"
//     processed over the whole group of cases): the pooled change
//     G[j,i] = sum_p delta[p,j] a[p,i] over all B patterns (Sections 3, 4.1),
//     then either G += tile (bp_backward) or directly the momentum update of
//     Section 6.2.1 (training launches), so the pooled change never leaves
//     registers.
//
// A training launch is a persistent cooperative kernel that loops over any
// number of groups with a grid barrier between the phases; every wait in the
// barrier is bounded and latches kFlagTimeout instead of hanging.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdio>

#include "bp_internal.h"

namespace bp {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kTJ = 8;            // weight-tile rows (output units)
constexpr int kTI = 32;           // weight-tile columns (input units + bias)
constexpr int kPC = 256;          // patterns per staged chunk in the weight phase
constexpr size_t kGradSmem = 2ull * kPC * (kTJ + kTI) * sizeof(float);

constexpr unsigned long long kWaitNs = 2000000000ull;   // 2 s per barrier wait
constexpr unsigned kWaitIters = 1u << 26;

// ------------------------------------------------------------ small helpers
__device__ __forceinline__ float sigmoid_f(float x) { return 1.0f / (1.0f + expf(-x)); }

__device__ __forceinline__ unsigned ld_acquire(const unsigned* p) {
    unsigned v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void st_release(unsigned* p, unsigned v) {
    asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ unsigned atom_add_acq_rel(unsigned* p, unsigned v) {
    unsigned old;
    asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], %2;"
                 : "=r"(old) : "l"(p), "r"(v) : "memory");
    return old;
}
__device__ __forceinline__ unsigned long long global_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Sense-reversing grid barrier for a cooperative launch.  Returns false (in
// every thread of the CTA) if the wait ran out; the caller must then return.
__device__ bool grid_barrier(unsigned* bar, int* flags) {
    __shared__ int s_ok;
    __syncthreads();
    if (threadIdx.x == 0) {
        int ok = 1;
        const unsigned gen = ld_acquire(bar + 1);
        const unsigned prev = atom_add_acq_rel(bar, 1u);
        if (prev == gridDim.x - 1) {
            atomicExch(bar, 0u);
            st_release(bar + 1, gen + 1u);
        } else {
            const unsigned long long t0 = global_ns();
            unsigned it = 0;
            while (ld_acquire(bar + 1) == gen) {
                ++it;
                if (it > kWaitIters || ((it & 63u) == 0 && global_ns() - t0 > kWaitNs)) {
                    atomicOr(flags, kFlagTimeout);
                    ok = 0;
                    break;
                }
                if (it > 256) __nanosleep(64);
            }
        }
        s_ok = ok;
    }
    __syncthreads();
    return s_ok != 0;
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

// Butterfly reduce-scatter of 32 per-lane values: afterwards lane k holds in
// v[0] the warp-wide sum of value k.  A binary-tree sum of each dot product
// (Section 10.3), 31 shuffles for 32 sums.
__device__ __forceinline__ void reduce_scatter32(float (&v)[32], int lane) {
#pragma unroll
    for (int half = 16; half >= 1; half >>= 1) {
        const bool up = (lane & half) != 0;
#pragma unroll
        for (int k = 0; k < half; ++k) {
            const float send = up ? v[k] : v[k + half];
            const float keep = up ? v[k + half] : v[k];
            v[k] = keep + __shfl_xor_sync(0xffffffffu, send, half);
        }
    }
}

// ------------------------------------------------------------ pattern phase
// Forward through one layer for PG patterns held in shared memory:
// out[p][j] = sigma(sum_i W[j][i] in[p][i] + b[j]).  A warp owns 32/PG units at
// a time; lanes stride over the inputs.
template <int PG>
__device__ void forward_layer(const float* __restrict__ W, const float* __restrict__ b,
                              int n_in, int n_out, const float* s_in, float* s_out) {
    constexpr int UJ = 32 / PG;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int j0 = warp * UJ; j0 < n_out; j0 += kWarps * UJ) {
        float acc[32];
#pragma unroll
        for (int k = 0; k < 32; ++k) acc[k] = 0.f;
        for (int i = lane; i < n_in; i += 32) {
            float a[PG];
#pragma unroll
            for (int p = 0; p < PG; ++p) a[p] = s_in[p * n_in + i];
#pragma unroll
            for (int u = 0; u < UJ; ++u) {
                const int j = min(j0 + u, n_out - 1);   // rows past the end are discarded
                const float w = __ldcg(W + (size_t)j * n_in + i);
#pragma unroll
                for (int p = 0; p < PG; ++p) acc[u * PG + p] = fmaf(w, a[p], acc[u * PG + p]);
            }
        }
        reduce_scatter32(acc, lane);
        const int u = lane / PG, p = lane % PG;
        const int j = j0 + u;
        if (j < n_out) s_out[p * n_out + j] = sigmoid_f(acc[0] + __ldcg(b + j));
    }
}

// Runs the pattern phase for this CTA's groups of `B` patterns.
//   do_fwd: forward pass from X (else the activations are reloaded from scratch)
//   do_bwd: deltas against T, written to scratch
//   Y: if not null, the outputs are copied there ([B, n_L] packed)
// Returns this CTA's summed squared error (valid in thread 0).
template <int PG>
__device__ float pattern_phase(const F32View& v, const float* __restrict__ X,
                               const float* __restrict__ T, int B, bool do_fwd, bool do_bwd,
                               float* __restrict__ Y, float* smem) {
    const int L = v.L;
    const int tid = threadIdx.x;
    int sa[BP_MAX_SIZES], sd[BP_MAX_SIZES];
    {
        int off = 0;
        for (int l = 0; l <= L; ++l) { sa[l] = off; off += PG * v.n[l]; }
        for (int l = 1; l <= L; ++l) { sd[l] = off; off += PG * v.n[l]; }
    }
    float sse = 0.f;
    const int ngroups = (B + PG - 1) / PG;
    for (int g = blockIdx.x; g < ngroups; g += gridDim.x) {
        const int p0 = g * PG;
        const int np = min(PG, B - p0);
        if (do_fwd) {
            const int n0 = v.n[0];
            for (int e = tid; e < PG * n0; e += kThreads) {
                const int p = e / n0, i = e - p * n0;
                smem[sa[0] + e] = (p < np) ? __ldg(X + (size_t)(p0 + p) * n0 + i) : 0.f;
            }
            __syncthreads();
            for (int l = 1; l <= L; ++l) {
                forward_layer<PG>(v.theta + v.woff[l], v.theta + v.boff[l], v.n[l - 1], v.n[l],
                                  smem + sa[l - 1], smem + sa[l]);
                __syncthreads();
            }
            for (int l = 1; l <= L; ++l) {
                const int n = v.n[l];
                const int pitch = (n + 3) & ~3;
                float* dst = v.A + v.soff[l];
                for (int e = tid; e < PG * n; e += kThreads) {
                    const int p = e / n, i = e - p * n;
                    if (p < np) dst[(size_t)(p0 + p) * pitch + i] = smem[sa[l] + e];
                }
            }
            if (Y != nullptr) {
                const int n = v.n[L];
                for (int e = tid; e < PG * n; e += kThreads) {
                    const int p = e / n, k = e - p * n;
                    if (p < np) Y[(size_t)(p0 + p) * n + k] = smem[sa[L] + e];
                }
            }
        } else {
            for (int l = 1; l <= L; ++l) {
                const int n = v.n[l];
                const int pitch = (n + 3) & ~3;
                const float* src = v.A + v.soff[l];
                for (int e = tid; e < PG * n; e += kThreads) {
                    const int p = e / n, i = e - p * n;
                    smem[sa[l] + e] = (p < np) ? __ldcg(src + (size_t)(p0 + p) * pitch + i) : 0.f;
                }
            }
            __syncthreads();
        }
        if (do_bwd) {
            // output delta and error sum (Section 3, fn. 5)
            const int nL = v.n[L];
            for (int e = tid; e < PG * nL; e += kThreads) {
                const int p = e / nL, k = e - p * nL;
                float d = 0.f;
                if (p < np) {
                    const float o = smem[sa[L] + e];
                    const float err = __ldg(T + (size_t)(p0 + p) * nL + k) - o;
                    sse = fmaf(err, err, sse);
                    d = err * o * (1.f - o);
                }
                smem[sd[L] + e] = d;
            }
            __syncthreads();
            // hidden deltas, output side first; no delta for the input layer
            for (int l = L - 1; l >= 1; --l) {
                const int n = v.n[l], nn = v.n[l + 1];
                const float* Wn = v.theta + v.woff[l + 1];
                for (int i = tid; i < n; i += kThreads) {
                    float acc[PG];
#pragma unroll
                    for (int p = 0; p < PG; ++p) acc[p] = 0.f;
                    for (int j = 0; j < nn; ++j) {
                        const float w = __ldcg(Wn + (size_t)j * n + i);
#pragma unroll
                        for (int p = 0; p < PG; ++p)
                            acc[p] = fmaf(smem[sd[l + 1] + p * nn + j], w, acc[p]);
                    }
#pragma unroll
                    for (int p = 0; p < PG; ++p) {
                        const float a = smem[sa[l] + p * n + i];
                        smem[sd[l] + p * n + i] = acc[p] * a * (1.f - a);
                    }
                }
                __syncthreads();
            }
            for (int l = 1; l <= L; ++l) {
                const int n = v.n[l];
                const int pitch = (n + 3) & ~3;
                float* dst = v.D + v.soff[l];
                for (int e = tid; e < PG * n; e += kThreads) {
                    const int p = e / n, i = e - p * n;
                    if (p < np) dst[(size_t)(p0 + p) * pitch + i] = smem[sd[l] + e];
                }
            }
        }
        __syncthreads();
    }
    return block_sum(sse);
}

// ------------------------------------------------------------ weight phase
__device__ __forceinline__ void cp_async4(float* dst, const float* src) {
    const unsigned d = (unsigned)__cvta_generic_to_shared(dst);
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(d), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async16(float* dst, const float* src) {
    const unsigned d = (unsigned)__cvta_generic_to_shared(dst);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(d), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

// Stage patterns [c*kPC, c*kPC + pc) of a weight tile: sD[pp][0..8) = delta rows
// j0.., sA[pp][0..32) = activation columns i0.. (zeros past the ends).
__device__ void stage_chunk(float* sD, float* sA, const float* Dl, int pitch_out, int n_out, int j0,
                            const float* Ain, int pitch_in, int n_in, int i0, bool in_is_x,
                            int p0, int pc) {
    const int tid = threadIdx.x;
    // deltas: two float4 per pattern row (scratch rows are 16-byte aligned)
    for (int e = tid; e < kPC * 2; e += kThreads) {
        const int pp = e >> 1, q = (e & 1) * 4;
        float* dst = sD + pp * kTJ + q;
        if (pp < pc && j0 + q < pitch_out) {
            cp_async16(dst, Dl + (size_t)(p0 + pp) * pitch_out + j0 + q);
        } else {
            dst[0] = dst[1] = dst[2] = dst[3] = 0.f;
        }
    }
    if (!in_is_x) {
        for (int e = tid; e < kPC * 8; e += kThreads) {
            const int pp = e >> 3, q = (e & 7) * 4;
            float* dst = sA + pp * kTI + q;
            if (pp < pc && i0 + q < pitch_in) {
                cp_async16(dst, Ain + (size_t)(p0 + pp) * pitch_in + i0 + q);
            } else {
                dst[0] = dst[1] = dst[2] = dst[3] = 0.f;
            }
        }
    } else {
        // caller's input rows: any pitch, read-only for the whole launch
        for (int e = tid; e < kPC * kTI; e += kThreads) {
            const int pp = e >> 5, q = e & 31;
            float* dst = sA + pp * kTI + q;
            if (pp < pc && i0 + q < n_in) {
                cp_async4(dst, Ain + (size_t)(p0 + pp) * n_in + i0 + q);
            } else {
                *dst = 0.f;
            }
        }
    }
    (void)n_out;
}

// Pooled change of every weight over the B patterns of the group, then either
// accumulate into G (fused == false) or apply the update directly.
__device__ void weight_phase(const F32View& v, const float* __restrict__ X, int B, bool fused,
                             bool fold_g, float* smem) {
    const int tid = threadIdx.x;
    const int tj = tid >> 5, ti = tid & 31;
    float* sD[2] = {smem, smem + kPC * kTJ};
    float* sA[2] = {smem + 2 * kPC * kTJ, smem + 2 * kPC * kTJ + kPC * kTI};
    const int L = v.L;
    const int ntiles = v.tile0[L + 1];
    const int nchunks = (B + kPC - 1) / kPC;
    for (int t = blockIdx.x; t < ntiles; t += gridDim.x) {
        int l = 1;
        while (t >= v.tile0[l + 1]) ++l;
        const int lt = t - v.tile0[l];
        const int jb = lt / v.tcols[l], ib = lt - jb * v.tcols[l];
        const int n_in = v.n[l - 1], n_out = v.n[l];
        const int j0 = jb * kTJ, i0 = ib * kTI;
        const bool in_is_x = (l == 1);
        const float* Ain = in_is_x ? X : v.A + v.soff[l - 1];
        const int pitch_in = in_is_x ? n_in : ((n_in + 3) & ~3);
        const float* Dl = v.D + v.soff[l];
        const int pitch_out = (n_out + 3) & ~3;
        const int i = i0 + ti, j = j0 + tj;
        const bool bias_col = (i == n_in);

        float acc0 = 0.f, acc1 = 0.f, acc2 = 0.f, acc3 = 0.f;
        stage_chunk(sD[0], sA[0], Dl, pitch_out, n_out, j0, Ain, pitch_in, n_in, i0, in_is_x, 0,
                    min(kPC, B));
        cp_async_commit();
        for (int c = 0; c < nchunks; ++c) {
            if (c + 1 < nchunks) {
                const int p0 = (c + 1) * kPC;
                stage_chunk(sD[(c + 1) & 1], sA[(c + 1) & 1], Dl, pitch_out, n_out, j0, Ain,
                            pitch_in, n_in, i0, in_is_x, p0, min(kPC, B - p0));
                cp_async_commit();
                cp_async_wait<1>();
            } else {
                cp_async_wait<0>();
            }
            __syncthreads();
            const float* d = sD[c & 1] + tj;
            const float* a = sA[c & 1] + ti;
            const int pc = min(kPC, B - c * kPC);
            int pp = 0;
            if (!bias_col) {
                for (; pp + 4 <= pc; pp += 4) {
                    acc0 = fmaf(d[(pp + 0) * kTJ], a[(pp + 0) * kTI], acc0);
                    acc1 = fmaf(d[(pp + 1) * kTJ], a[(pp + 1) * kTI], acc1);
                    acc2 = fmaf(d[(pp + 2) * kTJ], a[(pp + 2) * kTI], acc2);
                    acc3 = fmaf(d[(pp + 3) * kTJ], a[(pp + 3) * kTI], acc3);
                }
                for (; pp < pc; ++pp) acc0 = fmaf(d[pp * kTJ], a[pp * kTI], acc0);
            } else {
                // the true unit's activation is 1
                for (; pp + 4 <= pc; pp += 4) {
                    acc0 += d[(pp + 0) * kTJ];
                    acc1 += d[(pp + 1) * kTJ];
                    acc2 += d[(pp + 2) * kTJ];
                    acc3 += d[(pp + 3) * kTJ];
                }
                for (; pp < pc; ++pp) acc0 += d[pp * kTJ];
            }
            __syncthreads();
        }
        const float g = (acc0 + acc1) + (acc2 + acc3);
        if (j < n_out && i <= n_in) {
            const long long idx = bias_col ? v.boff[l] + j : v.woff[l] + (long long)j * n_in + i;
            if (!fused) {
                v.G[idx] += g;
            } else {
                float gt = g;
                if (fold_g) {
                    gt += v.G[idx];
                    v.G[idx] = 0.f;
                }
                const float vel = v.lr * v.grad_scale * gt + v.momentum * v.V[idx];
                v.V[idx] = vel;
                v.theta[idx] += vel;
            }
        }
    }
}

// Error sum of the group by the first warp of CTA 0: lane-strided partial sums
// then a fixed butterfly (the same order on every run).
__device__ void reduce_sse(const F32View& v, int nparts, float* sse_out) {
    if (blockIdx.x == 0 && threadIdx.x < 32) {
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
template <int PG>
__global__ void __launch_bounds__(kThreads) k_forward(F32View v, const float* X, int B, float* Y) {
    extern __shared__ float smem[];
    pattern_phase<PG>(v, X, nullptr, B, true, false, Y, smem);
}

template <int PG>
__global__ void __launch_bounds__(kThreads) k_deltas(F32View v, const float* T, int B) {
    extern __shared__ float smem[];
    const float e = pattern_phase<PG>(v, nullptr, T, B, false, true, nullptr, smem);
    if (threadIdx.x == 0) v.sse_part[blockIdx.x] = e;
}

__global__ void __launch_bounds__(kThreads)
    k_accumulate(F32View v, const float* X, int B, int nparts, float* sse_out) {
    extern __shared__ float smem[];
    reduce_sse(v, nparts, sse_out);
    weight_phase(v, X, B, false, false, smem);
}

__global__ void __launch_bounds__(kThreads) k_update(F32View v, long long n) {
    const float a = v.lr * v.grad_scale, m = v.momentum;
    for (long long k = blockIdx.x * (long long)kThreads + threadIdx.x; k < n;
         k += (long long)gridDim.x * kThreads) {
        const float vel = a * v.G[k] + m * v.V[k];
        v.V[k] = vel;
        v.theta[k] += vel;
        v.G[k] = 0.f;
    }
}

template <int PG>
__global__ void __launch_bounds__(kThreads)
    k_train(F32View v, const float* X, const float* T, int n_patterns, int minibatch,
            int n_steps, float* sse_out, int fold_g) {
    extern __shared__ float smem[];
    // A latched timeout means an earlier launch left the barrier half-way; do
    // nothing until bp_check() has cleared the latch and reset the barrier.
    if (__ldcg(v.flags) & kFlagTimeout) return;
    const int n0 = v.n[0], nL = v.n[v.L];
    for (int s = 0; s < n_steps; ++s) {
        const long long p0 = (long long)s * minibatch;
        const int B = (int)min((long long)minibatch, (long long)n_patterns - p0);
        const float* Xs = X + p0 * n0;
        const float* Ts = T + p0 * nL;
        const float e = pattern_phase<PG>(v, Xs, Ts, B, true, true, nullptr, smem);
        if (threadIdx.x == 0) v.sse_part[blockIdx.x] = e;
        if (!grid_barrier(v.bar, v.flags)) return;
        reduce_sse(v, gridDim.x, sse_out != nullptr ? sse_out + s : nullptr);
        weight_phase(v, Xs, B, true, fold_g != 0 && s == 0, smem);
        if (s + 1 < n_steps) {
            if (!grid_barrier(v.bar, v.flags)) return;
        }
    }
}

template <int PG>
cudaError_t set_smem_attr(size_t bytes) {
    cudaError_t e;
    if ((e = cudaFuncSetAttribute(k_forward<PG>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)bytes)) != cudaSuccess)
        return e;
    if ((e = cudaFuncSetAttribute(k_deltas<PG>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)bytes)) != cudaSuccess)
        return e;
    return cudaFuncSetAttribute(k_train<PG>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)bytes);
}

}  // namespace

// ------------------------------------------------------------ host side
// Dynamic shared memory a CTA may use: the opt-in limit (227 KB on sm_103a)
// minus room for the kernels' static shared arrays.
constexpr size_t kStaticSmemReserve = 1024;
constexpr size_t kSmemLimit = 227 * 1024 - kStaticSmemReserve;

size_t f32_smem_bytes(const int* n, int L, int pg) {
    size_t units = 0;
    for (int l = 0; l <= L; ++l) units += (size_t)n[l];
    for (int l = 1; l <= L; ++l) units += (size_t)n[l];
    const size_t pattern = units * (size_t)pg * sizeof(float);
    return pattern > kGradSmem ? pattern : kGradSmem;
}

int f32_max_pg(const int* n, int L) {
    int best = 0;
    for (int pg = 1; pg <= 8; pg *= 2)
        if (f32_smem_bytes(n, L, pg) <= kSmemLimit) best = pg;
    return best;
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
    return cudaFuncSetAttribute(k_accumulate, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)kGradSmem);
}

F32Plan f32_plan(const F32View& v, int batch, int num_sms) {
    F32Plan p;
    const int maxpg = f32_max_pg(v.n, v.L);
    const int want = (batch + num_sms - 1) / num_sms;
    int pg = 1;
    while (pg < want && pg < maxpg) pg *= 2;
    p.pg = pg;
    p.grid = num_sms;
    p.smem = f32_smem_bytes(v.n, v.L, pg);
    return p;
}

cudaError_t f32_forward(const F32View& v, const float* X, int batch, float* Y, const F32Plan& plan,
                        cudaStream_t s) {
    const int groups = (batch + plan.pg - 1) / plan.pg;
    const int grid = groups < plan.grid ? groups : plan.grid;
    switch (plan.pg) {
        case 1: k_forward<1><<<grid, kThreads, plan.smem, s>>>(v, X, batch, Y); break;
        case 2: k_forward<2><<<grid, kThreads, plan.smem, s>>>(v, X, batch, Y); break;
        case 4: k_forward<4><<<grid, kThreads, plan.smem, s>>>(v, X, batch, Y); break;
        default: k_forward<8><<<grid, kThreads, plan.smem, s>>>(v, X, batch, Y); break;
    }
    return cudaGetLastError();
}

cudaError_t f32_backward(const F32View& v, const float* X, const float* T, int batch,
                         float* sse_out, const F32Plan& plan, cudaStream_t s) {
    const int groups = (batch + plan.pg - 1) / plan.pg;
    const int grid = groups < plan.grid ? groups : plan.grid;
    switch (plan.pg) {
        case 1: k_deltas<1><<<grid, kThreads, plan.smem, s>>>(v, T, batch); break;
        case 2: k_deltas<2><<<grid, kThreads, plan.smem, s>>>(v, T, batch); break;
        case 4: k_deltas<4><<<grid, kThreads, plan.smem, s>>>(v, T, batch); break;
        default: k_deltas<8><<<grid, kThreads, plan.smem, s>>>(v, T, batch); break;
    }
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const int tiles = v.tile0[v.L + 1];
    const int ggrid = tiles < plan.grid ? tiles : plan.grid;
    k_accumulate<<<ggrid, kThreads, kGradSmem, s>>>(v, X, batch, grid, sse_out);
    return cudaGetLastError();
}

cudaError_t f32_update(const F32View& v, long long n_params, cudaStream_t s) {
    long long blocks = (n_params + kThreads - 1) / kThreads;
    if (blocks > 4096) blocks = 4096;
    if (blocks < 1) blocks = 1;
    k_update<<<(int)blocks, kThreads, 0, s>>>(v, n_params);
    return cudaGetLastError();
}

cudaError_t f32_train(const F32View& v, const float* X, const float* T, int n_patterns,
                      int minibatch, int n_steps, float* sse_out, bool fold_g,
                      const F32Plan& plan, cudaStream_t s) {
    int fold = fold_g ? 1 : 0;
    F32View vv = v;
    void* args[] = {(void*)&vv, (void*)&X, (void*)&T, (void*)&n_patterns, (void*)&minibatch,
                    (void*)&n_steps, (void*)&sse_out, (void*)&fold};
    const void* fn;
    switch (plan.pg) {
        case 1: fn = (const void*)k_train<1>; break;
        case 2: fn = (const void*)k_train<2>; break;
        case 4: fn = (const void*)k_train<4>; break;
        default: fn = (const void*)k_train<8>; break;
    }
    return cudaLaunchCooperativeKernel(fn, dim3(plan.grid), dim3(kThreads), args, plan.smem, s);
}

}  // namespace bp
