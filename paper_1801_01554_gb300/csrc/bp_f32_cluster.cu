// float32 training launch on thread-block clusters (sm_103a): weights stay in
// shared memory for the whole launch.
//
// The paper's two forms of parallelism meet here.  Across clusters it is the
// case parallelism of Section 4.1: every cluster holds a full copy of the net,
// runs its share of each group's patterns, and the pooled changes of all
// copies are summed before every copy applies the same update (Section 4.4's
// summation, here a fixed-order sum through L2 after one grid barrier).
// Inside a cluster the net is split by units, as Section 4.2 splits it into
// bundles: CTA r of C owns units [r*ceil(n_l/C), ...) of every layer l, with
// their incoming weights, bias ("true unit" weight, Section 6.3), previous
// change V and pooled change G, all in its shared memory.
//
// Per chunk of patterns in a cluster:
//   forward (Section 3): own units from the full previous layer; the slices
//     of a layer are all-gathered over distributed shared memory;
//   output delta (t - o) o (1 - o) and the error sum (Section 3, fn. 5);
//   hidden deltas (Section 3): partial sums over own units of layer l for
//     every unit of layer l-1, reduce-scattered over distributed shared memory
//     in a fixed rank order; none for the input units (Section 6.1);
//   pooled change of own weights, accumulated over the chunks (Section 3).
// Per group: each CTA writes its pooled change, one bounded grid barrier, then
// every copy sums the clusters' changes in cluster order and applies the
// momentum update of Section 6.2.1 to its weights in shared memory.
#include <cooperative_groups.h>
#include <cuda_runtime.h>

#include <cmath>

#include "bp_internal.h"

namespace cg = cooperative_groups;

namespace bp {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr unsigned long long kWaitNs = 2000000000ull;
constexpr unsigned kWaitIters = 1u << 26;

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
__device__ __forceinline__ void cp_async4(float* dst, const float* src) {
    const unsigned d = (unsigned)__cvta_generic_to_shared(dst);
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(d), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
    asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
}

// Bounded grid barrier (thread 0 waits).  Returns 1 if it completed.
__device__ int grid_barrier_t0(unsigned* bar, int* flags, unsigned nblocks) {
    const unsigned gen = ld_acquire(bar + 1);
    const unsigned prev = atom_add_acq_rel(bar, 1u);
    if (prev == nblocks - 1) {
        atomicExch(bar, 0u);
        st_release(bar + 1, gen + 1u);
        return 1;
    }
    const unsigned long long t0 = global_ns();
    unsigned it = 0;
    while (ld_acquire(bar + 1) == gen) {
        ++it;
        if (it > kWaitIters || ((it & 63u) == 0 && global_ns() - t0 > kWaitNs)) {
            atomicOr(flags, kFlagTimeout);
            return 0;
        }
        if (it > 512) __nanosleep(32);
    }
    return 1;
}

__device__ float block_sum(float x, float* red) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    __syncthreads();
    if (lane == 0) red[warp] = x;
    __syncthreads();
    float r = 0.f;
    if (threadIdx.x == 0)
        for (int w = 0; w < kWarps; ++w) r += red[w];
    return r;
}

}  // namespace

// Shared-memory carve of one CTA (computed on the host, passed in the kernel
// parameters so that the kernel indexes it without local memory).
//   own units per layer are padded to a multiple of 8 (two float4)
static void cl_make_carve(ClCarve& c, const int* n, int L, int C, int Pc, int R) {
    c.L = L;
    c.C = C;
    c.Pc = Pc;
    c.R = R;
    int off = 0;
    for (int l = 0; l <= L; ++l) {
        c.n[l] = n[l];
        c.ucap[l] = (n[l] + C - 1) / C;
        c.nup[l] = (c.ucap[l] + 7) & ~7;
        c.pf[l] = n[l] | 1;   // odd pitch: lanes on consecutive patterns hit distinct banks
        c.rp[l] = c.ucap[l] | 1;
        int blk = ((Pc * c.rp[l]) + 3) & ~3;
        if ((blk & 31) == 0) blk += 4;   // neighbouring rank blocks start in other banks
        c.blk[l] = blk;
    }
    c.slice = 0;
    for (int l = 1; l <= L; ++l) {
        c.wsz[l] = (n[l - 1] + 1) * c.nup[l];
        c.wt[l] = off;
        off += 3 * c.wsz[l];   // W^T, V^T, G^T of own units (last row: bias)
        c.soff[l] = c.slice;
        c.slice += c.wsz[l];
    }
    for (int l = 1; l <= L; ++l) {   // offset of input unit j in its activation buffer
        c.joff[l] = off;
        off += (n[l - 1] + 4) & ~3;
    }
    for (int l = 2; l <= L; ++l) {   // column of input unit j in the partial-sum rows
        c.sidx[l] = off;
        off += (n[l - 1] + 3) & ~3;
    }
    // ---- per-chunk buffers; after the last chunk of a group they are dead and
    // the staging ring of the copies' pooled changes reuses them
    const int chunk0 = off;
    c.full[0] = off;          // the input chunk, row-major [Pc][pf0]
    off += Pc * c.pf[0];
    c.tin = off;              // targets of own output units, [Pc][nup_L]
    off += Pc * c.nup[L];
    for (int l = 1; l < L; ++l) {   // activations: one block per rank, [Pc][rp] each
        c.full[l] = off;
        off += C * c.blk[l];
    }
    for (int l = 1; l <= L; ++l) {
        c.dn[l] = off;
        off += Pc * c.nup[l];
    }
    for (int l = 2; l <= L; ++l) {   // partial sums for layer l-1: [Pc][C * nup_{l-1}]
        c.S[l] = off;
        off += Pc * C * c.nup[l - 1];
    }
    int red = 0;
    for (int l = 1; l <= L; ++l) {
        int ks = kThreads / Pc;
        if (ks < 1) ks = 1;
        if (ks > n[l - 1]) ks = n[l - 1];
        c.ks[l] = ks;
        const int r = ks * Pc * c.nup[l];
        if (r > red) red = r;
    }
    c.red = off;
    off += red;
    c.stg = chunk0;           // staging of R copies' pooled changes (aliases the chunk)
    const int stg_end = chunk0 + R * c.slice;
    c.total = off > stg_end ? off : stg_end;
}

namespace {

__device__ __forceinline__ void mbar_init(uint64_t* bar, unsigned count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(
                     (unsigned)__cvta_generic_to_shared(bar)),
                 "r"(count)
                 : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, unsigned parity) {
    unsigned done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"((unsigned)__cvta_generic_to_shared(bar)), "r"(parity)
        : "memory");
    return done != 0;
}

__device__ __forceinline__ int units_of(int n, int ucap, int r) { return min(ucap, max(0, n - r * ucap)); }

__device__ __forceinline__ void fma8(float (&acc)[8], float a, const float* w) {
    const float4 w0 = *reinterpret_cast<const float4*>(w);
    const float4 w1 = *reinterpret_cast<const float4*>(w + 4);
    acc[0] = fmaf(a, w0.x, acc[0]);
    acc[1] = fmaf(a, w0.y, acc[1]);
    acc[2] = fmaf(a, w0.z, acc[2]);
    acc[3] = fmaf(a, w0.w, acc[3]);
    acc[4] = fmaf(a, w1.x, acc[4]);
    acc[5] = fmaf(a, w1.y, acc[5]);
    acc[6] = fmaf(a, w1.z, acc[6]);
    acc[7] = fmaf(a, w1.w, acc[7]);
}

__global__ void __launch_bounds__(kThreads, 1)
    k_train_cl(const __grid_constant__ ClArgs a, const float* __restrict__ X,
               const float* __restrict__ T, int n_patterns, int minibatch, int n_steps,
               float* sse_out, int fold_g) {
    extern __shared__ __align__(16) float sm[];
    __shared__ float red8[kWarps];
    __shared__ int s_fail[2];
    __shared__ int s_stop;
    __shared__ __align__(8) uint64_t s_bar;
    // the carve and layer sizes are indexed by a run-time layer number: keep a
    // copy in shared memory rather than indexing the kernel parameters
    __shared__ ClCarve c;
    __shared__ int s_n[BP_MAX_SIZES];
    {
        const int* src = reinterpret_cast<const int*>(&a.cv);
        int* dst = reinterpret_cast<int*>(&c);
        for (int k = threadIdx.x; k < (int)(sizeof(ClCarve) / sizeof(int)); k += blockDim.x) dst[k] = src[k];
        if (threadIdx.x < BP_MAX_SIZES) s_n[threadIdx.x] = a.n[threadIdx.x];
        __syncthreads();
    }
    cg::cluster_group cluster = cg::this_cluster();
    const int C = c.C;
    const int rank = (int)cluster.block_rank();
    const int cl = blockIdx.x / C;
    const int NC = gridDim.x / C;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int L = a.L;
    const int Pc = c.Pc;

    if (tid == 0) {
        // latched timeout: an earlier launch left the barrier half-way.  Rank 0
        // decides for the whole cluster so that no CTA is left alone at a
        // cluster barrier.
        s_stop = (__ldcg(a.flags) & kFlagTimeout) ? 1 : 0;
        mbar_init(&s_bar, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    // unit-offset tables
    for (int l = 1; l <= L; ++l) {
        int* jo = reinterpret_cast<int*>(sm + c.joff[l]);
        const int nin = s_n[l - 1];
        if (l == 1) {
            for (int j = tid; j < nin; j += kThreads) jo[j] = j;
        } else {
            const int ucap = c.ucap[l - 1], blk = c.blk[l - 1], nupm = c.nup[l - 1];
            int* si = reinterpret_cast<int*>(sm + c.sidx[l]);
            for (int j = tid; j < nin; j += kThreads) {
                jo[j] = (j / ucap) * blk + (j % ucap);
                si[j] = (j / ucap) * nupm + (j % ucap);
            }
        }
    }
    cluster.sync();
    if (*cluster.map_shared_rank(&s_stop, 0)) {
        cluster.sync();
        return;
    }
    unsigned bar_phase = 0;

    // own weights, V and a zero G into shared memory (transposed: row j = input)
    for (int l = 1; l <= L; ++l) {
        const int n_in = s_n[l - 1], nup = c.nup[l];
        const int u0 = rank * c.ucap[l], nu = units_of(s_n[l], c.ucap[l], rank);
        float* W = sm + c.wt[l];
        float* Vt = W + c.wsz[l];
        float* Gt = Vt + c.wsz[l];
        for (int e = tid; e < c.wsz[l]; e += kThreads) {
            const int j = e / nup, u = e - j * nup;
            float w = 0.f, v = 0.f;
            if (u < nu) {
                const long long idx = (j < n_in) ? a.woff[l] + (long long)(u0 + u) * n_in + j
                                                 : a.boff[l] + u0 + u;
                w = a.theta[idx];
                v = a.V[idx];
            }
            W[e] = w;
            Vt[e] = v;
            Gt[e] = 0.f;
        }
    }
    __syncthreads();

    const int n0 = s_n[0], nL = s_n[L];
    const int uL0 = rank * c.ucap[L], nuL = units_of(nL, c.ucap[L], rank);
    float sse = 0.f;
#pragma unroll 1
    for (int s = 0; s < n_steps; ++s) {
        const long long g0 = (long long)s * minibatch;
        const int B = (int)min((long long)minibatch, (long long)n_patterns - g0);
        const int p_lo = (int)((long long)B * cl / NC), p_hi = (int)((long long)B * (cl + 1) / NC);
        sse = 0.f;
#pragma unroll 1
        for (int q0 = p_lo; q0 < p_hi; q0 += Pc) {
            const int pc = min(Pc, p_hi - q0);
            const long long prow = g0 + q0;   // first pattern of the chunk
            // ---- input chunk and the targets of own output units
            {
                float* xin = sm + c.full[0];
                const int pf = c.pf[0];
                for (int p = warp; p < pc; p += kWarps) {
                    const float* src = X + (prow + p) * n0;
                    for (int j = lane; j < n0; j += 32) cp_async4(xin + p * pf + j, src + j);
                }
                float* tin = sm + c.tin;
                const int nupL = c.nup[L];
                for (int e = tid; e < pc * nuL; e += kThreads) {
                    const int p = e / nuL, u = e - p * nuL;
                    cp_async4(tin + p * nupL + u, T + (prow + p) * nL + uL0 + u);
                }
                cp_async_wait_all();
                __syncthreads();
            }
            // ---- forward: thread = (pattern, slice of the inputs), 8 units at a time
#pragma unroll 1
            for (int l = 1; l <= L; ++l) {
                const int n_in = s_n[l - 1], nup = c.nup[l], ks = c.ks[l];
                const float* W = sm + c.wt[l];
                const int* jo = reinterpret_cast<const int*>(sm + c.joff[l]);
                const float* inb = sm + c.full[l - 1];
                const int pin = (l == 1) ? c.pf[0] : c.rp[l - 1];
                float* red = sm + c.red;
                for (int it = tid; it < Pc * ks; it += kThreads) {
                    const int p = it % Pc, kq = it / Pc;
                    const int j0 = kq * n_in / ks, j1 = (kq + 1) * n_in / ks;
                    const float* ip = inb + p * pin;
                    for (int g = 0; g < nup; g += 8) {
                        float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
                        if (p < pc) {
                            if (l == 1) {
#pragma unroll 4
                                for (int j = j0; j < j1; ++j) fma8(acc, ip[j], W + j * nup + g);
                            } else {
#pragma unroll 2
                                for (int j = j0; j < j1; ++j) fma8(acc, ip[jo[j]], W + j * nup + g);
                            }
                        }
                        float* rp_ = red + (kq * Pc + p) * nup + g;
                        *reinterpret_cast<float4*>(rp_) = make_float4(acc[0], acc[1], acc[2], acc[3]);
                        *reinterpret_cast<float4*>(rp_ + 4) = make_float4(acc[4], acc[5], acc[6], acc[7]);
                    }
                }
                __syncthreads();
                const float* bias = W + n_in * nup;
                const int nu = units_of(s_n[l], c.ucap[l], rank);
                if (l < L) {
                    // own block of layer l, then all-gather the other blocks
                    const int rp = c.rp[l], blk = c.blk[l];
                    float* full = sm + c.full[l];
                    float* own = full + rank * blk;
                    for (int e = tid; e < Pc * nu; e += kThreads) {
                        const int p = e / nu, u = e - p * nu;
                        float sum = 0.f;
                        for (int kq = 0; kq < ks; ++kq) sum += red[(kq * Pc + p) * nup + u];
                        own[p * rp + u] = (p < pc) ? sigmoid_f(sum + bias[u]) : 0.f;
                    }
                    cluster.sync();   // every block of layer l is written
                    const int blk4 = blk >> 2;
                    const int tot = C * blk4;
                    for (int e = tid; e < tot; e += 4 * kThreads) {
                        float4 v[4];
                        int dst[4];
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            const int ee = e + k * kThreads;
                            const int r = ee / blk4;
                            dst[k] = -1;
                            if (ee < tot && r != rank) {
                                dst[k] = ee;
                                v[k] = reinterpret_cast<const float4*>(cluster.map_shared_rank(full, r))[ee];
                            }
                        }
#pragma unroll
                        for (int k = 0; k < 4; ++k)
                            if (dst[k] >= 0) reinterpret_cast<float4*>(full)[dst[k]] = v[k];
                    }
                    __syncthreads();
                } else {
                    // output layer: delta and error sum of own output units
                    float* dn = sm + c.dn[L];
                    const float* tin = sm + c.tin;
                    for (int e = tid; e < Pc * nup; e += kThreads) {
                        const int p = e / nup, u = e - p * nup;
                        float d = 0.f;
                        if (p < pc && u < nu) {
                            float sum = 0.f;
                            for (int kq = 0; kq < ks; ++kq) sum += red[(kq * Pc + p) * nup + u];
                            const float o = sigmoid_f(sum + bias[u]);
                            const float err = tin[p * nup + u] - o;
                            sse = fmaf(err, err, sse);
                            d = err * o * (1.f - o);
                        }
                        dn[e] = d;
                    }
                    __syncthreads();
                }
            }
            // ---- hidden deltas, output side first
#pragma unroll 1
            for (int l = L; l >= 2; --l) {
                const int n_in = s_n[l - 1], nup = c.nup[l], nupm = c.nup[l - 1];
                const float* W = sm + c.wt[l];
                const float* dn = sm + c.dn[l];
                float* S = sm + c.S[l];
                const int* si = reinterpret_cast<const int*>(sm + c.sidx[l]);
                const int ps = C * nupm;
                // partial sums over own units of layer l, for every unit of layer l-1
                for (int p = warp; p < pc; p += kWarps) {
                    const float* dp = dn + p * nup;
                    float* Sp = S + p * ps;
                    for (int j = lane; j < n_in; j += 32) {
                        const float* wj = W + j * nup;
                        float acc = 0.f;
                        for (int g = 0; g < nup; g += 4) {
                            const float4 d = *reinterpret_cast<const float4*>(dp + g);
                            const float4 w = *reinterpret_cast<const float4*>(wj + g);
                            acc = fmaf(d.x, w.x, acc);
                            acc = fmaf(d.y, w.y, acc);
                            acc = fmaf(d.z, w.z, acc);
                            acc = fmaf(d.w, w.w, acc);
                        }
                        Sp[si[j]] = acc;
                    }
                }
                cluster.sync();   // every CTA's partial sums are written
                // own units of layer l-1: sum the partials of all ranks in rank
                // order (4 floats per remote load)
                const int num = units_of(n_in, c.ucap[l - 1], rank);
                float* dm = sm + c.dn[l - 1];
                const float* act = sm + c.full[l - 1] + rank * c.blk[l - 1];
                const int rpa = c.rp[l - 1];
                const int nq = nupm >> 2;
                for (int e = tid; e < Pc * nq; e += kThreads) {
                    const int p = e / nq, q = e - p * nq;
                    float4 sum = make_float4(0.f, 0.f, 0.f, 0.f);
                    if (p < pc) {
                        const int col = p * ps + rank * nupm + q * 4;
#pragma unroll 4
                        for (int r = 0; r < C; ++r) {
                            const float4 v =
                                *reinterpret_cast<const float4*>(cluster.map_shared_rank(S, r) + col);
                            sum.x += v.x;
                            sum.y += v.y;
                            sum.z += v.z;
                            sum.w += v.w;
                        }
                    }
                    const float sv[4] = {sum.x, sum.y, sum.z, sum.w};
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        const int u = q * 4 + k;
                        float d = 0.f;
                        if (p < pc && u < num) {
                            const float av = act[p * rpa + u];
                            d = sv[k] * av * (1.f - av);
                        }
                        dm[p * nupm + u] = d;
                    }
                }
                __syncthreads();
            }
            // ---- pooled change of own weights over the chunk: thread = input unit
#pragma unroll 1
            for (int l = 1; l <= L; ++l) {
                const int n_in = s_n[l - 1], nup = c.nup[l];
                const float* dn = sm + c.dn[l];
                float* Gt = sm + c.wt[l] + 2 * c.wsz[l];
                const int rows = n_in + 1;
                const int* jo = reinterpret_cast<const int*>(sm + c.joff[l]);
                const float* inb = sm + c.full[l - 1];
                const int pin = (l == 1) ? c.pf[0] : c.rp[l - 1];
                const int ng = nup >> 3;
                for (int it = tid; it < rows * ng; it += kThreads) {
                    const int j = it % rows, g = (it / rows) * 8;
                    float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
                    if (j < n_in) {
                        const float* ip = inb + jo[j];
#pragma unroll 2
                        for (int p = 0; p < pc; ++p) fma8(acc, ip[p * pin], dn + p * nup + g);
                    } else {
#pragma unroll 2
                        for (int p = 0; p < pc; ++p) fma8(acc, 1.f, dn + p * nup + g);
                    }
                    float* gp = Gt + j * nup + g;
#pragma unroll
                    for (int k = 0; k < 8; ++k) gp[k] += acc[k];
                }
            }
            __syncthreads();
        }
        // ---- this copy's pooled change (one contiguous slice per CTA) and error sum
        const int buf = s & 1;
        const size_t slice_stride = (size_t)c.slice;
        {
            float* dst = a.gpart + (((size_t)buf * NC + cl) * C + rank) * slice_stride;
            for (int l = 1; l <= L; ++l) {
                float4* G4 = reinterpret_cast<float4*>(sm + c.wt[l] + 2 * c.wsz[l]);
                float4* d4 = reinterpret_cast<float4*>(dst + c.soff[l]);
                for (int e = tid; e < (c.wsz[l] >> 2); e += kThreads) {
                    d4[e] = G4[e];
                    G4[e] = make_float4(0.f, 0.f, 0.f, 0.f);
                }
            }
        }
        const float e = block_sum(sse, red8);
        if (tid == 0) {
            a.sse_part[(size_t)buf * gridDim.x + blockIdx.x] = e;
            __threadfence();   // this CTA's pooled change is visible GPU-wide
        }
        // hierarchical grid barrier: the cluster first, then one arrival per cluster
        cluster.sync();
        if (rank == 0 && tid == 0) s_fail[buf] = grid_barrier_t0(a.bar, a.flags, NC) ? 0 : 1;
        cluster.sync();
        int fail = 0;
        if (tid == 0) fail = cluster.map_shared_rank(s_fail, 0)[buf];
        fail = __syncthreads_or(fail);
        if (fail) {
            cluster.sync();
            return;
        }
        if (blockIdx.x == gridDim.x - 1 && tid < 32) {
            // error sum of the group, by the last CTA (the last rank owns the
            // fewest units): lane-strided partial sums, then a fixed butterfly,
            // so that every run adds in the same order
            const float* sp = a.sse_part + (size_t)buf * gridDim.x;
            float tot = 0.f;
            for (int k = tid; k < (int)gridDim.x; k += 32) tot += __ldcg(sp + k);
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) tot += __shfl_xor_sync(0xffffffffu, tot, o);
            if (tid == 0) {
                if (sse_out != nullptr) sse_out[s] = tot;
                if (!isfinite(tot)) atomicOr(a.flags, kFlagNonfinite);
            }
        }
        // ---- sum of all copies' changes in cluster order: bulk copies of this
        // rank's slice from every cluster, R at a time, into the staging ring
        float* stg = sm + c.stg;
        const unsigned slice_bytes = (unsigned)(c.slice * sizeof(float));
#pragma unroll 1
        for (int k0 = 0; k0 < NC; k0 += c.R) {
            const int nk = min(c.R, NC - k0);
            if (tid == 0) {
                asm volatile("fence.proxy.async.global;" ::: "memory");
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                const unsigned b = (unsigned)__cvta_generic_to_shared(&s_bar);
                asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(b),
                             "r"(slice_bytes * (unsigned)nk)
                             : "memory");
                for (int k = 0; k < nk; ++k) {
                    const float* src =
                        a.gpart + (((size_t)buf * NC + (k0 + k)) * C + rank) * slice_stride;
                    const unsigned d = (unsigned)__cvta_generic_to_shared(stg + (size_t)k * c.slice);
                    asm volatile(
                        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], "
                        "%2, [%3];" ::"r"(d),
                        "l"(src), "r"(slice_bytes), "r"(b)
                        : "memory");
                }
            }
            // bounded wait for the copies
            {
                bool done = mbar_try_wait(&s_bar, bar_phase);
                const unsigned long long t0 = done ? 0ull : global_ns();
                unsigned it = 0;
                while (!done) {
                    done = mbar_try_wait(&s_bar, bar_phase);
                    if (!done && ((++it & 255u) == 0) && global_ns() - t0 > kWaitNs) {
                        if (tid == 0) atomicOr(a.flags, kFlagTimeout);
                        break;
                    }
                }
                bar_phase ^= 1u;
            }
            const int s4 = c.slice >> 2;
            for (int l = 1; l <= L; ++l) {
                float4* G4 = reinterpret_cast<float4*>(sm + c.wt[l] + 2 * c.wsz[l]);
                const float4* sl = reinterpret_cast<const float4*>(stg + c.soff[l]);
                const int n4 = c.wsz[l] >> 2;
                for (int e4 = tid; e4 < n4; e4 += kThreads) {
                    float4 g = G4[e4];
                    for (int k = 0; k < nk; ++k) {
                        const float4 v = sl[(size_t)k * s4 + e4];
                        g.x += v.x;
                        g.y += v.y;
                        g.z += v.z;
                        g.w += v.w;
                    }
                    G4[e4] = g;
                }
            }
            __syncthreads();   // the staging ring is read before it is refilled
        }
        // ---- momentum update of own weights (Section 6.2.1); padding columns
        // hold zeros in W, V and G and stay zero
        const float lr_gs = a.lr * a.grad_scale, mom = a.momentum;
        const bool fold = (fold_g != 0) && (s == 0);
        for (int l = 1; l <= L; ++l) {
            float* W = sm + c.wt[l];
            float* Vt = W + c.wsz[l];
            float* Gt = Vt + c.wsz[l];
            if (fold) {
                const int n_in = s_n[l - 1], nup = c.nup[l];
                const int u0 = rank * c.ucap[l], nu = units_of(s_n[l], c.ucap[l], rank);
                for (int e = tid; e < c.wsz[l]; e += kThreads) {
                    const int j = e / nup, u = e - j * nup;
                    if (u < nu) {
                        const long long idx = (j < n_in) ? a.woff[l] + (long long)(u0 + u) * n_in + j
                                                         : a.boff[l] + u0 + u;
                        Gt[e] += a.G[idx];
                    }
                }
            }
            for (int e = tid; e < c.wsz[l]; e += kThreads) {
                const float vel = lr_gs * Gt[e] + mom * Vt[e];
                Vt[e] = vel;
                W[e] += vel;
                Gt[e] = 0.f;
            }
        }
        __syncthreads();
    }
    // ---- the first copy writes the weights and V back
    if (cl == 0) {
        for (int l = 1; l <= L; ++l) {
            const int n_in = s_n[l - 1], nup = c.nup[l];
            const int u0 = rank * c.ucap[l], nu = units_of(s_n[l], c.ucap[l], rank);
            const float* W = sm + c.wt[l];
            const float* Vt = W + c.wsz[l];
            const int rows = n_in + 1;
            for (int it = tid; it < nu * rows; it += kThreads) {
                const int u = it / rows, j = it - u * rows;
                const long long idx = (j < n_in) ? a.woff[l] + (long long)(u0 + u) * n_in + j
                                                 : a.boff[l] + u0 + u;
                a.theta[idx] = W[j * nup + u];
                a.V[idx] = Vt[j * nup + u];
            }
        }
    }
    cluster.sync();   // no CTA leaves while another may still read its shared memory
}

}  // namespace

// ------------------------------------------------------------ host side
static size_t cl_smem_bytes(const int* n, int L, int C, int Pc, int R) {
    ClCarve c;
    cl_make_carve(c, n, L, C, Pc, R);
    return (size_t)c.total * sizeof(float);
}

size_t cl_slice_floats(const int* n, int L, int C) {
    ClCarve c;
    cl_make_carve(c, n, L, C, 32, 1);
    return (size_t)c.slice;
}

cudaError_t cl_setup(int /*device*/) {
    cudaError_t e =
        cudaFuncSetAttribute(k_train_cl, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
    return cudaFuncSetAttribute(k_train_cl, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)kClSmemLimit);
}

static int max_clusters(int C, size_t smem) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(C, 1, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = C;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    int n = 0;
    const cudaError_t e = cudaOccupancyMaxActiveClusters(&n, k_train_cl, &cfg);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return 0;
    }
    return n;
}

ClPlan cl_plan(const int* n, int L, int batch, int num_sms) {
    ClPlan best{};
    best.ok = false;
    const int sizes[2] = {16, 8};
    for (int ci = 0; ci < 2; ++ci) {
        const int C = sizes[ci];
        // need room for at least a 32-pattern chunk and one staged copy
        if (cl_smem_bytes(n, L, C, 32, 1) > kClSmemLimit) continue;
        // clusters that can be resident at once with a full-size carve (one CTA
        // per SM): the grid barrier needs every cluster resident
        int NC = max_clusters(C, kClSmemLimit);
        if (NC * C > num_sms) NC = num_sms / C;
        if (NC > kClMaxCopies) NC = kClMaxCopies;
        if (NC < 1) continue;
        // chunk: the patterns a copy gets per group (a multiple of 8, at most
        // 256), shrunk until it fits; then as many staged copies as fit
        const int per = (batch + NC - 1) / NC;
        int pc = ((per + 7) / 8) * 8;
        if (pc > 256) pc = 256;
        if (pc < 32) pc = 32;
        while (pc > 32 && cl_smem_bytes(n, L, C, pc, 1) > kClSmemLimit) pc -= 8;
        int R = 1;
        while (R < NC && cl_smem_bytes(n, L, C, pc, R + 1) <= kClSmemLimit) ++R;
        ClPlan p;
        p.ok = true;
        p.C = C;
        p.NC = NC;
        p.Pc = pc;
        p.R = R;
        p.smem = cl_smem_bytes(n, L, C, pc, R);
        // prefer 16-CTA clusters unless they leave most of the GPU idle
        if (!best.ok || NC * C > 2 * best.NC * best.C) best = p;
        if (C == 16 && NC * C * 4 >= num_sms * 3) break;
    }
    return best;
}

cudaError_t f32_train_cluster(const ClArgs& args, const float* X, const float* T, int n_patterns,
                              int minibatch, int n_steps, float* sse_out, bool fold_g,
                              const ClPlan& plan, cudaStream_t s) {
    ClArgs a = args;
    cl_make_carve(a.cv, a.n, a.L, plan.C, plan.Pc, plan.R);
    int fold = fold_g ? 1 : 0;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(plan.NC * plan.C, 1, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = plan.smem;
    cfg.stream = s;
    cudaLaunchAttribute at[2];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = plan.C;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    at[1].id = cudaLaunchAttributeCooperative;
    at[1].val.cooperative = 1;
    cfg.attrs = at;
    cfg.numAttrs = 2;
    auto launch = [&]() {
        return cudaLaunchKernelEx(&cfg, k_train_cl, a, X, T, n_patterns, minibatch, n_steps,
                                  sse_out, fold);
    };
    cudaError_t e = launch();
    if (e == cudaErrorNotSupported || e == cudaErrorInvalidValue) {
        // Cluster launches that cannot also be cooperative: the grid is still
        // sized to the clusters the device holds at once (occupancy query above),
        // and every wait of the grid barrier is bounded.
        cudaGetLastError();
        cfg.numAttrs = 1;
        e = launch();
    }
    if (e != cudaSuccess) return e;
    if (fold_g && a.G != nullptr) e = cudaMemsetAsync(a.G, 0, (size_t)a.P * sizeof(float), s);
    return e;
}

}  // namespace bp
