// Internal declarations shared by the translation units of libbp.so.
#pragma once

#include <cuda_runtime.h>
#include <cstdint>

#include "bp.h"

namespace bp {

constexpr int kMaxL = BP_MAX_SIZES - 1;   // weight layers

// Bits of the device-side error word latched by kernels.
constexpr int kFlagTimeout = 1;     // a bounded wait ran out
constexpr int kFlagNonfinite = 2;   // an error sum was NaN/Inf

// Device view of a float32 net, passed to kernels by value.
//   theta/V/G: flat parameter vectors (layer order, W_l row-major then b_l).
//   A, D: scratch activations/deltas; rows of layer l start at soff[l] and hold
//         n[l] floats per pattern, capacity `cap` patterns.
//   Gradient tiles: layer l owns tiles [tile0[l], tile0[l+1]) of 8 rows x 32
//   columns of the [n_l, n_{l-1} + 1] matrix (last column = bias).
struct F32View {
    int L;
    int cap;
    int n[BP_MAX_SIZES];
    long long woff[BP_MAX_SIZES];
    long long boff[BP_MAX_SIZES];
    long long soff[BP_MAX_SIZES];
    int tile0[BP_MAX_SIZES + 1];
    int tcols[BP_MAX_SIZES];
    float* theta;
    float* V;
    float* G;
    float* A;
    float* D;
    float* sse_part;      // one partial error sum per CTA of the pattern phase
    unsigned* bar;        // grid barrier: [0] arrivals, [1] generation
    int* flags;           // latched error bits
    float lr, momentum, grad_scale;
};

// Launch geometry chosen on the host for a group size.
struct F32Plan {
    int pg;          // patterns per CTA group (1, 2, 4 or 8)
    int grid;        // CTAs of the persistent launch
    size_t smem;     // dynamic shared memory bytes
};

// --- float32 path (bp_f32.cu) -------------------------------------------
// Largest group size (patterns per CTA pass) whose activations fit in shared memory.
int f32_max_pg(const int* n, int L);
size_t f32_smem_bytes(const int* n, int L, int pg);
cudaError_t f32_setup(int device);   // opt-in shared memory limits, once per process
F32Plan f32_plan(const F32View& v, int batch, int num_sms);

cudaError_t f32_forward(const F32View& v, const float* X, int batch, float* Y,
                        const F32Plan& plan, cudaStream_t s);
cudaError_t f32_backward(const F32View& v, const float* X, const float* T, int batch,
                         float* sse_out, const F32Plan& plan, cudaStream_t s);
cudaError_t f32_update(const F32View& v, long long n_params, cudaStream_t s);
// Persistent cooperative launch running `n_steps` groups of `minibatch` patterns
// (the last may be ragged), one update after each.  fold_g: G holds a pending
// change to add into the first update.
cudaError_t f32_train(const F32View& v, const float* X, const float* T, int n_patterns,
                      int minibatch, int n_steps, float* sse_out, bool fold_g,
                      const F32Plan& plan, cudaStream_t s);

// Message returned by bp_last_error() on the calling thread (bp_api.cu).
void set_error_message(const char* msg);

// --- float32 path on thread-block clusters (bp_f32_cluster.cu) -------------
constexpr size_t kClSmemLimit = 227 * 1024 - 1024;   // dynamic shared memory per CTA
constexpr int kClMaxCopies = 19;                     // clusters (net copies) at most

// Shared-memory carve of a CTA (offsets in floats), computed on the host.
struct ClCarve {
    int L, C, Pc, R;
    int slice, stg, red, total;
    int n[BP_MAX_SIZES], ucap[BP_MAX_SIZES], nup[BP_MAX_SIZES], pf[BP_MAX_SIZES];
    int rp[BP_MAX_SIZES], blk[BP_MAX_SIZES];
    int wt[BP_MAX_SIZES], wsz[BP_MAX_SIZES], soff[BP_MAX_SIZES];
    int full[BP_MAX_SIZES], dn[BP_MAX_SIZES], S[BP_MAX_SIZES], joff[BP_MAX_SIZES];
    int sidx[BP_MAX_SIZES], ks[BP_MAX_SIZES];
    int tin;
};

// Arguments of the cluster training kernel.
struct ClArgs {
    int L;
    int n[BP_MAX_SIZES];
    long long woff[BP_MAX_SIZES];
    long long boff[BP_MAX_SIZES];
    long long P;          // parameters
    ClCarve cv;           // set from the plan at launch
    float* theta;
    float* V;
    float* G;             // pending pooled change (read only when folded in)
    float* gpart;         // [2][clusters][C][slice]: each CTA's pooled change
    float* sse_part;      // [2][CTAs]
    unsigned* bar;
    int* flags;
    float lr, momentum, grad_scale;
};

struct ClPlan {
    bool ok;
    int C;        // CTAs per cluster
    int NC;       // clusters = copies of the net
    int Pc;       // patterns per chunk
    int R;        // copies staged per round
    size_t smem;
};

cudaError_t cl_setup(int device);
size_t cl_slice_floats(const int* n, int L, int C);   // floats of one CTA's slice
ClPlan cl_plan(const int* n, int L, int batch, int num_sms);
cudaError_t f32_train_cluster(const ClArgs& a, const float* X, const float* T, int n_patterns,
                              int minibatch, int n_steps, float* sse_out, bool fold_g,
                              const ClPlan& plan, cudaStream_t s);

}  // namespace bp
