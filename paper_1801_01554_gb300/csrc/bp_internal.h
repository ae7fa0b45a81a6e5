// Internal declarations shared by the translation units of libbp.so.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>
#include <cstdint>

#include "bp.h"

namespace bp {

constexpr int kMaxL = BP_MAX_SIZES - 1;   // weight layers

// Bits of the device-side error word latched by kernels.
constexpr int kFlagTimeout = 1;     // a bounded wait ran out
constexpr int kFlagNonfinite = 2;   // an error sum was NaN/Inf
constexpr int kFlagBounds = 4;      // a check of the checked build (-DBP_CHECK) failed

// Words of the grid-barrier state (two used, padded to 16 bytes).
constexpr int kBarWords = 4;

// Device view of a float32 net, passed to kernels by value.
//   theta/V/G: flat parameter vectors in the padded device layout: layer by
//              layer, W_l as [n_l][kp_l] rows with kp_l = apitch_{l-1}, where
//              column n_{l-1} holds the bias b_l (the true unit's weight) and
//              the columns after it are zero; P floats in all, a multiple of 4
//              (also the size of its shared-memory copy, wsm).  The API's
//              packed layout (W_l row-major, then b_l; Pp floats) is converted
//              on the way in and out.
//   A: activations of layers 0..L for `cap` patterns, layer l at aoff[l] in
//      acb[l] column blocks of [cap][32] floats (columns 32b .. 32b + 31;
//      column n_l holds the true unit's 1, columns past it are 0).  Inside a
//      pattern's 128-byte block row the 16-byte chunk k sits at k ^ (p mod 8),
//      so that the weight phase's lanes read 32 consecutive rows without bank
//      conflicts; a chunk of a tile is one contiguous bulk copy.
//   D: deltas of layers 1..L at doff[l] in dtb[l] blocks of [cap][8] floats
//      (an even number of blocks per layer), chunk k of a 32-byte block row at
//      k ^ ((p / 4) mod 2).
//   apitch[l] = n_l + 1 and dpitch[l] = n_l rounded up to 4 are the row
//   pitches of the same rows in shared memory.
//   Gradient tiles: layer l owns tiles [tile0[l], tile0[l+1]) of 8 rows x 32
//   columns of the [n_l, n_{l-1} + 1] matrix (last column = bias), and tiles
//   [tile0w[l], tile0w[l+1]) of 16 rows x 32 columns in the balanced form.
struct F32View {
    int L;
    int cap;
    int n[BP_MAX_SIZES];
    int kp[BP_MAX_SIZES];          // row pitch of W_l in the padded layout
    long long woff[BP_MAX_SIZES];  // padded offset of W_l
    long long pw[BP_MAX_SIZES];    // packed offset of W_l
    long long pb[BP_MAX_SIZES];    // packed offset of b_l
    long long P;                   // padded parameter count
    long long Pp;                  // packed parameter count
    int wsm;
    int apitch[BP_MAX_SIZES];
    int dpitch[BP_MAX_SIZES];
    int acb[BP_MAX_SIZES];         // 32-column blocks of layer l's activations
    int dtb[BP_MAX_SIZES];         // 8-column blocks of layer l's deltas
    long long aoff[BP_MAX_SIZES];
    long long doff[BP_MAX_SIZES];
    long long a_floats, d_floats;
    int tile0[BP_MAX_SIZES + 1];
    int tile0w[BP_MAX_SIZES + 1];  // the same for the balanced weight phase's 16-row tiles
    int tcols[BP_MAX_SIZES];
    float* theta;
    float* V;
    float* G;
    float* A;
    float* D;
    float* sse_part;      // one partial error sum per CTA of the pattern phase
    float* wpart;         // balanced weight phase (large groups): [CTA][2][16 x 32] tile sums, or null
    unsigned* bar;        // grid barrier: [0] count at the end of the last launch, [1] arrival count
    int* flags;           // latched error bits
    float lr, momentum, grad_scale;
    int sig_table;        // 1: table-lookup logistic (Section 4.3) in the forward pass
    float guard;          // > 0: fault guard of Section 8 (|change| > guard is zeroed)
    unsigned* faults;     // changes the guard zeroed (flags[1])
    unsigned long long wait_ns;   // checked build: grid-barrier and weight-phase wait limit (0: the default 2 s)
    int debug_stall;              // checked build: the weight phase's first chunk never completes (test hook)
};

// Offsets (floats, each a multiple of 4) of a CTA's pattern buffers for PG
// patterns, computed on the host: activation rows sa[l] ([PG][apitch_l],
// l = 0..L), delta rows sd[l] ([PG][dpitch_l], l = 1..L), the same deltas
// pattern-minor sdt[l] ([n_l][PG], l = 2..L, read by the hidden deltas below
// them) and target rows st ([PG][n_L]); `total` floats in all.
struct PatLayout {
    int sa[BP_MAX_SIZES];
    int sd[BP_MAX_SIZES];
    int sdt[BP_MAX_SIZES];
    int st;
    int total;
};

// Launch geometry chosen on the host for a group size.
struct F32Plan {
    int pg;          // patterns per CTA pass (1, 2, 4 or 8)
    int grid;        // CTAs of the launch
    int w_in_smem;   // the weights are copied into shared memory
    size_t smem;     // dynamic shared memory bytes
    PatLayout q;     // pattern buffers
    int split;       // training launches use the balanced weight phase (large minibatches)
};

// --- float32 path (bp_f32.cu) -------------------------------------------
// Fills the layout fields of v for the layer sizes and capacity; returns the
// scratch floats A and D need together.
long long f32_layout(F32View& v, const int* n, int L, int cap);
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
// Packed <-> padded parameter layouts (see F32View), on the host and on the device.
void f32_pad_host(const F32View& v, const float* packed, float* padded);
void f32_unpad_host(const F32View& v, const float* padded, float* packed);
cudaError_t f32_pad_device(const F32View& v, const float* packed, float* padded, cudaStream_t s);
cudaError_t f32_unpad_device(const F32View& v, const float* padded, float* packed, cudaStream_t s);
// Persistent cooperative launch running `n_steps` groups of `minibatch` patterns
// (the last may be ragged), one update after each.  fold_g: G holds a pending
// change to add into the first update.
cudaError_t f32_train(const F32View& v, const float* X, const float* T, int n_patterns,
                      int minibatch, int n_steps, float* sse_out, bool fold_g,
                      const F32Plan& plan, cudaStream_t s);

// Groups of at most 4 patterns on one CTA, with the weights resident in its
// shared memory for the whole launch (f32_small_ok says whether the net fits;
// no pending change G is folded in).
bool f32_small_ok(const F32View& v, int minibatch);
cudaError_t f32_train_small(const F32View& v, const float* X, const float* T, int n_patterns,
                            int minibatch, int n_steps, float* sse_out, cudaStream_t s);

// Diagnostic mode (Section 8): num_sms CTAs each run the forward pass and error
// of all `batch` patterns; per-CTA error sums to d_sse, SM ids to d_sm.
cudaError_t f32_diagnose(const F32View& v, const float* X, const float* T, int batch, float* d_sse,
                         int* d_sm, int num_sms, cudaStream_t s);

// Message returned by bp_last_error() on the calling thread (bp_api.cu).
void set_error_message(const char* msg);

// cuTensorMapEncodeTiled from the driver, looked up once (bp_api.cu); null if
// the driver does not provide it.
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder();

}  // namespace bp
