/*
 * bp.h -- C ABI of libbp.so: the batch back-propagation training step of a
 * fully connected sigmoid multi-layer perceptron on one GB300 (sm_103a).
 *
 * The method is the one of Witbrock & Zagha, "An Implementation of
 * Back-Propagation Learning on GF11" (CMU-CS-89-208):
 *   - forward pass: a_j = 1 / (1 + exp(-(sum_i w_ji a_i + b_j)))       (Section 3, fn. 4)
 *   - error: summed squared difference E = sum (t - o)^2              (Section 3, fn. 5)
 *   - output delta (t - o) o (1 - o); hidden delta (W^T delta) h (1 - h);
 *     no delta for input units (Section 6.1, "Cycles backward/case")
 *   - pooled weight change summed over every pattern of a group       (Sections 3, 4.1)
 *   - update with learning rate and momentum, then the pooled change
 *     is zeroed (Section 6.2.1):
 *         V <- lr * grad_scale * G + momentum * V ;  W <- W + V ;  G <- 0
 *     G is the pooled sum of delta * activation (minus the gradient of E/2),
 *     V starts at zero, grad_scale is 1 (a sum, as the paper pools) unless set.
 * The bias of a unit is its weight from the always-on "true" unit (Section 6.3)
 * and is trained and counted like every other connection.
 *
 * Conventions shared by every entry point
 *   - Layer sizes n_0 (inputs) ... n_L (outputs), 2 <= n_layers <= BP_MAX_SIZES.
 *   - Parameter vectors ("theta", and V, G of the same shape) are flat float32
 *     arrays in layer order: for l = 1..L, W_l as n_l rows of n_{l-1} floats
 *     (row-major), then the n_l bias weights b_l.  Length = bp_num_params().
 *   - Patterns are row-major: X is [batch, n_0], T and Y are [batch, n_L].
 *     Their element type is float32 for BP_F32 nets and bfloat16 (raw uint16
 *     bits, round-to-nearest-even) for BP_BF16 nets.  Targets are in [0, 1].
 *   - Alignment: device pattern buffers (X, T, Y) start on a 16-byte boundary
 *     for BP_BF16 nets (their rows move in 16-byte pieces) and on a 4-byte
 *     boundary for BP_F32 nets; error-sum buffers on a 4-byte boundary.  Other
 *     pointers are rejected with BP_EINVAL before any work is queued.
 *   - Device pointers ("d_") are caller-owned CUDA device memory on the current
 *     device; the library never frees them.  Host pointers ("h_") are caller-
 *     owned host memory (pinned memory makes the copies asynchronous).
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *     Compute entry points are asynchronous with respect to the host; the
 *     device buffers they read must stay valid until the stream reaches them.
 *     A BP_BF16 net's backward pass forks part of its work (the input
 *     transpose) onto a stream of the net's own and joins it back into
 *     `stream` before the call's next dependent kernel, so that the call's
 *     work is ordered on `stream` as a whole (stream capture included).
 *   - A net must not be used from two host threads at once.
 *   - Every call returns a bp_status; on failure bp_last_error() holds a
 *     message for the calling thread.  Argument errors are detected before any
 *     work is queued.  Errors raised by a kernel (a bounded device-side wait
 *     that ran out, a non-finite error sum) are latched on the device and
 *     reported by bp_check().
 */
#ifndef BP_H
#define BP_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define BP_MAX_SIZES 9            /* n_0 .. n_8: at most 8 weight layers */

typedef struct bp_net bp_net;     /* opaque; owns device W, b, V, G and scratch */

typedef enum {
    BP_OK = 0,
    BP_EINVAL = 1,      /* NULL pointer, size <= 0, batch above capacity, bad hparam */
    BP_ENOMEM = 2,      /* a device or host allocation failed */
    BP_ECUDA = 3,       /* a CUDA runtime/driver call failed (message in bp_last_error) */
    BP_ESHAPE = 4,      /* layer sizes or batch not supported by this net's dtype path */
    BP_ETIMEOUT = 5,    /* a bounded device-side wait ran out; that launch did no more work */
    BP_ENONFINITE = 6,  /* the error sum of a group came out NaN or Inf */
    BP_ESTATE = 7       /* call order violated (e.g. bp_backward without bp_forward) */
} bp_status;

typedef enum {
    BP_F32 = 0,   /* float32 everywhere; SIMT FFMA kernels */
    BP_BF16 = 1   /* bfloat16 activations/deltas/weight copies on tcgen05 tensor
                     cores with float32 accumulation; float32 master W, b, V, G */
} bp_dtype;

/* Create a net (Section 6.2: the host program turns a network's topology into
 * the routines that train it; Section 6.2.1: the update routine takes the
 * learning rate and momentum).  Weights, V and G start at zero (set them with
 * bp_set_weights).
 * layer_sizes: host array of n_layers ints, each >= 1 (n_0 inputs ... n_L
 * outputs; every layer fully connected to the next, plus the true unit).
 * lr, momentum: the rates of the update routine (Section 6.2.1), finite.
 * dtype: a bp_dtype.  BP_BF16 needs every n_l to be a multiple of 8 (16-byte
 * rows for the tensor-memory copies); any batch size works.
 * max_batch: the largest group any later call may pass (sizes device scratch).
 * Errors: BP_EINVAL (bad argument), BP_ESHAPE (sizes unsupported by dtype),
 * BP_ENOMEM, BP_ECUDA.  *out is set only on BP_OK. */
bp_status bp_create(const int* layer_sizes, int n_layers, float lr, float momentum,
                    int dtype, int max_batch, bp_net** out);

/* Free every device buffer of the net (the counterpart of bp_create, Section
 * 6.2).  NULL-safe.  Synchronises the device.  Caller buffers are untouched. */
void bp_destroy(bp_net* net);

/* Learning rate, momentum and the factor applied to G in the update routine
 * of Section 6.2.1 (grad_scale 1 = the pooled sum of Sections 3 and 4.1,
 * 1/B = a mean).  No device work; the net is not touched on failure.  Takes
 * effect for work queued after the call.  Errors: BP_EINVAL if a value is not
 * finite. */
bp_status bp_set_hparams(bp_net* net, float lr, float momentum, float grad_scale);

/* Squashing function of the forward pass (Section 4.3, Figure 3).
 *   BP_SIGMOID_LOGISTIC (default): 1 / (1 + e^-x), with CUDA's expf.
 *   BP_SIGMOID_TABLE: the GF11's table-lookup logistic: net inputs outside
 *     [-15, 15] take the logistic at -15 or 15; inside, the input is remapped
 *     to [0, 255], its integer part picks one of 256 precomputed values of the
 *     logistic at equally spaced points and its fractional part interpolates
 *     linearly to the next one.  Its error against the logistic is at most
 *     h^2/8 * max|s''| = 1.66e-4 (h = 30/255).  The deltas use a (1 - a) of the
 *     activations it produces.
 * Takes effect for work queued after the call.  Errors: BP_EINVAL for an
 * unknown mode, or BP_SIGMOID_TABLE on a BP_BF16 net (float32 nets only). */
enum { BP_SIGMOID_LOGISTIC = 0, BP_SIGMOID_TABLE = 1 };
bp_status bp_set_sigmoid(bp_net* net, int mode);

/* Fault guard of Section 8: before each update, every total weight change of
 * the group (the pooled change G, before the learning rate) outside
 * [-threshold, threshold], or not a number, is set to zero and counted; the
 * weight then keeps only its momentum term.  threshold = 0 turns the guard off
 * (the default).  Both dtypes.  Takes effect for work queued after the call.
 * Errors: BP_EINVAL for a negative or NaN threshold. */
bp_status bp_set_guard(bp_net* net, float threshold);

/* Number of weight changes the fault guard has zeroed since the net was created
 * or the count was last reset (reset != 0 resets it after reading).
 * Synchronises the device.  Errors: BP_EINVAL, BP_ECUDA. */
bp_status bp_get_faults(bp_net* net, int64_t* count, int reset);

/* Diagnostic mode (Section 8): every CTA of one launch, one per SM, runs the
 * forward pass and the summed squared error of the same `batch` patterns
 * (device d_X [batch, n_0], d_T [batch, n_L]) with the net's weights, without
 * exchanging anything with the others, as each GF11 processor ran the same
 * training set alone.  The per-CTA error sums go to h_sse and the SM each CTA
 * ran on to h_sm (host arrays of `capacity` >= the SM count; either may be
 * NULL); *n_ctas receives the number of CTAs and *n_agree how many produced the
 * most common error sum, bit for bit (a healthy GPU: all of them).  Leaves the
 * weights alone.  Synchronous.  Float32 nets only.
 * Errors: BP_EINVAL (NULL pointers, a BP_BF16 net, capacity too small, batch
 * out of range), BP_ECUDA. */
bp_status bp_diagnose(bp_net* net, const void* d_X, const void* d_T, int batch, float* h_sse,
                      int* h_sm, int capacity, int* n_ctas, int* n_agree);

/* The host's vote of the diagnostic mode: the value that most of values[0, n)
 * equal bit for bit goes to *mode (may be NULL; ties: the earliest such value)
 * and its count to *n_agree.  Host only.  Errors: BP_EINVAL. */
bp_status bp_vote(const float* values, int n, float* mode, int* n_agree);

/* Number of float32 values in a parameter vector (W and b of every layer): the
 * connection count W of Section 7.1, bias connections included (13,826 for
 * 203-60-26, as Section 6.3 prints).  0 for a NULL net. */
int64_t bp_num_params(const bp_net* net);

/* Synchronous copies between host float32 arrays of bp_num_params() values and
 * the net's weights (theta), previous weight change (V) or pending pooled
 * change (G) -- the in-memory copies of the weights that Section 10.4 keeps
 * for checkpoint and recovery; V is the momentum term of Section 6.2.1 and G
 * the pooled change of Sections 3 and 4.1.  Layout: the packed parameter
 * vector above.  h_* are caller-owned host arrays, read or written in full.
 * They synchronise the device first.  bp_set_weights also refreshes the
 * bfloat16 weight copies of a BP_BF16 net.  Errors: BP_EINVAL (NULL), BP_ECUDA. */
bp_status bp_set_weights(bp_net* net, const float* h_theta);
bp_status bp_get_weights(const bp_net* net, float* h_theta);
bp_status bp_set_velocity(bp_net* net, const float* h_v);
bp_status bp_get_velocity(const bp_net* net, float* h_v);
bp_status bp_get_grads(const bp_net* net, float* h_g);

/* Forward pass (Section 3) of `batch` patterns d_X [batch, n_0] -> d_Y
 * [batch, n_L].  d_Y may be NULL.  The activations of every layer are kept in
 * the net's scratch for a following bp_backward, which also reads d_X again:
 * d_X must stay unchanged until then.  Errors: BP_EINVAL (batch < 1 or above
 * max_batch, NULL d_X), BP_ECUDA. */
bp_status bp_forward(bp_net* net, const void* d_X, int batch, void* d_Y, void* stream);

/* Backward pass for the group of the last bp_forward: output and hidden deltas
 * against targets d_T [batch, n_L], then G += the group's pooled change
 * (Sections 3, 4.1).  batch must equal the last forward's.  If d_sse is not
 * NULL, one float (the group's summed squared error) is written there.
 * Errors: BP_ESTATE (no forward, or a different batch), BP_EINVAL, BP_ECUDA. */
bp_status bp_backward(bp_net* net, const void* d_T, int batch, float* d_sse, void* stream);

/* Apply the pending pooled change: V <- lr*grad_scale*G + momentum*V;
 * W <- W + V; G <- 0 (Section 6.2.1). */
bp_status bp_update(bp_net* net, void* stream);

/* One whole training step on one group (Section 3's step with the pooled
 * change of Section 4.1 and the update of Section 6.2.1): forward, backward,
 * pooled change over the `batch` patterns and update, with any change already
 * pending in G folded in.  d_X [batch, n_0], d_T [batch, n_L] caller-owned
 * device buffers; d_sse NULL or one float (the group's summed squared error).
 * Errors: BP_EINVAL (NULL, batch out of [1, max_batch], misaligned buffers),
 * BP_ECUDA; kernel-side errors through bp_check. */
bp_status bp_train_batch(bp_net* net, const void* d_X, const void* d_T, int batch,
                         float* d_sse, void* stream);

/* One pass over n_patterns patterns taken in index order, one update per
 * minibatch (Section 3: changes pooled over a group of cases, then applied; a
 * group of 1 is the per-pattern update, and a ragged last minibatch is a group
 * of its own).  A BP_F32 net runs the whole pass as one persistent device
 * launch; a BP_BF16 net queues one chain of tensor-core kernels per minibatch.
 * d_X [n_patterns, n_0], d_T [n_patterns, n_L] caller-owned device buffers;
 * d_sse (may be NULL) receives ceil(n_patterns / minibatch) floats, the error
 * sum of each group.  minibatch <= max_batch.
 * Errors: BP_EINVAL, BP_ECUDA; kernel-side errors through bp_check. */
bp_status bp_train_epoch(bp_net* net, const void* d_X, const void* d_T, int n_patterns,
                         int minibatch, float* d_sse, void* stream);

/* bp_train_epoch on HOST buffers: copies h_X and h_T to device staging owned by
 * the net (grown on demand), runs the epoch, copies the ceil(n_patterns /
 * minibatch) error sums back to h_sse (may be NULL) and waits for the stream.
 * The epoch runs in up to 8 pieces of whole minibatches, each copied on a
 * stream of the net's own while the previous piece trains (the copies overlap
 * compute when h_X and h_T are pinned); pieces double from ceil(groups / 128)
 * minibatches, so that little of the copy waits in front of the first
 * update.  The updates are the same as one bp_train_epoch over the whole pass.
 * Errors as bp_train_epoch, plus BP_ENOMEM for the staging buffers and any
 * error latched by the epoch's kernels (as bp_check). */
bp_status bp_train_epoch_host(bp_net* net, const void* h_X, const void* h_T, int n_patterns,
                              int minibatch, float* h_sse, void* stream);

/* Wait for `stream`, then report and clear errors latched by earlier kernels
 * (the checks of Section 8: the host learns of a processor's failure and of an
 * error measure out of range before it trusts the weights):
 * BP_ETIMEOUT if a bounded wait ran out (the launch stopped early; its updates
 * so far stand and the grid barrier is reset for the next launch),
 * BP_ENONFINITE if an error sum was not finite, BP_ESTATE if a check of the
 * checked build failed, else BP_OK (or BP_ECUDA for an error from the CUDA
 * runtime).  After it returns, the latch is clear and the net usable. */
bp_status bp_check(bp_net* net, void* stream);

/* bp_train_epoch for callers that cannot allocate device memory.  The paper
 * has no counterpart to this entry point; it exists for callers such as code
 * running inside a host framework that owns the device allocator, processes
 * whose device memory budget was handed out up front, or plug-ins that may only
 * touch the buffers given to them.  It creates no bp_net and calls no
 * cudaMalloc, cudaFree or other allocating routine.
 *   Float32 nets only.  The caller passes every input and output:
 *     d_theta, d_V  float32 [bp_num_params] weights and previous weight change,
 *                   read and updated in place (start d_V at zero);
 *     d_X, d_T      float32 patterns [n_patterns, n_0] and targets [n_patterns, n_L];
 *     d_sse         NULL or ceil(n_patterns / minibatch) floats: error sums;
 *     d_status      NULL or one int: 0 when the launch finished cleanly, else the
 *                   latched error bits (1 = a bounded wait ran out, 2 = a
 *                   non-finite error sum).
 *   Scratch (activations, deltas, barrier, error word) lives in one static
 *   device array of 8 MiB, which every GPU that loads the library holds until the
 *   process exits.  Sizes whose scratch exceeds it are rejected with
 *   BP_EINVAL; the scratch takes 4 * (8 + roundup4(SMs) + 2 * Q + minibatch *
 *   (sum over l = 0..L of roundup32(n_l + 1) + sum over l = 1..L of roundup8(n_l)))
 *   bytes, where Q = sum over l = 1..L of n_l * roundup4(n_{l-1} + 1) holds a
 *   copy of the weights and of the weight changes in the kernel's row layout
 *   (for 203-120-26 on 152 SMs a minibatch of up to 3,808 patterns fits).
 *   The first call on a device looks up the array's device address and sets
 *   kernel attributes; make that first call before any stream capture.  All
 *   calls on a device share the array and find the previous call's contents:
 *   the call clears what must start at zero, and calls that overlap on the GPU
 *   (different streams, or several host threads) race on it.
 *   Every minibatch size runs on the grid-wide persistent kernel (152 CTAs and
 *   two grid barriers per group), including groups of 1-4 patterns, which
 *   bp_train_epoch sends to its one-CTA kernel.
 *   Asynchronous with respect to the host like bp_train_epoch.  Pointers are
 *   checked before any CUDA call: d_theta, d_V, d_X, d_T, d_sse and d_status
 *   must be 4-byte aligned.  Errors: BP_EINVAL, BP_ESHAPE, BP_ECUDA. */
bp_status bp_train_epoch_noalloc(const int* layer_sizes, int n_layers, float lr, float momentum,
                                 float grad_scale, float* d_theta, float* d_V, const float* d_X,
                                 const float* d_T, int n_patterns, int minibatch, float* d_sse,
                                 int* d_status, void* stream);

/* Test hook for the failure detection of Section 8 (a processor that stops
 * answering must be noticed, not waited for): float32 nets, checked builds
 * (-DBP_CHECK) only.  Sets the limit of the training kernel's grid-barrier
 * and weight-phase waits to wait_ns nanoseconds (0 restores the default of
 * 2 s).  unreachable == 1 moves the count that the next training launch's
 * barriers wait for out of reach, so that its first grid barrier runs out of
 * time; unreachable == 2 makes the first chunk copy of each CTA's weight phase
 * a copy that never comes (its barrier is armed for the bytes, no copy is
 * issued), so that the chunk waits run out.  Either way the launch latches the timeout,
 * every CTA returns with every copy it issued landed and no update applied,
 * and bp_check reports BP_ETIMEOUT and resets the barrier; 0 turns both off.
 * Synchronises the device.  Errors: BP_EINVAL (NULL, a BP_BF16 net),
 * BP_ESTATE (a library built without BP_CHECK: the hook does nothing there),
 * BP_ECUDA. */
bp_status bp_debug_wait_test(bp_net* net, unsigned long long wait_ns, int unreachable);

/* Message describing the last failure on the calling thread ("" if none).
 * The pointer stays valid until the thread's next call into the library. */
const char* bp_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* BP_H */
