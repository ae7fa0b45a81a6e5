// C ABI of libbp.so: argument checking, device state and dispatch to the
// float32 (bp_f32.cu) and bfloat16 (bp_bf16.cu) paths.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "bp.h"
#include "bp_bf16.h"
#include "bp_internal.h"

using namespace bp;

namespace {

thread_local std::string g_err;

bp_status fail(bp_status st, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    g_err = buf;
    return st;
}

bp_status cuda_fail(cudaError_t e, const char* what) {
    return fail(e == cudaErrorMemoryAllocation ? BP_ENOMEM : BP_ECUDA, "%s: %s (%s)", what,
                cudaGetErrorName(e), cudaGetErrorString(e));
}

#define BP_CUDA(call, what)                                  \
    do {                                                     \
        cudaError_t e_ = (call);                             \
        if (e_ != cudaSuccess) return cuda_fail(e_, what);   \
    } while (0)

std::mutex g_setup_mu;
bool g_f32_ready[64];

}  // namespace

struct bp_net {
    int dtype = BP_F32;
    int L = 0;
    int n[BP_MAX_SIZES] = {0};
    int max_batch = 0;
    int device = 0;
    int num_sms = 0;
    long long P = 0;    // parameters in the API's packed layout
    long long Pd = 0;   // floats of theta, V and G on the device (padded for float32)
    float lr = 0.f, momentum = 0.f, grad_scale = 1.f;
    // float32 master state (both paths)
    float* theta = nullptr;
    float* V = nullptr;
    float* G = nullptr;
    bool g_dirty = false;          // G holds a change not yet applied
    // float32 path scratch
    float* A = nullptr;
    float* D = nullptr;
    float* sse_part = nullptr;
    float* wpart = nullptr;
    unsigned* bar = nullptr;
    int* flags = nullptr;
    F32View view{};
    // bfloat16 path
    Bf16Net* bf = nullptr;
    // last forward, for bp_backward
    int fwd_batch = 0;
    const void* fwd_X = nullptr;
    // host-buffer epoch staging
    void* stage_X = nullptr;
    void* stage_T = nullptr;
    float* stage_sse = nullptr;
    size_t stage_x_bytes = 0, stage_t_bytes = 0, stage_sse_n = 0;
    // host-buffer epochs copy piece k + 1 on their own stream while piece k trains
    cudaStream_t copy_stream = nullptr;
    cudaEvent_t start_ev = nullptr;
    cudaEvent_t piece_ev[8] = {};
    int* diag_sm = nullptr;   // bp_diagnose: SM of each CTA
};

namespace {

size_t elem_size(const bp_net* net) { return net->dtype == BP_BF16 ? 2 : 4; }

void free_all(bp_net* net) {
    cudaFree(net->theta);
    cudaFree(net->V);
    cudaFree(net->G);
    cudaFree(net->A);
    cudaFree(net->D);
    cudaFree(net->sse_part);
    cudaFree(net->wpart);
    cudaFree(net->bar);
    cudaFree(net->flags);
    cudaFree(net->stage_X);
    cudaFree(net->stage_T);
    cudaFree(net->stage_sse);
    for (cudaEvent_t& e : net->piece_ev)
        if (e) cudaEventDestroy(e);
    if (net->start_ev) cudaEventDestroy(net->start_ev);
    if (net->copy_stream) cudaStreamDestroy(net->copy_stream);
    cudaFree(net->diag_sm);
    if (net->bf) bf16_destroy(net->bf);
}

void refresh_view(bp_net* net) {
    net->view.lr = net->lr;
    net->view.momentum = net->momentum;
    net->view.grad_scale = net->grad_scale;
}

bp_status check_batch(const bp_net* net, int batch) {
    if (batch < 1) return fail(BP_EINVAL, "batch must be >= 1 (got %d)", batch);
    if (batch > net->max_batch)
        return fail(BP_EINVAL, "batch %d exceeds the net's max_batch %d", batch, net->max_batch);
    return BP_OK;
}

// Pattern and output buffers: the bf16 kernels move rows in 16-byte pieces, the
// float32 kernels in 4-byte words.  The error sums are float32 words.
bp_status check_align(const bp_net* net, const void* X, const void* T, const void* Y,
                      const float* sse) {
    const uintptr_t a = net->dtype == BP_BF16 ? 16 : 4;
    const void* p[3] = {X, T, Y};
    const char* what[3] = {"X", "T", "Y"};
    for (int k = 0; k < 3; ++k)
        if (((uintptr_t)p[k] & (a - 1)) != 0)
            return fail(BP_EINVAL, "%s must be %d-byte aligned for this net's dtype", what[k], (int)a);
    if (((uintptr_t)sse & 3) != 0) return fail(BP_EINVAL, "the error-sum buffer must be 4-byte aligned");
    return BP_OK;
}

}  // namespace

extern "C" {

const char* bp_last_error(void) { return g_err.c_str(); }

bp_status bp_create(const int* sizes, int n_layers, float lr, float momentum, int dtype,
                    int max_batch, bp_net** out) {
    g_err.clear();
    if (out == nullptr || sizes == nullptr) return fail(BP_EINVAL, "NULL argument");
    if (n_layers < 2 || n_layers > BP_MAX_SIZES)
        return fail(BP_EINVAL, "n_layers must be in [2, %d] (got %d)", BP_MAX_SIZES, n_layers);
    for (int l = 0; l < n_layers; ++l)
        if (sizes[l] < 1) return fail(BP_EINVAL, "layer size %d is %d; must be >= 1", l, sizes[l]);
    if (max_batch < 1) return fail(BP_EINVAL, "max_batch must be >= 1 (got %d)", max_batch);
    if (dtype != BP_F32 && dtype != BP_BF16) return fail(BP_EINVAL, "unknown dtype %d", dtype);
    if (!std::isfinite(lr) || !std::isfinite(momentum))
        return fail(BP_EINVAL, "lr and momentum must be finite");

    bp_net* net = new bp_net();
    net->dtype = dtype;
    net->L = n_layers - 1;
    for (int l = 0; l < n_layers; ++l) net->n[l] = sizes[l];
    net->max_batch = max_batch;
    net->lr = lr;
    net->momentum = momentum;
    net->grad_scale = 1.f;
    long long P = 0;
    for (int l = 1; l <= net->L; ++l) P += (long long)(sizes[l - 1] + 1) * sizes[l];
    net->P = P;
    net->Pd = P;

    auto bail = [&](bp_status st) {
        free_all(net);
        delete net;
        return st;
    };
    cudaError_t e = cudaGetDevice(&net->device);
    if (e != cudaSuccess) return bail(cuda_fail(e, "cudaGetDevice"));
    e = cudaDeviceGetAttribute(&net->num_sms, cudaDevAttrMultiProcessorCount, net->device);
    if (e != cudaSuccess) return bail(cuda_fail(e, "cudaDeviceGetAttribute"));

    if (dtype == BP_F32) {
        if (f32_max_pg(net->n, net->L) < 1)
            return bail(fail(BP_ESHAPE,
                             "float32 path keeps one pattern's activations and deltas in "
                             "shared memory; these layer sizes need more than 227 KB"));
        {
            std::lock_guard<std::mutex> lk(g_setup_mu);
            if (net->device < 64 && !g_f32_ready[net->device]) {
                e = f32_setup(net->device);
                if (e != cudaSuccess) return bail(cuda_fail(e, "float32 kernel setup"));
                g_f32_ready[net->device] = true;
            }
        }
    } else {
        bp_status st = bf16_check_shape(net->n, net->L, max_batch);
        if (st != BP_OK) return bail(fail(st, "%s", bf16_last_message()));
    }

    // float32 nets keep their parameters in the padded device layout
    if (dtype == BP_F32) {
        f32_layout(net->view, net->n, net->L, max_batch);
        net->Pd = net->view.P;
    }
    const long long Pd = net->Pd;
    e = cudaMalloc(&net->theta, Pd * sizeof(float));
    if (e == cudaSuccess) e = cudaMalloc(&net->V, Pd * sizeof(float));
    if (e == cudaSuccess) e = cudaMalloc(&net->G, Pd * sizeof(float));
    if (e != cudaSuccess) return bail(cuda_fail(e, "cudaMalloc(parameters)"));
    e = cudaMemset(net->theta, 0, Pd * sizeof(float));
    if (e == cudaSuccess) e = cudaMemset(net->V, 0, Pd * sizeof(float));
    if (e == cudaSuccess) e = cudaMemset(net->G, 0, Pd * sizeof(float));
    if (e != cudaSuccess) return bail(cuda_fail(e, "cudaMemset(parameters)"));

    if (dtype == BP_F32) {
        F32View& v = net->view;
        e = cudaMalloc(&net->A, v.a_floats * sizeof(float));
        if (e == cudaSuccess) e = cudaMalloc(&net->D, v.d_floats * sizeof(float));
        if (e == cudaSuccess) e = cudaMalloc(&net->sse_part, (size_t)net->num_sms * 4 * sizeof(float));
        if (e == cudaSuccess) e = cudaMalloc(&net->wpart, (size_t)net->num_sms * 2 * 512 * sizeof(float));
        if (e == cudaSuccess) e = cudaMalloc(&net->bar, (size_t)bp::kBarWords * sizeof(unsigned));
        if (e == cudaSuccess) e = cudaMalloc(&net->flags, 4 * sizeof(int));
        if (e != cudaSuccess) return bail(cuda_fail(e, "cudaMalloc(scratch)"));
        e = cudaMemset(net->bar, 0, (size_t)bp::kBarWords * sizeof(unsigned));
        if (e == cudaSuccess) e = cudaMemset(net->flags, 0, 4 * sizeof(int));
        if (e == cudaSuccess) e = cudaMemset(net->A, 0, v.a_floats * sizeof(float));
        if (e == cudaSuccess) e = cudaMemset(net->D, 0, v.d_floats * sizeof(float));
        if (e != cudaSuccess) return bail(cuda_fail(e, "cudaMemset(scratch)"));
        v.theta = net->theta;
        v.V = net->V;
        v.G = net->G;
        v.A = net->A;
        v.D = net->D;
        v.sse_part = net->sse_part;
        v.wpart = net->wpart;
        v.bar = net->bar;
        v.flags = net->flags;
        v.faults = reinterpret_cast<unsigned*>(net->flags + 1);
        refresh_view(net);
    } else {
        Bf16Net* b = nullptr;
        bp_status st = bf16_create(net->n, net->L, max_batch, net->num_sms, net->theta, net->V,
                                   net->G, &b);
        if (st != BP_OK) return bail(fail(st, "%s", bf16_last_message()));
        net->bf = b;
        e = cudaMalloc(&net->flags, 4 * sizeof(int));
        if (e == cudaSuccess) e = cudaMemset(net->flags, 0, 4 * sizeof(int));
        if (e != cudaSuccess) return bail(cuda_fail(e, "cudaMalloc(flags)"));
        bf16_set_flags(b, net->flags);
    }
    *out = net;
    return BP_OK;
}

void bp_destroy(bp_net* net) {
    if (net == nullptr) return;
    cudaDeviceSynchronize();
    free_all(net);
    delete net;
}

bp_status bp_set_hparams(bp_net* net, float lr, float momentum, float grad_scale) {
    if (net == nullptr) return fail(BP_EINVAL, "NULL net");
    if (!std::isfinite(lr) || !std::isfinite(momentum) || !std::isfinite(grad_scale))
        return fail(BP_EINVAL, "hyper-parameters must be finite");
    net->lr = lr;
    net->momentum = momentum;
    net->grad_scale = grad_scale;
    refresh_view(net);
    return BP_OK;
}

bp_status bp_set_sigmoid(bp_net* net, int mode) {
    if (net == nullptr) return fail(BP_EINVAL, "NULL net");
    if (mode != BP_SIGMOID_LOGISTIC && mode != BP_SIGMOID_TABLE)
        return fail(BP_EINVAL, "unknown sigmoid mode %d", mode);
    if (mode == BP_SIGMOID_TABLE && net->dtype != BP_F32)
        return fail(BP_EINVAL, "the table-lookup sigmoid is implemented for float32 nets only");
    net->view.sig_table = mode == BP_SIGMOID_TABLE ? 1 : 0;
    return BP_OK;
}

bp_status bp_set_guard(bp_net* net, float threshold) {
    if (net == nullptr) return fail(BP_EINVAL, "NULL net");
    if (!(threshold >= 0.f)) return fail(BP_EINVAL, "guard threshold must be >= 0 (0 turns it off)");
    net->view.guard = threshold;
    if (net->bf) bf16_set_guard(net->bf, threshold);
    return BP_OK;
}

bp_status bp_get_faults(bp_net* net, int64_t* count, int reset) {
    if (net == nullptr || count == nullptr) return fail(BP_EINVAL, "NULL argument");
    BP_CUDA(cudaDeviceSynchronize(), "bp_get_faults");
    unsigned c = 0;
    BP_CUDA(cudaMemcpy(&c, net->flags + 1, sizeof(unsigned), cudaMemcpyDeviceToHost), "bp_get_faults");
    *count = (int64_t)c;
    if (reset) BP_CUDA(cudaMemset(net->flags + 1, 0, sizeof(unsigned)), "bp_get_faults");
    return BP_OK;
}

bp_status bp_vote(const float* values, int n, float* mode, int* n_agree) {
    if (values == nullptr || n < 1 || n_agree == nullptr) return fail(BP_EINVAL, "bad argument");
    // the value most CTAs produced, bit for bit (ties: the first such value)
    int best = 0, best_count = 0;
    for (int i = 0; i < n; ++i) {
        int c = 0;
        for (int k = 0; k < n; ++k) c += std::memcmp(&values[i], &values[k], sizeof(float)) == 0;
        if (c > best_count) {
            best = i;
            best_count = c;
        }
    }
    if (mode != nullptr) *mode = values[best];
    *n_agree = best_count;
    return BP_OK;
}

bp_status bp_diagnose(bp_net* net, const void* d_X, const void* d_T, int batch, float* h_sse,
                      int* h_sm, int capacity, int* n_ctas, int* n_agree) {
    if (net == nullptr || d_X == nullptr || d_T == nullptr || n_ctas == nullptr || n_agree == nullptr)
        return fail(BP_EINVAL, "NULL argument");
    if (net->dtype != BP_F32) return fail(BP_EINVAL, "the diagnostic mode is implemented for float32 nets");
    bp_status st = check_batch(net, batch);
    if (st == BP_OK) st = check_align(net, d_X, d_T, nullptr, nullptr);
    if (st != BP_OK) return st;
    const int n = net->num_sms;
    if ((h_sse != nullptr || h_sm != nullptr) && capacity < n)
        return fail(BP_EINVAL, "capacity %d is below the %d CTAs of the launch", capacity, n);
    if (net->diag_sm == nullptr) BP_CUDA(cudaMalloc(&net->diag_sm, n * sizeof(int)), "cudaMalloc(diagnose)");
    BP_CUDA(f32_diagnose(net->view, (const float*)d_X, (const float*)d_T, batch, net->sse_part,
                         net->diag_sm, n, 0),
            "bp_diagnose");
    std::vector<float> sse(n);
    std::vector<int> sm(n);
    BP_CUDA(cudaMemcpy(sse.data(), net->sse_part, n * sizeof(float), cudaMemcpyDeviceToHost), "bp_diagnose");
    BP_CUDA(cudaMemcpy(sm.data(), net->diag_sm, n * sizeof(int), cudaMemcpyDeviceToHost), "bp_diagnose");
    if (h_sse != nullptr) std::memcpy(h_sse, sse.data(), n * sizeof(float));
    if (h_sm != nullptr) std::memcpy(h_sm, sm.data(), n * sizeof(int));
    *n_ctas = n;
    return bp_vote(sse.data(), n, nullptr, n_agree);
}

int64_t bp_num_params(const bp_net* net) { return net ? (int64_t)net->P : 0; }

// Copies a parameter vector between the caller's packed layout (host) and the
// net's device layout (padded for float32 nets).
static bp_status copy_params(const bp_net* net, float* dst, const float* src, bool to_device,
                             const char* what) {
    if (net == nullptr || dst == nullptr || src == nullptr) return fail(BP_EINVAL, "NULL argument");
    BP_CUDA(cudaDeviceSynchronize(), what);
    if (net->dtype != BP_F32) {
        BP_CUDA(cudaMemcpy(dst, src, net->P * sizeof(float),
                           to_device ? cudaMemcpyHostToDevice : cudaMemcpyDeviceToHost),
                what);
        return BP_OK;
    }
    std::vector<float> tmp((size_t)net->Pd);
    if (to_device) {
        f32_pad_host(net->view, src, tmp.data());
        BP_CUDA(cudaMemcpy(dst, tmp.data(), net->Pd * sizeof(float), cudaMemcpyHostToDevice), what);
    } else {
        BP_CUDA(cudaMemcpy(tmp.data(), src, net->Pd * sizeof(float), cudaMemcpyDeviceToHost), what);
        f32_unpad_host(net->view, tmp.data(), dst);
    }
    return BP_OK;
}

bp_status bp_set_weights(bp_net* net, const float* h) {
    if (net == nullptr) return fail(BP_EINVAL, "NULL net");
    bp_status st = copy_params(net, net->theta, h, true, "bp_set_weights");
    if (st != BP_OK) return st;
    if (net->bf) {
        BP_CUDA(bf16_refresh_weights(net->bf, nullptr), "bp_set_weights(bf16 copies)");
        BP_CUDA(cudaDeviceSynchronize(), "bp_set_weights");
    }
    return BP_OK;
}
bp_status bp_get_weights(const bp_net* net, float* h) {
    if (net == nullptr) return fail(BP_EINVAL, "NULL net");
    return copy_params(net, h, net->theta, false, "bp_get_weights");
}
bp_status bp_set_velocity(bp_net* net, const float* h) {
    if (net == nullptr) return fail(BP_EINVAL, "NULL net");
    return copy_params(net, net->V, h, true, "bp_set_velocity");
}
bp_status bp_get_velocity(const bp_net* net, float* h) {
    if (net == nullptr) return fail(BP_EINVAL, "NULL net");
    return copy_params(net, h, net->V, false, "bp_get_velocity");
}
bp_status bp_get_grads(const bp_net* net, float* h) {
    if (net == nullptr) return fail(BP_EINVAL, "NULL net");
    return copy_params(net, h, net->G, false, "bp_get_grads");
}

bp_status bp_forward(bp_net* net, const void* d_X, int batch, void* d_Y, void* stream) {
    if (net == nullptr || d_X == nullptr) return fail(BP_EINVAL, "NULL argument");
    bp_status st = check_batch(net, batch);
    if (st == BP_OK) st = check_align(net, d_X, nullptr, d_Y, nullptr);
    if (st != BP_OK) return st;
    cudaStream_t s = (cudaStream_t)stream;
    if (net->dtype == BP_F32) {
        const F32Plan plan = f32_plan(net->view, batch, net->num_sms);
        BP_CUDA(f32_forward(net->view, (const float*)d_X, batch, (float*)d_Y, plan, s),
                "bp_forward");
    } else {
        BP_CUDA(bf16_forward(net->bf, d_X, batch, d_Y, s), "bp_forward");
    }
    net->fwd_batch = batch;
    net->fwd_X = d_X;
    return BP_OK;
}

bp_status bp_backward(bp_net* net, const void* d_T, int batch, float* d_sse, void* stream) {
    if (net == nullptr || d_T == nullptr) return fail(BP_EINVAL, "NULL argument");
    bp_status st = check_batch(net, batch);
    if (st == BP_OK) st = check_align(net, nullptr, d_T, nullptr, d_sse);
    if (st != BP_OK) return st;
    if (net->fwd_batch == 0) return fail(BP_ESTATE, "bp_backward needs a preceding bp_forward");
    if (net->fwd_batch != batch)
        return fail(BP_ESTATE, "bp_backward batch %d differs from the last forward's %d", batch,
                    net->fwd_batch);
    cudaStream_t s = (cudaStream_t)stream;
    if (net->dtype == BP_F32) {
        const F32Plan plan = f32_plan(net->view, batch, net->num_sms);
        BP_CUDA(f32_backward(net->view, (const float*)net->fwd_X, (const float*)d_T, batch, d_sse,
                             plan, s),
                "bp_backward");   // the forward kept its inputs in scratch
    } else {
        BP_CUDA(bf16_backward(net->bf, net->fwd_X, d_T, batch, d_sse, net->g_dirty, s),
                "bp_backward");
    }
    net->g_dirty = true;
    return BP_OK;
}

bp_status bp_update(bp_net* net, void* stream) {
    if (net == nullptr) return fail(BP_EINVAL, "NULL net");
    cudaStream_t s = (cudaStream_t)stream;
    if (net->dtype == BP_F32) {
        BP_CUDA(f32_update(net->view, net->Pd, s), "bp_update");
    } else {
        BP_CUDA(bf16_update(net->bf, net->lr, net->momentum, net->grad_scale, s), "bp_update");
    }
    net->g_dirty = false;
    return BP_OK;
}

static bp_status run_epoch(bp_net* net, const void* d_X, const void* d_T, int n_patterns,
                           int minibatch, float* d_sse, cudaStream_t s) {
    const int n_steps = (int)(((long long)n_patterns + minibatch - 1) / minibatch);
    if (net->dtype == BP_F32 && !net->g_dirty && f32_small_ok(net->view, minibatch)) {
        // groups of a few patterns: one CTA keeps the weights resident
        BP_CUDA(f32_train_small(net->view, (const float*)d_X, (const float*)d_T, n_patterns,
                                minibatch, n_steps, d_sse, s),
                "training launch");
    } else if (net->dtype == BP_F32) {
        const F32Plan plan = f32_plan(net->view, minibatch, net->num_sms);
        BP_CUDA(f32_train(net->view, (const float*)d_X, (const float*)d_T, n_patterns, minibatch,
                          n_steps, d_sse, net->g_dirty, plan, s),
                "training launch");
    } else {
        BP_CUDA(bf16_train(net->bf, d_X, d_T, n_patterns, minibatch, d_sse, net->lr, net->momentum,
                           net->grad_scale, net->g_dirty, s),
                "training launch");
    }
    net->g_dirty = false;
    net->fwd_batch = 0;
    return BP_OK;
}

bp_status bp_train_batch(bp_net* net, const void* d_X, const void* d_T, int batch, float* d_sse,
                         void* stream) {
    if (net == nullptr || d_X == nullptr || d_T == nullptr) return fail(BP_EINVAL, "NULL argument");
    bp_status st = check_batch(net, batch);
    if (st == BP_OK) st = check_align(net, d_X, d_T, nullptr, d_sse);
    if (st != BP_OK) return st;
    return run_epoch(net, d_X, d_T, batch, batch, d_sse, (cudaStream_t)stream);
}

bp_status bp_train_epoch(bp_net* net, const void* d_X, const void* d_T, int n_patterns,
                         int minibatch, float* d_sse, void* stream) {
    if (net == nullptr || d_X == nullptr || d_T == nullptr) return fail(BP_EINVAL, "NULL argument");
    if (n_patterns < 1) return fail(BP_EINVAL, "n_patterns must be >= 1 (got %d)", n_patterns);
    bp_status st = check_batch(net, minibatch);
    if (st == BP_OK) st = check_align(net, d_X, d_T, nullptr, d_sse);
    if (st != BP_OK) return st;
    return run_epoch(net, d_X, d_T, n_patterns, minibatch, d_sse, (cudaStream_t)stream);
}

bp_status bp_check(bp_net* net, void* stream) {
    if (net == nullptr) return fail(BP_EINVAL, "NULL net");
    cudaStream_t s = (cudaStream_t)stream;
    BP_CUDA(cudaStreamSynchronize(s), "bp_check");
    int flags = 0;
    BP_CUDA(cudaMemcpy(&flags, net->flags, sizeof(int), cudaMemcpyDeviceToHost), "bp_check");
    if (flags == 0) return BP_OK;
    BP_CUDA(cudaMemset(net->flags, 0, sizeof(int)), "bp_check");
    if (net->bar)
        BP_CUDA(cudaMemset(net->bar, 0, (size_t)bp::kBarWords * sizeof(unsigned)), "bp_check");
    if (flags & kFlagTimeout)
        return fail(BP_ETIMEOUT, "a bounded device-side wait ran out; the launch stopped early");
    if (flags & kFlagBounds)
        return fail(BP_ESTATE, "a bounds check of the checked build failed; the phase was skipped");
    return fail(BP_ENONFINITE, "the summed squared error of a group was not finite");
}

bp_status bp_debug_wait_test(bp_net* net, unsigned long long wait_ns, int unreachable) {
    if (net == nullptr) return fail(BP_EINVAL, "NULL net");
    if (net->dtype != BP_F32) return fail(BP_EINVAL, "the wait test hook is for float32 nets");
#ifdef BP_CHECK
    BP_CUDA(cudaDeviceSynchronize(), "bp_debug_wait_test");
    net->view.wait_ns = wait_ns;
    net->view.debug_stall = unreachable == 2 ? 1 : 0;
    if (unreachable == 1) {
        // barrier k of the next launch waits for bar[0] + k * grid arrivals
        unsigned words[2] = {0, 0};
        BP_CUDA(cudaMemcpy(words, net->bar, sizeof words, cudaMemcpyDeviceToHost), "bp_debug_wait_test");
        words[0] = words[1] + 0x40000000u;
        BP_CUDA(cudaMemcpy(net->bar, words, sizeof(unsigned), cudaMemcpyHostToDevice), "bp_debug_wait_test");
    }
    return BP_OK;
#else
    (void)wait_ns;
    (void)unreachable;
    return fail(BP_ESTATE, "bp_debug_wait_test works only in a library built with -DBP_CHECK");
#endif
}

bp_status bp_train_epoch_host(bp_net* net, const void* h_X, const void* h_T, int n_patterns,
                              int minibatch, float* h_sse, void* stream) {
    if (net == nullptr || h_X == nullptr || h_T == nullptr) return fail(BP_EINVAL, "NULL argument");
    if (n_patterns < 1) return fail(BP_EINVAL, "n_patterns must be >= 1 (got %d)", n_patterns);
    bp_status st = check_batch(net, minibatch);
    if (st != BP_OK) return st;
    cudaStream_t s = (cudaStream_t)stream;
    const size_t xb = (size_t)n_patterns * net->n[0] * elem_size(net);
    const size_t tb = (size_t)n_patterns * net->n[net->L] * elem_size(net);
    const size_t ns = (size_t)(((long long)n_patterns + minibatch - 1) / minibatch);
    if (xb > net->stage_x_bytes || tb > net->stage_t_bytes || ns > net->stage_sse_n) {
        BP_CUDA(cudaStreamSynchronize(s), "bp_train_epoch_host");
        if (xb > net->stage_x_bytes) {
            cudaFree(net->stage_X);
            net->stage_X = nullptr;
            net->stage_x_bytes = 0;
            BP_CUDA(cudaMalloc(&net->stage_X, xb), "cudaMalloc(staging)");
            net->stage_x_bytes = xb;
        }
        if (tb > net->stage_t_bytes) {
            cudaFree(net->stage_T);
            net->stage_T = nullptr;
            net->stage_t_bytes = 0;
            BP_CUDA(cudaMalloc(&net->stage_T, tb), "cudaMalloc(staging)");
            net->stage_t_bytes = tb;
        }
        if (ns > net->stage_sse_n) {
            cudaFree(net->stage_sse);
            net->stage_sse = nullptr;
            net->stage_sse_n = 0;
            BP_CUDA(cudaMalloc(&net->stage_sse, ns * sizeof(float)), "cudaMalloc(staging)");
            net->stage_sse_n = ns;
        }
    }
    if (net->copy_stream == nullptr) {
        BP_CUDA(cudaStreamCreateWithFlags(&net->copy_stream, cudaStreamNonBlocking), "copy stream");
        BP_CUDA(cudaEventCreateWithFlags(&net->start_ev, cudaEventDisableTiming), "copy events");
        for (cudaEvent_t& e : net->piece_ev)
            BP_CUDA(cudaEventCreateWithFlags(&e, cudaEventDisableTiming), "copy events");
    }
    // The epoch runs in up to 8 pieces of whole minibatches: the copy of piece
    // k + 1 (on the net's copy stream) overlaps the training of piece k (on the
    // caller's stream), which waits for its own piece only.  Pieces double in
    // size from f = ceil(steps / 128) minibatches (f, 2f, .. 64f, then the rest,
    // at most f), so that only 1/128 of the epoch's copy is exposed and no copy
    // is more than twice the training it hides behind.  The staging buffers may
    // still be read by work queued earlier on the caller's stream.
    BP_CUDA(cudaEventRecord(net->start_ev, s), "copy events");
    BP_CUDA(cudaStreamWaitEvent(net->copy_stream, net->start_ev, 0), "copy events");
    const long long n_steps = (long long)ns;
    const size_t xrow = (size_t)net->n[0] * elem_size(net);
    const size_t trow = (size_t)net->n[net->L] * elem_size(net);
    const long long first = (n_steps + 127) / 128;
    long long step0 = 0;
    for (int k = 0; k < 8 && step0 < n_steps; ++k) {
        const long long steps_k = k == 7 ? n_steps - step0 : std::min(first << k, n_steps - step0);
        const long long p0 = step0 * minibatch;
        const long long np = std::min((long long)n_patterns - p0, steps_k * minibatch);
        char* dx = (char*)net->stage_X + p0 * xrow;
        char* dt = (char*)net->stage_T + p0 * trow;
        BP_CUDA(cudaMemcpyAsync(dx, (const char*)h_X + p0 * xrow, np * xrow, cudaMemcpyHostToDevice,
                                net->copy_stream),
                "copy X");
        BP_CUDA(cudaMemcpyAsync(dt, (const char*)h_T + p0 * trow, np * trow, cudaMemcpyHostToDevice,
                                net->copy_stream),
                "copy T");
        BP_CUDA(cudaEventRecord(net->piece_ev[k], net->copy_stream), "copy events");
        BP_CUDA(cudaStreamWaitEvent(s, net->piece_ev[k], 0), "copy events");
        st = run_epoch(net, dx, dt, (int)np, minibatch, net->stage_sse + step0, s);
        if (st != BP_OK) return st;
        step0 += steps_k;
    }
    if (h_sse != nullptr)
        BP_CUDA(cudaMemcpyAsync(h_sse, net->stage_sse, ns * sizeof(float), cudaMemcpyDeviceToHost, s),
                "copy error sums");
    return bp_check(net, stream);
}

}  // extern "C"

namespace bp {
// Lets other translation units report a message through bp_last_error().
void set_error_message(const char* msg) { g_err = msg; }

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
    static std::once_flag once;
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    std::call_once(once, [] {
        cudaDriverEntryPointQueryResult q;
        void* p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}
}  // namespace bp
