// bp_train_epoch_noalloc: the float32 training launch for callers that cannot
// allocate device memory.
//
// Some callers cannot call cudaMalloc at all: code running inside a captured
// region of a host framework that owns the allocator, memory-budgeted
// processes whose device memory was handed out up front, or plug-ins that may
// only touch buffers given to them.  This entry point takes every input and
// output from the caller and keeps its scratch (activations, deltas, per-CTA
// error sums, the grid barrier and the error word) in one file-scope device
// array of fixed size instead of allocating it.
#include <cuda_runtime.h>

#include <cstdio>
#include <mutex>

#include "bp.h"
#include "bp_internal.h"

namespace bp {
namespace {

// 8 MiB of scratch.  Every GPU that loads the library holds this array until
// the process exits; every call on a device shares it.
constexpr size_t kNoallocScratchBytes = 8u << 20;
constexpr size_t kNoallocScratchFloats = kNoallocScratchBytes / sizeof(float);

static __device__ __align__(256) float g_noalloc_scratch[kNoallocScratchFloats];

constexpr int kMaxDevices = 64;
std::mutex g_noalloc_mu;
float* g_scratch_addr[kMaxDevices];   // device address of the array, per device
int g_scratch_sms[kMaxDevices];

// Once per device, with that device current: the array's device address (the
// host-side name is only a stand-in) and the kernels' shared-memory limits.
bp_status noalloc_setup(int dev, float** addr, int* sms) {
    std::lock_guard<std::mutex> lk(g_noalloc_mu);
    if (g_scratch_addr[dev] == nullptr) {
        float* p = nullptr;
        cudaError_t e = cudaGetSymbolAddress((void**)&p, g_noalloc_scratch);
        if (e != cudaSuccess || p == nullptr) {
            set_error_message("bp_train_epoch_noalloc: cudaGetSymbolAddress of the static scratch failed");
            return BP_ECUDA;
        }
        int n = 0;
        e = cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
        if (e == cudaSuccess) e = f32_setup(dev);
        if (e != cudaSuccess) {
            set_error_message("bp_train_epoch_noalloc: device set-up failed");
            return BP_ECUDA;
        }
        g_scratch_sms[dev] = n;
        g_scratch_addr[dev] = p;
    }
    *addr = g_scratch_addr[dev];
    *sms = g_scratch_sms[dev];
    return BP_OK;
}

}  // namespace
}  // namespace bp

using namespace bp;

extern "C" bp_status bp_train_epoch_noalloc(const int* layer_sizes, int n_layers, float lr,
                                            float momentum, float grad_scale, float* d_theta,
                                            float* d_V, const float* d_X, const float* d_T,
                                            int n_patterns, int minibatch, float* d_sse,
                                            int* d_status, void* stream) {
    char msg[256];
    if (layer_sizes == nullptr || d_theta == nullptr || d_V == nullptr || d_X == nullptr ||
        d_T == nullptr) {
        set_error_message("bp_train_epoch_noalloc: NULL argument");
        return BP_EINVAL;
    }
    if (n_layers < 2 || n_layers > BP_MAX_SIZES) {
        set_error_message("bp_train_epoch_noalloc: n_layers out of range");
        return BP_EINVAL;
    }
    for (int l = 0; l < n_layers; ++l)
        if (layer_sizes[l] < 1) {
            set_error_message("bp_train_epoch_noalloc: layer sizes must be >= 1");
            return BP_EINVAL;
        }
    if (n_patterns < 1 || minibatch < 1) {
        set_error_message("bp_train_epoch_noalloc: n_patterns and minibatch must be >= 1");
        return BP_EINVAL;
    }
    // the kernels read and write these as float32 words (4-byte cp.async for
    // the pattern rows): refuse a misaligned pointer before any CUDA call
    {
        const void* p[6] = {d_theta, d_V, d_X, d_T, d_sse, d_status};
        const char* what[6] = {"d_theta", "d_V", "d_X", "d_T", "d_sse", "d_status"};
        for (int k = 0; k < 6; ++k)
            if (((uintptr_t)p[k] & 3u) != 0) {
                snprintf(msg, sizeof msg, "bp_train_epoch_noalloc: %s must be 4-byte aligned", what[k]);
                set_error_message(msg);
                return BP_EINVAL;
            }
    }
    const int L = n_layers - 1;
    if (f32_max_pg(layer_sizes, L) < 1) {
        set_error_message("bp_train_epoch_noalloc: one pattern's activations do not fit in shared memory");
        return BP_ESHAPE;
    }
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
        set_error_message("bp_train_epoch_noalloc: no usable current device");
        return BP_ECUDA;
    }
    float* base = nullptr;
    int sms = 0;
    bp_status st = noalloc_setup(dev, &base, &sms);
    if (st != BP_OK) return st;

    // scratch layout (floats, each part 16-byte aligned):
    // [error word, pad][barrier words][per-CTA error sums, padded]
    // [weights, padded layout][weight changes, padded layout][activation rows][delta rows]
    F32View v{};
    const long long soff = f32_layout(v, layer_sizes, L, minibatch);
    const long long bar_words = kBarWords;
    const long long head = 4 + bar_words + (((long long)sms + 3) & ~3LL) + 2 * v.P;
    const long long need = head + soff;
    if (need > (long long)kNoallocScratchFloats) {
        snprintf(msg, sizeof msg,
                 "bp_train_epoch_noalloc: these sizes and minibatch %d need %lld bytes of scratch; "
                 "the static scratch holds %zu bytes (use a smaller minibatch)",
                 minibatch, need * 4, kNoallocScratchBytes);
        set_error_message(msg);
        return BP_EINVAL;
    }
    v.flags = reinterpret_cast<int*>(base);
    v.faults = reinterpret_cast<unsigned*>(base + 1);   // the guard stays off here
    v.bar = reinterpret_cast<unsigned*>(base + 4);
    v.sse_part = base + 4 + bar_words;
    float* theta_pad = base + 4 + bar_words + (((long long)sms + 3) & ~3LL);
    float* V_pad = theta_pad + v.P;
    v.A = base + head;
    v.D = base + head + v.a_floats;
    // the kernel works on padded copies of the caller's (packed) weights and
    // weight changes, copied back when it is done
    v.theta = theta_pad;
    v.V = V_pad;
    v.G = nullptr;   // nothing pending: the launch never reads G
    v.lr = lr;
    v.momentum = momentum;
    v.grad_scale = grad_scale;

    cudaStream_t s = (cudaStream_t)stream;
    // the array keeps the last call's contents: the error word and the barrier
    // must start at zero
    cudaError_t e = cudaMemsetAsync(base, 0, (size_t)(4 + bar_words) * sizeof(float), s);
    if (e == cudaSuccess) e = f32_pad_device(v, d_theta, theta_pad, s);
    if (e == cudaSuccess) e = f32_pad_device(v, d_V, V_pad, s);
    if (e == cudaSuccess) {
        const F32Plan plan = f32_plan(v, minibatch, sms);
        const int n_steps = (int)(((long long)n_patterns + minibatch - 1) / minibatch);
        e = f32_train(v, d_X, d_T, n_patterns, minibatch, n_steps, d_sse, false, plan, s);
    }
    if (e == cudaSuccess) e = f32_unpad_device(v, theta_pad, d_theta, s);
    if (e == cudaSuccess) e = f32_unpad_device(v, V_pad, d_V, s);
    if (e == cudaSuccess && d_status != nullptr)
        e = cudaMemcpyAsync(d_status, base, sizeof(int), cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) {
        snprintf(msg, sizeof msg, "bp_train_epoch_noalloc: %s", cudaGetErrorString(e));
        set_error_message(msg);
        return BP_ECUDA;
    }
    return BP_OK;
}
