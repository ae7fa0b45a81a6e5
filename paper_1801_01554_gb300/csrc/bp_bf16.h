// bfloat16 tensor-core path of libbp.so (tcgen05 + TMA GEMMs with fused
// back-propagation epilogues).  Internal interface used by bp_api.cu.
#pragma once

#include <cuda_runtime.h>

#include "bp.h"

namespace bp {

struct Bf16Net;

// Shape rules of the path; on failure bf16_last_message() says why.
bp_status bf16_check_shape(const int* n, int L, int max_batch);
const char* bf16_last_message();

// theta, V, G: the net's float32 master vectors (owned by the caller).
bp_status bf16_create(const int* n, int L, int max_batch, int num_sms, float* theta, float* V,
                      float* G, Bf16Net** out);
void bf16_destroy(Bf16Net* b);
void bf16_set_flags(Bf16Net* b, int* flags);   // flags[0] error bits, flags[1] fault count
void bf16_set_guard(Bf16Net* b, float guard);  // fault guard of Section 8 (0: off)

// Rewrite the bfloat16 weight copies from the float32 master weights.
cudaError_t bf16_refresh_weights(Bf16Net* b, cudaStream_t s);
cudaError_t bf16_forward(Bf16Net* b, const void* X, int batch, void* Y, cudaStream_t s);
cudaError_t bf16_backward(Bf16Net* b, const void* X, const void* T, int batch, float* sse,
                          bool g_dirty, cudaStream_t s);
cudaError_t bf16_update(Bf16Net* b, float lr, float momentum, float grad_scale, cudaStream_t s);
cudaError_t bf16_train(Bf16Net* b, const void* X, const void* T, int n_patterns, int minibatch,
                       float* sse, float lr, float momentum, float grad_scale, bool g_dirty,
                       cudaStream_t s);

}  // namespace bp
