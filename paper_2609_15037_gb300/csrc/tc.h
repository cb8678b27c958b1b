// Tensor-core (tcgen05 / TMEM / TMA) path of the step for bf16 gradients.
#pragma once

#include "internal.h"

namespace moara {

struct TcState;

// Whether a module of this shape can run on the tensor-core kernels.
bool tc_supported(int m, int n, int r, int B, int dtype, int decompose);

// Hook used to time the tensor-core launches with CUDA events.
struct TcProfile {
    bool on;
    void (*mark)(void* ctx, int phase, cudaStream_t s, bool begin);
    void* ctx;
};

TcState* tc_create(int device, int* d_status);
void tc_destroy(TcState* st);
int tc_register(TcState* st, int id, const ModDev& md, const moara_hparams& hp);
int tc_step(TcState* st, const moara_hparams& hp, int n_mod, const int* ids, const void* const* G,
            float bc1, float bc2, float lr, int first_step, cudaStream_t s, int64_t* launches,
            const TcProfile& prof);
const char* tc_last_error(const TcState* st);

}  // namespace moara
