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
// One module's operands of the refresh products on tensor cores.
struct TcProdItem {
    const uint16_t* Vhi;   // m x n bf16 (V, or G when the refresh source is G)
    const uint16_t* Vlo;   // m x n bf16 residual, or null when Vhi is exact
    const uint16_t* Qbf;   // m x l bf16 (op 0)
    const uint16_t* Zbf;   // n x l bf16 (op 1)
    float* out;            // n x l (op 0) or m x l (op 1), fp32
    int m, n, l;
};

// op 0: out = V^T Qbf;  op 1: out = V Zbf.  Requires n % 8 == 0 and l % 8 == 0
// (TMA row pitch) and 16-byte aligned planes.
int tc_refresh_products(TcState* st, int op, const TcProdItem* items, int count, cudaStream_t s,
                        int64_t* launches);

// V = Decompose(G, B) direction as two bf16 planes (V_hi, V_lo) for the
// refresh products; G bf16 m x n, B in {8, ..., 128}.
struct TcSplitItem {
    const void* G;
    uint16_t* Vhi;
    uint16_t* Vlo;
    int m, n;
};
int tc_split_v(TcState* st, const TcSplitItem* items, int count, int B, float decomp_eps, cudaStream_t s,
               int64_t* launches);

const char* tc_last_error(const TcState* st);

}  // namespace moara
