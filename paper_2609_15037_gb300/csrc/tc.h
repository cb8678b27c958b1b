// Tensor-core (tcgen05 / TMEM / TMA) path of the step for bf16 gradients.
#pragma once

#include "internal.h"

namespace moara {

struct TcState;

// Whether a module of this shape can run on the tensor-core kernels.
bool tc_supported(int m, int n, int r, int B, int dtype, int decompose, int state_dtype);

// Hook used to time the tensor-core launches with CUDA events.
struct TcProfile {
    bool on;
    void (*mark)(void* ctx, int phase, cudaStream_t s, bool begin);
    void* ctx;
};

TcState* tc_create(int device, int* d_status);
void tc_destroy(TcState* st);
int tc_register(TcState* st, int id, const ModDev& md, const moara_hparams& hp);
// Global-norm clipping computed inside the step from the decomposition's
// block norms (no extra pass over G): the step writes {norm, coefficient} to
// state after every module's decomposition and before Optimizer_M.
struct TcClipFuse {
    float* state;           // device {total norm, coefficient}
    double* partials;       // device scratch of kNormParts doubles
    const float* extra;     // device sum of squares of other gradients, or null
    float max_norm;
};
// Largest number of modules one fused-clipping step takes.
int tc_group_limit();

// clip: device clipping coefficient of this step's gradients, or null;
// fuse: clipping from the block norms (decomposition on, at most
// tc_group_limit() modules), or null
int tc_step(TcState* st, const moara_hparams& hp, int n_mod, const int* ids, const void* const* G,
            float bc1, float bc2, float lr, int first_step, const float* clip, const TcClipFuse* fuse,
            cudaStream_t s, int64_t* launches, const TcProfile& prof);
// One problem of the refresh GEMM on tensor cores: out = op(A) B, bf16
// operands, fp32 accumulation.
struct TcGemmItem {
    const uint16_t* A;     // K-major: M x K row-major;  MN-major: K x M row-major
    const uint16_t* A_lo;  // residual plane of A in the same layout, or null
    const uint16_t* B;     // K x N row-major
    float* out;            // M x N row-major fp32, or null
    uint16_t* out_bf16;    // M x N row-major bf16, or null
    int M, N, K;
    int ktri;              // B upper triangular: column j needs k <= j only
    uint16_t* out_lo;      // M x N row-major bf16 residual out - bf16(out), or null
    int lower;             // 1: only output tiles on or below the diagonal (M = N)
};

// Grouped launch of TcGemmItems (A read K-major when a_kmajor, else
// MN-major).  A's row pitch (K or M) and N must be multiples of 8 and every
// plane 16-byte aligned; returns MOARA_ERR_UNSUPPORTED otherwise.
int tc_gemm_bf16(TcState* st, int a_kmajor, const TcGemmItem* items, int count, cudaStream_t s,
                 int64_t* launches);

// Alignment diagnostic S(W, t) = cos(G, Rep_B(M) (.) (P P^T V)) of §3.2 for
// modules on the tensor-core path (bf16 G, B in {8, ..., 128}); uses each
// module's workspace as scratch and writes S for module q to S_out[q]
// (device).  acc: device scratch of 3 * n_mod doubles.
int tc_alignment(TcState* st, const moara_hparams& hp, int n_mod, const int* ids, const void* const* G,
                 float* S_out, double* acc, cudaStream_t s, int64_t* launches);

// One problem of the split-precision GEMM: out (M x N fp32) = A B with A
// stored K x M and B stored K x N, each as three consecutive bf16 planes
// (hi, mid, lo; plane strides a_plane / b_plane elements) whose sum is the
// fp32 operand.
struct TcSplitGemmItem {
    const uint16_t* A;
    const uint16_t* B;
    size_t a_plane, b_plane;
    float* out;
    int M, N, K;
    int ktri;              // B upper triangular: column j needs k <= j only
    int ldo;               // row pitch of out (elements); 0: N
    int sub;               // 1: out -= A B instead of out = A B
    int lower;             // 1: only output tiles on or below the diagonal
};

// Grouped launch; M and N multiples of 8, planes 16-byte aligned.
// planes = 3: hi + mid + lo (fp32-accurate); planes = 2: hi + mid only
// (16 significant bits, three products per k-step).
int tc_gemm_split3(TcState* st, const TcSplitGemmItem* items, int count, int planes, cudaStream_t s,
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

// out (cols x rows, bf16) = in^T for in (rows x cols, bf16, row-major)
cudaError_t tc_transpose_bf16(const uint16_t* in, uint16_t* out, int rows, int cols, cudaStream_t s,
                              int64_t* launches);

const char* tc_last_error(const TcState* st);

// Clock cycles a bounded wait of the refresh / alignment product kernels (KR,
// KS) spins before it gives up and records MOARA_ERR_DEVICE_TIMEOUT; <= 0
// restores the default (~2 s).
void tc_set_wait_limit(TcState* st, long long cycles);

}  // namespace moara
