// Internal declarations shared by the host API and the kernel translation
// units of libmoara.  Plain C++ structs passed to kernels by value (grouped
// launches) or stored in the context's device table.
#pragma once

#include <cstddef>
#include <cstdint>

#include <cuda_runtime.h>

#include "../../include/moara.h"

namespace moara {

// Largest number of problems a grouped launch carries in its parameter block
// (kernel parameters up to 32 KB are allowed on sm_70+ with CUDA >= 12.1).
constexpr int kMaxGroup = 224;

// Device-side image of one registered module.
struct ModDev {
    int m, n, r, kb;        // kb = ceil(n / B)
    int dtype;              // MOARA_DTYPE_*
    int right;              // 1: right projector Q (n x r) in P / Pb, moments m x r
    float* W;
    float* P;
    uint16_t* Pb;
    float* exp_avg;
    float* exp_avg_sq;
    float* mag_avg;
    float* mag_avg_sq;
    float* ws_N;            // r x n update of the direction branch (fp32 or bf16)
    float* ws_dM;           // m x kb update of the magnitude branch
    float* ws_inv;          // m x kb inverse block scales 1 / (||g|| + eps)
    uint16_t* ws_Vhi;       // m x n direction matrix V in bf16 (tensor-core path)
    uint16_t* ws_Vlo;       // m x n bf16 residual V - V_hi (first Adam step)
    uint16_t* ws_Qt;        // r x n bf16 transpose of a right projector (tall modules), or null
};

// Workspace carve-up of one module (byte offsets, 256-byte aligned).
struct WsLayout {
    size_t off_N, off_dM, off_inv, off_Vhi, off_Vlo, off_Qt, total;   // off_Qt = 0: none
};
WsLayout workspace_layout(int m, int n, int r, int B);

// ---------------------------------------------------------------- decompose
struct DecompItem {
    const void* G;
    float* inv;       // m x kb, written
    float* mag_avg;   // m x kb, updated when do_mag
    float* mag_avg_sq;
    float* dM;        // m x kb, written when do_mag
    int m, n, kb, dtype;
};

struct DecompBatch {
    int count;
    int B;
    int do_mag;
    float decomp_eps, beta1, beta2, adam_eps, bc1, bc2;
    const float* clip;    // gradient clipping coefficient (device), applied to M before Optimizer_M, or null
    long long item_start[kMaxGroup + 1];
    DecompItem p[kMaxGroup];
};

// ------------------------------------------------------------- SIMT GEMM
// C (M x N) = op(A) (M x K) * op(B) (K x N), fp32 accumulate.
enum Epi { EPI_STORE = 0, EPI_ADAM = 1, EPI_UPDATE = 2, EPI_STORE_NEG = 3, EPI_SUB = 4 };

// Triangular operands of the SIMT GEMM (zeros stored explicitly): the K loop
// of an output tile at (m0, n0) covers only the range that can be nonzero.
enum KTri {
    KTRI_NONE = 0,
    KTRI_B_UPPER = 1,     // B[k][j] = 0 for k > j:  k < n0 + tile width
    KTRI_B_LOWER = 2,     // B[k][j] = 0 for k < j:  k >= n0
    KTRI_A_LOWER = 3,     // A[i][k] = 0 for k > i:  k < m0 + tile height
};

struct GemmProb {
    const void* A;
    const void* Bm;
    float* C;
    const float* a_inv;   // block scales applied to A (V operand) or null
    const float* b_inv;   // block scales applied to B or null
    float* aux0;          // EPI_ADAM: exp_avg    EPI_UPDATE: W
    float* aux1;          // EPI_ADAM: exp_avg_sq
    const float* aux2;    // EPI_UPDATE: dM (m x kb) or null (no magnitude)
    int M, N, K;
    int lda, ldb, ldc;
    int kb;               // blocks per row of the scaled operand / of dM
    int a_bf16, b_bf16;
    int lower_only;       // skip output tiles strictly above the diagonal
    int k_tri;            // triangular operand: the K range of an output tile shrinks (KTRI_*)
    uint16_t* c_bf16;     // EPI_STORE: also write C rounded to bf16 here (same layout), or null
};

struct GemmBatch {
    int count;
    int B;                        // block size (scales, dM repetition)
    int log2B;                    // log2(B) when B is a power of two, else -1 (set at launch)
    float beta1, beta2, adam_eps, bc1, bc2;
    float step_scale;             // lr * alpha (EPI_UPDATE)
    const float* clip;            // EPI_ADAM: clipping coefficient (device) applied to R, or null
    int tiles_n[kMaxGroup];
    int tile_start[kMaxGroup + 1];
    GemmProb p[kMaxGroup];
};

// Operand layouts of the SIMT GEMM.
//   A: KCONTIG  A[i][k] = A[i*lda + k];  MCONTIG  A[i][k] = A[k*lda + i]
//   B: NCONTIG  B[k][j] = B[k*ldb + j];  KCONTIG  B[k][j] = B[j*ldb + k]
enum ALayout { A_KCONTIG = 0, A_MCONTIG = 1 };
enum BLayout { B_NCONTIG = 0, B_KCONTIG = 1 };

struct GemmKind {
    int a_layout, b_layout, a_scale, b_scale, a_bf16, b_bf16, epi;
    int narrow = 0;       // 128 x 64 output tiles, four CTAs per SM (plain fp32 operands, short K)
};

// Host launchers (return cudaError_t of the launch).
cudaError_t launch_decompose(const DecompBatch& b, cudaStream_t s, int64_t* launches);
cudaError_t launch_gemm(const GemmKind& kind, GemmBatch& b, cudaStream_t s, int64_t* launches);
int gemm_tile_m();
int gemm_tile_n();

cudaError_t launch_f32_to_bf16(const float* src, float* dst_f32, uint16_t* dst_bf16,
                               long long count, cudaStream_t s, int64_t* launches);

// ------------------------------------------------------- gradient clipping
// Sum of squared gradient entries over a group of gradients, in chunks of
// kNormChunk elements; chunk c goes to CTA c % kNormParts of the launch, so
// the partial sums (one double per CTA) and their total are reproducible.
constexpr int kNormChunk = 16384;
constexpr int kNormParts = 1216;

struct GradNormBatch {
    int count;
    long long chunk_start[kMaxGroup + 1];
    const void* G[kMaxGroup];
    long long elems[kMaxGroup];
    int dtype[kMaxGroup];
};

cudaError_t launch_grad_sq(const GradNormBatch& b, double* partials, cudaStream_t s, int64_t* launches);
// state[0] = sqrt(sum of partials[0..n) + *extra), state[1] = min(1, max_norm / (state[0] + 1e-6))
cudaError_t launch_clip_finish(const double* partials, int n, const float* extra, float max_norm, float* state,
                               cudaStream_t s, int64_t* launches);

// ------------------------------------------------------------- refresh
struct RefreshItem {
    int m, n, r, l, kb, dtype;
    const void* G;
    float* inv;       // block scales (src V) or null (src G)
    float* Omega;     // n x l
    float* Qa; float* Qb;   // m x l
    float* Za; float* Zb;   // n x l
    float* Cg;        // l x l Gram / Cholesky factor
    float* Tt;        // l x l temporary of the blocked triangular inverse
    float* scal;      // per-problem scalars (diagonal shift)
    float* Linv;      // l x l
    float* Cr;        // l x l Rayleigh-Ritz matrix
    float* Xa; float* Xb;   // l x l
    float* ritz;      // l
    int* perm;        // l
    int* fail;        // 1 int
    float* P;         // m x r destination
    uint16_t* Pb;     // m x r bf16 destination (may be null)
    uint64_t key;     // RNG key (seed, module, refresh count)
    int tc;           // products with V on tensor cores
    int trans;        // right projector: the refresh runs on V^T (m, n above are V's n, m)
    const uint16_t* Vhi;    // m x n bf16 planes of V (or G) for the tensor-core products
    uint16_t* Vhi_w;        // writable view of Vhi when V is formed here (null otherwise)
    uint16_t* Vlo;          // residual plane, or null when Vhi is exact
    uint16_t* Qbf;    // m x l bf16 copy of the latest orthonormal Q
    uint16_t* Zbf;    // n x l bf16 copy of the latest Z (or of Omega)
    uint16_t* Cp;     // 3 x l x l bf16 planes of the Rayleigh-Ritz matrix
    uint16_t* P1;     // 3 x l x l planes of X / W / W^T
    uint16_t* P2;     // 3 x l x l planes of Linv^T
};

size_t refresh_ws_bytes(int m, int n, int r, int l, int B, int src_v);
void refresh_carve(RefreshItem& it, void* base, int m, int n, int r, int l, int B, int src_v);

// Small dense kernels (one CTA per problem).
struct SmallBatch {
    int count;
    int l[kMaxGroup];
    int rows[kMaxGroup];
    float* a[kMaxGroup];
    float* b[kMaxGroup];
    float* c[kMaxGroup];
    int* fail[kMaxGroup];
    int* iaux[kMaxGroup];
    uint16_t* h[kMaxGroup];
    int ld[kMaxGroup];    // row pitch of a (split3), 0: l
    float shift_rel;      // diagonal shift: shift_rel * sqrt(rows) * trace
    uint64_t key[kMaxGroup];
};

cudaError_t launch_philox_gaussian(const SmallBatch& b, cudaStream_t s, int64_t* launches);
// Inverts the diagonal blocks [64j, 64j+64) of each lower-triangular a into c.
constexpr int kTriBase = 64;
cudaError_t launch_tri_inverse_diag(const SmallBatch& b, cudaStream_t s, int64_t* launches);
// Blocked Cholesky pieces: the diagonal shift shift_rel*sqrt(rows)*trace(a)
// into b[0]; and the factorisation of the diagonal block starting at j0
// (a: matrix, b: shift, c: inverse of the factor's block, written in place).
cudaError_t launch_trace_shift(const SmallBatch& b, cudaStream_t s, int64_t* launches);
cudaError_t launch_chol_diag(const SmallBatch& b, int j0, cudaStream_t s, int64_t* launches);
cudaError_t launch_set_identity(const SmallBatch& b, cudaStream_t s, int64_t* launches);
cudaError_t launch_ritz_sort(const SmallBatch& b, cudaStream_t s, int64_t* launches);
// Exact Rayleigh-Ritz (Jacobi) on the leading min(64, l) columns of X (a)
// with W = C X (b): both rotated in place by the eigenvectors of X_w^T W_w.
cudaError_t launch_lead_ritz(const SmallBatch& b, cudaStream_t s, int64_t* launches);
cudaError_t launch_gather_cols(const SmallBatch& b, cudaStream_t s, int64_t* launches);
cudaError_t launch_sign_fix_store(const SmallBatch& b, cudaStream_t s, int64_t* launches);
cudaError_t launch_transpose_bf16(const SmallBatch& b, cudaStream_t s, int64_t* launches);  // h = bf16(a^T)
// three bf16 planes (hi, mid, lo) of a (rows x l) at h, or of its transpose
cudaError_t launch_split3(const SmallBatch& b, int transpose, cudaStream_t s, int64_t* launches);

}  // namespace moara
