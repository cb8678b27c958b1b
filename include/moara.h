/*
 * moara.h -- C ABI of the MoARa-on-GaLore projected-Adam optimizer step for
 * NVIDIA GB300 (sm_103a).
 *
 * The library implements the training-phase body of Algorithm 1 of the paper
 * ("Overall procedure of MoARa") for every registered 2-D weight:
 *
 *   M, V   <- Decompose(G, B)                 (§3.1; Appendix B.1)
 *   P      <- TruncatedSVD(V, r)  every T steps (Algorithm 1; T = 200, App. D.2)
 *   Vt     <- P^T V ; dVt <- Adam(Vt) ; dV <- P dVt      (Algorithm 1)
 *   dM     <- Adam(M)                                    (Algorithm 1; App. D.2)
 *   W      <- W - lr * alpha * (Rep_B(dM) (.) dV)        (Algorithm 1; §3.1)
 *
 * plus the helpers of the setup phase (Phase 3 rank reallocation, §3.2) and
 * the optimizer-state memory model (Appendix G).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - Matrices are dense row-major.  A weight W is m x n in PyTorch nn.Linear
 *   (out, in) order; blocks of B contiguous columns run along each row
 *   (Appendix B.1), k = ceil(n / B) blocks per row.
 * - "device pointer" means memory of the CUDA device the context was created
 *   on; the caller allocates and owns every such buffer.  The library only
 *   allocates a small context-owned table (module descriptors, a device status
 *   word), in moara_create.
 * - Work is enqueued asynchronously on the caller's stream (a cudaStream_t
 *   passed as void*; NULL is the legacy default stream).  Apart from
 *   moara_get_device_status, no entry point synchronizes with the device.
 * - Every function returns MOARA_OK (0) or a negative MOARA_ERR_* code.  On
 *   an error nothing has been enqueued and the context state is unchanged;
 *   moara_last_error() describes the first failed check.
 * - bf16 data is passed as raw 16-bit patterns (uint16_t storage).
 */
#ifndef MOARA_H_
#define MOARA_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes ------------------------------------------------------ */
#define MOARA_OK                   0
#define MOARA_ERR_INVALID_ARG     -1  /* null pointer, bad enum, bad scalar      */
#define MOARA_ERR_SHAPE           -2  /* m, n < 1, B < 1, T < 1, size overflow    */
#define MOARA_ERR_RANK            -3  /* r < 1 or r > min(m, n)                  */
#define MOARA_ERR_ALIGN           -4  /* device pointer not 16-byte aligned       */
#define MOARA_ERR_UNKNOWN_MODULE  -5  /* module id not registered in the context  */
#define MOARA_ERR_CUDA            -6  /* a CUDA runtime call failed               */
#define MOARA_ERR_DEVICE_TIMEOUT  -7  /* a bounded device-side wait ran out       */
#define MOARA_ERR_WORKSPACE       -8  /* workspace missing or too small           */
#define MOARA_ERR_UNSUPPORTED     -9  /* valid request the library cannot serve   */

/* ---- enums ------------------------------------------------------------- */
#define MOARA_PROJ_LEFT    0
#define MOARA_PROJ_SMALLER 1

#define MOARA_DTYPE_F32    0   /* 32-bit IEEE float gradient                     */
#define MOARA_DTYPE_BF16   1   /* bfloat16 gradient                              */

#define MOARA_REFRESH_SRC_V  0 /* SVD of the direction matrix V (Algorithm 1)   */
#define MOARA_REFRESH_SRC_G  1 /* SVD of the raw gradient G (plain GaLore)      */

#define MOARA_PREC_AUTO     0  /* bf16 tensor cores for bf16 G, fp32 otherwise  */
#define MOARA_PREC_FP32     1  /* every product in fp32 FMA (SIMT)              */
#define MOARA_PREC_BF16_TC  2  /* bf16 operands, fp32 accumulate (tcgen05)      */

#define MOARA_DRULE_N      0   /* d_W = n  (left projector, state r x n)        */
#define MOARA_DRULE_MAX    1   /* d_W = max(m, n) (smaller side projected)      */

/* Module types in Algorithm 1's order; bit i of a mask selects type i. */
#define MOARA_MOD_Q     0
#define MOARA_MOD_K     1
#define MOARA_MOD_V     2
#define MOARA_MOD_O     3
#define MOARA_MOD_GATE  4
#define MOARA_MOD_UP    5
#define MOARA_MOD_DOWN  6

/* ---- hyper-parameters (Algorithm 1 "Require"; Appendix D.2) ------------- */
typedef struct moara_hparams {
    float beta1;            /* Adam beta1 (0.9, App. D.2)                         */
    float beta2;            /* Adam beta2 (0.999)                                 */
    float adam_eps;         /* Adam eps (1e-6), added to sqrt(v_hat)             */
    float decomp_eps;       /* eps of the block normalisation (1e-12, App. B.1)  */
    float scale;            /* GaLore scale alpha (0.25, App. D.2)               */
    int   block_size;       /* B >= 1 (§3.1; 32/64/128 by model scale)           */
    int   refresh_interval; /* T_SVD >= 1 (200)                                  */
    int   decompose;        /* 1: MoARa decomposition; 0: plain GaLore step      */
    int   refresh_src;      /* MOARA_REFRESH_SRC_V (default) or _G               */
    int   oversample;       /* p >= 0: extra sketch columns of the refresh       */
    int   power_iters;      /* q >= 0: power iterations of the refresh           */
    int   ritz_iters;       /* orthogonal iterations of the Rayleigh-Ritz stage  */
    int   precision;        /* MOARA_PREC_*                                      */
    uint64_t seed;          /* key of the refresh's Gaussian test matrix         */
    float clip_norm;        /* global-norm gradient clipping threshold (App. D.2:
                               1.0 for the 7B runs); <= 0 (default): off.  A step
                               with clipping scales every gradient of the call by
                               min(1, clip_norm / (||G||_total + 1e-6)), where
                               ||G||_total^2 sums the squared entries of all the
                               call's gradients plus the optional extra term of
                               moara_set_clip_extra (torch.nn.utils.clip_grad_norm_). */
    int   state_dtype;      /* MOARA_DTYPE_F32 (default): W and the direction
                               moments in fp32; MOARA_DTYPE_BF16: both in bf16
                               (the paper's runs keep 2-byte states and apply
                               the update to bf16 weights, App. D.2 / App. G),
                               updated in fp32 and stored rounded to nearest
                               even; tensor-core modules only (bf16 G, B >= 32);
                               the magnitude moments stay fp32. */
    int   proj_rule;        /* MOARA_PROJ_LEFT (default): projector P (m x r) on
                               the left of every weight; MOARA_PROJ_SMALLER:
                               GaLore's rule, a right projector Q (n x r) for
                               tall weights (m > n), R = V Q (m x r), dV = N Q^T;
                               tensor-core modules only (the paper's memory
                               model counts r * max(m, n) state entries, App. G). */
} moara_hparams;

/* One registered weight.  All pointers are device pointers, 16-byte aligned,
 * owned by the caller, and must stay valid while the module is registered.
 *   W           m x n  fp32, updated in place by moara_step_grouped
 *   P           m x r  fp32 projector with orthonormal columns (written by the
 *               refresh or by moara_load_projector)
 *   P_bf16      m x r  bf16 copy of P used as tensor-core operand; may be NULL
 *               when precision is MOARA_PREC_FP32
 *   exp_avg     r x n  fp32 first moment of the direction branch (zeroed by
 *   exp_avg_sq  r x n  fp32 second moment          the caller before step 1)
 *   mag_avg     m x k  fp32 first moment of the magnitude branch (k=ceil(n/B));
 *   mag_avg_sq  m x k  fp32 second moment          unused when decompose = 0
 *   workspace   moara_workspace_bytes() bytes of scratch, private to the module
 * With hparams.state_dtype = MOARA_DTYPE_BF16, W, exp_avg and exp_avg_sq
 * point to bf16 arrays of the same shapes (the pointer types stay float*).
 * With hparams.proj_rule = MOARA_PROJ_SMALLER and m > n, P and P_bf16 hold
 * the right projector Q (n x r) and exp_avg / exp_avg_sq are m x r.
 */
typedef struct moara_module_desc {
    int m, n, r;
    int grad_dtype;         /* MOARA_DTYPE_F32 or MOARA_DTYPE_BF16 */
    float*    W;
    float*    P;
    uint16_t* P_bf16;
    float*    exp_avg;
    float*    exp_avg_sq;
    float*    mag_avg;
    float*    mag_avg_sq;
    void*     workspace;
    size_t    workspace_bytes;
} moara_module_desc;

typedef struct moara_ctx moara_ctx;

/* Fills *out with the paper's defaults (App. D.2: beta 0.9/0.999, eps 1e-6,
 * alpha 0.25, T 200; App. B.1: decomp eps 1e-12; B = 128) and the refresh
 * defaults p = 32, q = 4, ritz_iters = 3, precision AUTO, seed 0. */
int moara_default_hparams(moara_hparams* out);

/* Creates a context on CUDA device `device` (the current device is restored
 * on return).  Validates hp (betas in [0,1), eps >= 0, B >= 1, T >= 1,
 * p, q >= 0).  Allocates the module table and the device status word.
 * *out is NULL on error. */
int moara_create(moara_ctx** out, const moara_hparams* hp, int device);

/* Releases the context-owned device memory.  Caller buffers are untouched.
 * Accepts NULL.  Work still queued on a stream must have completed. */
void moara_destroy(moara_ctx* ctx);

/* Copies the context's hyper-parameters into *out. */
int moara_get_hparams(const moara_ctx* ctx, moara_hparams* out);

/* Optimizer-state bytes of one m x n target matrix (Appendix G):
 *   2*b_V*r*d_W  (+ 2*b_M*m*ceil(n/B) when decompose != 0)
 * with d_W = n (MOARA_DRULE_N) or max(m, n) (MOARA_DRULE_MAX).  Host only;
 * MOARA_ERR_SHAPE on overflow of size_t. */
int moara_state_bytes(int m, int n, int r, int block_size, int b_V, int b_M,
                      int d_rule, int decompose, size_t* out);

/* Phase 3 of Algorithm 1 (§3.2; App. C final allocation): donors (bits of
 * donor_mask) get r_base - delta_r, receivers r_base + delta_r*|D|/|R|, the
 * rest r_base.  An uneven split is floored and the remainder given one by one
 * to receivers in module order, so sum(out_ranks) == 7*r_base.  Host only.
 * Errors: overlapping masks, donors without receivers, delta_r outside
 * [0, r_base), masks with bits above MOARA_MOD_DOWN. */
int moara_rank_table(int r_base, uint32_t donor_mask, uint32_t receiver_mask,
                     int delta_r, int out_ranks[7]);

/* Bytes of per-module scratch a module of this shape needs (Adam update of
 * the direction branch r x n, magnitude update m x k, block scales m x k,
 * and the direction matrix V as two m x n bf16 planes for the tensor-core
 * projection). */
int moara_workspace_bytes(int m, int n, int r, int block_size, size_t* out);

/* Registers a weight (see moara_module_desc).  Checks shapes (r <= min(m,n)),
 * dtype, alignment, workspace size; copies the descriptor into the context's
 * device table with a synchronous copy (do this before any graph capture).
 * *module_id receives a dense id 0, 1, 2, ... */
int moara_init_module(moara_ctx* ctx, const moara_module_desc* desc,
                      int* module_id);

/* Writes P (fp32) and its bf16 copy from a caller device buffer P_src
 * (m x r fp32 row-major; may alias desc.P).  For callers that supply the
 * projector themselves instead of running the refresh. */
int moara_load_projector(moara_ctx* ctx, int module_id, const float* P_src,
                         void* stream);

/* Bytes of shared scratch the refresh of one module of this shape needs with
 * the context's p and q (Gaussian sketch, range basis, Gram and Cholesky
 * factors).  The refresh processes modules in groups that fit the workspace
 * set with moara_set_refresh_workspace. */
int moara_refresh_workspace_bytes(const moara_ctx* ctx, int m, int n, int r,
                                  size_t* out);

/* Hands the context a caller-owned device buffer used as refresh scratch. */
int moara_set_refresh_workspace(moara_ctx* ctx, void* ptr, size_t bytes);

/* TruncatedSVD(V, r) of Algorithm 1 for the listed modules: P <- top-r left
 * singular vectors of V = Decompose(G, B) (or of G with refresh_src = G),
 * computed by randomized subspace iteration (Gaussian sketch with p extra
 * columns, q power iterations, CholeskyQR orthonormalisation, Rayleigh-Ritz
 * on the sketch).  Columns come in descending singular-value order, each
 * of unit length and signed so that its largest-magnitude entry is positive
 * (the lowest row on ties).  Writes P and P_bf16; a module whose
 * factorisation meets a non-positive pivot keeps its previous P.  G[i] is the m x n gradient of module ids[i] (device, dtype of the
 * module).  MOARA_ERR_WORKSPACE if one module does not fit the workspace. */
int moara_refresh_projector(moara_ctx* ctx, int n_mod, const int* ids,
                            const void* const* G, void* stream);

/* One optimizer step at Adam step t (1-based) for the listed modules, all in
 * one grouped launch per kernel.  G[i] is module ids[i]'s gradient (device,
 * m x n, the module's dtype, read only).  lr is this step's learning rate
 * (the schedule is the caller's).  With auto_refresh != 0 every module whose
 * (t - 1) mod T == 0 first runs moara_refresh_projector (the refresh reads
 * the same G and happens before projecting, as in Algorithm 1).
 * Updates W, the four moment buffers, and on refresh steps P and P_bf16.
 * A NaN or Inf in G propagates: a non-finite entry of G at (i, j) makes the
 * update of every column of j's block non-finite (row i's block norm enters
 * the direction projection of those columns); with decompose = 0 only
 * column j is affected. */
int moara_step_grouped(moara_ctx* ctx, int n_mod, const int* ids,
                       const void* const* G, int64_t t, float lr,
                       int auto_refresh, void* stream);

/* The same step with the gradients in host memory: G_host[i] is module
 * ids[i]'s gradient in page-locked host memory (m x n, the module's dtype).
 * The modules are taken in order, in chunks of at most chunk_bytes of
 * gradient (a larger module is a chunk of its own).  Each chunk is copied on
 * an internal stream into one of two device staging buffers while the step
 * kernels of the previous chunk run on `stream`, so the transfer overlaps the
 * computation.  The staging buffers (2 x the largest chunk) are allocated on
 * first use and kept until moara_destroy.  Asynchronous like
 * cudaMemcpyAsync: G_host must stay valid and unchanged until the work
 * enqueued on `stream` by this call has finished. */
int moara_step_grouped_host(moara_ctx* ctx, int n_mod, const int* ids,
                            const void* const* G_host, int64_t t, float lr,
                            int auto_refresh, size_t chunk_bytes, void* stream);

/* Global-norm clipping state (hparams.clip_norm > 0; App. D.2).
 *
 * moara_set_clip_extra: `extra_sq` is a device float holding the sum of
 * squared gradient entries of parameters the library does not own (the
 * embedding, norms, ...); every clipped step reads it stream-ordered, so the
 * caller writes it on the step's stream before the step.  NULL (the default)
 * means 0.  The pointer must stay valid while clipped steps run.
 *
 * moara_clip_state: `*state` receives the address of a context-owned device
 * array {total norm, coefficient} written by every clipped step (before any
 * of the step's updates), for scaling the caller's other gradients with the
 * same coefficient.  Valid until moara_destroy.
 *
 * Clipping needs every gradient of the step on the device before the first
 * update: moara_step_grouped_host and moara_step_static_scratch return
 * MOARA_ERR_UNSUPPORTED when clip_norm > 0.  The refresh is unaffected (the
 * singular subspace of c G and of V is that of G). */
int moara_set_clip_extra(moara_ctx* ctx, const float* extra_sq);
int moara_clip_state(moara_ctx* ctx, const float** state);

/* N-D flatten rule of App. B ("Flattening"): a gradient of shape
 * (s_0, s_1, ..., s_{k-1}) is treated as the m x n matrix with m = s_0 and
 * n = s_1 * ... * s_{k-1} (the row axis kept, blocks along the flattened
 * columns); a 1-D shape gives m = s_0, n = 1.  Host only.  Errors:
 * MOARA_ERR_INVALID_ARG for ndim < 1, a NULL pointer or a non-positive extent,
 * MOARA_ERR_SHAPE when m or n exceeds INT_MAX. */
int moara_flatten_shape(int ndim, const int64_t* shape, int* m, int* n);

/* Alignment diagnostic S(W, t) (§3.2, the module-alignment equation; App. C
 * "Profiling-based rank allocation"): for each module q of the call,
 *   S_q = cos(G_q, Rep_B(M) (.) (P P^T V)),  (M, V) = Decompose(G_q, B),
 * with the module's current projector P (its bf16 copy) and the context's
 * block size B (V Q Q^T for a module with a right projector Q); the cosine is the Frobenius inner product over ||G|| ||.||
 * (0 when either norm is 0).  The paper averages S over profiling steps and
 * matrices of a module type (S_tau) to rank the modules; that average is the
 * caller's.
 *
 * G: device pointers to the modules' gradients (bf16, m x n row-major).
 * S_out: device array of n_mod floats, written stream-ordered.
 * Scratch: each module's workspace (its contents are rewritten by the next
 * step anyway) and three doubles per module owned by the context (allocated
 * on first use or when a call has more modules than before; growing them
 * waits for `stream`).
 * Errors: MOARA_ERR_UNSUPPORTED (nothing launched) when a module is not on
 * the tensor-core path (bf16 gradient, n and r multiples of 8, B in {8, 16,
 * 32, 64, 128}); the usual argument errors otherwise. */
int moara_alignment(moara_ctx* ctx, int n_mod, const int* ids, const void* const* G, float* S_out,
                    void* stream);

/* Reads and clears the device status word (0, or a MOARA_ERR_* code a kernel
 * recorded, e.g. MOARA_ERR_DEVICE_TIMEOUT from a bounded wait).  Synchronizes
 * `stream`.  *status receives the code. */
int moara_get_device_status(moara_ctx* ctx, int* status, void* stream);

/* Text of the last failed check in this context ("" if none).  The pointer
 * stays valid until the next call on the context. */
const char* moara_last_error(const moara_ctx* ctx);

/* Static text for a MOARA_* status code. */
const char* moara_status_string(int code);

/* Number of kernel launches the context has enqueued since creation. */
int64_t moara_launch_count(const moara_ctx* ctx);

/* Failure-detection hook (the paper has no counterpart).  Every wait of the
 * library's kernels on an mbarrier is bounded; when the bound passes without
 * progress the kernel records MOARA_ERR_DEVICE_TIMEOUT in the device status
 * word, waits (with the default bound) for its own copies and tensor-core
 * work in flight, frees its tensor memory and returns, leaving the context
 * usable.  This call sets the bound, in SM clock cycles, of the waits of the
 * tensor-core products of the projector refresh and of moara_alignment (the
 * single-CTA kernels) for launches enqueued afterwards; cycles <= 0 restores
 * the default (2^32 cycles, about 2 s).  A bound shorter than the kernels'
 * own latency (a few hundred cycles) makes them give up on purpose, which is
 * how the failure path is tested; their outputs are then undefined until the
 * next call with the default bound.  The step kernels' two-CTA pairs keep the
 * default bound.  Returns MOARA_ERR_UNSUPPORTED without tensor-core state. */
int moara_set_wait_limit(moara_ctx* ctx, int64_t cycles);

/* Per-kernel timing with CUDA events recorded on the launching stream around
 * every launch of the step and refresh kernels (enable != 0 turns it on).
 * Phases: MOARA_PHASE_*.  Adds two event records per launch; no effect on
 * results. */
#define MOARA_PHASE_DECOMPOSE     0  /* block norms + magnitude Adam (fp32 path)     */
#define MOARA_PHASE_PROJECT       1  /* R = P^T V + direction Adam (fp32 path)       */
#define MOARA_PHASE_BACKPROJECT   2  /* dV = P N + weight update (fp32 path)         */
#define MOARA_PHASE_REFRESH       3  /* one whole refresh call                       */
#define MOARA_PHASE_TC_PROJECT    4  /* tensor-core projection kernel                */
#define MOARA_PHASE_TC_BACKPROJECT 5 /* tensor-core back-projection kernel           */
#define MOARA_PHASE_TC_DECOMPOSE  6  /* tensor-core path: block norms, magnitude Adam, V in bf16 */
#define MOARA_PHASE_TC_REFRESH    7  /* refresh products V^T Q, V Z on tensor cores (inside REFRESH) */
#define MOARA_PHASE_TC_DECOMPOSE_OVERLAP 8  /* decomposition of later module parts on the library's
                                               auxiliary stream, concurrent with K1 / K2 of earlier
                                               parts (event time on that stream, not additive)      */
#define MOARA_PHASE_CLIP_NORM     9  /* global gradient norm and clipping coefficient      */
#define MOARA_NUM_PHASES          10
int moara_profile_enable(moara_ctx* ctx, int enable);

/* Waits for the recorded events, writes the summed milliseconds and launch
 * counts per phase (arrays of MOARA_NUM_PHASES), and clears the record. */
int moara_profile_read(moara_ctx* ctx, double ms[MOARA_NUM_PHASES], int64_t launches[MOARA_NUM_PHASES]);

/* One optimizer step of a single weight that allocates no device memory.
 *
 * For callers that cannot allocate device memory when they run the step:
 * code embedded in a host application that reserves the GPU's memory up
 * front through its own pool (and forbids allocations outside it), or a step
 * loop that must not pay the device-wide synchronisation that cudaMalloc and
 * cudaFree can imply.  Such callers cannot create a context (moara_create
 * allocates) or hand over a per-module workspace; this entry point takes the
 * buffers directly and keeps its scratch -- the direction update N (r x n
 * floats), the magnitude update and the block scales (m x ceil(n/B) floats
 * each) -- in a 16 MiB array compiled into the library, which every GPU that
 * loads the library holds until the process exits.  The paper has no
 * counterpart; the computation is that of moara_step_grouped on the fp32
 * path (MOARA_PREC_FP32), without the refresh.
 *
 *   hp          hyper-parameters (block size, betas, eps, scale, decompose)
 *   m, n, r     shape and rank, 1 <= r <= min(m, n)
 *   grad_dtype  MOARA_DTYPE_F32 or MOARA_DTYPE_BF16
 *   G           m x n gradient (read);  W  m x n fp32 (updated)
 *   P           m x r fp32 projector (read)
 *   exp_avg, exp_avg_sq   r x n fp32 (updated)
 *   mag_avg, mag_avg_sq   m x ceil(n/B) fp32 (updated; unused if decompose = 0)
 *   t, lr       1-based Adam step and learning rate; stream as elsewhere
 * All pointers are device pointers on the calling thread's current device,
 * 16-byte aligned.  Returns MOARA_ERR_WORKSPACE when
 * 4*(r*n + 2*m*ceil(n/B)) bytes (each part rounded up to 256 bytes) exceed
 * the 16 MiB array; nothing is launched then.  The first call on a device
 * looks up the array's device address (once per device, then cached).  With
 * lazy module loading, the CUDA default, that first call is also what loads
 * the library's module holding the array onto the device and so reserves the
 * 16 MiB there: a caller whose memory pool takes the GPU's free memory should
 * make one accepted call before reserving its pool, and before any stream
 * capture.  Later calls on that device allocate nothing.  The cached address
 * is that of the device's primary context; after cudaDeviceReset it is stale
 * and this entry point must not be called again in the process.  All calls
 * share the one array: calls whose kernels overlap on the GPU (different
 * streams, or different host threads on the same device) race on it and must
 * be serialised by the caller.  No scratch value is carried from one call to
 * the next.  Only the left projector is taken: with proj_rule =
 * MOARA_PROJ_SMALLER and m > n the call returns MOARA_ERR_UNSUPPORTED.
 * hp->precision is ignored (the fp32 path always runs), and so are the
 * refresh fields; clip_norm > 0 and bf16 states return MOARA_ERR_UNSUPPORTED. */
int moara_step_static_scratch(const moara_hparams* hp, int m, int n, int r, int grad_dtype,
                              const void* G, float* W, const float* P, float* exp_avg,
                              float* exp_avg_sq, float* mag_avg, float* mag_avg_sq, int64_t t,
                              float lr, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* MOARA_H_ */
