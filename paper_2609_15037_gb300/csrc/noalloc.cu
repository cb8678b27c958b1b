// One-module optimizer step whose scratch lives in a fixed device array
// compiled into the library, for callers that cannot allocate device memory
// when they run the step.  It launches the same fp32 kernels as the grouped
// step (decomposition + magnitude Adam, projection + direction Adam,
// back-projection + weight update); only the origin of the scratch differs.
#include <cmath>
#include <mutex>

#include "internal.h"

namespace {

// 16 MiB of scratch: the direction update N (r x n floats) followed by the
// magnitude update dM and the block scales (m x ceil(n/B) floats each).  Every
// GPU that loads the library keeps this array until the process exits.
constexpr size_t kStaticScratchFloats = size_t(4) << 20;
static __device__ __align__(256) float g_static_scratch[kStaticScratchFloats];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
float* g_scratch_addr[kMaxDevices] = {};

// Device address of the array on the current device.  In host code the
// array's name is only a host-side stand-in, so the address is looked up once
// per device (the first call on that device) with that device current.  With
// lazy module loading (the CUDA default) that first lookup is also what loads
// this file's module on the device and reserves the 16 MiB there.  The cached
// address belongs to the device's primary context: after cudaDeviceReset (or
// any reset of the primary context) the module is loaded again, possibly at
// another address, and the cached one is stale -- such a caller must not use
// this entry point again in the same process.
int scratch_address(float** out) {
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return MOARA_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    if (g_scratch_addr[dev] == nullptr) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_static_scratch) != cudaSuccess || p == nullptr) return MOARA_ERR_CUDA;
        g_scratch_addr[dev] = static_cast<float*>(p);
    }
    *out = g_scratch_addr[dev];
    return MOARA_OK;
}

bool aligned16(const void* p) { return p != nullptr && (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

size_t round64(size_t x) { return (x + 63) / 64 * 64; }

}  // namespace

extern "C" int moara_step_static_scratch(const moara_hparams* hp, int m, int n, int r, int grad_dtype,
                                         const void* G, float* W, const float* P, float* exp_avg,
                                         float* exp_avg_sq, float* mag_avg, float* mag_avg_sq, int64_t t,
                                         float lr, void* stream) {
    if (hp == nullptr) return MOARA_ERR_INVALID_ARG;
    // the same hyper-parameter checks as moara_create
    if (!(hp->beta1 >= 0.0f && hp->beta1 < 1.0f) || !(hp->beta2 >= 0.0f && hp->beta2 < 1.0f) ||
        !(hp->adam_eps >= 0.0f) || !std::isfinite(hp->adam_eps) || !(hp->decomp_eps >= 0.0f) ||
        !std::isfinite(hp->decomp_eps) || !std::isfinite(hp->scale) || !std::isfinite(hp->clip_norm) ||
        (hp->decompose != 0 && hp->decompose != 1))
        return MOARA_ERR_INVALID_ARG;
    if (hp->proj_rule != MOARA_PROJ_LEFT && hp->proj_rule != MOARA_PROJ_SMALLER) return MOARA_ERR_INVALID_ARG;
    if (hp->precision != MOARA_PREC_AUTO && hp->precision != MOARA_PREC_FP32 && hp->precision != MOARA_PREC_BF16_TC)
        return MOARA_ERR_INVALID_ARG;
    if (m < 1 || n < 1 || hp->block_size < 1) return MOARA_ERR_SHAPE;
    if (r < 1 || r > (m < n ? m : n)) return MOARA_ERR_RANK;
    // only the left projector P (m x r) is taken here; the smaller-side rule
    // would give a tall weight a right projector
    if (hp->proj_rule == MOARA_PROJ_SMALLER && m > n) return MOARA_ERR_UNSUPPORTED;
    if (grad_dtype != MOARA_DTYPE_F32 && grad_dtype != MOARA_DTYPE_BF16) return MOARA_ERR_INVALID_ARG;
    if (t < 1 || !std::isfinite(lr)) return MOARA_ERR_INVALID_ARG;
    if (hp->clip_norm > 0.0f) return MOARA_ERR_UNSUPPORTED;   // global-norm clipping needs the whole step
    if (hp->state_dtype != MOARA_DTYPE_F32) return MOARA_ERR_UNSUPPORTED;   // fp32 states only here
    if (!aligned16(G) || !aligned16(W) || !aligned16(P) || !aligned16(exp_avg) || !aligned16(exp_avg_sq))
        return G && W && P && exp_avg && exp_avg_sq ? MOARA_ERR_ALIGN : MOARA_ERR_INVALID_ARG;
    if (hp->decompose && (!aligned16(mag_avg) || !aligned16(mag_avg_sq)))
        return mag_avg && mag_avg_sq ? MOARA_ERR_ALIGN : MOARA_ERR_INVALID_ARG;

    const int B = hp->block_size;
    const int kb = (n + B - 1) / B;
    const size_t off_dM = round64(static_cast<size_t>(r) * n);
    const size_t off_inv = off_dM + round64(static_cast<size_t>(m) * kb);
    const size_t need = off_inv + static_cast<size_t>(m) * kb;
    if (need > kStaticScratchFloats) return MOARA_ERR_WORKSPACE;

    float* scratch = nullptr;
    int rc = scratch_address(&scratch);
    if (rc != MOARA_OK) return rc;
    float* N = scratch;
    float* dM = scratch + off_dM;
    float* inv = scratch + off_inv;

    cudaStream_t s = static_cast<cudaStream_t>(stream);
    int64_t launches = 0;
    const double bc1 = 1.0 - std::pow(static_cast<double>(hp->beta1), static_cast<double>(t));
    const double bc2 = 1.0 - std::pow(static_cast<double>(hp->beta2), static_cast<double>(t));
    const int bf = grad_dtype == MOARA_DTYPE_BF16 ? 1 : 0;

    // Every scratch element read below is written earlier in this call (block
    // scales and dM for all (row, block) pairs, N for all r x n entries), so
    // nothing carried over from the previous call is used.
    if (hp->decompose) {
        moara::DecompBatch db{};
        db.count = 1;
        db.B = B;
        db.do_mag = 1;
        db.decomp_eps = hp->decomp_eps;
        db.beta1 = hp->beta1;
        db.beta2 = hp->beta2;
        db.adam_eps = hp->adam_eps;
        db.bc1 = static_cast<float>(bc1);
        db.bc2 = static_cast<float>(bc2);
        db.item_start[0] = 0;
        db.item_start[1] = static_cast<long long>(m) * kb;
        db.p[0] = moara::DecompItem{G, inv, mag_avg, mag_avg_sq, dM, m, n, kb, grad_dtype};
        if (moara::launch_decompose(db, s, &launches) != cudaSuccess) return MOARA_ERR_CUDA;
    }
    {
        moara::GemmBatch b{};
        b.count = 1;
        b.B = B;
        b.beta1 = hp->beta1;
        b.beta2 = hp->beta2;
        b.adam_eps = hp->adam_eps;
        b.bc1 = static_cast<float>(bc1);
        b.bc2 = static_cast<float>(bc2);
        moara::GemmProb& p = b.p[0];
        p.A = P;
        p.Bm = G;
        p.b_inv = hp->decompose ? inv : nullptr;
        p.C = N;
        p.aux0 = exp_avg;
        p.aux1 = exp_avg_sq;
        p.M = r; p.N = n; p.K = m;
        p.lda = r; p.ldb = n; p.ldc = n;
        p.kb = kb;
        p.b_bf16 = bf;
        moara::GemmKind k{moara::A_MCONTIG, moara::B_NCONTIG, 0, hp->decompose, 0, bf, moara::EPI_ADAM};
        if (moara::launch_gemm(k, b, s, &launches) != cudaSuccess) return MOARA_ERR_CUDA;
    }
    {
        moara::GemmBatch b{};
        b.count = 1;
        b.B = B;
        b.step_scale = lr * hp->scale;
        moara::GemmProb& p = b.p[0];
        p.A = P;
        p.Bm = N;
        p.aux0 = W;
        p.aux2 = hp->decompose ? dM : nullptr;
        p.M = m; p.N = n; p.K = r;
        p.lda = r; p.ldb = n; p.ldc = n;
        p.kb = kb;
        moara::GemmKind k{moara::A_KCONTIG, moara::B_NCONTIG, 0, 0, 0, 0, moara::EPI_UPDATE};
        if (moara::launch_gemm(k, b, s, &launches) != cudaSuccess) return MOARA_ERR_CUDA;
    }
    return MOARA_OK;
}
