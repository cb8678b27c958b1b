// Host side of libmoara: argument validation, the context and its device
// module table, the memory model and rank table helpers, and the sequencing of
// the step and refresh kernels.  Declarations and contracts are in moara.h.
#include <algorithm>
#include <climits>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <limits>
#include <new>
#include <string>
#include <array>
#include <vector>

#include "internal.h"
#include "tc.h"

struct moara_ctx {
    int device = 0;
    moara_hparams hp{};
    std::vector<moara_module_desc> mods;
    std::vector<moara::ModDev> moddev;
    std::vector<int64_t> refresh_count;
    moara::ModDev* d_mods = nullptr;
    int cap = 0;
    int* d_status = nullptr;
    int* h_status = nullptr;
    void* refresh_ws = nullptr;
    size_t refresh_ws_bytes = 0;
    std::string last_error;
    int64_t launches = 0;
    moara::TcState* tc = nullptr;
    // host-gradient step: two device staging buffers, a copy stream, events
    void* stage[2] = {nullptr, nullptr};
    size_t stage_bytes = 0;
    cudaStream_t copy_stream = nullptr;
    cudaEvent_t copy_done[2] = {nullptr, nullptr};
    cudaEvent_t compute_done[2] = {nullptr, nullptr};
    // per-kernel CUDA-event timing (moara_profile_enable)
    bool prof = false;
    struct Rec { int phase; cudaEvent_t a, b; };
    std::vector<Rec> recs;
    std::vector<cudaEvent_t> free_events;
    cudaEvent_t open_event = nullptr;
    double prof_ms[MOARA_NUM_PHASES] = {0};
    int64_t prof_n[MOARA_NUM_PHASES] = {0};
    // alignment diagnostic: three double accumulators per module of a call
    double* align_acc = nullptr;
    int align_cap = 0;
    // global-norm clipping: {total norm, coefficient}, per-CTA partial sums,
    // the caller's extra sum of squares
    float* d_clip = nullptr;
    double* d_clip_part = nullptr;
    int clip_part_cap = 0;
    const float* clip_extra = nullptr;
};

namespace {

constexpr int kMaxModules = 65536;

int fail(moara_ctx* ctx, int code, const char* fmt, ...) {
    if (ctx != nullptr) {
        char buf[512];
        va_list ap;
        va_start(ap, fmt);
        std::vsnprintf(buf, sizeof(buf), fmt, ap);
        va_end(ap);
        ctx->last_error = buf;
    }
    return code;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

int blocks_of(int n, int B) { return (n + B - 1) / B; }

struct DeviceGuard {
    int prev = -1;
    explicit DeviceGuard(int dev) {
        if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
        if (prev != dev) cudaSetDevice(dev);
    }
    ~DeviceGuard() {
        int cur = -1;
        if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
    }
};

int check_hparams(moara_ctx* ctx, const moara_hparams* hp) {
    if (hp == nullptr) return fail(ctx, MOARA_ERR_INVALID_ARG, "hparams is NULL");
    if (!(hp->beta1 >= 0.0f && hp->beta1 < 1.0f) || !(hp->beta2 >= 0.0f && hp->beta2 < 1.0f))
        return fail(ctx, MOARA_ERR_INVALID_ARG, "betas must lie in [0, 1)");
    if (!(hp->adam_eps >= 0.0f) || !std::isfinite(hp->adam_eps))
        return fail(ctx, MOARA_ERR_INVALID_ARG, "adam_eps must be finite and >= 0");
    if (!(hp->decomp_eps >= 0.0f) || !std::isfinite(hp->decomp_eps))
        return fail(ctx, MOARA_ERR_INVALID_ARG, "decomp_eps must be finite and >= 0");
    if (!std::isfinite(hp->scale)) return fail(ctx, MOARA_ERR_INVALID_ARG, "scale must be finite");
    if (hp->block_size < 1) return fail(ctx, MOARA_ERR_SHAPE, "block_size must be >= 1");
    if (hp->refresh_interval < 1) return fail(ctx, MOARA_ERR_SHAPE, "refresh_interval must be >= 1");
    if (hp->decompose != 0 && hp->decompose != 1)
        return fail(ctx, MOARA_ERR_INVALID_ARG, "decompose must be 0 or 1");
    if (hp->refresh_src != MOARA_REFRESH_SRC_V && hp->refresh_src != MOARA_REFRESH_SRC_G)
        return fail(ctx, MOARA_ERR_INVALID_ARG, "unknown refresh_src");
    if (hp->oversample < 0 || hp->power_iters < 0 || hp->ritz_iters < 0)
        return fail(ctx, MOARA_ERR_INVALID_ARG, "oversample, power_iters, ritz_iters must be >= 0");
    if (hp->oversample > 4096 || hp->power_iters > 64 || hp->ritz_iters > 256)
        return fail(ctx, MOARA_ERR_INVALID_ARG, "refresh parameters out of range");
    if (hp->precision != MOARA_PREC_AUTO && hp->precision != MOARA_PREC_FP32 &&
        hp->precision != MOARA_PREC_BF16_TC)
        return fail(ctx, MOARA_ERR_INVALID_ARG, "unknown precision");
    if (!std::isfinite(hp->clip_norm)) return fail(ctx, MOARA_ERR_INVALID_ARG, "clip_norm must be finite");
    if (hp->state_dtype != MOARA_DTYPE_F32 && hp->state_dtype != MOARA_DTYPE_BF16)
        return fail(ctx, MOARA_ERR_INVALID_ARG, "state_dtype must be MOARA_DTYPE_F32 or MOARA_DTYPE_BF16");
    if (hp->proj_rule != MOARA_PROJ_LEFT && hp->proj_rule != MOARA_PROJ_SMALLER)
        return fail(ctx, MOARA_ERR_INVALID_ARG, "unknown proj_rule");
    if (hp->state_dtype == MOARA_DTYPE_BF16 && hp->precision == MOARA_PREC_FP32)
        return fail(ctx, MOARA_ERR_UNSUPPORTED, "bf16 states run on the tensor-core path only");
    return MOARA_OK;
}

int cuda_fail(moara_ctx* ctx, cudaError_t e, const char* what) {
    return fail(ctx, MOARA_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

cudaEvent_t take_event(moara_ctx* ctx) {
    if (!ctx->free_events.empty()) {
        cudaEvent_t e = ctx->free_events.back();
        ctx->free_events.pop_back();
        return e;
    }
    cudaEvent_t e = nullptr;
    cudaEventCreate(&e);
    return e;
}

// Records an event pair around the launches made in its scope when profiling.
struct ProfScope {
    moara_ctx* ctx;
    int phase;
    cudaStream_t s;
    cudaEvent_t a = nullptr;
    ProfScope(moara_ctx* c, int ph, cudaStream_t st) : ctx(c), phase(ph), s(st) {
        if (ctx->prof) {
            a = take_event(ctx);
            cudaEventRecord(a, s);
        }
    }
    ~ProfScope() {
        if (a != nullptr) {
            cudaEvent_t b = take_event(ctx);
            cudaEventRecord(b, s);
            ctx->recs.push_back({phase, a, b});
        }
    }
};

// Whether module `mi` runs its step on tensor cores.
bool use_tc(const moara_ctx* ctx, int mi) {
    const moara_module_desc& d = ctx->mods[mi];
    if (ctx->hp.precision == MOARA_PREC_FP32) return false;
    if (ctx->hp.precision == MOARA_PREC_AUTO && d.grad_dtype != MOARA_DTYPE_BF16) return false;
    return moara::tc_supported(d.m, d.n, d.r, ctx->hp.block_size, d.grad_dtype, ctx->hp.decompose,
                               ctx->hp.state_dtype) &&
           d.P_bf16 != nullptr && ctx->tc != nullptr;
}

}  // namespace

namespace moara {

WsLayout workspace_layout(int m, int n, int r, int B) {
    const int kb = blocks_of(n, B);
    WsLayout w{};
    size_t off = 0;
    // N: r x n, or m x r for a right projector (sized for either on a tall weight)
    w.off_N = off;   off = align_up(off + sizeof(float) * (size_t)r * std::max(n, m), 256);
    w.off_dM = off;  off = align_up(off + sizeof(float) * (size_t)m * kb, 256);
    w.off_inv = off; off = align_up(off + sizeof(float) * (size_t)m * kb, 256);
    w.off_Vhi = off; off = align_up(off + sizeof(uint16_t) * (size_t)m * n, 256);
    w.off_Vlo = off; off = align_up(off + sizeof(uint16_t) * (size_t)m * n, 256);
    w.off_Qt = 0;
    if (m > n) { w.off_Qt = off; off = align_up(off + sizeof(uint16_t) * (size_t)r * n, 256); }   // Q^T
    w.total = off;
    return w;
}

size_t refresh_ws_bytes(int m, int n, int r, int l, int B, int src_v) {
    (void)r;
    const int kb = blocks_of(n, B);
    size_t off = 0;
    auto add = [&](size_t bytes) { off = align_up(off + bytes, 256); };
    if (src_v) add(sizeof(float) * (size_t)m * kb);
    add(sizeof(float) * (size_t)n * l);  // Za (also Omega)
    add(sizeof(float) * (size_t)n * l);  // Zb
    add(2 * sizeof(float) * (size_t)m * l + align_up(sizeof(uint16_t) * (size_t)m * l, 16));  // Qa, Qbf, Qb
    add(sizeof(uint16_t) * (size_t)n * l);  // Zbf
    for (int i = 0; i < 3; ++i) add(3 * sizeof(uint16_t) * (size_t)l * l);   // Cp, P1, P2
    for (int i = 0; i < 6; ++i) add(sizeof(float) * (size_t)l * l);
    add(sizeof(float) * 16);
    add(sizeof(float) * (size_t)l);
    add(sizeof(int) * (size_t)l);
    add(sizeof(int) * 4);
    return off;
}

void refresh_carve(RefreshItem& it, void* base, int m, int n, int r, int l, int B, int src_v) {
    (void)r;
    const int kb = blocks_of(n, B);
    char* p = static_cast<char*>(base);
    size_t off = 0;
    auto take = [&](size_t bytes) { char* q = p + off; off = align_up(off + bytes, 256); return q; };
    it.inv = src_v ? reinterpret_cast<float*>(take(sizeof(float) * (size_t)m * kb)) : nullptr;
    it.Za = reinterpret_cast<float*>(take(sizeof(float) * (size_t)n * l));
    it.Omega = it.Za;
    it.Zb = reinterpret_cast<float*>(take(sizeof(float) * (size_t)n * l));
    // Qa, Qbf, Qb back to back (Qb 16-byte aligned after Qbf): Qbf + Qb
    // hold the three bf16 planes of a tall Q (3 m l entries) for the
    // tensor-core CholeskyQR pass
    const size_t qbf_bytes = align_up(sizeof(uint16_t) * (size_t)m * l, 16);
    it.Qa = reinterpret_cast<float*>(take(2 * sizeof(float) * (size_t)m * l + qbf_bytes));
    it.Qbf = reinterpret_cast<uint16_t*>(it.Qa + (size_t)m * l);
    it.Qb = reinterpret_cast<float*>(reinterpret_cast<char*>(it.Qbf) + qbf_bytes);
    it.Zbf = reinterpret_cast<uint16_t*>(take(sizeof(uint16_t) * (size_t)n * l));
    it.Cp = reinterpret_cast<uint16_t*>(take(3 * sizeof(uint16_t) * (size_t)l * l));
    it.P1 = reinterpret_cast<uint16_t*>(take(3 * sizeof(uint16_t) * (size_t)l * l));
    it.P2 = reinterpret_cast<uint16_t*>(take(3 * sizeof(uint16_t) * (size_t)l * l));
    it.Cg = reinterpret_cast<float*>(take(sizeof(float) * (size_t)l * l));
    it.Linv = reinterpret_cast<float*>(take(sizeof(float) * (size_t)l * l));
    it.Tt = reinterpret_cast<float*>(take(sizeof(float) * (size_t)l * l));
    it.scal = reinterpret_cast<float*>(take(sizeof(float) * 16));
    it.Cr = reinterpret_cast<float*>(take(sizeof(float) * (size_t)l * l));
    it.Xa = reinterpret_cast<float*>(take(sizeof(float) * (size_t)l * l));
    it.Xb = reinterpret_cast<float*>(take(sizeof(float) * (size_t)l * l));
    it.ritz = reinterpret_cast<float*>(take(sizeof(float) * (size_t)l));
    it.perm = reinterpret_cast<int*>(take(sizeof(int) * (size_t)l));
    it.fail = reinterpret_cast<int*>(take(sizeof(int) * 4));
}

}  // namespace moara

namespace {

int refresh_l(const moara_ctx* ctx, int m, int n, int r) {
    long long l = (long long)r + ctx->hp.oversample;
    l = std::min<long long>(l, std::min(m, n));
    return static_cast<int>(std::max<long long>(l, r));
}

// ------------------------------------------------------------------ refresh
// Panel width of the fast blocked Cholesky (tensor-core trailing updates).
constexpr int kFastPanel = 256;
constexpr int kTriTcMin = 512;   // triangular-inverse levels from this block size run on tensor cores

struct RefreshRunner {
    moara_ctx* ctx;
    cudaStream_t s;
    std::vector<moara::RefreshItem> it;
    int src_v;
    cudaError_t err = cudaSuccess;

    void chk(cudaError_t e) { if (err == cudaSuccess && e != cudaSuccess) err = e; }

    template <class F>
    void gemm(const moara::GemmKind& kind, F fill) {
        moara::GemmBatch b{};
        b.count = static_cast<int>(it.size());
        b.B = ctx->hp.block_size;
        for (int i = 0; i < b.count; ++i) {
            b.p[i] = moara::GemmProb{};
            fill(i, b.p[i]);
        }
        chk(moara::launch_gemm(kind, b, s, &ctx->launches));
    }

    moara::SmallBatch small() {
        moara::SmallBatch b{};
        b.count = static_cast<int>(it.size());
        return b;
    }

    // X_out = X_in * chol(X_in^T X_in + shift)^-T for every item (rows(i) x l).
    // Only the lower triangle of the Gram matrix is formed (the Cholesky
    // factorisation reads no more), and the product with the lower-triangular
    // inverse skips its zero upper part.  `bf` (per item, may hold nulls)
    // receives a bf16 copy of X_out for the tensor-core products.
    void cholqr_pass(std::vector<float*>& Xin, std::vector<float*>& Xout,
                     const std::vector<int>& rows, float shift_rel,
                     const std::vector<uint16_t*>* bf = nullptr) {
        moara::GemmKind gram{moara::A_MCONTIG, moara::B_NCONTIG, 0, 0, 0, 0, moara::EPI_STORE};
        gemm(gram, [&](int i, moara::GemmProb& p) {
            const int l = it[i].l;
            p.A = Xin[i]; p.Bm = Xin[i]; p.C = it[i].Cg;
            p.M = l; p.N = l; p.K = rows[i]; p.lda = l; p.ldb = l; p.ldc = l;
            p.lower_only = 1;
        });
        cholesky_blocked(rows, shift_rel);
        tri_inverse(/*have_diag=*/true);
        moara::GemmKind apply{moara::A_KCONTIG, moara::B_KCONTIG, 0, 0, 0, 0, moara::EPI_STORE};
        gemm(apply, [&](int i, moara::GemmProb& p) {
            const int l = it[i].l;
            p.A = Xin[i]; p.Bm = it[i].Linv; p.C = Xout[i];
            p.M = rows[i]; p.N = l; p.K = l; p.lda = l; p.ldb = l; p.ldc = l;
            p.k_tri = moara::KTRI_B_UPPER;
            p.c_bf16 = bf != nullptr ? (*bf)[i] : nullptr;
        });
    }

    // Linv <- Cg^-1 for the lower-triangular Cholesky factor in Cg: diagonal
    // 64 x 64 blocks in shared memory, then the off-diagonal blocks level by
    // level (block size s = 64, 128, ...) with two grouped GEMMs per level:
    //   T = L[D, A] Linv[A, A];  Linv[D, A] = -Linv[D, D] T.
    // Lower Cholesky factor of Cg (+ shift on the diagonal) in place, by 64-wide
    // panels: factor the diagonal block (its inverse goes to the diagonal block
    // of Linv), solve the panel below it, update the trailing matrix.
    void cholesky_blocked(const std::vector<int>& rows, float shift_rel, bool fast = false) {
        int lmax = 0;
        moara::SmallBatch sb = small();
        sb.shift_rel = shift_rel;
        for (size_t i = 0; i < it.size(); ++i) {
            chk(cudaMemsetAsync(it[i].Linv, 0, sizeof(float) * (size_t)it[i].l * it[i].l, s));
            sb.l[i] = it[i].l; sb.rows[i] = rows[i]; sb.a[i] = it[i].Cg; sb.b[i] = it[i].scal;
            sb.c[i] = it[i].Linv; sb.fail[i] = it[i].fail;
            lmax = std::max(lmax, it[i].l);
        }
        chk(moara::launch_trace_shift(sb, s, &ctx->launches));
        const int nb = moara::kTriBase;
        moara::GemmKind solve{moara::A_KCONTIG, moara::B_KCONTIG, 0, 0, 0, 0, moara::EPI_STORE, 1};
        moara::GemmKind upd{moara::A_KCONTIG, moara::B_KCONTIG, 0, 0, 0, 0, moara::EPI_SUB, 1};
        for (int j0 = 0; j0 < lmax; j0 += nb) {
            chk(moara::launch_chol_diag(sb, j0, s, &ctx->launches));
            // fast: the 64-wide steps update only the rest of their
            // kFastPanel-wide panel; the trailing matrix past the panel gets
            // one tensor-core update per panel
            const int pend = fast ? (j0 / kFastPanel + 1) * kFastPanel : lmax;
            for (int pass = 0; pass < 2; ++pass) {
                moara::GemmBatch b{};
                b.B = 1;
                for (int i = 0; i < static_cast<int>(it.size()); ++i) {
                    const auto& x = it[i];
                    const long long l = x.l;
                    const int j1 = j0 + nb;
                    if (j1 >= x.l) continue;
                    const int cend = std::min(x.l, pend);
                    if (pass == 1 && cend <= j1) continue;
                    moara::GemmProb& p = b.p[b.count++];
                    p = moara::GemmProb{};
                    p.lda = p.ldb = p.ldc = x.l;
                    if (pass == 0) {      // L[j1:, panel] = A[j1:, panel] * Ljj^-T (in place)
                        p.A = x.Cg + j1 * l + j0;
                        p.Bm = x.Linv + j0 * l + j0;
                        p.C = x.Cg + j1 * l + j0;
                        p.M = x.l - j1; p.N = nb; p.K = nb;
                    } else {              // A[j1:, j1:cend] -= L[j1:, panel] L[j1:cend, panel]^T (lower tiles)
                        p.A = x.Cg + j1 * l + j0;
                        p.Bm = x.Cg + j1 * l + j0;
                        p.C = x.Cg + j1 * l + j1;
                        p.M = x.l - j1; p.N = cend - j1; p.K = nb;
                        p.lower_only = 1;
                    }
                }
                if (b.count > 0) chk(moara::launch_gemm(pass == 0 ? solve : upd, b, s, &ctx->launches));
            }
            if (fast && j0 + nb == pend) trailing_update_tc(pend);
        }
    }

    // A[pe:, pe:] -= L[pe:, pe - kFastPanel : pe] L[pe:, ...]^T (lower tiles)
    // for every item with l > pe, as a two-plane split-precision product
    // (16 significant bits): the panel's transposed planes go to P1.
    void trailing_update_tc(int pe) {
        moara::SmallBatch sq{};
        std::vector<moara::TcSplitGemmItem> g;
        for (size_t i = 0; i < it.size(); ++i) {
            const auto& x = it[i];
            if (x.l <= pe) continue;
            const int rest = x.l - pe;
            const int q = sq.count++;
            sq.a[q] = x.Cg + (size_t)pe * x.l + (pe - kFastPanel);
            sq.h[q] = x.P1;
            sq.rows[q] = rest;
            sq.l[q] = kFastPanel;
            sq.ld[q] = x.l;
            const size_t pl = (size_t)rest * kFastPanel;
            moara::TcSplitGemmItem item{x.P1, x.P1, pl, pl, x.Cg + (size_t)pe * x.l + pe, rest, rest, kFastPanel, 0};
            item.ldo = x.l;
            item.sub = 1;
            item.lower = 1;
            g.push_back(item);
        }
        if (g.empty()) return;
        chk(moara::launch_split3(sq, 1, s, &ctx->launches));
        ks_run(g, 2);
    }

    // One level of the blocked triangular inverse on tensor cores, for the
    // pairs (module, a0, d0, dn) of block size sz:
    //   T[D, A] = L[D, A] Linv[A, A];  Linv[D, A] = -Linv[D, D] T[D, A],
    // both as three-plane (24-bit) split-precision products.  Each pair's
    // operands are split into the module's P1 (A side) and P2 (B side)
    // planes at running offsets.  A level's pairs of one module cover
    // disjoint row blocks D, so the A sides need at most 3 sz (l - sz) <=
    // 3 l^2 / 4 entries; the B side of the first product, 3 sz^2 per pair
    // over at most (l - sz) / (2 sz) + 1 pairs, stays within 3 l^2.
    // Linv[D, A] is still zero here, so "out -= A B" gives the negated product.
    template <class PairAt>
    void tri_level_tc(int sz, size_t npairs, PairAt pair_at) {
        for (int pass = 0; pass < 2; ++pass) {
            std::vector<size_t> off_a(it.size(), 0), off_b(it.size(), 0);
            std::vector<moara::TcSplitGemmItem> items;
            moara::SmallBatch sa{}, sb{};
            auto flush_splits = [&]() {
                if (sa.count > 0) chk(moara::launch_split3(sa, 1, s, &ctx->launches));
                if (sb.count > 0) chk(moara::launch_split3(sb, 0, s, &ctx->launches));
                sa = moara::SmallBatch{};
                sb = moara::SmallBatch{};
            };
            for (size_t q = 0; q < npairs; ++q) {
                const std::array<int, 4> pr = pair_at(q);
                const auto& x = it[pr[0]];
                const long long l = x.l;
                const int a0 = pr[1], d0 = pr[2], dn = pr[3];
                const int K = pass == 0 ? sz : dn;
                // A is read as K x M (the transpose of the left factor), B as K x N
                const float* asrc = pass == 0 ? x.Cg + d0 * l + a0 : x.Linv + d0 * l + d0;
                const float* bsrc = pass == 0 ? x.Linv + a0 * l + a0 : x.Tt + d0 * l + a0;
                uint16_t* ap = x.P1 + off_a[pr[0]];
                uint16_t* bp = x.P2 + off_b[pr[0]];
                off_a[pr[0]] += 3 * (size_t)K * dn;
                off_b[pr[0]] += 3 * (size_t)K * sz;
                if (sa.count == moara::kMaxGroup) flush_splits();
                const int ia = sa.count++, ib = sb.count++;
                sa.a[ia] = const_cast<float*>(asrc); sa.h[ia] = ap; sa.rows[ia] = dn; sa.l[ia] = K; sa.ld[ia] = x.l;
                sb.a[ib] = const_cast<float*>(bsrc); sb.h[ib] = bp; sb.rows[ib] = K; sb.l[ib] = sz; sb.ld[ib] = x.l;
                moara::TcSplitGemmItem g{ap, bp, (size_t)K * dn, (size_t)K * sz,
                                         pass == 0 ? x.Tt + d0 * l + a0 : x.Linv + d0 * l + a0, dn, sz, K, 0};
                g.ldo = x.l;
                g.sub = pass == 1 ? 1 : 0;
                items.push_back(g);
            }
            flush_splits();
            ks_run(items, 3);
        }
    }

    void tri_inverse(bool have_diag) {
        int lmax = 0;
        for (auto& x : it) {
            if (!have_diag) chk(cudaMemsetAsync(x.Linv, 0, sizeof(float) * (size_t)x.l * x.l, s));
            lmax = std::max(lmax, x.l);
        }
        if (!have_diag) {
            moara::SmallBatch sb = small();
            for (size_t i = 0; i < it.size(); ++i) { sb.l[i] = it[i].l; sb.a[i] = it[i].Cg; sb.c[i] = it[i].Linv; }
            chk(moara::launch_tri_inverse_diag(sb, s, &ctx->launches));
        }
        moara::GemmKind mul{moara::A_KCONTIG, moara::B_NCONTIG, 0, 0, 0, 0, moara::EPI_STORE};
        moara::GemmKind neg{moara::A_KCONTIG, moara::B_NCONTIG, 0, 0, 0, 0, moara::EPI_STORE_NEG};
        const bool tc = !it.empty() && it[0].tc && ctx->tc != nullptr;
        for (int sz = moara::kTriBase; sz < lmax; sz *= 2) {
            struct Pair { int mod, a0, d0, dn; };
            std::vector<Pair> pairs;
            for (int i = 0; i < static_cast<int>(it.size()); ++i) {
                const int l = it[i].l;
                for (int a0 = 0; a0 + sz < l; a0 += 2 * sz)
                    pairs.push_back({i, a0, a0 + sz, std::min(sz, l - a0 - sz)});
            }
            if (tc && sz >= kTriTcMin) {
                tri_level_tc(sz, pairs.size(), [&](size_t q) {
                    const Pair& pr = pairs[q];
                    return std::array<int, 4>{pr.mod, pr.a0, pr.d0, pr.dn};
                });
                continue;
            }
            for (int pass = 0; pass < 2; ++pass) {
                for (size_t c0 = 0; c0 < pairs.size(); c0 += moara::kMaxGroup) {
                    moara::GemmBatch b{};
                    b.count = static_cast<int>(std::min<size_t>(moara::kMaxGroup, pairs.size() - c0));
                    b.B = 1;
                    for (int q = 0; q < b.count; ++q) {
                        const Pair& pr = pairs[c0 + q];
                        const auto& x = it[pr.mod];
                        const long long l = x.l;
                        moara::GemmProb& p = b.p[q];
                        p = moara::GemmProb{};
                        p.lda = p.ldb = p.ldc = x.l;
                        if (pass == 0) {          // T[D, A] = L[D, A] Linv[A, A]  (Linv[A, A] lower)
                            p.A = x.Cg + pr.d0 * l + pr.a0;
                            p.Bm = x.Linv + pr.a0 * l + pr.a0;
                            p.C = x.Tt + pr.d0 * l + pr.a0;
                            p.M = pr.dn; p.N = sz; p.K = sz;
                            p.k_tri = moara::KTRI_B_LOWER;
                        } else {                  // Linv[D, A] = -Linv[D, D] T[D, A]  (Linv[D, D] lower)
                            p.A = x.Linv + pr.d0 * l + pr.d0;
                            p.Bm = x.Tt + pr.d0 * l + pr.a0;
                            p.C = x.Linv + pr.d0 * l + pr.a0;
                            p.M = pr.dn; p.N = sz; p.K = pr.dn;
                            p.k_tri = moara::KTRI_A_LOWER;
                        }
                    }
                    chk(moara::launch_gemm(pass == 0 ? mul : neg, b, s, &ctx->launches));
                }
            }
        }
    }

    // CholeskyQR2 with a shifted first pass; result lands in `b` (and its bf16
    // copy in `bf` when given).
    void cholqr2s(std::vector<float*>& a, std::vector<float*>& b, const std::vector<int>& rows,
                  const std::vector<uint16_t*>* bf = nullptr) {
        const float u = 5.9604645e-08f;   // fp32 unit roundoff
        cholqr_pass(a, b, rows, 2.0f * u);
        cholqr_pass(b, a, rows, 0.0f, bf);
        std::swap(a, b);
    }

    // ---------------------------------------------- tensor-core helpers
    void tc_gemm(int a_kmajor, const std::vector<moara::TcGemmItem>& items) {
        if (items.empty()) return;
        ProfScope ps(ctx, MOARA_PHASE_TC_REFRESH, s);
        if (moara::tc_gemm_bf16(ctx->tc, a_kmajor, items.data(), static_cast<int>(items.size()), s,
                                &ctx->launches) != MOARA_OK)
            chk(cudaErrorLaunchFailure);
    }

    // out (n x l) = V^T X with X (m x l) in bf16; fp32 and/or bf16 output
    // (`lo` false: V_hi alone, for products whose output is rounded to bf16
    // anyway, the intermediate iterates of the subspace iteration)
    void tc_vt_times(const std::vector<uint16_t*>& X, const std::vector<float*>& out,
                     const std::vector<uint16_t*>& out_bf, bool lo = true) {
        // V stored m x n is read MN-major; for a transposed item (V^T) the
        // same product is V X with V read K-major
        std::vector<moara::TcGemmItem> g[2];
        for (size_t i = 0; i < it.size(); ++i) {
            const auto& x = it[i];
            g[x.trans ? 1 : 0].push_back({x.Vhi, lo ? x.Vlo : nullptr, X[i], out[i], out_bf[i], x.n, x.l, x.m, 0});
        }
        tc_gemm(0, g[0]);
        tc_gemm(1, g[1]);
    }

    // out (m x l) = V Z with Z (n x l) in bf16
    void tc_v_times(const std::vector<uint16_t*>& Z, const std::vector<float*>& out,
                    const std::vector<uint16_t*>& out_bf, bool lo = true) {
        std::vector<moara::TcGemmItem> g[2];
        for (size_t i = 0; i < it.size(); ++i) {
            const auto& x = it[i];
            g[x.trans ? 1 : 0].push_back({x.Vhi, lo ? x.Vlo : nullptr, Z[i], out[i], out_bf[i], x.m, x.l, x.n, 0});
        }
        tc_gemm(1, g[0]);
        tc_gemm(0, g[1]);
    }

    // One shifted CholeskyQR pass on tensor cores: X_out = X_in R^-1 with
    // R^T R = X_in^T X_in + shift, X_in and X_out bf16 (rows x l).  The Gram
    // matrix of the bf16 X_in is exact up to fp32 accumulation; R^-1 is
    // applied in bf16.  Upper-triangular R keeps the nested column spans of
    // X_in, which is all the subspace iteration needs from this step.
    void tc_cholqr_pass(const std::vector<uint16_t*>& Xin, const std::vector<uint16_t*>& Xout,
                        const std::vector<int>& rows, float shift_rel) {
        std::vector<moara::TcGemmItem> gram;
        for (size_t i = 0; i < it.size(); ++i) {
            const int l = it[i].l;
            moara::TcGemmItem g{Xin[i], nullptr, Xin[i], it[i].Cg, nullptr, l, l, rows[i], 0};
            g.lower = 1;                    // the Cholesky reads the lower triangle only
            gram.push_back(g);
        }
        tc_gemm(0, gram);
        cholesky_blocked(rows, shift_rel, /*fast=*/true);
        tri_inverse(/*have_diag=*/true);
        {   // (R^-1) in bf16: the transpose of the lower-triangular Linv, into Tt
            moara::SmallBatch sb = small();
            for (size_t i = 0; i < it.size(); ++i) {
                sb.a[i] = it[i].Linv; sb.h[i] = reinterpret_cast<uint16_t*>(it[i].Tt); sb.l[i] = it[i].l;
            }
            chk(moara::launch_transpose_bf16(sb, s, &ctx->launches));
        }
        std::vector<moara::TcGemmItem> apply;
        for (size_t i = 0; i < it.size(); ++i) {
            const int l = it[i].l;
            apply.push_back({Xin[i], nullptr, reinterpret_cast<const uint16_t*>(it[i].Tt), nullptr, Xout[i],
                             rows[i], l, l, 1});
        }
        tc_gemm(1, apply);
    }

    // ------------------------------------- split-precision l x l products
    void split3(const std::vector<float*>& src, const std::vector<uint16_t*>& dst, int transpose) {
        moara::SmallBatch sb = small();
        for (size_t i = 0; i < it.size(); ++i) {
            sb.a[i] = src[i]; sb.h[i] = dst[i]; sb.rows[i] = it[i].l; sb.l[i] = it[i].l;
        }
        chk(moara::launch_split3(sb, transpose, s, &ctx->launches));
    }

    // planes = 3: fp32-accurate operands; 2: hi + mid (16 bits), for iterates
    // that a later fp32-accurate pass corrects
    void ks_run(const std::vector<moara::TcSplitGemmItem>& g, int planes) {
        ProfScope ps(ctx, MOARA_PHASE_TC_REFRESH, s);
        if (moara::tc_gemm_split3(ctx->tc, g.data(), static_cast<int>(g.size()), planes, s, &ctx->launches) !=
            MOARA_OK)
            chk(cudaErrorLaunchFailure);
    }

    // out = A B (l x l) from three-plane operands (A stored K x M, B K x N)
    void ks_gemm(const std::vector<uint16_t*>& A, const std::vector<uint16_t*>& B, const std::vector<float*>& out,
                 int ktri, int planes) {
        std::vector<moara::TcSplitGemmItem> g;
        for (size_t i = 0; i < it.size(); ++i) {
            const int l = it[i].l;
            const size_t pl = (size_t)l * l;
            g.push_back({A[i], B[i], pl, pl, out[i], l, l, l, ktri});
        }
        ks_run(g, planes);
    }

    // Shifted CholeskyQR pass of a tall X (rows x l, rows % 8 == 0) with the
    // Gram matrix X^T X (K = rows) and the triangular apply X R^-1 as
    // split-precision tensor-core products; X is replaced in place (the apply
    // reads only the planes).  `pl` holds 3 * rows * l bf16 entries: the
    // planes of X for the Gram matrix, then those of X^T for the apply.
    void ks_cholqr_tall(std::vector<float*>& X, const std::vector<uint16_t*>& pl, const std::vector<int>& rows,
                        float shift_rel, int planes, bool fast_chol = true) {
        const size_t n_it = it.size();
        auto split_rows = [&](int transpose) {
            moara::SmallBatch sb = small();
            for (size_t i = 0; i < n_it; ++i) {
                sb.a[i] = X[i]; sb.h[i] = pl[i]; sb.rows[i] = rows[i]; sb.l[i] = it[i].l;
            }
            chk(moara::launch_split3(sb, transpose, s, &ctx->launches));
        };
        split_rows(0);                      // X stored K x M (and K x N): rows x l
        std::vector<moara::TcSplitGemmItem> g;
        for (size_t i = 0; i < n_it; ++i) {
            const int l = it[i].l;
            const size_t pm = (size_t)rows[i] * l;
            g.push_back({pl[i], pl[i], pm, pm, it[i].Cg, l, l, rows[i], 0});
        }
        ks_run(g, planes);                  // Gram X^T X
        cholesky_blocked(rows, shift_rel, fast_chol);
        tri_inverse(/*have_diag=*/true);
        std::vector<float*> linv(n_it);
        std::vector<uint16_t*> p2(n_it);
        for (size_t i = 0; i < n_it; ++i) { linv[i] = it[i].Linv; p2[i] = it[i].P2; }
        split3(linv, p2, 1);                // B = Linv^T (upper triangular)
        split_rows(1);                      // A = X stored K x M: its transpose, l x rows
        g.clear();
        for (size_t i = 0; i < n_it; ++i) {
            const int l = it[i].l;
            g.push_back({pl[i], p2[i], (size_t)rows[i] * l, (size_t)l * l, X[i], rows[i], l, l, 1});
        }
        ks_run(g, planes);
    }

    // One CholeskyQR pass on an l x l matrix with the Gram matrix and the
    // triangular apply as split-precision tensor-core products (fp32-accurate):
    // Xout = Win R^-1, R^T R = Win^T Win + shift.
    void ks_cholqr_pass(std::vector<float*>& Win, std::vector<float*>& Xout, const std::vector<int>& rows_l,
                        float shift_rel, int planes, bool fast_chol = true) {
        std::vector<uint16_t*> p1(it.size()), p2(it.size());
        for (size_t i = 0; i < it.size(); ++i) { p1[i] = it[i].P1; p2[i] = it[i].P2; }
        std::vector<float*> cg(it.size());
        for (size_t i = 0; i < it.size(); ++i) cg[i] = it[i].Cg;
        split3(Win, p1, 0);                 // W (as A = W^T, MN-major, and as B)
        ks_gemm(p1, p1, cg, 0, planes);     // Gram W^T W
        cholesky_blocked(rows_l, shift_rel, fast_chol);
        tri_inverse(/*have_diag=*/true);
        std::vector<float*> linv(it.size());
        for (size_t i = 0; i < it.size(); ++i) linv[i] = it[i].Linv;
        split3(linv, p2, 1);                // B = Linv^T (upper triangular)
        split3(Win, p1, 1);                 // A = W read MN-major: its transpose
        ks_gemm(p1, p2, Xout, 1, planes);
    }

    void run() {
        const int n_it = static_cast<int>(it.size());
        const moara_hparams& hp = ctx->hp;
        const bool tc = n_it > 0 && it[0].tc;   // groups are all tensor-core or all fp32
        for (auto& x : it) chk(cudaMemsetAsync(x.fail, 0, sizeof(int), s));
        // Decompose(G, B) when the source is V: fp32 block scales for the fp32
        // products, bf16 planes V_hi + V_lo for the tensor-core ones
        if (src_v && !tc) {
            moara::DecompBatch db{};
            db.count = n_it; db.B = hp.block_size; db.do_mag = 0; db.decomp_eps = hp.decomp_eps;
            long long acc = 0;
            for (int i = 0; i < n_it; ++i) {
                db.item_start[i] = acc;
                db.p[i] = moara::DecompItem{it[i].G, it[i].inv, nullptr, nullptr, nullptr,
                                            it[i].m, it[i].n, it[i].kb, it[i].dtype};
                acc += (long long)it[i].m * it[i].kb;
            }
            db.item_start[n_it] = acc;
            chk(moara::launch_decompose(db, s, &ctx->launches));
        }
        if (src_v && tc) {
            std::vector<moara::TcSplitItem> sp;
            for (auto& x : it) sp.push_back({x.G, x.Vhi_w, x.Vlo, x.trans ? x.n : x.m, x.trans ? x.m : x.n});
            if (moara::tc_split_v(ctx->tc, sp.data(), n_it, hp.block_size, hp.decomp_eps, s, &ctx->launches) !=
                MOARA_OK)
                chk(cudaErrorLaunchFailure);
        }
        // Gaussian test matrix Omega (n x l)
        {
            moara::SmallBatch sb = small();
            for (int i = 0; i < n_it; ++i) {
                sb.a[i] = it[i].Omega; sb.rows[i] = it[i].n; sb.l[i] = it[i].l; sb.key[i] = it[i].key;
            }
            chk(moara::launch_philox_gaussian(sb, s, &ctx->launches));
        }
        std::vector<float*> Qa(n_it), Qb(n_it), Za(n_it), Zb(n_it), Xa(n_it), Xb(n_it);
        std::vector<int> rows_m(n_it), rows_n(n_it), rows_l(n_it);
        std::vector<uint16_t*> qbf(n_it), zbf(n_it), ybf(n_it), zraw(n_it);
        std::vector<float*> nof(n_it, nullptr);
        std::vector<uint16_t*> nob(n_it, nullptr);
        for (int i = 0; i < n_it; ++i) {
            Qa[i] = it[i].Qa; Qb[i] = it[i].Qb; Za[i] = it[i].Za; Zb[i] = it[i].Zb;
            Xa[i] = it[i].Xa; Xb[i] = it[i].Xb;
            rows_m[i] = it[i].m; rows_n[i] = it[i].n; rows_l[i] = it[i].l;
            qbf[i] = it[i].Qbf; zbf[i] = it[i].Zbf;
            // bf16 iterates of the tensor-core power iterations live in the
            // fp32 buffers (4 bytes per entry hold the 2-byte plane)
            ybf[i] = reinterpret_cast<uint16_t*>(it[i].Qa);
            zraw[i] = reinterpret_cast<uint16_t*>(it[i].Za);
        }
        const float u_rnd = 5.9604645e-08f;   // fp32 unit roundoff
        // split-precision tensor-core products with the tall Q need its row
        // count to be a multiple of 8 (TMA row pitch of Q^T)
        bool tall_ks = tc;
        for (int i = 0; i < n_it; ++i) tall_ks = tall_ks && rows_m[i] % 8 == 0;
        if (tc) {
            // Subspace iteration with every product and every intermediate
            // orthonormalisation on tensor cores; only the last Y gets the
            // fp32 CholeskyQR2 that makes Q orthonormal for the Rayleigh-Ritz step.
            for (int i = 0; i < n_it; ++i)
                chk(moara::launch_f32_to_bf16(it[i].Omega, nullptr, it[i].Zbf, (long long)it[i].n * it[i].l, s,
                                              &ctx->launches));
            const int q_it = hp.power_iters;
            if (q_it == 0) {
                tc_v_times(zbf, Qa, nob);
            } else {
                // the iterates rounded to bf16 take V_hi alone; the last Y and
                // the Rayleigh-Ritz product take V_hi + V_lo
                tc_v_times(zbf, nof, ybf, false);
                tc_cholqr_pass(ybf, qbf, rows_m, 2.0f * u_rnd);
                for (int q = 0; q < q_it; ++q) {
                    tc_vt_times(qbf, nof, zraw, false);
                    tc_cholqr_pass(zraw, zbf, rows_n, 2.0f * u_rnd);
                    if (q + 1 < q_it) {
                        tc_v_times(zbf, nof, ybf, false);
                        tc_cholqr_pass(ybf, qbf, rows_m, 2.0f * u_rnd);
                    } else {
                        tc_v_times(zbf, Qa, nob);
                    }
                }
            }
            if (tall_ks) {
                // shifted first pass on tensor cores (the planes of Q fill the
                // Qbf / Qb pair), the pass that fixes Q's orthonormality on the
                // fp32 units
                std::vector<uint16_t*> qpl(n_it);
                for (int i = 0; i < n_it; ++i) qpl[i] = it[i].Qbf;
                ks_cholqr_tall(Qa, qpl, rows_m, 2.0f * u_rnd, 2);
                // the second pass with three-plane (24-bit) operands and an
                // fp32 Cholesky: the tensor cores' accumulation leaves the
                // Gram matrix's diagonal short by ~1e-5 (relative), which
                // scales Q's columns alike and is removed by the unit-length
                // store of P; the off-diagonal orthogonality it gives is that
                // of the fp32 pass
                ks_cholqr_tall(Qa, qpl, rows_m, 0.0f, 3, /*fast_chol=*/false);
                for (int i = 0; i < n_it; ++i)                  // Q in Qb (fp32) and qbf
                    chk(moara::launch_f32_to_bf16(Qa[i], Qb[i], qbf[i], (long long)it[i].m * it[i].l, s,
                                                  &ctx->launches));
            } else {
                cholqr2s(Qa, Qb, rows_m, &qbf);             // Q in Qb (fp32) and qbf
            }
            // Rayleigh-Ritz matrix C = Z^T Z with Z = V^T Q (bf16 operands)
            tc_vt_times(qbf, nof, zraw);
            std::vector<moara::TcGemmItem> gram;
            for (int i = 0; i < n_it; ++i)
                gram.push_back({zraw[i], nullptr, zraw[i], it[i].Cr, nullptr, it[i].l, it[i].l, it[i].n, 0});
            tc_gemm(0, gram);
        } else {
            // Y = V * Z  (m x l), fp32 SIMT products (V scaled on the fly)
            auto v_times = [&](std::vector<float*>& rhs, std::vector<float*>& out) {
                for (int d = 0; d < 2; ++d) {  // per-dtype sub-batches
                    std::vector<int> sel;
                    for (int i = 0; i < n_it; ++i) if ((it[i].dtype == MOARA_DTYPE_BF16) == (d == 1)) sel.push_back(i);
                    if (sel.empty()) continue;
                    moara::GemmKind k{moara::A_KCONTIG, moara::B_NCONTIG, src_v, 0, d, 0, moara::EPI_STORE};
                    moara::GemmBatch b{};
                    b.count = static_cast<int>(sel.size());
                    b.B = hp.block_size;
                    for (int q = 0; q < b.count; ++q) {
                        const auto& x = it[sel[q]];
                        moara::GemmProb& p = b.p[q];
                        p = moara::GemmProb{};
                        p.A = x.G; p.a_inv = x.inv; p.Bm = rhs[sel[q]]; p.C = out[sel[q]];
                        p.M = x.m; p.N = x.l; p.K = x.n; p.lda = x.n; p.ldb = x.l; p.ldc = x.l; p.kb = x.kb;
                        p.a_bf16 = d;
                    }
                    chk(moara::launch_gemm(k, b, s, &ctx->launches));
                }
            };
            // Z = V^T * Q  (n x l)
            auto vt_times = [&](std::vector<float*>& rhs, std::vector<float*>& out) {
                for (int d = 0; d < 2; ++d) {
                    std::vector<int> sel;
                    for (int i = 0; i < n_it; ++i) if ((it[i].dtype == MOARA_DTYPE_BF16) == (d == 1)) sel.push_back(i);
                    if (sel.empty()) continue;
                    moara::GemmKind k{moara::A_MCONTIG, moara::B_NCONTIG, src_v, 0, d, 0, moara::EPI_STORE};
                    moara::GemmBatch b{};
                    b.count = static_cast<int>(sel.size());
                    b.B = hp.block_size;
                    for (int q = 0; q < b.count; ++q) {
                        const auto& x = it[sel[q]];
                        moara::GemmProb& p = b.p[q];
                        p = moara::GemmProb{};
                        p.A = x.G; p.a_inv = x.inv; p.Bm = rhs[sel[q]]; p.C = out[sel[q]];
                        p.M = x.n; p.N = x.l; p.K = x.m; p.lda = x.n; p.ldb = x.l; p.ldc = x.l; p.kb = x.kb;
                        p.a_bf16 = d;
                    }
                    chk(moara::launch_gemm(k, b, s, &ctx->launches));
                }
            };
            v_times(Za, Qa);
            cholqr2s(Qa, Qb, rows_m);          // Q in Qb
            // power iterations Y = V (V^T Q): Z = V^T Q gets one shifted CholeskyQR
            // pass (enough to keep V Z well conditioned), Y the full two passes
            for (int q = 0; q < hp.power_iters; ++q) {
                vt_times(Qb, Za);
                cholqr_pass(Za, Zb, rows_n, 2.0f * u_rnd);   // Z in Zb
                v_times(Zb, Qa);
                cholqr2s(Qa, Qb, rows_m);                    // Q in Qb
            }
            // Rayleigh-Ritz matrix C = (V^T Q)^T (V^T Q)
            vt_times(Qb, Za);
            moara::GemmKind gram{moara::A_MCONTIG, moara::B_NCONTIG, 0, 0, 0, 0, moara::EPI_STORE};
            gemm(gram, [&](int i, moara::GemmProb& p) {
                const int l = it[i].l;
                p.A = Za[i]; p.Bm = Za[i]; p.C = it[i].Cr;
                p.M = l; p.N = l; p.K = it[i].n; p.lda = l; p.ldb = l; p.ldc = l;
            });
        }
        // Eigenvectors of C by orthogonal iteration X <- C X with CholeskyQR2
        // (shifted, then plain) every iteration: each X is orthonormal, so
        // directions of C below its rounding level only ever fill an
        // orthonormal completion.  Then the Ritz order.  On the tensor-core
        // path the l x l products run as split-precision (3 x bf16) MMAs.
        {
            moara::SmallBatch sb = small();
            for (int i = 0; i < n_it; ++i) { sb.a[i] = Xa[i]; sb.l[i] = it[i].l; }
            chk(moara::launch_set_identity(sb, s, &ctx->launches));
        }
        moara::GemmKind prod{moara::A_KCONTIG, moara::B_NCONTIG, 0, 0, 0, 0, moara::EPI_STORE};
        std::vector<uint16_t*> cp(n_it), p1(n_it);
        for (int i = 0; i < n_it; ++i) { cp[i] = it[i].Cp; p1[i] = it[i].P1; }
        std::vector<float*> cr(n_it);
        for (int i = 0; i < n_it; ++i) cr[i] = it[i].Cr;
        if (tc) split3(cr, cp, 0);          // C is symmetric: read MN-major as A
        for (int q = 0; q < hp.ritz_iters; ++q) {
            if (tc) {
                // the iterations before the last carry hi + mid planes (16
                // bits): the later iterations correct them
                const bool last = q + 1 == hp.ritz_iters;
                const int planes = last ? 3 : 2;
                split3(Xa, p1, 0);
                ks_gemm(cp, p1, Xb, 0, planes);          // W = C X
                ks_cholqr_pass(Xb, Xa, rows_l, 2.0f * u_rnd, planes);
                // the pass that fixes the final orthonormality of X: three
                // planes and an fp32 Cholesky (the tensor cores' short
                // diagonal of the Gram matrix scales the columns of X alike;
                // P's columns are stored at unit length)
                ks_cholqr_pass(Xa, Xb, rows_l, 0.0f, planes, /*fast_chol=*/!last);
                std::swap(Xa, Xb);                       // X in Xa
            } else {
                gemm(prod, [&](int i, moara::GemmProb& p) {
                    const int l = it[i].l;
                    p.A = it[i].Cr; p.Bm = Xa[i]; p.C = Xb[i];
                    p.M = l; p.N = l; p.K = l; p.lda = l; p.ldb = l; p.ldc = l;
                });
                cholqr2s(Xb, Xa, rows_l);      // X in Xa
            }
        }
        // Ritz values (Rayleigh quotients of the columns of X) and order:
        // W = C X into Xb
        if (tc) {
            split3(Xa, p1, 0);
            ks_gemm(cp, p1, Xb, 0, 3);
        } else {
            gemm(prod, [&](int i, moara::GemmProb& p) {
                const int l = it[i].l;
                p.A = it[i].Cr; p.Bm = Xa[i]; p.C = Xb[i];
                p.M = l; p.N = l; p.K = l; p.lda = l; p.ldb = l; p.ldc = l;
            });
        }
        {
            // exact Rayleigh-Ritz within the leading 64 columns (Jacobi), so
            // that the separated leading eigenvectors are exact whatever the
            // number of orthogonal iterations; then the Ritz order
            moara::SmallBatch sb = small();
            for (int i = 0; i < n_it; ++i) {
                sb.a[i] = Xa[i]; sb.b[i] = Xb[i]; sb.c[i] = it[i].ritz; sb.iaux[i] = it[i].perm;
                sb.l[i] = it[i].l;
            }
            chk(moara::launch_lead_ritz(sb, s, &ctx->launches));
            chk(moara::launch_ritz_sort(sb, s, &ctx->launches));
        }
        {   // Xs (l x r) = X[:, perm[:r]] into Xb
            moara::SmallBatch sb = small();
            for (int i = 0; i < n_it; ++i) {
                sb.a[i] = Xa[i]; sb.c[i] = Xb[i]; sb.iaux[i] = it[i].perm;
                sb.l[i] = it[i].l; sb.rows[i] = it[i].r;
            }
            chk(moara::launch_gather_cols(sb, s, &ctx->launches));
        }
        // P_tmp (m x r) = Q * Xs; the store below scales every column to unit
        // length
        std::vector<float*> ptmp(n_it);
        if (tall_ks) {
            // three-plane split-precision product: the planes of Q^T fill the
            // Qa / Qbf pair (Q itself is in Qb), those of Xs the P1 region;
            // P_tmp overwrites Q, which the product no longer reads.  The
            // tensor cores' accumulation leaves the column norms ~1e-5 short;
            // the unit-length store removes that.
            moara::SmallBatch sq = small(), sx = small();
            for (int i = 0; i < n_it; ++i) {
                sq.a[i] = Qb[i]; sq.h[i] = reinterpret_cast<uint16_t*>(it[i].Qa); sq.rows[i] = it[i].m;
                sq.l[i] = it[i].l;
                sx.a[i] = Xb[i]; sx.h[i] = it[i].P1; sx.rows[i] = it[i].l; sx.l[i] = it[i].r;
            }
            chk(moara::launch_split3(sq, 1, s, &ctx->launches));
            chk(moara::launch_split3(sx, 0, s, &ctx->launches));
            std::vector<moara::TcSplitGemmItem> g;
            for (int i = 0; i < n_it; ++i) {
                g.push_back({reinterpret_cast<uint16_t*>(it[i].Qa), it[i].P1, (size_t)it[i].m * it[i].l,
                             (size_t)it[i].l * it[i].r, Qb[i], it[i].m, it[i].r, it[i].l, 0});
                ptmp[i] = Qb[i];
            }
            ks_run(g, 3);
        } else {
            gemm(prod, [&](int i, moara::GemmProb& p) {
                p.A = Qb[i]; p.Bm = Xb[i]; p.C = Qa[i];
                p.M = it[i].m; p.N = it[i].r; p.K = it[i].l; p.lda = it[i].l; p.ldb = it[i].r; p.ldc = it[i].r;
            });
            ptmp = Qa;
        }
        {
            moara::SmallBatch sb = small();
            for (int i = 0; i < n_it; ++i) {
                sb.a[i] = ptmp[i]; sb.c[i] = it[i].P; sb.h[i] = it[i].Pb; sb.fail[i] = it[i].fail;
                sb.rows[i] = it[i].m; sb.l[i] = it[i].r;
            }
            chk(moara::launch_sign_fix_store(sb, s, &ctx->launches));
        }
    }
};

int do_refresh(moara_ctx* ctx, int n_mod, const int* ids, const void* const* G, cudaStream_t s) {
    const moara_hparams& hp = ctx->hp;
    const int src_v = (hp.refresh_src == MOARA_REFRESH_SRC_V && hp.decompose) ? 1 : 0;
    // Modules whose step runs on tensor cores refresh there too (their bf16
    // planes of Q and Z need l % 8 == 0 for the TMA row pitch); the others use
    // the fp32 path.  Each kind is grouped so that a group fits the workspace.
    std::vector<int> kinds[2];
    for (int i = 0; i < n_mod; ++i) {
        const moara_module_desc& d = ctx->mods[ids[i]];
        const int l = refresh_l(ctx, d.m, d.n, d.r);
        kinds[(use_tc(ctx, ids[i]) && (l % 8) == 0) ? 1 : 0].push_back(i);
    }
    for (int kind = 0; kind < 2; ++kind) {
        const std::vector<int>& sel = kinds[kind];
        size_t start = 0;
        while (start < sel.size()) {
            RefreshRunner rr{ctx, s, {}, src_v};
            size_t used = 0;
            size_t end = start;
            while (end < sel.size() && static_cast<int>(rr.it.size()) < moara::kMaxGroup) {
                const int gi = sel[end];
                const int id = ids[gi];
                const moara_module_desc& d = ctx->mods[id];
                const bool tr = ctx->moddev[id].right != 0;   // right projector: the refresh of V^T
                if (tr && kind == 0)
                    return fail(ctx, MOARA_ERR_UNSUPPORTED,
                                "module %d: a right projector is refreshed on tensor cores only (r + p a multiple of 8)",
                                id);
                const int rm = tr ? d.n : d.m, rn = tr ? d.m : d.n;
                const int l = refresh_l(ctx, d.m, d.n, d.r);
                const size_t need = align_up(moara::refresh_ws_bytes(rm, rn, d.r, l, hp.block_size, src_v), 256);
                if (used + need > ctx->refresh_ws_bytes) {
                    if (rr.it.empty())
                        return fail(ctx, MOARA_ERR_WORKSPACE,
                                    "refresh workspace of %zu bytes is smaller than the %zu bytes module %d needs",
                                    ctx->refresh_ws_bytes, need, id);
                    break;
                }
                moara::RefreshItem x{};
                x.m = rm; x.n = rn; x.r = d.r; x.l = l; x.kb = blocks_of(d.n, hp.block_size);
                x.trans = tr ? 1 : 0;
                x.dtype = d.grad_dtype; x.G = G[gi];
                moara::refresh_carve(x, static_cast<char*>(ctx->refresh_ws) + used, rm, rn, d.r, l,
                                     hp.block_size, src_v);
                x.P = d.P; x.Pb = d.P_bf16;
                const uint64_t cnt = static_cast<uint64_t>(ctx->refresh_count[id]++);
                x.key = hp.seed ^ (0x9E3779B97F4A7C15ull * (static_cast<uint64_t>(id) + 1)) ^
                        (cnt * 0xD1B54A32D192ED03ull);
                if (kind == 1) {
                    const moara::ModDev& md = ctx->moddev[id];
                    x.tc = 1;
                    if (src_v) {
                        x.Vhi = md.ws_Vhi; x.Vhi_w = md.ws_Vhi; x.Vlo = md.ws_Vlo;
                    } else {
                        x.Vhi = static_cast<const uint16_t*>(G[gi]); x.Vhi_w = nullptr; x.Vlo = nullptr;
                    }
                }
                rr.it.push_back(x);
                used += need;
                ++end;
            }
            rr.run();
            // a right projector's K2 operand is Q^T
            for (size_t q = start; q < end && rr.err == cudaSuccess; ++q) {
                const moara::ModDev& md = ctx->moddev[ids[sel[q]]];
                if (md.right) rr.chk(moara::tc_transpose_bf16(md.Pb, md.ws_Qt, md.n, md.r, s, &ctx->launches));
            }
            if (rr.err != cudaSuccess) {
                if (kind == 1 && ctx->tc != nullptr)
                    return fail(ctx, MOARA_ERR_CUDA, "tensor-core refresh: %s", moara::tc_last_error(ctx->tc));
                return cuda_fail(ctx, rr.err, "refresh launch");
            }
            start = end;
        }
    }
    return MOARA_OK;
}

// ------------------------------------------------------------------ step
int do_step_simt(moara_ctx* ctx, const std::vector<int>& sel, const int* ids, const void* const* G,
                 int64_t t, float lr, const float* clip, cudaStream_t s) {
    const moara_hparams& hp = ctx->hp;
    const double bc1 = 1.0 - std::pow((double)hp.beta1, (double)t);
    const double bc2 = 1.0 - std::pow((double)hp.beta2, (double)t);
    // longest K (= m for the projection) first
    std::vector<int> order(sel);
    std::stable_sort(order.begin(), order.end(), [&](int a, int b) {
        return ctx->mods[ids[a]].m > ctx->mods[ids[b]].m;
    });
    for (size_t c0 = 0; c0 < order.size(); c0 += moara::kMaxGroup) {
        const int cnt = static_cast<int>(std::min<size_t>(moara::kMaxGroup, order.size() - c0));
        if (hp.decompose) {
            moara::DecompBatch db{};
            db.count = cnt; db.B = hp.block_size; db.do_mag = 1; db.decomp_eps = hp.decomp_eps;
            db.beta1 = hp.beta1; db.beta2 = hp.beta2; db.adam_eps = hp.adam_eps;
            db.bc1 = static_cast<float>(bc1); db.bc2 = static_cast<float>(bc2);
            db.clip = clip;
            long long acc = 0;
            for (int q = 0; q < cnt; ++q) {
                const int i = order[c0 + q];
                const moara::ModDev& md = ctx->moddev[ids[i]];
                db.item_start[q] = acc;
                db.p[q] = moara::DecompItem{G[i], md.ws_inv, md.mag_avg, md.mag_avg_sq, md.ws_dM,
                                            md.m, md.n, md.kb, md.dtype};
                acc += (long long)md.m * md.kb;
            }
            db.item_start[cnt] = acc;
            cudaError_t e;
            {
                ProfScope ps(ctx, MOARA_PHASE_DECOMPOSE, s);
                e = moara::launch_decompose(db, s, &ctx->launches);
            }
            if (e != cudaSuccess) return cuda_fail(ctx, e, "decompose launch");
        }
        // projection + direction Adam, split by gradient dtype
        for (int d = 0; d < 2; ++d) {
            moara::GemmBatch b{};
            b.B = hp.block_size; b.beta1 = hp.beta1; b.beta2 = hp.beta2; b.adam_eps = hp.adam_eps;
            b.bc1 = static_cast<float>(bc1); b.bc2 = static_cast<float>(bc2);
            b.clip = hp.decompose ? nullptr : clip;   // with the decomposition V is unchanged
            for (int q = 0; q < cnt; ++q) {
                const int i = order[c0 + q];
                const moara::ModDev& md = ctx->moddev[ids[i]];
                if ((md.dtype == MOARA_DTYPE_BF16) != (d == 1)) continue;
                moara::GemmProb& p = b.p[b.count++];
                p = moara::GemmProb{};
                p.A = md.P; p.Bm = G[i]; p.b_inv = hp.decompose ? md.ws_inv : nullptr;
                p.C = md.ws_N; p.aux0 = md.exp_avg; p.aux1 = md.exp_avg_sq;
                p.M = md.r; p.N = md.n; p.K = md.m; p.lda = md.r; p.ldb = md.n; p.ldc = md.n;
                p.kb = md.kb; p.b_bf16 = d;
            }
            moara::GemmKind k{moara::A_MCONTIG, moara::B_NCONTIG, 0, hp.decompose, 0, d, moara::EPI_ADAM};
            if (b.count == 0) continue;
            cudaError_t e;
            {
                ProfScope ps(ctx, MOARA_PHASE_PROJECT, s);
                e = moara::launch_gemm(k, b, s, &ctx->launches);
            }
            if (e != cudaSuccess) return cuda_fail(ctx, e, "projection launch");
        }
        // back-projection + weight update
        {
            moara::GemmBatch b{};
            b.B = hp.block_size;
            b.step_scale = lr * hp.scale;
            for (int q = 0; q < cnt; ++q) {
                const int i = order[c0 + q];
                const moara::ModDev& md = ctx->moddev[ids[i]];
                moara::GemmProb& p = b.p[b.count++];
                p = moara::GemmProb{};
                p.A = md.P; p.Bm = md.ws_N; p.aux0 = md.W; p.aux2 = hp.decompose ? md.ws_dM : nullptr;
                p.M = md.m; p.N = md.n; p.K = md.r; p.lda = md.r; p.ldb = md.n; p.ldc = md.n; p.kb = md.kb;
            }
            moara::GemmKind k{moara::A_KCONTIG, moara::B_NCONTIG, 0, 0, 0, 0, moara::EPI_UPDATE};
            cudaError_t e;
            {
                ProfScope ps(ctx, MOARA_PHASE_BACKPROJECT, s);
                e = moara::launch_gemm(k, b, s, &ctx->launches);
            }
            if (e != cudaSuccess) return cuda_fail(ctx, e, "back-projection launch");
        }
    }
    return MOARA_OK;
}

int check_ids(moara_ctx* ctx, int n_mod, const int* ids, const void* const* G) {
    if (n_mod < 0) return fail(ctx, MOARA_ERR_INVALID_ARG, "n_mod must be >= 0");
    if (n_mod > 0 && (ids == nullptr || G == nullptr))
        return fail(ctx, MOARA_ERR_INVALID_ARG, "ids and G must not be NULL");
    std::vector<char> seen(ctx->mods.size(), 0);
    for (int i = 0; i < n_mod; ++i) {
        if (ids[i] < 0 || ids[i] >= static_cast<int>(ctx->mods.size()))
            return fail(ctx, MOARA_ERR_UNKNOWN_MODULE, "module id %d is not registered", ids[i]);
        if (seen[ids[i]]) return fail(ctx, MOARA_ERR_INVALID_ARG, "module id %d listed twice", ids[i]);
        seen[ids[i]] = 1;
        if (G[i] == nullptr) return fail(ctx, MOARA_ERR_INVALID_ARG, "G[%d] is NULL", i);
        if (!aligned16(G[i])) return fail(ctx, MOARA_ERR_ALIGN, "G[%d] is not 16-byte aligned", i);
    }
    return MOARA_OK;
}

}  // namespace

extern "C" {

int moara_default_hparams(moara_hparams* out) {
    if (out == nullptr) return MOARA_ERR_INVALID_ARG;
    std::memset(out, 0, sizeof(*out));
    out->beta1 = 0.9f;
    out->beta2 = 0.999f;
    out->adam_eps = 1e-6f;
    out->decomp_eps = 1e-12f;
    out->scale = 0.25f;
    out->block_size = 128;
    out->refresh_interval = 200;
    out->decompose = 1;
    out->refresh_src = MOARA_REFRESH_SRC_V;
    out->oversample = 32;
    out->power_iters = 4;
    out->ritz_iters = 3;
    out->precision = MOARA_PREC_AUTO;
    out->seed = 0;
    return MOARA_OK;
}

int moara_create(moara_ctx** out, const moara_hparams* hp, int device) {
    if (out == nullptr) return MOARA_ERR_INVALID_ARG;
    *out = nullptr;
    moara_ctx tmp;
    int rc = check_hparams(&tmp, hp);
    if (rc != MOARA_OK) return rc;
    int ndev = 0;
    if (cudaGetDeviceCount(&ndev) != cudaSuccess || device < 0 || device >= ndev) return MOARA_ERR_CUDA;
    moara_ctx* ctx = new (std::nothrow) moara_ctx();
    if (ctx == nullptr) return MOARA_ERR_INVALID_ARG;
    ctx->device = device;
    ctx->hp = *hp;
    DeviceGuard g(device);
    ctx->cap = 1024;
    if (cudaMalloc(&ctx->d_mods, sizeof(moara::ModDev) * ctx->cap) != cudaSuccess ||
        cudaMalloc(&ctx->d_status, sizeof(int) * 4) != cudaSuccess ||
        cudaMallocHost(&ctx->h_status, sizeof(int) * 4) != cudaSuccess ||
        cudaMemset(ctx->d_status, 0, sizeof(int) * 4) != cudaSuccess ||
        cudaMalloc(&ctx->d_clip, sizeof(float) * 2) != cudaSuccess ||
        cudaMemset(ctx->d_clip, 0, sizeof(float) * 2) != cudaSuccess) {
        moara_destroy(ctx);
        return MOARA_ERR_CUDA;
    }
    ctx->tc = moara::tc_create(device, ctx->d_status);
    *out = ctx;
    return MOARA_OK;
}

void moara_destroy(moara_ctx* ctx) {
    if (ctx == nullptr) return;
    DeviceGuard g(ctx->device);
    if (ctx->tc) moara::tc_destroy(ctx->tc);
    if (ctx->copy_stream) cudaStreamSynchronize(ctx->copy_stream);
    for (int b = 0; b < 2; ++b) {
        if (ctx->stage[b]) cudaFree(ctx->stage[b]);
        if (ctx->copy_done[b]) cudaEventDestroy(ctx->copy_done[b]);
        if (ctx->compute_done[b]) cudaEventDestroy(ctx->compute_done[b]);
    }
    if (ctx->copy_stream) cudaStreamDestroy(ctx->copy_stream);
    for (auto& r : ctx->recs) { cudaEventDestroy(r.a); cudaEventDestroy(r.b); }
    for (auto e : ctx->free_events) cudaEventDestroy(e);
    if (ctx->d_mods) cudaFree(ctx->d_mods);
    if (ctx->d_status) cudaFree(ctx->d_status);
    if (ctx->h_status) cudaFreeHost(ctx->h_status);
    if (ctx->align_acc) cudaFree(ctx->align_acc);
    if (ctx->d_clip) cudaFree(ctx->d_clip);
    if (ctx->d_clip_part) cudaFree(ctx->d_clip_part);
    delete ctx;
}

int moara_get_hparams(const moara_ctx* ctx, moara_hparams* out) {
    if (ctx == nullptr || out == nullptr) return MOARA_ERR_INVALID_ARG;
    *out = ctx->hp;
    return MOARA_OK;
}

int moara_state_bytes(int m, int n, int r, int block_size, int b_V, int b_M, int d_rule,
                      int decompose, size_t* out) {
    if (out == nullptr) return MOARA_ERR_INVALID_ARG;
    if (m < 1 || n < 1 || block_size < 1 || b_V < 0 || b_M < 0) return MOARA_ERR_SHAPE;
    if (r < 1 || r > std::min(m, n)) return MOARA_ERR_RANK;
    if (d_rule != MOARA_DRULE_N && d_rule != MOARA_DRULE_MAX) return MOARA_ERR_INVALID_ARG;
    const unsigned long long d = d_rule == MOARA_DRULE_N ? (unsigned long long)n
                                                         : (unsigned long long)std::max(m, n);
    const unsigned long long kb = (unsigned long long)blocks_of(n, block_size);
    const long double dir = 2.0L * b_V * (long double)r * d;
    const long double mag = decompose ? 2.0L * b_M * (long double)m * kb : 0.0L;
    const long double tot = dir + mag;
    if (tot > (long double)std::numeric_limits<size_t>::max()) return MOARA_ERR_SHAPE;
    *out = static_cast<size_t>(2ull * b_V * r * d + (decompose ? 2ull * b_M * m * kb : 0ull));
    return MOARA_OK;
}

int moara_rank_table(int r_base, uint32_t donor_mask, uint32_t receiver_mask, int delta_r,
                     int out_ranks[7]) {
    if (out_ranks == nullptr) return MOARA_ERR_INVALID_ARG;
    if (r_base < 1) return MOARA_ERR_RANK;
    if (((donor_mask | receiver_mask) >> 7) != 0) return MOARA_ERR_INVALID_ARG;
    if (donor_mask & receiver_mask) return MOARA_ERR_INVALID_ARG;
    if (delta_r < 0 || delta_r >= r_base) return MOARA_ERR_RANK;
    int nd = 0, nr = 0;
    for (int i = 0; i < 7; ++i) {
        nd += (donor_mask >> i) & 1;
        nr += (receiver_mask >> i) & 1;
    }
    if (nd > 0 && nr == 0) return MOARA_ERR_INVALID_ARG;
    const long long moved = (long long)delta_r * nd;
    const long long share = nr ? moved / nr : 0;
    long long rem = nr ? moved - share * nr : 0;
    for (int i = 0; i < 7; ++i) {
        long long v = r_base;
        if ((donor_mask >> i) & 1) v = r_base - delta_r;
        if ((receiver_mask >> i) & 1) {
            v = r_base + share + (rem > 0 ? 1 : 0);
            if (rem > 0) --rem;
        }
        if (v > std::numeric_limits<int>::max()) return MOARA_ERR_RANK;
        out_ranks[i] = static_cast<int>(v);
    }
    return MOARA_OK;
}

int moara_workspace_bytes(int m, int n, int r, int block_size, size_t* out) {
    if (out == nullptr) return MOARA_ERR_INVALID_ARG;
    if (m < 1 || n < 1 || block_size < 1) return MOARA_ERR_SHAPE;
    if (r < 1 || r > std::min(m, n)) return MOARA_ERR_RANK;
    *out = moara::workspace_layout(m, n, r, block_size).total;
    return MOARA_OK;
}

int moara_init_module(moara_ctx* ctx, const moara_module_desc* d, int* module_id) {
    if (ctx == nullptr) return MOARA_ERR_INVALID_ARG;
    if (d == nullptr || module_id == nullptr) return fail(ctx, MOARA_ERR_INVALID_ARG, "desc or module_id is NULL");
    if (d->m < 1 || d->n < 1) return fail(ctx, MOARA_ERR_SHAPE, "m and n must be >= 1 (got %d x %d)", d->m, d->n);
    if ((long long)d->m * d->n > (1LL << 40)) return fail(ctx, MOARA_ERR_SHAPE, "matrix too large");
    if (d->r < 1 || d->r > std::min(d->m, d->n))
        return fail(ctx, MOARA_ERR_RANK, "rank %d outside [1, min(m, n) = %d]", d->r, std::min(d->m, d->n));
    if (d->grad_dtype != MOARA_DTYPE_F32 && d->grad_dtype != MOARA_DTYPE_BF16)
        return fail(ctx, MOARA_ERR_INVALID_ARG, "unknown grad_dtype %d", d->grad_dtype);
    const void* req[] = {d->W, d->P, d->exp_avg, d->exp_avg_sq, d->workspace};
    const char* names[] = {"W", "P", "exp_avg", "exp_avg_sq", "workspace"};
    for (int i = 0; i < 5; ++i) {
        if (req[i] == nullptr) return fail(ctx, MOARA_ERR_INVALID_ARG, "%s is NULL", names[i]);
        if (!aligned16(req[i])) return fail(ctx, MOARA_ERR_ALIGN, "%s is not 16-byte aligned", names[i]);
    }
    if (ctx->hp.decompose) {
        if (d->mag_avg == nullptr || d->mag_avg_sq == nullptr)
            return fail(ctx, MOARA_ERR_INVALID_ARG, "mag_avg / mag_avg_sq are NULL with decompose = 1");
        if (!aligned16(d->mag_avg) || !aligned16(d->mag_avg_sq))
            return fail(ctx, MOARA_ERR_ALIGN, "mag_avg / mag_avg_sq not 16-byte aligned");
    }
    if (d->P_bf16 != nullptr && !aligned16(d->P_bf16))
        return fail(ctx, MOARA_ERR_ALIGN, "P_bf16 is not 16-byte aligned");
    if (ctx->hp.precision == MOARA_PREC_BF16_TC && d->P_bf16 == nullptr)
        return fail(ctx, MOARA_ERR_INVALID_ARG, "P_bf16 is required with precision BF16_TC");
    const bool right = ctx->hp.proj_rule == MOARA_PROJ_SMALLER && d->m > d->n;
    if (right && (d->grad_dtype != MOARA_DTYPE_BF16 || d->P_bf16 == nullptr || ctx->tc == nullptr ||
                  ctx->hp.precision == MOARA_PREC_FP32 ||
                  !moara::tc_supported(d->m, d->n, d->r, ctx->hp.block_size, d->grad_dtype, ctx->hp.decompose,
                                       ctx->hp.state_dtype)))
        return fail(ctx, MOARA_ERR_UNSUPPORTED,
                    "a right projector (m > n under MOARA_PROJ_SMALLER) needs the tensor-core path: bf16 gradient, "
                    "P_bf16, n and r multiples of 8");
    if (ctx->hp.state_dtype == MOARA_DTYPE_BF16 &&
        (d->grad_dtype != MOARA_DTYPE_BF16 || d->P_bf16 == nullptr || ctx->tc == nullptr ||
         !moara::tc_supported(d->m, d->n, d->r, ctx->hp.block_size, d->grad_dtype, ctx->hp.decompose,
                              ctx->hp.state_dtype)))
        return fail(ctx, MOARA_ERR_UNSUPPORTED,
                    "bf16 states need the tensor-core path: bf16 gradient, P_bf16, n and r multiples of 8, B >= 32");
    const moara::WsLayout wl = moara::workspace_layout(d->m, d->n, d->r, ctx->hp.block_size);
    if (d->workspace_bytes < wl.total)
        return fail(ctx, MOARA_ERR_WORKSPACE, "workspace of %zu bytes, %zu needed", d->workspace_bytes, wl.total);
    if (static_cast<int>(ctx->mods.size()) >= kMaxModules)
        return fail(ctx, MOARA_ERR_INVALID_ARG, "too many modules");

    DeviceGuard g(ctx->device);
    if (static_cast<int>(ctx->mods.size()) >= ctx->cap) {
        const int ncap = ctx->cap * 2;
        moara::ModDev* nd = nullptr;
        cudaError_t e = cudaMalloc(&nd, sizeof(moara::ModDev) * ncap);
        if (e != cudaSuccess) return cuda_fail(ctx, e, "cudaMalloc module table");
        if (!ctx->moddev.empty()) {
            e = cudaMemcpy(nd, ctx->moddev.data(), sizeof(moara::ModDev) * ctx->moddev.size(),
                           cudaMemcpyHostToDevice);
            if (e != cudaSuccess) { cudaFree(nd); return cuda_fail(ctx, e, "module table copy"); }
        }
        cudaFree(ctx->d_mods);
        ctx->d_mods = nd;
        ctx->cap = ncap;
    }
    moara::ModDev md{};
    md.m = d->m; md.n = d->n; md.r = d->r; md.kb = blocks_of(d->n, ctx->hp.block_size);
    md.dtype = d->grad_dtype;
    md.right = right ? 1 : 0;
    md.W = d->W; md.P = d->P; md.Pb = d->P_bf16;
    md.exp_avg = d->exp_avg; md.exp_avg_sq = d->exp_avg_sq;
    md.mag_avg = d->mag_avg; md.mag_avg_sq = d->mag_avg_sq;
    char* ws = static_cast<char*>(d->workspace);
    md.ws_N = reinterpret_cast<float*>(ws + wl.off_N);
    md.ws_dM = reinterpret_cast<float*>(ws + wl.off_dM);
    md.ws_inv = reinterpret_cast<float*>(ws + wl.off_inv);
    md.ws_Vhi = reinterpret_cast<uint16_t*>(ws + wl.off_Vhi);
    md.ws_Vlo = reinterpret_cast<uint16_t*>(ws + wl.off_Vlo);
    md.ws_Qt = wl.off_Qt != 0 ? reinterpret_cast<uint16_t*>(ws + wl.off_Qt) : nullptr;
    const int id = static_cast<int>(ctx->mods.size());
    cudaError_t e = cudaMemcpy(ctx->d_mods + id, &md, sizeof(md), cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "module table copy");
    if (ctx->tc) {
        int rc = moara::tc_register(ctx->tc, id, md, ctx->hp);
        if (rc != MOARA_OK) return fail(ctx, rc, "tensor-core registration of module %d failed", id);
    }
    ctx->mods.push_back(*d);
    ctx->moddev.push_back(md);
    ctx->refresh_count.push_back(0);
    *module_id = id;
    ctx->last_error.clear();
    return MOARA_OK;
}

int moara_load_projector(moara_ctx* ctx, int module_id, const float* P_src, void* stream) {
    if (ctx == nullptr) return MOARA_ERR_INVALID_ARG;
    if (module_id < 0 || module_id >= static_cast<int>(ctx->mods.size()))
        return fail(ctx, MOARA_ERR_UNKNOWN_MODULE, "module id %d is not registered", module_id);
    if (P_src == nullptr) return fail(ctx, MOARA_ERR_INVALID_ARG, "P_src is NULL");
    if (!aligned16(P_src)) return fail(ctx, MOARA_ERR_ALIGN, "P_src is not 16-byte aligned");
    DeviceGuard g(ctx->device);
    const moara::ModDev& md = ctx->moddev[module_id];
    const int rows = md.right ? md.n : md.m;      // P (m x r) or the right projector Q (n x r)
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = moara::launch_f32_to_bf16(P_src, md.P, md.Pb, (long long)rows * md.r, s, &ctx->launches);
    if (e == cudaSuccess && md.right) e = moara::tc_transpose_bf16(md.Pb, md.ws_Qt, md.n, md.r, s, &ctx->launches);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "projector copy");
    return MOARA_OK;
}

int moara_refresh_workspace_bytes(const moara_ctx* ctx, int m, int n, int r, size_t* out) {
    if (ctx == nullptr || out == nullptr) return MOARA_ERR_INVALID_ARG;
    if (m < 1 || n < 1) return MOARA_ERR_SHAPE;
    if (r < 1 || r > std::min(m, n)) return MOARA_ERR_RANK;
    const int src_v = (ctx->hp.refresh_src == MOARA_REFRESH_SRC_V && ctx->hp.decompose) ? 1 : 0;
    const bool tr = ctx->hp.proj_rule == MOARA_PROJ_SMALLER && m > n;   // refresh of V^T
    *out = align_up(moara::refresh_ws_bytes(tr ? n : m, tr ? m : n, r, refresh_l(ctx, m, n, r), ctx->hp.block_size,
                                            src_v), 256);
    return MOARA_OK;
}

int moara_set_refresh_workspace(moara_ctx* ctx, void* ptr, size_t bytes) {
    if (ctx == nullptr) return MOARA_ERR_INVALID_ARG;
    if (ptr == nullptr && bytes != 0) return fail(ctx, MOARA_ERR_INVALID_ARG, "NULL workspace with nonzero size");
    if (ptr != nullptr && (reinterpret_cast<uintptr_t>(ptr) & 255u) != 0)
        return fail(ctx, MOARA_ERR_ALIGN, "refresh workspace must be 256-byte aligned");
    ctx->refresh_ws = ptr;
    ctx->refresh_ws_bytes = bytes;
    return MOARA_OK;
}

int moara_refresh_projector(moara_ctx* ctx, int n_mod, const int* ids, const void* const* G, void* stream) {
    if (ctx == nullptr) return MOARA_ERR_INVALID_ARG;
    int rc = check_ids(ctx, n_mod, ids, G);
    if (rc != MOARA_OK) return rc;
    if (n_mod == 0) return MOARA_OK;
    if (ctx->refresh_ws == nullptr) return fail(ctx, MOARA_ERR_WORKSPACE, "no refresh workspace set");
    DeviceGuard g(ctx->device);
    ProfScope ps(ctx, MOARA_PHASE_REFRESH, static_cast<cudaStream_t>(stream));
    return do_refresh(ctx, n_mod, ids, G, static_cast<cudaStream_t>(stream));
}

}  // extern "C"

namespace {

// The step on validated arguments (device gradients), enqueued on s.
int step_impl(moara_ctx* ctx, int n_mod, const int* ids, const void* const* G, int64_t t, float lr,
              int auto_refresh, cudaStream_t s) {
    int rc = MOARA_OK;
    if (auto_refresh && ((t - 1) % ctx->hp.refresh_interval) == 0) {
        if (ctx->refresh_ws == nullptr) return fail(ctx, MOARA_ERR_WORKSPACE, "no refresh workspace set");
        ProfScope ps(ctx, MOARA_PHASE_REFRESH, s);
        rc = do_refresh(ctx, n_mod, ids, G, s);
        if (rc != MOARA_OK) return rc;
    }
    // global-norm clipping (App. D.2): the coefficient of this step's
    // gradients, before any update.  When every module runs on tensor cores
    // with the decomposition, the step takes it from the block norms of its
    // own decomposition (no extra pass over G); otherwise a norm pass first.
    const float* clip = nullptr;
    moara::TcClipFuse fuse{};
    bool fused = false;
    if (ctx->hp.clip_norm > 0.0f && ctx->hp.decompose && n_mod <= moara::tc_group_limit()) {
        fused = true;
        for (int i = 0; i < n_mod && fused; ++i) fused = use_tc(ctx, ids[i]);
    }
    if (ctx->hp.clip_norm > 0.0f) {
        const int need = fused ? 1 : (n_mod + moara::kMaxGroup - 1) / moara::kMaxGroup;
        if (ctx->clip_part_cap < need) {
            if (ctx->d_clip_part != nullptr) {
                cudaError_t e = cudaStreamSynchronize(s);   // an earlier step may still use them
                if (e != cudaSuccess) return cuda_fail(ctx, e, "clipping partial sums release");
                cudaFree(ctx->d_clip_part);
                ctx->d_clip_part = nullptr;
                ctx->clip_part_cap = 0;
            }
            cudaError_t e = cudaMalloc(&ctx->d_clip_part, sizeof(double) * moara::kNormParts * (size_t)need);
            if (e != cudaSuccess) return cuda_fail(ctx, e, "cudaMalloc of the clipping partial sums");
            ctx->clip_part_cap = need;
        }
        fuse = moara::TcClipFuse{ctx->d_clip, ctx->d_clip_part, ctx->clip_extra, ctx->hp.clip_norm};
    }
    if (ctx->hp.clip_norm > 0.0f && !fused) {
        ProfScope ps(ctx, MOARA_PHASE_CLIP_NORM, s);
        const int nb = (n_mod + moara::kMaxGroup - 1) / moara::kMaxGroup;
        for (int c0 = 0, bi = 0; c0 < n_mod; c0 += moara::kMaxGroup, ++bi) {
            moara::GradNormBatch nbt{};
            nbt.count = std::min(moara::kMaxGroup, n_mod - c0);
            long long acc = 0;
            for (int q = 0; q < nbt.count; ++q) {
                const moara_module_desc& d = ctx->mods[ids[c0 + q]];
                nbt.chunk_start[q] = acc;
                nbt.G[q] = G[c0 + q];
                nbt.elems[q] = (long long)d.m * d.n;
                nbt.dtype[q] = d.grad_dtype;
                acc += (nbt.elems[q] + moara::kNormChunk - 1) / moara::kNormChunk;
            }
            nbt.chunk_start[nbt.count] = acc;
            cudaError_t e = moara::launch_grad_sq(nbt, ctx->d_clip_part + (size_t)bi * moara::kNormParts, s,
                                                  &ctx->launches);
            if (e != cudaSuccess) return cuda_fail(ctx, e, "gradient norm launch");
        }
        cudaError_t e = moara::launch_clip_finish(ctx->d_clip_part, nb * moara::kNormParts, ctx->clip_extra,
                                                  ctx->hp.clip_norm, ctx->d_clip, s, &ctx->launches);
        if (e != cudaSuccess) return cuda_fail(ctx, e, "clipping coefficient launch");
        clip = ctx->d_clip + 1;
    }
    std::vector<int> simt, tcm;
    for (int i = 0; i < n_mod; ++i) (use_tc(ctx, ids[i]) ? tcm : simt).push_back(i);
    if (!tcm.empty()) {
        const double bc1 = 1.0 - std::pow((double)ctx->hp.beta1, (double)t);
        const double bc2 = 1.0 - std::pow((double)ctx->hp.beta2, (double)t);
        std::vector<int> mids(tcm.size());
        std::vector<const void*> gp(tcm.size());
        for (size_t q = 0; q < tcm.size(); ++q) { mids[q] = ids[tcm[q]]; gp[q] = G[tcm[q]]; }
        moara::TcProfile tp{ctx->prof, [](void* c, int ph, cudaStream_t st, bool begin) {
            moara_ctx* cx = static_cast<moara_ctx*>(c);
            if (begin) {
                cx->open_event = take_event(cx);
                cudaEventRecord(cx->open_event, st);
            } else {
                cudaEvent_t b = take_event(cx);
                cudaEventRecord(b, st);
                cx->recs.push_back({ph, cx->open_event, b});
            }
        }, ctx};
        rc = moara::tc_step(ctx->tc, ctx->hp, static_cast<int>(mids.size()), mids.data(), gp.data(),
                            static_cast<float>(bc1), static_cast<float>(bc2), lr, t == 1 ? 1 : 0, clip,
                            fused ? &fuse : nullptr, s, &ctx->launches, tp);
        if (rc != MOARA_OK) return fail(ctx, rc, "tensor-core step launch failed: %s", moara::tc_last_error(ctx->tc));
    }
    if (!simt.empty()) {
        rc = do_step_simt(ctx, simt, ids, G, t, lr, clip, s);
        if (rc != MOARA_OK) return rc;
    }
    return MOARA_OK;
}


// Two staging buffers of at least `bytes` each, the copy stream and events.
int ensure_staging(moara_ctx* ctx, size_t bytes) {
    if (ctx->copy_stream == nullptr) {
        cudaError_t e = cudaStreamCreateWithFlags(&ctx->copy_stream, cudaStreamNonBlocking);
        for (int b = 0; b < 2 && e == cudaSuccess; ++b) {
            e = cudaEventCreateWithFlags(&ctx->copy_done[b], cudaEventDisableTiming);
            if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ctx->compute_done[b], cudaEventDisableTiming);
        }
        if (e != cudaSuccess) return cuda_fail(ctx, e, "copy stream / events");
    }
    if (ctx->stage_bytes >= bytes) return MOARA_OK;
    // earlier steps may still read the old buffers
    for (int b = 0; b < 2; ++b) {
        if (ctx->stage[b] != nullptr) {
            cudaError_t e = cudaEventSynchronize(ctx->compute_done[b]);
            if (e != cudaSuccess) return cuda_fail(ctx, e, "staging buffer release");
            cudaFree(ctx->stage[b]);
            ctx->stage[b] = nullptr;
        }
    }
    ctx->stage_bytes = 0;
    for (int b = 0; b < 2; ++b) {
        cudaError_t e = cudaMalloc(&ctx->stage[b], bytes);
        if (e != cudaSuccess) return cuda_fail(ctx, e, "cudaMalloc of a gradient staging buffer");
    }
    ctx->stage_bytes = bytes;
    return MOARA_OK;
}

}  // namespace

extern "C" {

int moara_step_grouped(moara_ctx* ctx, int n_mod, const int* ids, const void* const* G, int64_t t,
                       float lr, int auto_refresh, void* stream) {
    if (ctx == nullptr) return MOARA_ERR_INVALID_ARG;
    int rc = check_ids(ctx, n_mod, ids, G);
    if (rc != MOARA_OK) return rc;
    if (t < 1) return fail(ctx, MOARA_ERR_INVALID_ARG, "step t must be >= 1 (got %lld)", (long long)t);
    if (!std::isfinite(lr)) return fail(ctx, MOARA_ERR_INVALID_ARG, "lr must be finite");
    if (n_mod == 0) return MOARA_OK;
    DeviceGuard g(ctx->device);
    return step_impl(ctx, n_mod, ids, G, t, lr, auto_refresh, static_cast<cudaStream_t>(stream));
}

int moara_step_grouped_host(moara_ctx* ctx, int n_mod, const int* ids, const void* const* G_host, int64_t t,
                            float lr, int auto_refresh, size_t chunk_bytes, void* stream) {
    if (ctx == nullptr) return MOARA_ERR_INVALID_ARG;
    int rc = check_ids(ctx, n_mod, ids, G_host);
    if (rc != MOARA_OK) return rc;
    if (t < 1) return fail(ctx, MOARA_ERR_INVALID_ARG, "step t must be >= 1 (got %lld)", (long long)t);
    if (!std::isfinite(lr)) return fail(ctx, MOARA_ERR_INVALID_ARG, "lr must be finite");
    if (chunk_bytes == 0) return fail(ctx, MOARA_ERR_INVALID_ARG, "chunk_bytes must be > 0");
    if (ctx->hp.clip_norm > 0.0f)
        return fail(ctx, MOARA_ERR_UNSUPPORTED,
                    "global-norm clipping needs all of the step's gradients on the device: use moara_step_grouped");
    if (n_mod == 0) return MOARA_OK;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    DeviceGuard g(ctx->device);
    // chunks of consecutive modules, at most chunk_bytes of gradient each
    // (a larger module forms its own chunk); 256-byte aligned offsets
    auto gbytes = [&](int i) {
        const moara_module_desc& d = ctx->mods[ids[i]];
        const size_t es = d.grad_dtype == MOARA_DTYPE_BF16 ? 2 : 4;
        return align_up(es * (size_t)d.m * d.n, 256);
    };
    std::vector<int> cstart{0};
    size_t cur = 0, maxc = 0;
    for (int i = 0; i < n_mod; ++i) {
        const size_t b = gbytes(i);
        if (cur > 0 && cur + b > chunk_bytes) {
            maxc = std::max(maxc, cur);
            cstart.push_back(i);
            cur = 0;
        }
        cur += b;
    }
    maxc = std::max(maxc, cur);
    cstart.push_back(n_mod);
    rc = ensure_staging(ctx, maxc);
    if (rc != MOARA_OK) return rc;
    std::vector<const void*> gdev(n_mod);
    for (size_t c = 0; c + 1 < cstart.size(); ++c) {
        const int b = static_cast<int>(c & 1);
        // the copy into buffer b waits for the step that last read it
        cudaError_t e = cudaStreamWaitEvent(ctx->copy_stream, ctx->compute_done[b], 0);
        size_t off = 0;
        for (int i = cstart[c]; i < cstart[c + 1] && e == cudaSuccess; ++i) {
            const moara_module_desc& d = ctx->mods[ids[i]];
            const size_t es = d.grad_dtype == MOARA_DTYPE_BF16 ? 2 : 4;
            void* dst = static_cast<char*>(ctx->stage[b]) + off;
            e = cudaMemcpyAsync(dst, G_host[i], es * (size_t)d.m * d.n, cudaMemcpyHostToDevice, ctx->copy_stream);
            gdev[i] = dst;
            off += gbytes(i);
        }
        if (e == cudaSuccess) e = cudaEventRecord(ctx->copy_done[b], ctx->copy_stream);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(s, ctx->copy_done[b], 0);
        if (e != cudaSuccess) return cuda_fail(ctx, e, "gradient upload");
        rc = step_impl(ctx, cstart[c + 1] - cstart[c], ids + cstart[c], gdev.data() + cstart[c], t, lr,
                       auto_refresh, s);
        if (rc != MOARA_OK) return rc;
        e = cudaEventRecord(ctx->compute_done[b], s);
        if (e != cudaSuccess) return cuda_fail(ctx, e, "step event");
    }
    return MOARA_OK;
}

int moara_set_clip_extra(moara_ctx* ctx, const float* extra_sq) {
    if (ctx == nullptr) return MOARA_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(extra_sq) & 3) != 0)
        return fail(ctx, MOARA_ERR_ALIGN, "extra_sq is not 4-byte aligned");
    ctx->clip_extra = extra_sq;
    return MOARA_OK;
}

int moara_clip_state(moara_ctx* ctx, const float** state) {
    if (ctx == nullptr || state == nullptr) return MOARA_ERR_INVALID_ARG;
    *state = ctx->d_clip;
    return MOARA_OK;
}

int moara_flatten_shape(int ndim, const int64_t* shape, int* m, int* n) {
    if (ndim < 1 || shape == nullptr || m == nullptr || n == nullptr) return MOARA_ERR_INVALID_ARG;
    for (int i = 0; i < ndim; ++i)
        if (shape[i] < 1) return MOARA_ERR_INVALID_ARG;
    if (shape[0] > INT_MAX) return MOARA_ERR_SHAPE;
    int64_t cols = 1;
    for (int i = 1; i < ndim; ++i) {
        if (cols > INT_MAX / shape[i]) return MOARA_ERR_SHAPE;
        cols *= shape[i];
    }
    *m = static_cast<int>(shape[0]);
    *n = static_cast<int>(cols);
    return MOARA_OK;
}

int moara_alignment(moara_ctx* ctx, int n_mod, const int* ids, const void* const* G, float* S_out,
                    void* stream) {
    if (ctx == nullptr) return MOARA_ERR_INVALID_ARG;
    int rc = check_ids(ctx, n_mod, ids, G);
    if (rc != MOARA_OK) return rc;
    if (n_mod == 0) return MOARA_OK;
    if (S_out == nullptr) return fail(ctx, MOARA_ERR_INVALID_ARG, "S_out is null");
    if ((reinterpret_cast<uintptr_t>(S_out) & 3) != 0) return fail(ctx, MOARA_ERR_ALIGN, "S_out is not 4-byte aligned");
    for (int i = 0; i < n_mod; ++i)
        if (!use_tc(ctx, ids[i]))
            return fail(ctx, MOARA_ERR_UNSUPPORTED,
                        "alignment: module %d is not on the tensor-core path (bf16 gradient, n and r multiples of 8)",
                        ids[i]);
    DeviceGuard g(ctx->device);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (ctx->align_cap < n_mod) {
        if (ctx->align_acc != nullptr) {
            // an earlier call may still use the old accumulators
            cudaError_t e = cudaStreamSynchronize(s);
            if (e != cudaSuccess) return cuda_fail(ctx, e, "alignment accumulator release");
            cudaFree(ctx->align_acc);
            ctx->align_acc = nullptr;
            ctx->align_cap = 0;
        }
        cudaError_t e = cudaMalloc(&ctx->align_acc, sizeof(double) * 3 * (size_t)n_mod);
        if (e != cudaSuccess) return cuda_fail(ctx, e, "cudaMalloc of the alignment accumulators");
        ctx->align_cap = n_mod;
    }
    rc = moara::tc_alignment(ctx->tc, ctx->hp, n_mod, ids, G, S_out, ctx->align_acc, s, &ctx->launches);
    if (rc != MOARA_OK) return fail(ctx, rc, "alignment: %s", moara::tc_last_error(ctx->tc));
    return MOARA_OK;
}

int moara_get_device_status(moara_ctx* ctx, int* status, void* stream) {
    if (ctx == nullptr || status == nullptr) return MOARA_ERR_INVALID_ARG;
    DeviceGuard g(ctx->device);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = cudaMemcpyAsync(ctx->h_status, ctx->d_status, sizeof(int), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(ctx->d_status, 0, sizeof(int), s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "status read");
    *status = ctx->h_status[0];
    return MOARA_OK;
}

const char* moara_last_error(const moara_ctx* ctx) {
    if (ctx == nullptr) return "context is NULL";
    return ctx->last_error.c_str();
}

const char* moara_status_string(int code) {
    switch (code) {
        case MOARA_OK: return "ok";
        case MOARA_ERR_INVALID_ARG: return "invalid argument";
        case MOARA_ERR_SHAPE: return "invalid shape";
        case MOARA_ERR_RANK: return "invalid rank";
        case MOARA_ERR_ALIGN: return "misaligned pointer";
        case MOARA_ERR_UNKNOWN_MODULE: return "unknown module";
        case MOARA_ERR_CUDA: return "CUDA error";
        case MOARA_ERR_DEVICE_TIMEOUT: return "device-side wait timed out";
        case MOARA_ERR_WORKSPACE: return "workspace missing or too small";
        case MOARA_ERR_UNSUPPORTED: return "unsupported";
        default: return "unknown status";
    }
}

int64_t moara_launch_count(const moara_ctx* ctx) { return ctx ? ctx->launches : -1; }

int moara_set_wait_limit(moara_ctx* ctx, int64_t cycles) {
    if (ctx == nullptr) return MOARA_ERR_INVALID_ARG;
    if (ctx->tc == nullptr) return fail(ctx, MOARA_ERR_UNSUPPORTED, "no tensor-core state on this device");
    moara::tc_set_wait_limit(ctx->tc, static_cast<long long>(cycles));
    return MOARA_OK;
}

int moara_profile_enable(moara_ctx* ctx, int enable) {
    if (ctx == nullptr) return MOARA_ERR_INVALID_ARG;
    ctx->prof = enable != 0;
    return MOARA_OK;
}

int moara_profile_read(moara_ctx* ctx, double ms[MOARA_NUM_PHASES], int64_t launches[MOARA_NUM_PHASES]) {
    if (ctx == nullptr || ms == nullptr || launches == nullptr) return MOARA_ERR_INVALID_ARG;
    DeviceGuard g(ctx->device);
    for (auto& r : ctx->recs) {
        cudaError_t e = cudaEventSynchronize(r.b);
        float t = 0.0f;
        if (e == cudaSuccess) e = cudaEventElapsedTime(&t, r.a, r.b);
        if (e != cudaSuccess) return cuda_fail(ctx, e, "profile event");
        ctx->prof_ms[r.phase] += t;
        ctx->prof_n[r.phase] += 1;
        ctx->free_events.push_back(r.a);
        ctx->free_events.push_back(r.b);
    }
    ctx->recs.clear();
    for (int i = 0; i < MOARA_NUM_PHASES; ++i) {
        ms[i] = ctx->prof_ms[i];
        launches[i] = ctx->prof_n[i];
        ctx->prof_ms[i] = 0.0;
        ctx->prof_n[i] = 0;
    }
    return MOARA_OK;
}

}  // extern "C"
