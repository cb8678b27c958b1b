// fp32 SIMT kernels of the step: block decomposition with the magnitude
// branch's Adam, and a grouped tiled GEMM whose operand loaders apply the
// block scales of the decomposition and whose epilogues run the direction
// branch's Adam or the weight update.  Every product is an fp32 FMA, so this
// path meets the all-fp32 tolerance; it also serves the refresh.
#include <cuda_bf16.h>

#include "internal.h"

namespace moara {

__device__ __forceinline__ float bf16_bits_to_f32(uint16_t h) {
    return __uint_as_float(static_cast<uint32_t>(h) << 16);
}

template <bool BF16>
__device__ __forceinline__ float load_elem(const void* base, long long idx) {
    if (BF16) {
        return bf16_bits_to_f32(__ldg(reinterpret_cast<const unsigned short*>(base) + idx));
    } else {
        return __ldg(reinterpret_cast<const float*>(base) + idx);
    }
}

// ---------------------------------------------------------------------------
// Decompose(G, B) of §3.1 / Appendix B.1 for every (row, block) item, plus
// Optimizer_M (Adam on the block magnitudes, Algorithm 1).  Writes the inverse
// scales 1 / (m_{i,b} + eps) used by the projection's operand loader.
// Columns past n (the right zero padding) contribute nothing to the norm.
// ---------------------------------------------------------------------------
__device__ __forceinline__ int find_item(const long long* start, int count, long long item) {
    int lo = 0, hi = count - 1;
    while (lo < hi) {
        int mid = (lo + hi + 1) >> 1;
        if (start[mid] <= item) lo = mid; else hi = mid - 1;
    }
    return lo;
}

__device__ __forceinline__ void finish_item(const DecompBatch& b, const DecompItem& it,
                                            long long local, float ss) {
    float mag = sqrtf(ss);
    it.inv[local] = 1.0f / (mag + b.decomp_eps);
    if (b.do_mag) {
        // a clipped gradient c G has block norms c M and the same direction V
        if (b.clip != nullptr) mag *= *b.clip;
        float ma = b.beta1 * it.mag_avg[local] + (1.0f - b.beta1) * mag;
        float mas = b.beta2 * it.mag_avg_sq[local] + (1.0f - b.beta2) * mag * mag;
        it.mag_avg[local] = ma;
        it.mag_avg_sq[local] = mas;
        it.dM[local] = (ma / b.bc1) / (sqrtf(mas / b.bc2) + b.adam_eps);
    }
}

// One thread per (row, block): used for B <= 32.
__global__ void __launch_bounds__(256) k_decompose_thread(const __grid_constant__ DecompBatch b) {
    const long long total = b.item_start[b.count];
    for (long long item = blockIdx.x * (long long)blockDim.x + threadIdx.x; item < total;
         item += (long long)gridDim.x * blockDim.x) {
        const int pi = find_item(b.item_start, b.count, item);
        const DecompItem& it = b.p[pi];
        const long long local = item - b.item_start[pi];
        const int row = static_cast<int>(local / it.kb);
        const int blk = static_cast<int>(local - (long long)row * it.kb);
        const int c0 = blk * b.B;
        const int c1 = min(c0 + b.B, it.n);
        const long long base = (long long)row * it.n;
        float ss = 0.0f;
        if (it.dtype == MOARA_DTYPE_BF16) {
            for (int c = c0; c < c1; ++c) { float x = load_elem<true>(it.G, base + c); ss = fmaf(x, x, ss); }
        } else {
            for (int c = c0; c < c1; ++c) { float x = load_elem<false>(it.G, base + c); ss = fmaf(x, x, ss); }
        }
        finish_item(b, it, local, ss);
    }
}

// One warp per (row, block): used for B > 32.
__global__ void __launch_bounds__(256) k_decompose_warp(const __grid_constant__ DecompBatch b) {
    const long long total = b.item_start[b.count];
    const int lane = threadIdx.x & 31;
    const long long warp0 = (blockIdx.x * (long long)blockDim.x + threadIdx.x) >> 5;
    const long long nwarps = ((long long)gridDim.x * blockDim.x) >> 5;
    for (long long item = warp0; item < total; item += nwarps) {
        const int pi = find_item(b.item_start, b.count, item);
        const DecompItem& it = b.p[pi];
        const long long local = item - b.item_start[pi];
        const int row = static_cast<int>(local / it.kb);
        const int blk = static_cast<int>(local - (long long)row * it.kb);
        const int c0 = blk * b.B;
        const int c1 = min(c0 + b.B, it.n);
        const long long base = (long long)row * it.n;
        float ss = 0.0f;
        if (it.dtype == MOARA_DTYPE_BF16) {
            for (int c = c0 + lane; c < c1; c += 32) { float x = load_elem<true>(it.G, base + c); ss = fmaf(x, x, ss); }
        } else {
            for (int c = c0 + lane; c < c1; c += 32) { float x = load_elem<false>(it.G, base + c); ss = fmaf(x, x, ss); }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
        if (lane == 0) finish_item(b, it, local, ss);
    }
}

cudaError_t launch_decompose(const DecompBatch& b, cudaStream_t s, int64_t* launches) {
    const long long total = b.item_start[b.count];
    if (total <= 0) return cudaSuccess;
    const int threads = 256;
    if (b.B > 32) {
        long long blocks = (total * 32 + threads - 1) / threads;
        if (blocks > 152LL * 64) blocks = 152LL * 64;
        k_decompose_warp<<<static_cast<unsigned>(blocks), threads, 0, s>>>(b);
    } else {
        long long blocks = (total + threads - 1) / threads;
        if (blocks > 152LL * 64) blocks = 152LL * 64;
        k_decompose_thread<<<static_cast<unsigned>(blocks), threads, 0, s>>>(b);
    }
    ++*launches;
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Grouped SIMT GEMM: 128 x 128 tile, BK = 8, 256 threads, 8 x 8 per thread,
// register-staged double buffering.  blockIdx.x enumerates the tiles of all
// problems of the batch (problems are ordered longest-K first by the host).
// ---------------------------------------------------------------------------
constexpr int TM = 128, TN = 128, TK = 16, TPAD = 4;
constexpr int NQ = TK * 128 / 256;   // elements of A (and of B) each thread stages per k-tile

int gemm_tile_m() { return TM; }
int gemm_tile_n() { return TN; }

// Index of the block holding column c: a shift when B is a power of two.
__device__ __forceinline__ int block_of(int c, int B, int log2B) { return log2B >= 0 ? (c >> log2B) : c / B; }

template <int ALAY, bool ASC, bool ABF, int BLAY, bool BSC, bool BBF>
struct TileLoader {
    float ra[NQ], rb[NQ];

    __device__ __forceinline__ void load(const GemmProb& p, int m0, int n0, int k0, int B, int log2B) {
        const int t = threadIdx.x;
#pragma unroll
        for (int q = 0; q < NQ; ++q) {
            int i, k;
            if (ALAY == A_KCONTIG) { k = t & (TK - 1); i = (t / TK) + (256 / TK) * q; }
            else                   { i = t & 127; k = (t >> 7) + 2 * q; }
            const int gi = m0 + i, gk = k0 + k;
            float v = 0.0f;
            if (gi < p.M && gk < p.K) {
                long long idx;
                int vrow, vcol;
                if (ALAY == A_KCONTIG) { idx = (long long)gi * p.lda + gk; vrow = gi; vcol = gk; }
                else                   { idx = (long long)gk * p.lda + gi; vrow = gk; vcol = gi; }
                v = load_elem<ABF>(p.A, idx);
                if (ASC) v *= __ldg(p.a_inv + (long long)vrow * p.kb + block_of(vcol, B, log2B));
            }
            ra[q] = v;
        }
#pragma unroll
        for (int q = 0; q < NQ; ++q) {
            int j, k;
            if (BLAY == B_NCONTIG) { j = t & 127; k = (t >> 7) + 2 * q; }
            else                   { k = t & (TK - 1); j = (t / TK) + (256 / TK) * q; }
            const int gj = n0 + j, gk = k0 + k;
            float v = 0.0f;
            if (gj < p.N && gk < p.K) {
                long long idx;
                int vrow, vcol;
                if (BLAY == B_NCONTIG) { idx = (long long)gk * p.ldb + gj; vrow = gk; vcol = gj; }
                else                   { idx = (long long)gj * p.ldb + gk; vrow = gj; vcol = gk; }
                v = load_elem<BBF>(p.Bm, idx);
                if (BSC) v *= __ldg(p.b_inv + (long long)vrow * p.kb + block_of(vcol, B, log2B));
            }
            rb[q] = v;
        }
    }

    __device__ __forceinline__ void store(float (*As)[TM + TPAD], float (*Bs)[TN + TPAD]) {
        const int t = threadIdx.x;
#pragma unroll
        for (int q = 0; q < NQ; ++q) {
            int i, k;
            if (ALAY == A_KCONTIG) { k = t & (TK - 1); i = (t / TK) + (256 / TK) * q; }
            else                   { i = t & 127; k = (t >> 7) + 2 * q; }
            As[k][i] = ra[q];
        }
#pragma unroll
        for (int q = 0; q < NQ; ++q) {
            int j, k;
            if (BLAY == B_NCONTIG) { j = t & 127; k = (t >> 7) + 2 * q; }
            else                   { k = t & (TK - 1); j = (t / TK) + (256 / TK) * q; }
            Bs[k][j] = rb[q];
        }
    }
};

template <int EPI>
__device__ __forceinline__ void epilogue(const GemmBatch& b, const GemmProb& p, int i, int j, float acc) {
    const long long o = (long long)i * p.ldc + j;
    if (EPI == EPI_STORE) {
        p.C[o] = acc;
        if (p.c_bf16 != nullptr) {
            __nv_bfloat16 h = __float2bfloat16_rn(acc);
            p.c_bf16[o] = *reinterpret_cast<uint16_t*>(&h);
        }
    } else if (EPI == EPI_STORE_NEG) {
        p.C[o] = -acc;
    } else if (EPI == EPI_SUB) {
        p.C[o] = p.C[o] - acc;
    } else if (EPI == EPI_ADAM) {
        // Optimizer_V (Algorithm 1): Adam on the projected direction R = acc
        // (of the clipped gradient when a clipping coefficient is given).
        if (b.clip != nullptr) acc *= *b.clip;
        float ea = b.beta1 * p.aux0[o] + (1.0f - b.beta1) * acc;
        float eas = b.beta2 * p.aux1[o] + (1.0f - b.beta2) * acc * acc;
        p.aux0[o] = ea;
        p.aux1[o] = eas;
        p.C[o] = (ea / b.bc1) / (sqrtf(eas / b.bc2) + b.adam_eps);
    } else {
        // W <- W - lr*alpha*(Rep_B(dM) (.) dV)  (Algorithm 1; Rep_B of §3.1).
        float u = acc;
        if (p.aux2 != nullptr) u *= p.aux2[(long long)i * p.kb + block_of(j, b.B, b.log2B)];
        p.aux0[o] = p.aux0[o] - b.step_scale * u;
    }
}

template <int ALAY, bool ASC, bool ABF, int BLAY, bool BSC, bool BBF, int EPI>
__global__ void __launch_bounds__(256, 2) k_gemm(const __grid_constant__ GemmBatch b) {
    __shared__ __align__(16) float As[2][TK][TM + TPAD];
    __shared__ __align__(16) float Bs[2][TK][TN + TPAD];

    // locate (problem, tile)
    const int tile = blockIdx.x;
    int lo = 0, hi = b.count - 1;
    while (lo < hi) {
        int mid = (lo + hi + 1) >> 1;
        if (b.tile_start[mid] <= tile) lo = mid; else hi = mid - 1;
    }
    const GemmProb& p = b.p[lo];
    const int local = tile - b.tile_start[lo];
    const int tn = b.tiles_n[lo];
    const int m0 = (local / tn) * TM;
    const int n0 = (local % tn) * TN;
    if (p.lower_only && n0 >= m0 + TM) return;

    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    float acc[8][8];
#pragma unroll
    for (int a = 0; a < 8; ++a)
#pragma unroll
        for (int c = 0; c < 8; ++c) acc[a][c] = 0.0f;

    TileLoader<ALAY, ASC, ABF, BLAY, BSC, BBF> ld;
    int kbeg = 0, kend = p.K;
    if (p.k_tri == KTRI_B_UPPER) kend = min(p.K, n0 + TN);
    else if (p.k_tri == KTRI_B_LOWER) kbeg = min(p.K, n0) & ~(TK - 1);
    else if (p.k_tri == KTRI_A_LOWER) kend = min(p.K, m0 + TM);
    const int ktiles = kend > kbeg ? (kend - kbeg + TK - 1) / TK : 0;
    if (ktiles > 0) {
        ld.load(p, m0, n0, kbeg, b.B, b.log2B);
        ld.store(As[0], Bs[0]);
    }
    __syncthreads();
    for (int kt = 0; kt < ktiles; ++kt) {
        const int cur = kt & 1;
        if (kt + 1 < ktiles) ld.load(p, m0, n0, kbeg + (kt + 1) * TK, b.B, b.log2B);
#pragma unroll
        for (int k = 0; k < TK; ++k) {
            float av[8], bv[8];
            const float4 a0 = *reinterpret_cast<const float4*>(&As[cur][k][ty * 4]);
            const float4 a1 = *reinterpret_cast<const float4*>(&As[cur][k][64 + ty * 4]);
            const float4 b0 = *reinterpret_cast<const float4*>(&Bs[cur][k][tx * 4]);
            const float4 b1 = *reinterpret_cast<const float4*>(&Bs[cur][k][64 + tx * 4]);
            av[0] = a0.x; av[1] = a0.y; av[2] = a0.z; av[3] = a0.w;
            av[4] = a1.x; av[5] = a1.y; av[6] = a1.z; av[7] = a1.w;
            bv[0] = b0.x; bv[1] = b0.y; bv[2] = b0.z; bv[3] = b0.w;
            bv[4] = b1.x; bv[5] = b1.y; bv[6] = b1.z; bv[7] = b1.w;
#pragma unroll
            for (int a = 0; a < 8; ++a)
#pragma unroll
                for (int c = 0; c < 8; ++c) acc[a][c] = fmaf(av[a], bv[c], acc[a][c]);
        }
        if (kt + 1 < ktiles) {
            ld.store(As[cur ^ 1], Bs[cur ^ 1]);
        }
        __syncthreads();
    }

    // Plain stores and read-modify-writes move four consecutive columns per
    // thread as one 16-byte access when the layout allows it.
    if (EPI == EPI_STORE || EPI == EPI_STORE_NEG || EPI == EPI_SUB) {
        const bool vec = (p.ldc & 3) == 0 && (reinterpret_cast<uintptr_t>(p.C) & 15) == 0 &&
                         (EPI != EPI_STORE || p.c_bf16 == nullptr ||
                          (reinterpret_cast<uintptr_t>(p.c_bf16) & 7) == 0);
        if (vec) {
#pragma unroll
            for (int a = 0; a < 8; ++a) {
                const int i = m0 + (a < 4 ? ty * 4 + a : 64 + ty * 4 + (a - 4));
                if (i >= p.M) continue;
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int j = n0 + h * 64 + tx * 4;
                    if (j + 3 < p.N) {
                        const long long o = (long long)i * p.ldc + j;
                        float4 v = make_float4(acc[a][4 * h], acc[a][4 * h + 1], acc[a][4 * h + 2],
                                               acc[a][4 * h + 3]);
                        float4* dst = reinterpret_cast<float4*>(p.C + o);
                        if (EPI == EPI_SUB) {
                            const float4 c = *dst;
                            v = make_float4(c.x - v.x, c.y - v.y, c.z - v.z, c.w - v.w);
                        } else if (EPI == EPI_STORE_NEG) {
                            v = make_float4(-v.x, -v.y, -v.z, -v.w);
                        }
                        *dst = v;
                        if (EPI == EPI_STORE && p.c_bf16 != nullptr) {
                            const __nv_bfloat162 lo = __floats2bfloat162_rn(v.x, v.y);
                            const __nv_bfloat162 hi = __floats2bfloat162_rn(v.z, v.w);
                            uint2 pk;
                            pk.x = *reinterpret_cast<const uint32_t*>(&lo);
                            pk.y = *reinterpret_cast<const uint32_t*>(&hi);
                            *reinterpret_cast<uint2*>(p.c_bf16 + o) = pk;
                        }
                    } else {
#pragma unroll
                        for (int c = 0; c < 4; ++c)
                            if (j + c < p.N) epilogue<EPI>(b, p, i, j + c, acc[a][4 * h + c]);
                    }
                }
            }
            return;
        }
    }
#pragma unroll
    for (int a = 0; a < 8; ++a) {
        const int i = m0 + (a < 4 ? ty * 4 + a : 64 + ty * 4 + (a - 4));
        if (i >= p.M) continue;
#pragma unroll
        for (int c = 0; c < 8; ++c) {
            const int j = n0 + (c < 4 ? tx * 4 + c : 64 + tx * 4 + (c - 4));
            if (j < p.N) epilogue<EPI>(b, p, i, j, acc[a][c]);
        }
    }
}

// ---------------------------------------------------------------------------
// Narrow variant for the blocked Cholesky's panel solve and trailing update
// (K = 64): 128 x 64 output tiles, 8 x 4 per thread, plain fp32 operands,
// four CTAs per SM, so more tiles are in flight to hide the short K loop's
// load and store latency.
// ---------------------------------------------------------------------------
constexpr int TN2 = 64;

template <int ALAY, int BLAY, int EPI>
__global__ void __launch_bounds__(256, 4) k_gemm_n64(const __grid_constant__ GemmBatch b) {
    __shared__ __align__(16) float As[2][TK][TM + TPAD];
    __shared__ __align__(16) float Bs[2][TK][TN2 + TPAD];
    const int tile = blockIdx.x;
    int lo = 0, hi = b.count - 1;
    while (lo < hi) {
        int mid = (lo + hi + 1) >> 1;
        if (b.tile_start[mid] <= tile) lo = mid; else hi = mid - 1;
    }
    const GemmProb& p = b.p[lo];
    const int local = tile - b.tile_start[lo];
    const int tn = b.tiles_n[lo];
    const int m0 = (local / tn) * TM;
    const int n0 = (local % tn) * TN2;
    if (p.lower_only && n0 >= m0 + TM) return;

    const int t = threadIdx.x;
    const int tx = t & 15, ty = t >> 4;
    float acc[8][4];
#pragma unroll
    for (int a = 0; a < 8; ++a)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[a][c] = 0.0f;

    int kbeg = 0, kend = p.K;
    if (p.k_tri == KTRI_B_UPPER) kend = min(p.K, n0 + TN2);
    else if (p.k_tri == KTRI_B_LOWER) kbeg = min(p.K, n0) & ~(TK - 1);
    else if (p.k_tri == KTRI_A_LOWER) kend = min(p.K, m0 + TM);
    const int ktiles = kend > kbeg ? (kend - kbeg + TK - 1) / TK : 0;
    const float* A = static_cast<const float*>(p.A);
    const float* Bm = static_cast<const float*>(p.Bm);
    float ra[NQ], rb[4];
    auto load = [&](int k0) {
#pragma unroll
        for (int q = 0; q < NQ; ++q) {
            int i, k;
            if (ALAY == A_KCONTIG) { k = t & (TK - 1); i = (t / TK) + (256 / TK) * q; }
            else                   { i = t & 127; k = (t >> 7) + 2 * q; }
            const int gi = m0 + i, gk = k0 + k;
            ra[q] = (gi < p.M && gk < p.K)
                        ? __ldg(A + (ALAY == A_KCONTIG ? (long long)gi * p.lda + gk : (long long)gk * p.lda + gi))
                        : 0.0f;
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            int j, k;
            if (BLAY == B_NCONTIG) { j = t & 63; k = (t >> 6) + 4 * q; }
            else                   { k = t & (TK - 1); j = (t / TK) + 16 * q; }
            const int gj = n0 + j, gk = k0 + k;
            rb[q] = (gj < p.N && gk < p.K)
                        ? __ldg(Bm + (BLAY == B_NCONTIG ? (long long)gk * p.ldb + gj : (long long)gj * p.ldb + gk))
                        : 0.0f;
        }
    };
    auto store = [&](int buf) {
#pragma unroll
        for (int q = 0; q < NQ; ++q) {
            int i, k;
            if (ALAY == A_KCONTIG) { k = t & (TK - 1); i = (t / TK) + (256 / TK) * q; }
            else                   { i = t & 127; k = (t >> 7) + 2 * q; }
            As[buf][k][i] = ra[q];
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            int j, k;
            if (BLAY == B_NCONTIG) { j = t & 63; k = (t >> 6) + 4 * q; }
            else                   { k = t & (TK - 1); j = (t / TK) + 16 * q; }
            Bs[buf][k][j] = rb[q];
        }
    };
    if (ktiles > 0) {
        load(kbeg);
        store(0);
    }
    __syncthreads();
    for (int kt = 0; kt < ktiles; ++kt) {
        const int cur = kt & 1;
        if (kt + 1 < ktiles) load(kbeg + (kt + 1) * TK);
#pragma unroll
        for (int k = 0; k < TK; ++k) {
            const float4 a0 = *reinterpret_cast<const float4*>(&As[cur][k][ty * 4]);
            const float4 a1 = *reinterpret_cast<const float4*>(&As[cur][k][64 + ty * 4]);
            const float4 b0 = *reinterpret_cast<const float4*>(&Bs[cur][k][tx * 4]);
            const float av[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
            const float bv[4] = {b0.x, b0.y, b0.z, b0.w};
#pragma unroll
            for (int a = 0; a < 8; ++a)
#pragma unroll
                for (int c = 0; c < 4; ++c) acc[a][c] = fmaf(av[a], bv[c], acc[a][c]);
        }
        if (kt + 1 < ktiles) store(cur ^ 1);
        __syncthreads();
    }
    const bool vec = (p.ldc & 3) == 0 && (reinterpret_cast<uintptr_t>(p.C) & 15) == 0 &&
                     (EPI != EPI_STORE || p.c_bf16 == nullptr);
#pragma unroll
    for (int a = 0; a < 8; ++a) {
        const int i = m0 + (a < 4 ? ty * 4 + a : 64 + ty * 4 + (a - 4));
        if (i >= p.M) continue;
        const int j = n0 + tx * 4;
        if (vec && j + 3 < p.N) {
            float4* dst = reinterpret_cast<float4*>(p.C + (long long)i * p.ldc + j);
            float4 v = make_float4(acc[a][0], acc[a][1], acc[a][2], acc[a][3]);
            if (EPI == EPI_SUB) {
                const float4 c = *dst;
                v = make_float4(c.x - v.x, c.y - v.y, c.z - v.z, c.w - v.w);
            } else if (EPI == EPI_STORE_NEG) {
                v = make_float4(-v.x, -v.y, -v.z, -v.w);
            }
            *dst = v;
        } else {
#pragma unroll
            for (int c = 0; c < 4; ++c)
                if (j + c < p.N) epilogue<EPI>(b, p, i, j + c, acc[a][c]);
        }
    }
}

template <int ALAY, int BLAY, int EPI>
static cudaError_t launch_n64(GemmBatch& b, cudaStream_t s, int64_t* launches) {
    int total = 0;
    for (int i = 0; i < b.count; ++i) {
        const GemmProb& p = b.p[i];
        const int tm = (p.M + TM - 1) / TM;
        const int tn = (p.N + TN2 - 1) / TN2;
        b.tiles_n[i] = tn;
        b.tile_start[i] = total;
        total += tm * tn;
    }
    b.tile_start[b.count] = total;
    if (total == 0) return cudaSuccess;
    k_gemm_n64<ALAY, BLAY, EPI><<<total, 256, 0, s>>>(b);
    ++*launches;
    return cudaGetLastError();
}

template <int ALAY, bool ASC, bool ABF, int BLAY, bool BSC, bool BBF, int EPI>
static cudaError_t launch_one(GemmBatch& b, cudaStream_t s, int64_t* launches) {
    b.log2B = -1;
    if (b.B > 0 && (b.B & (b.B - 1)) == 0) {
        int lg = 0;
        while ((1 << lg) < b.B) ++lg;
        b.log2B = lg;
    }
    int total = 0;
    for (int i = 0; i < b.count; ++i) {
        const GemmProb& p = b.p[i];
        const int tm = (p.M + TM - 1) / TM;
        const int tn = (p.N + TN - 1) / TN;
        b.tiles_n[i] = tn;
        b.tile_start[i] = total;
        total += tm * tn;
    }
    b.tile_start[b.count] = total;
    if (total == 0) return cudaSuccess;
    k_gemm<ALAY, ASC, ABF, BLAY, BSC, BBF, EPI><<<total, 256, 0, s>>>(b);
    ++*launches;
    return cudaGetLastError();
}

// Dispatch over the operand/epilogue combinations the library uses.
cudaError_t launch_gemm(const GemmKind& k, GemmBatch& b, cudaStream_t s, int64_t* launches) {
    if (b.count <= 0) return cudaSuccess;
    if (k.narrow && !k.a_scale && !k.b_scale && !k.a_bf16 && !k.b_bf16 && k.a_layout == A_KCONTIG &&
        k.b_layout == B_KCONTIG) {
        b.log2B = -1;
        if (k.epi == EPI_STORE) return launch_n64<A_KCONTIG, B_KCONTIG, EPI_STORE>(b, s, launches);
        if (k.epi == EPI_SUB) return launch_n64<A_KCONTIG, B_KCONTIG, EPI_SUB>(b, s, launches);
    }
#define MOARA_GEMM_CASE(AL, AS, AB, BL, BS, BB, EP)                                         \
    if (k.a_layout == AL && !!k.a_scale == AS && !!k.a_bf16 == AB && k.b_layout == BL &&   \
        !!k.b_scale == BS && !!k.b_bf16 == BB && k.epi == EP)                               \
        return launch_one<AL, AS, AB, BL, BS, BB, EP>(b, s, launches);
    // step: R = P^T V (+ Adam), V = G scaled (bf16 or f32) or G itself
    MOARA_GEMM_CASE(A_MCONTIG, false, false, B_NCONTIG, true, true, EPI_ADAM)
    MOARA_GEMM_CASE(A_MCONTIG, false, false, B_NCONTIG, true, false, EPI_ADAM)
    MOARA_GEMM_CASE(A_MCONTIG, false, false, B_NCONTIG, false, true, EPI_ADAM)
    MOARA_GEMM_CASE(A_MCONTIG, false, false, B_NCONTIG, false, false, EPI_ADAM)
    // step: dV = P N (+ weight update)
    MOARA_GEMM_CASE(A_KCONTIG, false, false, B_NCONTIG, false, false, EPI_UPDATE)
    // refresh: Y = V Omega, V scaled or raw, bf16 or f32
    MOARA_GEMM_CASE(A_KCONTIG, true, true, B_NCONTIG, false, false, EPI_STORE)
    MOARA_GEMM_CASE(A_KCONTIG, true, false, B_NCONTIG, false, false, EPI_STORE)
    MOARA_GEMM_CASE(A_KCONTIG, false, true, B_NCONTIG, false, false, EPI_STORE)
    // refresh: Z = V^T Q
    MOARA_GEMM_CASE(A_MCONTIG, true, true, B_NCONTIG, false, false, EPI_STORE)
    MOARA_GEMM_CASE(A_MCONTIG, true, false, B_NCONTIG, false, false, EPI_STORE)
    MOARA_GEMM_CASE(A_MCONTIG, false, true, B_NCONTIG, false, false, EPI_STORE)
    // plain fp32: Gram X^T X (MCONTIG), products X Y (KCONTIG), X L^-T (B KCONTIG)
    MOARA_GEMM_CASE(A_MCONTIG, false, false, B_NCONTIG, false, false, EPI_STORE)
    MOARA_GEMM_CASE(A_KCONTIG, false, false, B_NCONTIG, false, false, EPI_STORE)
    MOARA_GEMM_CASE(A_KCONTIG, false, false, B_KCONTIG, false, false, EPI_STORE)
    MOARA_GEMM_CASE(A_KCONTIG, false, false, B_NCONTIG, false, false, EPI_STORE_NEG)
    MOARA_GEMM_CASE(A_KCONTIG, false, false, B_KCONTIG, false, false, EPI_SUB)
#undef MOARA_GEMM_CASE
    return cudaErrorInvalidValue;
}

// ---------------------------------------------------------------------------
// Global gradient norm for clipping: sum of squares per chunk in fp32 (at
// most kNormChunk / 256 terms per thread), chunk sums added in fp64; fixed
// chunk-to-CTA assignment and reduction order.
// ---------------------------------------------------------------------------
__device__ __forceinline__ double block_sum_d(double v, double* red) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    __syncthreads();
    if (lane == 0) red[w] = v;
    __syncthreads();
    double t = 0.0;
    if (threadIdx.x == 0)
        for (int i = 0; i < (int)(blockDim.x >> 5); ++i) t += red[i];
    return t;
}

__global__ void __launch_bounds__(256) k_grad_sq(const __grid_constant__ GradNormBatch b, double* partials) {
    __shared__ double red[8];
    // a chunk is kNormChunk elements: 8 x 16 bytes per thread for bf16, 16 for
    // fp32; all of a thread's loads of a chunk are issued before the sums
    constexpr int VB = kNormChunk / (8 * 256);          // uint4 per thread, bf16
    constexpr int VF = kNormChunk / (4 * 256);          // float4 per thread, fp32
    static_assert(VB * 8 * 256 == kNormChunk && VF * 4 * 256 == kNormChunk, "chunk = whole vectors per thread");
    const long long total = b.chunk_start[b.count];
    double acc = 0.0;
    for (long long c = blockIdx.x; c < total; c += gridDim.x) {
        int lo = 0, hi = b.count - 1;
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (b.chunk_start[mid] <= c) lo = mid; else hi = mid - 1;
        }
        const long long e0 = (c - b.chunk_start[lo]) * kNormChunk;
        const long long e1 = min(e0 + (long long)kNormChunk, b.elems[lo]);
        float ss = 0.0f;
        if (b.dtype[lo] == MOARA_DTYPE_BF16) {
            const uint16_t* g = static_cast<const uint16_t*>(b.G[lo]);
            if (e1 - e0 == kNormChunk) {
                uint4 w[VB];
#pragma unroll
                for (int k = 0; k < VB; ++k)
                    w[k] = __ldcs(reinterpret_cast<const uint4*>(g + e0 + 8LL * (threadIdx.x + 256 * k)));
#pragma unroll
                for (int k = 0; k < VB; ++k) {
                    const uint32_t ww[4] = {w[k].x, w[k].y, w[k].z, w[k].w};
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        const float x = __uint_as_float(ww[q] << 16), y = __uint_as_float(ww[q] & 0xFFFF0000u);
                        ss = fmaf(x, x, ss);
                        ss = fmaf(y, y, ss);
                    }
                }
            } else {
                for (long long k = e0 + threadIdx.x; k < e1; k += blockDim.x) {
                    const float x = bf16_bits_to_f32(g[k]);
                    ss = fmaf(x, x, ss);
                }
            }
        } else {
            const float* g = static_cast<const float*>(b.G[lo]);
            if (e1 - e0 == kNormChunk) {
                float4 w[VF];
#pragma unroll
                for (int k = 0; k < VF; ++k)
                    w[k] = __ldcs(reinterpret_cast<const float4*>(g + e0 + 4LL * (threadIdx.x + 256 * k)));
#pragma unroll
                for (int k = 0; k < VF; ++k) {
                    ss = fmaf(w[k].x, w[k].x, ss);
                    ss = fmaf(w[k].y, w[k].y, ss);
                    ss = fmaf(w[k].z, w[k].z, ss);
                    ss = fmaf(w[k].w, w[k].w, ss);
                }
            } else {
                for (long long k = e0 + threadIdx.x; k < e1; k += blockDim.x) ss = fmaf(g[k], g[k], ss);
            }
        }
        acc += static_cast<double>(ss);
    }
    const double t = block_sum_d(acc, red);
    if (threadIdx.x == 0) partials[blockIdx.x] = t;
}

cudaError_t launch_grad_sq(const GradNormBatch& b, double* partials, cudaStream_t s, int64_t* launches) {
    k_grad_sq<<<kNormParts, 256, 0, s>>>(b, partials);
    ++*launches;
    return cudaGetLastError();
}

__global__ void __launch_bounds__(256) k_clip_finish(const double* partials, int n, const float* extra,
                                                     float max_norm, float* state) {
    __shared__ double red[8];
    double acc = 0.0;
    for (int i = threadIdx.x; i < n; i += blockDim.x) acc += partials[i];
    double t = block_sum_d(acc, red);
    if (threadIdx.x == 0) {
        if (extra != nullptr) t += static_cast<double>(*extra);
        const double norm = sqrt(t);
        const double coef = static_cast<double>(max_norm) / (norm + 1e-6);
        state[0] = static_cast<float>(norm);
        state[1] = static_cast<float>(coef < 1.0 ? coef : 1.0);
    }
}

cudaError_t launch_clip_finish(const double* partials, int n, const float* extra, float max_norm, float* state,
                               cudaStream_t s, int64_t* launches) {
    k_clip_finish<<<1, 256, 0, s>>>(partials, n, extra, max_norm, state);
    ++*launches;
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// fp32 -> (fp32 copy, bf16 round-to-nearest-even copy)
// ---------------------------------------------------------------------------
__global__ void k_f32_to_bf16(const float* __restrict__ src, float* dst_f32, uint16_t* dst_bf16,
                              long long count) {
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < count;
         i += (long long)gridDim.x * blockDim.x) {
        const float v = src[i];
        if (dst_f32 != nullptr && dst_f32 != src) dst_f32[i] = v;
        if (dst_bf16 != nullptr) {
            __nv_bfloat16 h = __float2bfloat16_rn(v);
            dst_bf16[i] = *reinterpret_cast<uint16_t*>(&h);
        }
    }
}

cudaError_t launch_f32_to_bf16(const float* src, float* dst_f32, uint16_t* dst_bf16,
                               long long count, cudaStream_t s, int64_t* launches) {
    if (count <= 0) return cudaSuccess;
    long long blocks = (count + 255) / 256;
    if (blocks > 152LL * 32) blocks = 152LL * 32;
    k_f32_to_bf16<<<static_cast<unsigned>(blocks), 256, 0, s>>>(src, dst_f32, dst_bf16, count);
    ++*launches;
    return cudaGetLastError();
}

}  // namespace moara
