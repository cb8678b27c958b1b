// Small dense kernels of the projector refresh (TruncatedSVD of Algorithm 1
// computed by randomized subspace iteration): the Gaussian test matrix, the
// diagonal blocks of the blocked Cholesky factorisation and of the triangular
// inverse used by CholeskyQR, the ordering of Ritz vectors, and the final sign
// convention.  One CTA per problem (or per diagonal block); the problems of a
// group run side by side in one launch.
#include <algorithm>
#include <cuda_bf16.h>

#include "internal.h"

namespace moara {

// ---------------------------------------------------------------------------
// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel random numbers: as easy
// as 1, 2, 3", SC'11): 10 rounds of the 4x32 S-box with the published
// multipliers and Weyl key increments.  Box-Muller turns pairs of uniforms
// into standard normals.
// ---------------------------------------------------------------------------
struct U4 { uint32_t x, y, z, w; };

__device__ __forceinline__ U4 philox4x32_10(U4 c, uint32_t k0, uint32_t k1) {
    const uint32_t M0 = 0xD2511F53u, M1 = 0xCD9E8D57u;
    const uint32_t W0 = 0x9E3779B9u, W1 = 0xBB67AE85u;
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        const uint32_t hi0 = __umulhi(M0, c.x), lo0 = M0 * c.x;
        const uint32_t hi1 = __umulhi(M1, c.z), lo1 = M1 * c.z;
        U4 n;
        n.x = hi1 ^ c.y ^ k0;
        n.y = lo1;
        n.z = hi0 ^ c.w ^ k1;
        n.w = lo0;
        c = n;
        k0 += W0;
        k1 += W1;
    }
    return c;
}

// uniform in (0, 1]: (x + 1) * 2^-32 with x the top 24 bits scaled
__device__ __forceinline__ float u01(uint32_t x) {
    return (static_cast<float>(x >> 8) + 1.0f) * (1.0f / 16777216.0f);
}

__global__ void k_philox_gaussian(const __grid_constant__ SmallBatch b) {
    const int pi = blockIdx.y;
    float* out = b.a[pi];
    const long long count = (long long)b.rows[pi] * b.l[pi];
    const uint32_t k0 = static_cast<uint32_t>(b.key[pi]);
    const uint32_t k1 = static_cast<uint32_t>(b.key[pi] >> 32);
    const long long groups = (count + 3) / 4;
    for (long long g = blockIdx.x * (long long)blockDim.x + threadIdx.x; g < groups;
         g += (long long)gridDim.x * blockDim.x) {
        U4 c{static_cast<uint32_t>(g), static_cast<uint32_t>(g >> 32), 0x4D6F4152u, 0x52616E64u};
        const U4 r = philox4x32_10(c, k0, k1);
        const float u1 = u01(r.x), u2 = u01(r.y), u3 = u01(r.z), u4 = u01(r.w);
        const float ra = sqrtf(-2.0f * logf(u1)), rb = sqrtf(-2.0f * logf(u3));
        float s2, c2, s4, c4;
        sincospif(2.0f * u2, &s2, &c2);
        sincospif(2.0f * u4, &s4, &c4);
        const float z[4] = {ra * c2, ra * s2, rb * c4, rb * s4};
        const long long base = g * 4;
#pragma unroll
        for (int q = 0; q < 4; ++q)
            if (base + q < count) out[base + q] = z[q];
    }
}

cudaError_t launch_philox_gaussian(const SmallBatch& b, cudaStream_t s, int64_t* launches) {
    if (b.count <= 0) return cudaSuccess;
    dim3 grid(64, b.count);
    k_philox_gaussian<<<grid, 256, 0, s>>>(b);
    ++*launches;
    return cudaGetLastError();
}

constexpr int kSmallThreads = 1024;

__device__ float block_sum(float v, float* red) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    __syncthreads();
    if (lane == 0) red[w] = v;
    __syncthreads();
    float t = 0.0f;
    if (w == 0) {
        t = (lane < static_cast<int>(blockDim.x >> 5)) ? red[lane] : 0.0f;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
        if (lane == 0) red[32] = t;
    }
    __syncthreads();
    return red[32];
}

// ---------------------------------------------------------------------------
// Diagonal blocks of a lower-triangular inverse: block j of problem y covers
// rows/cols [64j, min(64j + 64, l)); the block of a is inverted in shared
// memory by forward substitution and written to the same place in c.  The
// off-diagonal blocks are filled afterwards level by level with GEMMs:
//   inv([A 0; C D]) = [A^-1 0; -D^-1 C A^-1  D^-1].
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_tri_inverse_diag(const __grid_constant__ SmallBatch b) {
    __shared__ float Ls[kTriBase][kTriBase + 1];
    __shared__ float Xs[kTriBase][kTriBase + 1];
    const int pi = blockIdx.y;
    const int l = b.l[pi];
    const int i0 = blockIdx.x * kTriBase;
    if (i0 >= l) return;
    const int sz = min(kTriBase, l - i0);
    const float* L = b.a[pi];
    float* X = b.c[pi];
    for (int e = threadIdx.x; e < sz * sz; e += blockDim.x) {
        const int i = e / sz, c = e - i * sz;
        Ls[i][c] = L[(long long)(i0 + i) * l + i0 + c];
    }
    __syncthreads();
    // row by row; thread c owns column c
    for (int i = 0; i < sz; ++i) {
        if (threadIdx.x < sz) {
            const int c = threadIdx.x;
            float v = 0.0f;
            if (c <= i) {
                float acc = (c == i) ? 1.0f : 0.0f;
                for (int k = c; k < i; ++k) acc = fmaf(-Ls[i][k], Xs[k][c], acc);
                v = acc / Ls[i][i];
            }
            Xs[i][c] = v;
        }
        __syncthreads();
    }
    for (int e = threadIdx.x; e < sz * sz; e += blockDim.x) {
        const int i = e / sz, c = e - i * sz;
        X[(long long)(i0 + i) * l + i0 + c] = Xs[i][c];
    }
}

cudaError_t launch_tri_inverse_diag(const SmallBatch& b, cudaStream_t s, int64_t* launches) {
    if (b.count <= 0) return cudaSuccess;
    int lmax = 1;
    for (int i = 0; i < b.count; ++i) lmax = b.l[i] > lmax ? b.l[i] : lmax;
    dim3 grid((lmax + kTriBase - 1) / kTriBase, b.count);
    k_tri_inverse_diag<<<grid, 256, 0, s>>>(b);
    ++*launches;
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Blocked right-looking Cholesky.  k_trace_shift stores the diagonal shift of
// the shifted CholeskyQR pass; k_chol_diag factors the (at most 64 x 64)
// diagonal block at j0 in shared memory after the trailing updates of the
// earlier panels, checks its pivots, writes the factor in place and its
// inverse into the same block of c (the diagonal blocks of the triangular
// inverse).  The panel below the block and the trailing matrix are updated by
// grouped GEMMs on the host side.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_trace_shift(const __grid_constant__ SmallBatch b) {
    __shared__ float red[33];
    const int pi = blockIdx.x;
    const int l = b.l[pi];
    const float* A = b.a[pi];
    float tr = 0.0f;
    for (int i = threadIdx.x; i < l; i += blockDim.x) tr += A[(long long)i * l + i];
    tr = block_sum(tr, red);
    if (threadIdx.x == 0) b.b[pi][0] = b.shift_rel * sqrtf(static_cast<float>(b.rows[pi])) * tr;
}

cudaError_t launch_trace_shift(const SmallBatch& b, cudaStream_t s, int64_t* launches) {
    if (b.count <= 0) return cudaSuccess;
    k_trace_shift<<<b.count, 256, 0, s>>>(b);
    ++*launches;
    return cudaGetLastError();
}

// 128 threads, two per row: thread (i, h) keeps columns 32 h .. 32 h + 31 of
// row i of the block in registers (the two threads of a row are adjacent
// lanes of one warp).  The step loops stay rolled (a fully unrolled 64 x 64
// factorisation is too large for the instruction cache and stalls on
// instruction fetch): during the factorisation each row is shifted left by
// one column per step, the column crossing from the upper to the lower half
// by a lane shuffle, so the column being eliminated is always a[0] of the
// h = 0 thread and every register index is a compile-time constant; the
// finished column j of the factor is broadcast through shared memory from
// index 0, read as aligned 16-byte vectors.  The inverse then runs by
// forward substitution, thread (i, h) holding half of row i of the inverse;
// the finished row k is broadcast (its entries past k are exact zeros, so
// every row update may run over all 64 columns).  Each step costs two
// barriers of four warps.  The block moves between global and shared memory
// coalesced.
__global__ void __launch_bounds__(128) k_chol_diag(const __grid_constant__ SmallBatch b, int j0) {
    constexpr int NB = kTriBase;
    constexpr int HB = NB / 2;
    __shared__ float tile[NB][NB + 1];   // the block; the factor's lower part as it is finished
    __shared__ __align__(16) float bc[NB];   // broadcast column of the factor / row of the inverse
    __shared__ float piv;
    __shared__ int s_fail;
    const int pi = blockIdx.x;
    const int l = b.l[pi];
    if (j0 >= l) return;
    const int sz = min(NB, l - j0);
    float* A = b.a[pi];
    float* X = b.c[pi];
    const float shift = b.b[pi][0];
    const int t = threadIdx.x;
    const int i = t >> 1, h = t & 1, c0 = h * HB;
    const int lane = t & 31;
    // rows and columns past sz are padded with the identity
    for (int r = t >> 6; r < NB; r += 2) {
        const int c = t & 63;
        tile[r][c] = (r < sz && c < sz) ? A[(long long)(j0 + r) * l + j0 + c] + (r == c ? shift : 0.0f)
                                        : (r == c ? 1.0f : 0.0f);
    }
    if (t == 0) s_fail = 0;
    if (t < NB) bc[t] = 0.0f;
    __syncthreads();
    float a[HB];
#pragma unroll
    for (int k = 0; k < HB; ++k) a[k] = tile[i][c0 + k];
    // right-looking factorisation; at step j, a[k] of thread (i, h) holds
    // column j + 32 h + k of the updated row i.  A pivot that is not positive
    // and finite is replaced by 1 and marks the failure.
    const float4* col4 = reinterpret_cast<const float4*>(bc) + h * (HB / 4);
#pragma unroll 1
    for (int j = 0; j < NB; ++j) {
        if (i == j && h == 0) {
            float d = a[0];
            if (!(d > 0.0f) || !isfinite(d)) {
                d = 1.0f;
                s_fail = 1;
            }
            d = sqrtf(d);
            piv = d;
            tile[j][j] = d;
        }
        __syncthreads();
        float lij = 0.0f;
        if (i > j && h == 0) {
            lij = a[0] / piv;
            bc[i - j - 1] = lij;       // column j of L below the diagonal, from index 0
            tile[i][j] = lij;
        }
        lij = __shfl_sync(0xffffffffu, lij, lane & ~1);
        const float up = __shfl_sync(0xffffffffu, a[0], lane | 1);   // column j + 32, before its update
        __syncthreads();
        // row i -= L[i][j] * (column j of L)^T over columns j + 1 .., shifted
        // left by one: a[k] (column j + 32 h + k) takes bc[32 h + k - 1] =
        // L[j + 32 h + k][j].  Past index 62 - j, bc holds earlier columns'
        // values; they reach only slots of columns past the block or above
        // the diagonal (and rows i <= j, which are finished), none of which
        // is read again.
#pragma unroll
        for (int k = 1; k < HB; k += 4) {
            const float4 lk = col4[(k - 1) / 4];
            a[k - 1] = fmaf(-lij, lk.x, a[k]);
            a[k] = fmaf(-lij, lk.y, a[k + 1]);
            a[k + 1] = fmaf(-lij, lk.z, a[k + 2]);
            if (k + 3 < HB) a[k + 2] = fmaf(-lij, lk.w, a[k + 3]);
        }
        // the last slot: column j + 32 crosses from the upper half (h = 0
        // takes it, updated with bc[31]); past the block for h = 1
        a[HB - 1] = h == 0 ? fmaf(-lij, bc[HB - 1], up) : 0.0f;
    }
    // inverse by forward substitution: row k of the inverse is finished at
    // step k (divided by the pivot) and broadcast; rows below subtract
    // L[i][k] times it
    float x[HB];
#pragma unroll
    for (int c = 0; c < HB; ++c) x[c] = (c0 + c == i) ? 1.0f : 0.0f;
    float4* bc4 = reinterpret_cast<float4*>(bc) + h * (HB / 4);
#pragma unroll 1
    for (int k = 0; k < NB; ++k) {
        if (i == k) {
            const float inv = 1.0f / tile[k][k];
#pragma unroll
            for (int c = 0; c < HB; c += 4) {
                x[c] *= inv; x[c + 1] *= inv; x[c + 2] *= inv; x[c + 3] *= inv;
                bc4[c / 4] = make_float4(x[c], x[c + 1], x[c + 2], x[c + 3]);
            }
        }
        __syncthreads();
        if (i > k) {
            const float lik = tile[i][k];
#pragma unroll
            for (int c = 0; c < HB; c += 4) {
                const float4 r = bc4[c / 4];
                x[c] = fmaf(-lik, r.x, x[c]);
                x[c + 1] = fmaf(-lik, r.y, x[c + 1]);
                x[c + 2] = fmaf(-lik, r.z, x[c + 2]);
                x[c + 3] = fmaf(-lik, r.w, x[c + 3]);
            }
        }
        __syncthreads();
    }
    // the factor (zeros above the diagonal) in place, the inverse into c
#pragma unroll
    for (int k = 0; k < HB; ++k)
        if (c0 + k > i) tile[i][c0 + k] = 0.0f;
    __syncthreads();
    for (int r = t >> 6; r < sz; r += 2) {
        const int c = t & 63;
        if (c < sz) A[(long long)(j0 + r) * l + j0 + c] = tile[r][c];
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < HB; ++k) tile[i][c0 + k] = (c0 + k <= i) ? x[k] : 0.0f;
    __syncthreads();
    for (int r = t >> 6; r < sz; r += 2) {
        const int c = t & 63;
        if (c < sz) X[(long long)(j0 + r) * l + j0 + c] = tile[r][c];
    }
    if (t == 0 && s_fail && b.fail[pi] != nullptr) *b.fail[pi] = 1;
}

cudaError_t launch_chol_diag(const SmallBatch& b, int j0, cudaStream_t s, int64_t* launches) {
    if (b.count <= 0) return cudaSuccess;
    k_chol_diag<<<b.count, 128, 0, s>>>(b, j0);
    ++*launches;
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// h <- a^T rounded to bf16 (l x l): 32 x 32 tiles through shared memory.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_transpose_bf16(const __grid_constant__ SmallBatch b) {
    __shared__ float t[32][33];
    const int pi = blockIdx.z;
    const int l = b.l[pi];
    const float* src = b.a[pi];
    uint16_t* dst = b.h[pi];
    const int tiles = (l + 31) / 32;
    for (int tile = blockIdx.x; tile < tiles * tiles; tile += gridDim.x) {
        const int ti = tile / tiles, tj = tile - ti * tiles;
        const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
        for (int r = ty; r < 32; r += 8) {
            const int i = ti * 32 + r, j = tj * 32 + tx;
            t[r][tx] = (i < l && j < l) ? src[(long long)i * l + j] : 0.0f;
        }
        __syncthreads();
        for (int r = ty; r < 32; r += 8) {
            const int i = tj * 32 + r, j = ti * 32 + tx;   // dst row i = src column
            if (i < l && j < l) {
                __nv_bfloat16 h = __float2bfloat16_rn(t[tx][r]);
                dst[(long long)i * l + j] = *reinterpret_cast<uint16_t*>(&h);
            }
        }
        __syncthreads();
    }
}

cudaError_t launch_transpose_bf16(const SmallBatch& b, cudaStream_t s, int64_t* launches) {
    if (b.count <= 0) return cudaSuccess;
    k_transpose_bf16<<<dim3(128, 1, b.count), 256, 0, s>>>(b);
    ++*launches;
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Three bf16 planes of an fp32 matrix (rows x l, row-major, row pitch ld or
// l): hi = bf16(x), mid = bf16(x - hi), lo = bf16(x - hi - mid), so
// hi + mid + lo carries 24 significant bits.  With `transpose` the planes hold the l x rows transpose.
// Planes are consecutive at h, each rows * l elements.  32 x 32 tiles through
// shared memory keep both sides coalesced.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_split3(const __grid_constant__ SmallBatch b, int transpose) {
    __shared__ float t[32][33];
    const int pi = blockIdx.z;
    const int rows = b.rows[pi], cols = b.l[pi];
    const long long lds = b.ld[pi] > 0 ? b.ld[pi] : cols;
    const float* src = b.a[pi];
    uint16_t* dst = b.h[pi];
    const long long plane = (long long)rows * cols;
    const int tr = (rows + 31) / 32, tc = (cols + 31) / 32;
    const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
    // stores: thread (ty2, tx2) writes output rows ty2 and ty2 + 16 of the
    // tile, columns 2 tx2 and 2 tx2 + 1, as 4-byte pairs where aligned
    const int tx2 = threadIdx.x & 15, ty2 = threadIdx.x >> 4;
    const int orows = transpose ? cols : rows, ocols = transpose ? rows : cols;
    for (int tile = blockIdx.x; tile < tr * tc; tile += gridDim.x) {
        const int ti = tile / tc, tj = tile - ti * tc;
        for (int r = ty; r < 32; r += 8) {
            const int i = ti * 32 + r, j = tj * 32 + tx;
            t[r][tx] = (i < rows && j < cols) ? src[(long long)i * lds + j] : 0.0f;
        }
        __syncthreads();
        for (int rr = ty2; rr < 32; rr += 16) {
            const int i = (transpose ? tj : ti) * 32 + rr;          // output row
            const int j = (transpose ? ti : tj) * 32 + 2 * tx2;     // output column of the pair
            if (i < orows && j < ocols) {
                const float x0 = transpose ? t[2 * tx2][rr] : t[rr][2 * tx2];
                const float x1 = transpose ? t[2 * tx2 + 1][rr] : t[rr][2 * tx2 + 1];
                uint16_t h[3], g[3];
                {
                    const __nv_bfloat16 a0 = __float2bfloat16_rn(x0);
                    const float r0 = x0 - __bfloat162float(a0);
                    const __nv_bfloat16 a1 = __float2bfloat16_rn(r0);
                    const __nv_bfloat16 a2 = __float2bfloat16_rn(r0 - __bfloat162float(a1));
                    h[0] = *reinterpret_cast<const uint16_t*>(&a0);
                    h[1] = *reinterpret_cast<const uint16_t*>(&a1);
                    h[2] = *reinterpret_cast<const uint16_t*>(&a2);
                }
                {
                    const __nv_bfloat16 a0 = __float2bfloat16_rn(x1);
                    const float r0 = x1 - __bfloat162float(a0);
                    const __nv_bfloat16 a1 = __float2bfloat16_rn(r0);
                    const __nv_bfloat16 a2 = __float2bfloat16_rn(r0 - __bfloat162float(a1));
                    g[0] = *reinterpret_cast<const uint16_t*>(&a0);
                    g[1] = *reinterpret_cast<const uint16_t*>(&a1);
                    g[2] = *reinterpret_cast<const uint16_t*>(&a2);
                }
                const long long o = (long long)i * ocols + j;
                if (j + 1 < ocols && ((o | plane) & 1) == 0 && (reinterpret_cast<uintptr_t>(dst) & 3) == 0) {
#pragma unroll
                    for (int q = 0; q < 3; ++q)
                        *reinterpret_cast<uint32_t*>(dst + q * plane + o) =
                            static_cast<uint32_t>(h[q]) | (static_cast<uint32_t>(g[q]) << 16);
                } else {
#pragma unroll
                    for (int q = 0; q < 3; ++q) {
                        dst[q * plane + o] = h[q];
                        if (j + 1 < ocols) dst[q * plane + o + 1] = g[q];
                    }
                }
            }
        }
        __syncthreads();
    }
}

cudaError_t launch_split3(const SmallBatch& b, int transpose, cudaStream_t s, int64_t* launches) {
    if (b.count <= 0) return cudaSuccess;
    // as many blocks per item as the largest item has 32 x 32 tiles (at most 256)
    long long tiles = 1;
    for (int q = 0; q < b.count; ++q)
        tiles = std::max(tiles, (long long)((b.rows[q] + 31) / 32) * ((b.l[q] + 31) / 32));
    k_split3<<<dim3(static_cast<unsigned>(std::min(256LL, tiles)), 1, b.count), 256, 0, s>>>(b, transpose);
    ++*launches;
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// a <- I (l x l)
// ---------------------------------------------------------------------------
__global__ void k_set_identity(const __grid_constant__ SmallBatch b) {
    const int pi = blockIdx.y;
    const int l = b.l[pi];
    float* X = b.a[pi];
    const long long n = (long long)l * l;
    for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < n;
         e += (long long)gridDim.x * blockDim.x) {
        const long long i = e / l, c = e - i * l;
        X[e] = (i == c) ? 1.0f : 0.0f;
    }
}

cudaError_t launch_set_identity(const SmallBatch& b, cudaStream_t s, int64_t* launches) {
    if (b.count <= 0) return cudaSuccess;
    k_set_identity<<<dim3(32, b.count), 256, 0, s>>>(b);
    ++*launches;
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Ritz values d_j = x_j^T (C x_j) / x_j^T x_j from X (a) and W = C X (b), then the
// descending order: iaux[rank] = j, rank_j = #{i : d_i > d_j, or d_i == d_j
// and i < j}.  Ritz values go to c.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kSmallThreads) k_ritz_sort(const __grid_constant__ SmallBatch b) {
    const int pi = blockIdx.x;
    const int l = b.l[pi];
    const float* X = b.a[pi];
    const float* W = b.b[pi];
    float* d = b.c[pi];
    int* perm = b.iaux[pi];
    for (int j = threadIdx.x; j < l; j += blockDim.x) {
        float acc = 0.0f, nrm = 0.0f;
        for (int i = 0; i < l; ++i) {
            const float x = X[(long long)i * l + j];
            acc = fmaf(x, W[(long long)i * l + j], acc);
            nrm = fmaf(x, x, nrm);
        }
        d[j] = nrm > 0.0f ? acc / nrm : 0.0f;
    }
    __syncthreads();
    __threadfence_block();
    for (int j = threadIdx.x; j < l; j += blockDim.x) {
        const float dj = d[j];
        int rank = 0;
        for (int i = 0; i < l; ++i) {
            const float di = d[i];
            rank += (di > dj || (di == dj && i < j)) ? 1 : 0;
        }
        perm[rank] = j;
    }
}

// ---------------------------------------------------------------------------
// Exact Rayleigh-Ritz on the leading w = min(64, l) columns of an orthonormal
// X (a, l x l) with W = C X (b): H = X_w^T W_w (w x w, symmetric), its
// eigen-decomposition H = J diag(h) J^T by the cyclic Jacobi method (Golub
// and Van Loan, Matrix Computations, 4th ed., §8.5: one rotation per index
// pair zeroes H_pq; the pairs of a sweep are scheduled as a round-robin
// tournament so that the w / 2 rotations of a round touch disjoint rows and
// columns and run in parallel), then X_w <- X_w J and W_w <- W_w J.  The
// orthogonal iteration before it leaves span(X_w) close to the leading
// invariant subspace of C; within it the individual eigenvectors of
// separated eigenvalues are then exact up to rounding.  One CTA per
// problem, everything in shared memory, rows of X and W streamed in chunks.
// ---------------------------------------------------------------------------
constexpr int kLeadW = 64;
constexpr int kLeadChunk = 16;            // rows of X / W per chunk

__global__ void __launch_bounds__(kSmallThreads) k_lead_ritz(const __grid_constant__ SmallBatch b) {
    __shared__ float H[kLeadW][kLeadW + 1];
    __shared__ float J[kLeadW][kLeadW + 1];
    __shared__ float xs[kLeadChunk][kLeadW];
    __shared__ float ws[kLeadChunk][kLeadW];
    __shared__ float rc[kLeadW / 2], rs_[kLeadW / 2];
    __shared__ int rp[kLeadW / 2], rq[kLeadW / 2];
    __shared__ float red[33];
    const int pi = blockIdx.x;
    const int l = b.l[pi];
    const int w = l < kLeadW ? l : kLeadW;
    const int wp = w + (w & 1);                    // even player count (a dummy index when w is odd)
    float* X = b.a[pi];
    float* W = b.b[pi];
    const int t = threadIdx.x;
    // H = X_w^T W_w: thread t owns entries t, t + 1024, ... of the w x w block
    float acc[4] = {0.0f, 0.0f, 0.0f, 0.0f};
    for (int r0 = 0; r0 < l; r0 += kLeadChunk) {
        for (int e = t; e < kLeadChunk * kLeadW; e += blockDim.x) {
            const int i = e / kLeadW, j = e % kLeadW;
            const bool in = r0 + i < l && j < w;
            xs[i][j] = in ? X[(long long)(r0 + i) * l + j] : 0.0f;
            ws[i][j] = in ? W[(long long)(r0 + i) * l + j] : 0.0f;
        }
        __syncthreads();
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int e = t + u * blockDim.x;
            if (e < w * w) {
                const int p = e / w, q = e % w;
#pragma unroll 4
                for (int i = 0; i < kLeadChunk; ++i) acc[u] = fmaf(xs[i][p], ws[i][q], acc[u]);
            }
        }
        __syncthreads();
    }
    for (int e = t; e < kLeadW * kLeadW; e += blockDim.x) {
        const int p = e / kLeadW, q = e % kLeadW;
        H[p][q] = 0.0f;
        J[p][q] = (p == q) ? 1.0f : 0.0f;
    }
    __syncthreads();
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const int e = t + u * blockDim.x;
        if (e < w * w) H[e / w][e % w] = acc[u];
    }
    __syncthreads();
    // symmetrise (the two triangles differ by rounding)
    for (int e = t; e < w * w; e += blockDim.x) {
        const int p = e / w, q = e % w;
        if (p < q) {
            const float v = 0.5f * (H[p][q] + H[q][p]);
            H[p][q] = v;
            H[q][p] = v;
        }
    }
    __syncthreads();
    const int npairs = wp / 2;
    for (int sweep = 0; sweep < 20; ++sweep) {
        // stop once the off-diagonal mass is below fp32 resolution of the diagonal
        float off = 0.0f, dia = 0.0f;
        for (int e = t; e < w * w; e += blockDim.x) {
            const int p = e / w, q = e % w;
            const float v = H[p][q];
            if (p == q) dia = fmaf(v, v, dia); else off = fmaf(v, v, off);
        }
        off = block_sum(off, red);
        dia = block_sum(dia, red);
        if (!(off > 1e-14f * dia)) break;          // also ends on a non-finite H
        for (int round = 0; round < wp - 1; ++round) {
            if (t < npairs) {
                // tournament: player 0 fixed, the others rotate by one each round
                auto player = [&](int pos) { return pos == 0 ? 0 : 1 + (pos - 1 + round) % (wp - 1); };
                int p = player(t), q = player(wp - 1 - t);
                if (p > q) { const int x = p; p = q; q = x; }
                float c = 1.0f, sn = 0.0f;
                if (q < w) {
                    const float hpq = H[p][q];
                    if (fabsf(hpq) > 1e-30f) {
                        const float tau = (H[q][q] - H[p][p]) / (2.0f * hpq);
                        const float tt = (tau >= 0.0f ? 1.0f : -1.0f) / (fabsf(tau) + sqrtf(1.0f + tau * tau));
                        c = 1.0f / sqrtf(1.0f + tt * tt);
                        sn = tt * c;
                    }
                }
                rp[t] = p; rq[t] = q; rc[t] = c; rs_[t] = sn;
            }
            __syncthreads();
            // columns: H <- H G, J <- J G
            for (int e = t; e < npairs * kLeadW; e += blockDim.x) {
                const int k = e / kLeadW, row = e % kLeadW;
                const int p = rp[k], q = rq[k];
                if (q >= w || row >= w) continue;
                const float c = rc[k], sn = rs_[k];
                const float hp = H[row][p], hq = H[row][q];
                H[row][p] = c * hp - sn * hq;
                H[row][q] = sn * hp + c * hq;
                const float jp = J[row][p], jq = J[row][q];
                J[row][p] = c * jp - sn * jq;
                J[row][q] = sn * jp + c * jq;
            }
            __syncthreads();
            // rows: H <- G^T H
            for (int e = t; e < npairs * kLeadW; e += blockDim.x) {
                const int k = e / kLeadW, col = e % kLeadW;
                const int p = rp[k], q = rq[k];
                if (q >= w || col >= w) continue;
                const float c = rc[k], sn = rs_[k];
                const float hp = H[p][col], hq = H[q][col];
                H[p][col] = c * hp - sn * hq;
                H[q][col] = sn * hp + c * hq;
            }
            __syncthreads();
        }
    }
    // X_w <- X_w J, W_w <- W_w J, chunk by chunk
    for (int r0 = 0; r0 < l; r0 += kLeadChunk) {
        for (int e = t; e < kLeadChunk * kLeadW; e += blockDim.x) {
            const int i = e / kLeadW, j = e % kLeadW;
            const bool in = r0 + i < l && j < w;
            xs[i][j] = in ? X[(long long)(r0 + i) * l + j] : 0.0f;
            ws[i][j] = in ? W[(long long)(r0 + i) * l + j] : 0.0f;
        }
        __syncthreads();
        float ox = 0.0f, ow = 0.0f;
        const int i = t / kLeadW, j = t % kLeadW;     // 1024 threads = 16 rows x 64 columns
        if (j < w) {
            for (int k = 0; k < w; ++k) {
                ox = fmaf(xs[i][k], J[k][j], ox);
                ow = fmaf(ws[i][k], J[k][j], ow);
            }
        }
        __syncthreads();
        if (j < w && r0 + i < l) {
            X[(long long)(r0 + i) * l + j] = ox;
            W[(long long)(r0 + i) * l + j] = ow;
        }
        __syncthreads();
    }
}

cudaError_t launch_lead_ritz(const SmallBatch& b, cudaStream_t s, int64_t* launches) {
    if (b.count <= 0) return cudaSuccess;
    k_lead_ritz<<<b.count, kSmallThreads, 0, s>>>(b);
    ++*launches;
    return cudaGetLastError();
}

cudaError_t launch_ritz_sort(const SmallBatch& b, cudaStream_t s, int64_t* launches) {
    if (b.count <= 0) return cudaSuccess;
    k_ritz_sort<<<b.count, kSmallThreads, 0, s>>>(b);
    ++*launches;
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// c[:, q] = a[:, iaux[q]] for q < rows (a is l x l, c is l x rows).
// ---------------------------------------------------------------------------
__global__ void k_gather_cols(const __grid_constant__ SmallBatch b) {
    const int pi = blockIdx.y;
    const int l = b.l[pi], r = b.rows[pi];
    const float* X = b.a[pi];
    float* Xs = b.c[pi];
    const int* perm = b.iaux[pi];
    const long long n = (long long)l * r;
    for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < n;
         e += (long long)gridDim.x * blockDim.x) {
        const long long i = e / r, q = e - i * r;
        Xs[e] = X[i * l + perm[q]];
    }
}

cudaError_t launch_gather_cols(const SmallBatch& b, cudaStream_t s, int64_t* launches) {
    if (b.count <= 0) return cudaSuccess;
    k_gather_cols<<<dim3(64, b.count), 256, 0, s>>>(b);
    ++*launches;
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Final projector: each column of a (rows x l, here l = r columns) is scaled
// to unit length and signed so that its largest-magnitude entry is positive
// (lowest row wins ties), then stored to c (fp32) and h (bf16).  Skipped when
// the problem's fail flag is set, which leaves the previous projector in place.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_sign_fix_store(const __grid_constant__ SmallBatch b) {
    // a CTA owns 32 columns: lane = column, the 8 warps split the rows, so
    // every row segment is one coalesced 128-byte load
    __shared__ float s_best[8][32];
    __shared__ int s_bi[8][32];
    __shared__ float s_ss[8][32];
    __shared__ float s_sgn[32];
    const int pi = blockIdx.y;
    const int rows = b.rows[pi], r = b.l[pi];
    if (b.fail[pi] != nullptr && *b.fail[pi] != 0) return;
    const float* Pt = b.a[pi];
    float* P = b.c[pi];
    uint16_t* Pb = b.h[pi];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int q0 = blockIdx.x * 32; q0 < r; q0 += gridDim.x * 32) {
        const int q = q0 + lane;
        const bool col = q < r;
        // largest |entry| of the column over this warp's rows (ascending, so
        // the lowest row wins ties)
        float best = -1.0f, ss = 0.0f;
        int bi = 0x7fffffff;
        if (col)
            for (int i = warp; i < rows; i += 8) {
                const float v = Pt[(long long)i * r + q];
                const float a = fabsf(v);
                ss = fmaf(v, v, ss);
                if (a > best) { best = a; bi = i; }
            }
        s_best[warp][lane] = best;
        s_bi[warp][lane] = bi;
        s_ss[warp][lane] = ss;
        __syncthreads();
        if (warp == 0) {
            for (int w = 1; w < 8; ++w) {
                const float ob = s_best[w][lane];
                const int oi = s_bi[w][lane];
                ss += s_ss[w][lane];
                if (ob > best || (ob == best && oi < bi)) { best = ob; bi = oi; }
            }
            const float sg = (col && bi < rows && Pt[(long long)bi * r + q] < 0.0f) ? -1.0f : 1.0f;
            // unit length (a zero or non-finite column is left unscaled)
            const float nrm = sqrtf(ss);
            s_sgn[lane] = (nrm > 0.0f && isfinite(nrm)) ? sg / nrm : sg;
        }
        __syncthreads();
        const float sgnv = s_sgn[lane];
        if (col)
            for (int i = warp; i < rows; i += 8) {
                const float v = Pt[(long long)i * r + q] * sgnv;
                P[(long long)i * r + q] = v;
                if (Pb != nullptr) {
                    __nv_bfloat16 h = __float2bfloat16_rn(v);
                    Pb[(long long)i * r + q] = *reinterpret_cast<uint16_t*>(&h);
                }
            }
        __syncthreads();   // the shared arrays are reused by the next column group
    }
}

cudaError_t launch_sign_fix_store(const SmallBatch& b, cudaStream_t s, int64_t* launches) {
    if (b.count <= 0) return cudaSuccess;
    k_sign_fix_store<<<dim3(64, b.count), 256, 0, s>>>(b);
    ++*launches;
    return cudaGetLastError();
}

}  // namespace moara
