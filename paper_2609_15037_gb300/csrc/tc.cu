// Tensor-core path of the optimizer step for bf16 gradients (sm_103a):
//
//  K1  R = P^T V with V = Decompose(G, B) formed in shared memory in bf16
//      (at the first Adam step as the pair V_hi + V_lo, two MMAs; P is
//      exact in bf16), then
//      Optimizer_V (Adam) on R in the epilogue; writes the Adam update N as
//      bf16.  The block norms computed for V also drive Optimizer_M (Adam on
//      the block magnitudes M), done once per (row, block) by the CTAs of the
//      first rank tile.  (Algorithm 1; §3.1 / Appendix B.1.)
//  K2  dV = P N, then W <- W - lr*alpha*(Rep_B(dM) (.) dV) in the epilogue,
//      reading and writing W once.  (Algorithm 1.)
//
// Both kernels are persistent and warp specialised: one warp issues TMA tile
// loads into a 4-stage shared-memory ring, one thread issues tcgen05.mma into
// double-buffered TMEM accumulators, and epilogue warps drain TMEM while the
// next tile's MMAs run.  Every mbarrier wait is bounded; on expiry the kernel
// records MOARA_ERR_DEVICE_TIMEOUT in the context's status word, drains its
// own TMA copies and MMAs, frees TMEM and returns.
#include <cuda.h>
#include <cuda_bf16.h>

#include <algorithm>
#include <cstring>
#include <map>
#include <string>
#include <vector>

#include "tc.h"
#include "tc_ptx.cuh"

namespace moara {

namespace {

constexpr int kTcGroup = 224;                 // modules per launch (G maps in params)
constexpr long long kWaitLimit = 1LL << 32;   // ~2 s of SM clocks

struct TcMod {
    int m, n, r, kb;
    float* W;
    float* exp_avg;
    float* exp_avg_sq;
    float* mag_avg;
    float* mag_avg_sq;
    uint16_t* Nb;     // r x n bf16 Adam update of the direction branch
    float* dM;        // m x kb Adam update of the magnitude branch
};

struct TcTile {
    int mod, slot, t0, t1;
};

// ------------------------------------------------------------------- K1
constexpr int K1_BM = 256, K1_BN = 128, K1_BK = 64, K1_STAGES = 3;
constexpr int K1_A_BYTES = K1_BM * K1_BK * 2;           // 32 KB: four 64-row chunks of P^T
constexpr int K1_B_BYTES = K1_BK * K1_BN * 2;           // 16 KB: two 64-column chunks of G
// stage: A | B (G, then V_hi after the transform) | V_lo (V - V_hi in bf16)
constexpr int K1_STAGE_BYTES = K1_A_BYTES + 2 * K1_B_BYTES;
constexpr int K1_TX_BYTES = K1_A_BYTES + K1_B_BYTES;    // bytes the TMA brings per stage
constexpr int K1_WARPS = 18;                            // 0 TMA, 1 MMA, 2-9 transform, 10-17 epilogue
constexpr int K1_THREADS = K1_WARPS * 32;
constexpr int GUARD_BYTES = 16384;
constexpr int K1_SMEM = 1024 + K1_STAGES * K1_STAGE_BYTES + GUARD_BYTES + 2048;

struct K1Params {
    CUtensorMap gmap[kTcGroup];        // G of each launch slot: dims {n, m}, box {64, 64}
    const int* cta_start;              // tiles of CTA c: tiles[cta_start[c] .. cta_start[c+1])
    const TcTile* tiles;
    const TcMod* mods;
    const CUtensorMap* maps;           // per module: [0] P for K1, [1] P for K2, [2] N, [3] W
    int* status;
    float beta1, beta2, adam_eps, bc1, bc2, decomp_eps;
    int hilo;                          // project V_hi + V_lo (first Adam step) or V_hi only
};

// ------------------------------------------------------------------- K2
constexpr int K2_BM = 128, K2_BN = 256, K2_BK = 64, K2_STAGES = 3;
constexpr int K2_A_BYTES = K2_BM * K2_BK * 2;           // 16 KB: P rows, K-major
constexpr int K2_B_BYTES = K2_BK * K2_BN * 2;           // 32 KB: four 64-column chunks of N
constexpr int K2_STAGE_BYTES = K2_A_BYTES + K2_B_BYTES;
// W streams through a ring of 128-row x 32-column fp32 chunks (TMA in and out)
constexpr int K2_WCOLS = 32, K2_WBUF = 4;
constexpr int K2_WBYTES = K2_BM * K2_WCOLS * 4;         // 16 KB
constexpr int K2_WARPS = 12;                            // 0 TMA, 1 MMA, 2 W loader, 3 W storer, 4-11 epilogue
constexpr int K2_THREADS = K2_WARPS * 32;
constexpr int K2_GUARD = 8192;
constexpr int K2_SMEM = 1024 + K2_STAGES * K2_STAGE_BYTES + K2_WBUF * K2_WBYTES + K2_GUARD + 2048;

struct K2Params {
    const int* cta_start;
    const TcTile* tiles;
    const TcMod* mods;
    const CUtensorMap* maps;
    int* status;
    float step_scale;                  // lr * alpha
    int decompose;
};

struct SmemCtl {
    uint64_t full[4];
    uint64_t xform[4];
    uint64_t empty[4];   // sized for up to four stages
    uint64_t accf[2];
    uint64_t acce[2];
    uint64_t drain;
    uint64_t wfull[4];
    uint64_t wdone[4];
    uint64_t wempty[4];
    uint32_t tmem_base;
    int abort;
};

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
    return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

__device__ __forceinline__ bool wait_drain(uint32_t bar, uint32_t parity) {
    const long long t0 = clock64();
    while (!ptx::mbar_try_wait(bar, parity)) {
        if (clock64() - t0 > kWaitLimit) return false;
    }
    return true;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&h);
}

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

// ===========================================================================
// K1: projection R = P^T V with the decomposition fused into the B operand,
// direction-branch Adam in the epilogue, magnitude-branch Adam in the
// transform warps.
// ===========================================================================
template <int BLK, bool DECOMP>
__global__ void __launch_bounds__(K1_THREADS, 1) k1_project(const __grid_constant__ K1Params p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = align1024(smem_raw);
    SmemCtl* ctl = reinterpret_cast<SmemCtl*>(smem + K1_STAGES * K1_STAGE_BYTES + GUARD_BYTES);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    volatile int* abort_flag = &ctl->abort;

    if (threadIdx.x == 0) {
        for (int s = 0; s < K1_STAGES; ++s) {
            ptx::mbar_init(ptx::smem_u32(&ctl->full[s]), 1);
            ptx::mbar_init(ptx::smem_u32(&ctl->xform[s]), 256);
            ptx::mbar_init(ptx::smem_u32(&ctl->empty[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            ptx::mbar_init(ptx::smem_u32(&ctl->accf[b]), 1);
            ptx::mbar_init(ptx::smem_u32(&ctl->acce[b]), 8);
        }
        ptx::mbar_init(ptx::smem_u32(&ctl->drain), 1);
        ctl->abort = 0;
        ptx::fence_barrier_init();
    }
    if (warp == 1) {
        ptx::tmem_alloc(ptx::smem_u32(&ctl->tmem_base), 512);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = ctl->tmem_base;

    if (warp == 0) {
        // ------------------------------------------------------ TMA producer
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            uint32_t issued = 0, last_par = 0;
            bool ok = true;
            for (int t = p.cta_start[blockIdx.x]; t < p.cta_start[blockIdx.x + 1] && ok; ++t) {
                const TcTile tl = p.tiles[t];
                const TcMod& md = p.mods[tl.mod];
                const CUtensorMap* pmap = &p.maps[tl.mod * 4 + 0];
                const CUtensorMap* gmap = &p.gmap[tl.slot];
                const int r0 = tl.t0 * K1_BM, n0 = tl.t1 * K1_BN;
                const int nk = (md.m + K1_BK - 1) / K1_BK;
                for (int kb = 0; kb < nk; ++kb) {
                    if (!ptx::mbar_wait(ptx::smem_u32(&ctl->empty[stage]), phase ^ 1, abort_flag, p.status,
                                        MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit)) { ok = false; break; }
                    const uint32_t fb = ptx::smem_u32(&ctl->full[stage]);
                    ptx::mbar_arrive_expect_tx(fb, K1_TX_BYTES);
                    const uint32_t a = ptx::smem_u32(smem + stage * K1_STAGE_BYTES);
                    const uint32_t b = a + K1_A_BYTES;
#pragma unroll
                    for (int c = 0; c < 4; ++c) ptx::tma_load_2d(a + c * 8192, pmap, fb, r0 + 64 * c, kb * K1_BK);
#pragma unroll
                    for (int c = 0; c < 2; ++c) ptx::tma_load_2d(b + c * 8192, gmap, fb, n0 + 64 * c, kb * K1_BK);
                    issued |= 1u << stage;
                    last_par = (last_par & ~(1u << stage)) | (phase << stage);
                    if (++stage == K1_STAGES) { stage = 0; phase ^= 1; }
                }
            }
            if (!ok) {   // let the copies already in flight land before the CTA exits
                for (int s = 0; s < K1_STAGES; ++s)
                    if (issued & (1u << s)) wait_drain(ptx::smem_u32(&ctl->full[s]), (last_par >> s) & 1);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc = ptx::idesc_bf16(128, K1_BN, 1, 1);
            int stage = 0;
            uint32_t phase = 0;
            int buf = 0;
            uint32_t acc_phase = 0;
            bool ok = true;
            for (int t = p.cta_start[blockIdx.x]; t < p.cta_start[blockIdx.x + 1] && ok; ++t) {
                const TcTile tl = p.tiles[t];
                const TcMod& md = p.mods[tl.mod];
                const int r0 = tl.t0 * K1_BM;
                const int nh = (r0 + 128 < md.r) ? 2 : 1;
                const int nk = (md.m + K1_BK - 1) / K1_BK;
                if (!ptx::mbar_wait(ptx::smem_u32(&ctl->acce[buf]), acc_phase ^ 1, abort_flag, p.status,
                                    MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit)) { ok = false; break; }
                ptx::tc_fence_after();
                const uint32_t d0 = tmem + buf * 256;
                for (int kb = 0; kb < nk; ++kb) {
                    const uint32_t wb = DECOMP ? ptx::smem_u32(&ctl->xform[stage]) : ptx::smem_u32(&ctl->full[stage]);
                    if (!ptx::mbar_wait(wb, phase, abort_flag, p.status, MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit)) {
                        ok = false;
                        break;
                    }
                    ptx::tc_fence_after();
                    const uint32_t a = ptx::smem_u32(smem + stage * K1_STAGE_BYTES);
                    const uint32_t b = a + K1_A_BYTES;
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk) {
                        const uint64_t bdesc = ptx::smem_desc_sw128(b + kk * 2048, 8192, 1024);
                        const uint64_t ldesc = ptx::smem_desc_sw128(b + K1_B_BYTES + kk * 2048, 8192, 1024);
                        for (int h = 0; h < nh; ++h) {
                            const uint64_t adesc = ptx::smem_desc_sw128(a + h * 16384 + kk * 2048, 8192, 1024);
                            ptx::mma_f16(d0 + h * 128, adesc, bdesc, idesc, (kb | kk) != 0);
                            // P^T V_lo: the bf16 rounding residual of V, so that R carries
                            // about 16 significant bits (P is exact in bf16)
                            if (DECOMP && p.hilo) ptx::mma_f16(d0 + h * 128, adesc, ldesc, idesc, 1);
                        }
                    }
                    ptx::mma_commit(ptx::smem_u32(&ctl->empty[stage]));
                    if (++stage == K1_STAGES) { stage = 0; phase ^= 1; }
                }
                if (!ok) break;
                ptx::mma_commit(ptx::smem_u32(&ctl->accf[buf]));
                if (++buf == 2) { buf = 0; acc_phase ^= 1; }
            }
            // wait for every MMA this thread issued before TMEM is released
            ptx::mma_commit(ptx::smem_u32(&ctl->drain));
            wait_drain(ptx::smem_u32(&ctl->drain), 0);
        }
    } else if (warp < 10) {
        // ------------------------------------------------- transform warps
        if (DECOMP) {
            // 256 threads: lane bits 0-2 = row within an 8-row group, bit 3 = unit
            // half (16-byte units 0-3 or 4-7 of the 128-byte row), bit 4 =
            // 64-column chunk, warp = 8-row group.  Each quarter-warp then touches
            // 8 distinct rows of one chunk (conflict-free under the 128-byte
            // swizzle); the threads sharing a block are lanes ^ 8 and ^ 16.
            const int tid = threadIdx.x - 64;           // 0..255
            const int k = ((tid >> 5) << 3) | (tid & 7);  // row within the stage (0..63)
            const int hu = (tid >> 3) & 1;              // unit half
            const int hc = (tid >> 4) & 1;              // 64-column chunk
            const uint32_t x = static_cast<uint32_t>(k & 7);
            constexpr int UB = BLK / 8;                 // 16-byte units per block
            constexpr int UPB = UB < 4 ? UB : 4;        // units of a block held by this thread
            constexpr int NBT = 4 / UPB;                // blocks (or block parts) per thread
            int stage = 0;
            uint32_t phase = 0;
            bool ok = true;
            for (int t = p.cta_start[blockIdx.x]; t < p.cta_start[blockIdx.x + 1] && ok; ++t) {
                const TcTile tl = p.tiles[t];
                const TcMod& md = p.mods[tl.mod];
                const int n0 = tl.t1 * K1_BN;
                const bool do_mag = (tl.t0 == 0);
                const int mm = md.m, mkb = md.kb;
                float* const mag_avg = md.mag_avg;
                float* const mag_avg_sq = md.mag_avg_sq;
                float* const dMp = md.dM;
                const int nk = (mm + K1_BK - 1) / K1_BK;
                const bool owner = (UB < 8) || (hu == 0 && (UB < 16 || hc == 0));
                const bool mag_here = do_mag && owner;
                const int gb0 = (n0 + hc * 64 + hu * 32) / BLK;
                // the magnitude moments of the next stage are loaded one stage ahead,
                // so their latency is not on the path to the MMA
                float pma[NBT], pmas[NBT];
#pragma unroll
                for (int bl = 0; bl < NBT; ++bl) { pma[bl] = 0.0f; pmas[bl] = 0.0f; }
                if (mag_here && k < mm) {
#pragma unroll
                    for (int bl = 0; bl < NBT; ++bl) {
                        const int gb = gb0 + (UB < 8 ? bl : 0);
                        if (gb < mkb) {
                            pma[bl] = mag_avg[(long long)k * mkb + gb];
                            pmas[bl] = mag_avg_sq[(long long)k * mkb + gb];
                        }
                    }
                }
                for (int kb = 0; kb < nk; ++kb) {
                    float cma[NBT], cmas[NBT];
#pragma unroll
                    for (int bl = 0; bl < NBT; ++bl) { cma[bl] = pma[bl]; cmas[bl] = pmas[bl]; }
                    const int nrow = (kb + 1) * K1_BK + k;
                    if (mag_here && nrow < mm) {
#pragma unroll
                        for (int bl = 0; bl < NBT; ++bl) {
                            const int gb = gb0 + (UB < 8 ? bl : 0);
                            if (gb < mkb) {
                                pma[bl] = mag_avg[(long long)nrow * mkb + gb];
                                pmas[bl] = mag_avg_sq[(long long)nrow * mkb + gb];
                            }
                        }
                    }
                    const bool got = ptx::mbar_wait(ptx::smem_u32(&ctl->full[stage]), phase, abort_flag, p.status,
                                                    MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit);
                    if (!__all_sync(0xffffffffu, got)) { ok = false; break; }
                    uint8_t* row = smem + stage * K1_STAGE_BYTES + K1_A_BYTES + hc * 8192 + k * 128;
                    uint4 d[4];
#pragma unroll
                    for (int u = 0; u < 4; ++u)
                        d[u] = *reinterpret_cast<const uint4*>(row + (((hu * 4 + u) ^ x) << 4));
                    float ssu[4];
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        const uint32_t w[4] = {d[u].x, d[u].y, d[u].z, d[u].w};
                        float s2 = 0.0f;
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const float lo = bf_lo(w[e]), hi = bf_hi(w[e]);
                            s2 = fmaf(lo, lo, s2);
                            s2 = fmaf(hi, hi, s2);
                        }
                        ssu[u] = s2;
                    }
                    float ssb[NBT];
#pragma unroll
                    for (int bl = 0; bl < NBT; ++bl) {
                        float s2 = 0.0f;
#pragma unroll
                        for (int u = 0; u < UPB; ++u) s2 += ssu[bl * UPB + u];
                        ssb[bl] = s2;
                    }
                    if (UB >= 8) ssb[0] += __shfl_xor_sync(0xffffffffu, ssb[0], 8);    // other unit half
                    if (UB >= 16) ssb[0] += __shfl_xor_sync(0xffffffffu, ssb[0], 16);  // other chunk
                    float inv[NBT];
                    float mag[NBT];
#pragma unroll
                    for (int bl = 0; bl < NBT; ++bl) {
                        mag[bl] = sqrtf(ssb[bl]);
                        inv[bl] = 1.0f / (mag[bl] + p.decomp_eps);
                    }
                    uint8_t* lrow = row + K1_B_BYTES;
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        const float sc = inv[u / UPB];
                        const uint32_t w[4] = {d[u].x, d[u].y, d[u].z, d[u].w};
                        uint32_t hi[4], lo[4];
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const float v0 = bf_lo(w[e]) * sc, v1 = bf_hi(w[e]) * sc;
                            hi[e] = pack_bf16x2(v0, v1);
                            lo[e] = pack_bf16x2(v0 - bf_lo(hi[e]), v1 - bf_hi(hi[e]));
                        }
                        const uint32_t off = ((hu * 4 + u) ^ x) << 4;
                        *reinterpret_cast<uint4*>(row + off) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
                        if (p.hilo) *reinterpret_cast<uint4*>(lrow + off) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
                    }
                    ptx::fence_proxy_async_smem();
                    ptx::mbar_arrive(ptx::smem_u32(&ctl->xform[stage]));
                    // Optimizer_M on the block magnitudes, once per (row, block)
                    const int grow = kb * K1_BK + k;
                    if (mag_here && grow < mm) {
#pragma unroll
                        for (int bl = 0; bl < NBT; ++bl) {
                            const int gb = gb0 + (UB < 8 ? bl : 0);
                            if (gb < mkb) {
                                const long long o = (long long)grow * mkb + gb;
                                const float ma = p.beta1 * cma[bl] + (1.0f - p.beta1) * mag[bl];
                                const float mas = p.beta2 * cmas[bl] + (1.0f - p.beta2) * mag[bl] * mag[bl];
                                mag_avg[o] = ma;
                                mag_avg_sq[o] = mas;
                                dMp[o] = (ma / p.bc1) / (sqrtf(mas / p.bc2) + p.adam_eps);
                            }
                        }
                    }
                    if (++stage == K1_STAGES) { stage = 0; phase ^= 1; }
                }
            }
        }
    } else {
        // ------------------------------------------------- epilogue warps
        const int ew = warp - 10;                      // 0..7
        const int q = warp & 3;                        // TMEM lane quarter of this warp
        const int h = ew >> 2;                         // accumulator half (rows 0-127 / 128-255)
        int buf = 0;
        uint32_t acc_phase = 0;
        bool ok = true;
        for (int t = p.cta_start[blockIdx.x]; t < p.cta_start[blockIdx.x + 1] && ok; ++t) {
            const TcTile tl = p.tiles[t];
            const TcMod& md = p.mods[tl.mod];
            const int r0 = tl.t0 * K1_BM, n0 = tl.t1 * K1_BN;
            const bool got = ptx::mbar_wait(ptx::smem_u32(&ctl->accf[buf]), acc_phase, abort_flag, p.status,
                                            MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit);
            if (!__all_sync(0xffffffffu, got)) { ok = false; break; }
            ptx::tc_fence_after();
            const bool half_valid = (r0 + h * 128) < md.r;
            if (half_valid) {
                const int a = r0 + h * 128 + q * 32 + lane;
                const bool row_ok = a < md.r;
#pragma unroll 1
                for (int c = 0; c < K1_BN / 16; ++c) {
                    float v[16];
                    __syncwarp();
                    ptx::tmem_ld16(tmem + (static_cast<uint32_t>(q * 32) << 16) + buf * 256 + h * 128 + c * 16, v);
                    const int j0 = n0 + c * 16;
                    if (!row_ok || j0 >= md.n) continue;
                    const long long o = (long long)a * md.n + j0;
                    if (j0 + 16 <= md.n) {
                        float4* ea4 = reinterpret_cast<float4*>(md.exp_avg + o);
                        float4* es4 = reinterpret_cast<float4*>(md.exp_avg_sq + o);
                        float ea[16], es[16];
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const float4 x = ea4[e], y = es4[e];
                            ea[4 * e] = x.x; ea[4 * e + 1] = x.y; ea[4 * e + 2] = x.z; ea[4 * e + 3] = x.w;
                            es[4 * e] = y.x; es[4 * e + 1] = y.y; es[4 * e + 2] = y.z; es[4 * e + 3] = y.w;
                        }
                        uint32_t nb[8];
                        float nv[16];
#pragma unroll
                        for (int e = 0; e < 16; ++e) {
                            ea[e] = p.beta1 * ea[e] + (1.0f - p.beta1) * v[e];
                            es[e] = p.beta2 * es[e] + (1.0f - p.beta2) * v[e] * v[e];
                            nv[e] = (ea[e] / p.bc1) / (sqrtf(es[e] / p.bc2) + p.adam_eps);
                        }
#pragma unroll
                        for (int e = 0; e < 8; ++e) nb[e] = pack_bf16x2(nv[2 * e], nv[2 * e + 1]);
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            ea4[e] = make_float4(ea[4 * e], ea[4 * e + 1], ea[4 * e + 2], ea[4 * e + 3]);
                            es4[e] = make_float4(es[4 * e], es[4 * e + 1], es[4 * e + 2], es[4 * e + 3]);
                        }
                        uint4* n4 = reinterpret_cast<uint4*>(md.Nb + o);
                        n4[0] = make_uint4(nb[0], nb[1], nb[2], nb[3]);
                        n4[1] = make_uint4(nb[4], nb[5], nb[6], nb[7]);
                    } else {
#pragma unroll
                        for (int e = 0; e < 16; ++e) {
                            if (j0 + e >= md.n) continue;
                            const float ea = p.beta1 * md.exp_avg[o + e] + (1.0f - p.beta1) * v[e];
                            const float es = p.beta2 * md.exp_avg_sq[o + e] + (1.0f - p.beta2) * v[e] * v[e];
                            md.exp_avg[o + e] = ea;
                            md.exp_avg_sq[o + e] = es;
                            const float nv = (ea / p.bc1) / (sqrtf(es / p.bc2) + p.adam_eps);
                            __nv_bfloat16 hb = __float2bfloat16_rn(nv);
                            md.Nb[o + e] = *reinterpret_cast<uint16_t*>(&hb);
                        }
                    }
                }
            }
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(ptx::smem_u32(&ctl->acce[buf]));
            if (++buf == 2) { buf = 0; acc_phase ^= 1; }
        }
    }

    ptx::tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, 512);
    }
}

// ===========================================================================
// K2: back-projection dV = P N and the weight update in the epilogue.
// ===========================================================================
template <int BLK>
__global__ void __launch_bounds__(K2_THREADS, 1) k2_backproject(const __grid_constant__ K2Params p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = align1024(smem_raw);
    uint8_t* wring = smem + K2_STAGES * K2_STAGE_BYTES;
    SmemCtl* ctl = reinterpret_cast<SmemCtl*>(wring + K2_WBUF * K2_WBYTES + K2_GUARD);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    volatile int* abort_flag = &ctl->abort;

    if (threadIdx.x == 0) {
        for (int s = 0; s < K2_STAGES; ++s) {
            ptx::mbar_init(ptx::smem_u32(&ctl->full[s]), 1);
            ptx::mbar_init(ptx::smem_u32(&ctl->empty[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            ptx::mbar_init(ptx::smem_u32(&ctl->accf[b]), 1);
            ptx::mbar_init(ptx::smem_u32(&ctl->acce[b]), 8);
        }
        for (int b = 0; b < K2_WBUF; ++b) {
            ptx::mbar_init(ptx::smem_u32(&ctl->wfull[b]), 1);
            ptx::mbar_init(ptx::smem_u32(&ctl->wdone[b]), 8);
            ptx::mbar_init(ptx::smem_u32(&ctl->wempty[b]), 1);
        }
        ptx::mbar_init(ptx::smem_u32(&ctl->drain), 1);
        ctl->abort = 0;
        ptx::fence_barrier_init();
    }
    if (warp == 1) {
        ptx::tmem_alloc(ptx::smem_u32(&ctl->tmem_base), 512);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = ctl->tmem_base;
    const int t_begin = p.cta_start[blockIdx.x], t_end = p.cta_start[blockIdx.x + 1];

    if (warp == 0) {
        // ------------------------------------------------ operand TMA producer
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            uint32_t issued = 0, last_par = 0;
            bool ok = true;
            for (int t = t_begin; t < t_end && ok; ++t) {
                const TcTile tl = p.tiles[t];
                const TcMod& md = p.mods[tl.mod];
                const CUtensorMap* amap = &p.maps[tl.mod * 4 + 1];
                const CUtensorMap* bmap = &p.maps[tl.mod * 4 + 2];
                const int i0 = tl.t0 * K2_BM, n0 = tl.t1 * K2_BN;
                const int nk = (md.r + K2_BK - 1) / K2_BK;
                for (int kb = 0; kb < nk; ++kb) {
                    if (!ptx::mbar_wait(ptx::smem_u32(&ctl->empty[stage]), phase ^ 1, abort_flag, p.status,
                                        MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit)) { ok = false; break; }
                    const uint32_t fb = ptx::smem_u32(&ctl->full[stage]);
                    ptx::mbar_arrive_expect_tx(fb, K2_STAGE_BYTES);
                    const uint32_t a = ptx::smem_u32(smem + stage * K2_STAGE_BYTES);
                    const uint32_t b = a + K2_A_BYTES;
                    ptx::tma_load_2d(a, amap, fb, kb * K2_BK, i0);
#pragma unroll
                    for (int c = 0; c < 4; ++c) ptx::tma_load_2d(b + c * 8192, bmap, fb, n0 + 64 * c, kb * K2_BK);
                    issued |= 1u << stage;
                    last_par = (last_par & ~(1u << stage)) | (phase << stage);
                    if (++stage == K2_STAGES) { stage = 0; phase ^= 1; }
                }
            }
            if (!ok) {
                for (int s = 0; s < K2_STAGES; ++s)
                    if (issued & (1u << s)) wait_drain(ptx::smem_u32(&ctl->full[s]), (last_par >> s) & 1);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc = ptx::idesc_bf16(128, K2_BN, 0, 1);
            int stage = 0;
            uint32_t phase = 0;
            int buf = 0;
            uint32_t acc_phase = 0;
            bool ok = true;
            for (int t = t_begin; t < t_end && ok; ++t) {
                const TcTile tl = p.tiles[t];
                const TcMod& md = p.mods[tl.mod];
                const int nk = (md.r + K2_BK - 1) / K2_BK;
                if (!ptx::mbar_wait(ptx::smem_u32(&ctl->acce[buf]), acc_phase ^ 1, abort_flag, p.status,
                                    MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit)) { ok = false; break; }
                ptx::tc_fence_after();
                const uint32_t d0 = tmem + buf * 256;
                for (int kb = 0; kb < nk; ++kb) {
                    if (!ptx::mbar_wait(ptx::smem_u32(&ctl->full[stage]), phase, abort_flag, p.status,
                                        MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit)) { ok = false; break; }
                    ptx::tc_fence_after();
                    const uint32_t a = ptx::smem_u32(smem + stage * K2_STAGE_BYTES);
                    const uint32_t b = a + K2_A_BYTES;
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk) {
                        const uint64_t adesc = ptx::smem_desc_sw128(a + kk * 32, 16, 1024);
                        const uint64_t bdesc = ptx::smem_desc_sw128(b + kk * 2048, 8192, 1024);
                        ptx::mma_f16(d0, adesc, bdesc, idesc, (kb | kk) != 0);
                    }
                    ptx::mma_commit(ptx::smem_u32(&ctl->empty[stage]));
                    if (++stage == K2_STAGES) { stage = 0; phase ^= 1; }
                }
                if (!ok) break;
                ptx::mma_commit(ptx::smem_u32(&ctl->accf[buf]));
                if (++buf == 2) { buf = 0; acc_phase ^= 1; }
            }
            ptx::mma_commit(ptx::smem_u32(&ctl->drain));
            wait_drain(ptx::smem_u32(&ctl->drain), 0);
        }
    } else if (warp == 2) {
        // ------------------------------------------- W chunk loader (TMA in)
        if (lane == 0) {
            uint32_t g = 0;
            uint32_t issued = 0, last_par = 0;
            bool ok = true;
            for (int t = t_begin; t < t_end && ok; ++t) {
                const TcTile tl = p.tiles[t];
                const TcMod& md = p.mods[tl.mod];
                const CUtensorMap* wmap = &p.maps[tl.mod * 4 + 3];
                const int i0 = tl.t0 * K2_BM, n0 = tl.t1 * K2_BN;
                const int nc = min(K2_BN / K2_WCOLS, (md.n - n0 + K2_WCOLS - 1) / K2_WCOLS);
                for (int c = 0; c < nc; ++c, ++g) {
                    const int b = g % K2_WBUF;
                    const uint32_t ph = (g / K2_WBUF) & 1;
                    if (!ptx::mbar_wait(ptx::smem_u32(&ctl->wempty[b]), ph ^ 1, abort_flag, p.status,
                                        MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit)) { ok = false; break; }
                    const uint32_t fb = ptx::smem_u32(&ctl->wfull[b]);
                    ptx::mbar_arrive_expect_tx(fb, K2_WBYTES);
                    ptx::tma_load_2d(ptx::smem_u32(wring + b * K2_WBYTES), wmap, fb, n0 + c * K2_WCOLS, i0);
                    issued |= 1u << b;
                    last_par = (last_par & ~(1u << b)) | (ph << b);
                }
            }
            if (!ok) {
                for (int b = 0; b < K2_WBUF; ++b)
                    if (issued & (1u << b)) wait_drain(ptx::smem_u32(&ctl->wfull[b]), (last_par >> b) & 1);
            }
        }
    } else if (warp == 3) {
        // ------------------------------------------ W chunk storer (TMA out)
        if (lane == 0) {
            uint32_t g = 0;
            bool ok = true;
            for (int t = t_begin; t < t_end && ok; ++t) {
                const TcTile tl = p.tiles[t];
                const TcMod& md = p.mods[tl.mod];
                const CUtensorMap* wmap = &p.maps[tl.mod * 4 + 3];
                const int i0 = tl.t0 * K2_BM, n0 = tl.t1 * K2_BN;
                const int nc = min(K2_BN / K2_WCOLS, (md.n - n0 + K2_WCOLS - 1) / K2_WCOLS);
                for (int c = 0; c < nc; ++c, ++g) {
                    const int b = g % K2_WBUF;
                    const uint32_t ph = (g / K2_WBUF) & 1;
                    if (!ptx::mbar_wait(ptx::smem_u32(&ctl->wdone[b]), ph, abort_flag, p.status,
                                        MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit)) { ok = false; break; }
                    ptx::tma_store_2d(wmap, ptx::smem_u32(wring + b * K2_WBYTES), n0 + c * K2_WCOLS, i0);
                    ptx::bulk_commit_group();
                    ptx::bulk_wait_read_all();            // the chunk may be refilled once read
                    ptx::mbar_arrive(ptx::smem_u32(&ctl->wempty[b]));
                }
            }
            ptx::bulk_wait_all();
        }
    } else {
        // ------------------------------------------------- epilogue warps
        // 8 warps: TMEM lane quarter q = warp % 4, column half ch of each
        // 32-column chunk; each thread updates 16 values of its W row in the
        // swizzled shared-memory chunk: W -= lr * alpha * dM * (P N).
        const int ew = warp - 4;                        // 0..7
        const int q = warp & 3;
        const int ch = ew >> 2;
        const int il = q * 32 + lane;                   // row within the tile
        constexpr int NDM = BLK >= 16 ? 1 : 16 / BLK;   // dM values per thread and chunk
        int buf = 0;
        uint32_t acc_phase = 0;
        uint32_t g = 0;
        bool ok = true;
        for (int t = t_begin; t < t_end && ok; ++t) {
            const TcTile tl = p.tiles[t];
            const TcMod& md = p.mods[tl.mod];
            const int mm = md.m, nn = md.n, mkb = md.kb;
            const float* const dMp = md.dM;
            const int i0 = tl.t0 * K2_BM, n0 = tl.t1 * K2_BN;
            const int i = i0 + il;
            const bool row_ok = i < mm;
            const int nc = min(K2_BN / K2_WCOLS, (nn - n0 + K2_WCOLS - 1) / K2_WCOLS);
            const bool got = ptx::mbar_wait(ptx::smem_u32(&ctl->accf[buf]), acc_phase, abort_flag, p.status,
                                            MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit);
            if (!__all_sync(0xffffffffu, got)) { ok = false; break; }
            ptx::tc_fence_after();
            for (int c = 0; c < nc; ++c, ++g) {
                const int b = g % K2_WBUF;
                const uint32_t ph = (g / K2_WBUF) & 1;
                const int j0 = n0 + c * K2_WCOLS + ch * 16;
                float dm[NDM];
#pragma unroll
                for (int d = 0; d < NDM; ++d) {
                    const int jb = (j0 + 8 * d) / BLK;
                    dm[d] = (p.decompose && row_ok && jb < mkb) ? dMp[(long long)i * mkb + jb] : 1.0f;
                }
                float v[16];
                __syncwarp();
                ptx::tmem_ld16(tmem + (static_cast<uint32_t>(q * 32) << 16) + buf * 256 + c * K2_WCOLS + ch * 16, v);
                const bool gotw = ptx::mbar_wait(ptx::smem_u32(&ctl->wfull[b]), ph, abort_flag, p.status,
                                                 MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit);
                if (!__all_sync(0xffffffffu, gotw)) { ok = false; break; }
                uint8_t* wrow = wring + b * K2_WBYTES + il * 128;
                const uint32_t x = static_cast<uint32_t>(il & 7);
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    float4* w4 = reinterpret_cast<float4*>(wrow + (((ch * 4 + u) ^ x) << 4));
                    float4 w = *w4;
                    const float d0 = dm[NDM == 1 ? 0 : (u * 4) / BLK];
                    w.x -= p.step_scale * (d0 * v[4 * u + 0]);
                    w.y -= p.step_scale * (d0 * v[4 * u + 1]);
                    w.z -= p.step_scale * (d0 * v[4 * u + 2]);
                    w.w -= p.step_scale * (d0 * v[4 * u + 3]);
                    *w4 = w;
                }
                ptx::fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive(ptx::smem_u32(&ctl->wdone[b]));
            }
            if (!ok) break;
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(ptx::smem_u32(&ctl->acce[buf]));
            if (++buf == 2) { buf = 0; acc_phase ^= 1; }
        }
    }

    ptx::tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, 512);
    }
}

// ---------------------------------------------------------------- host side
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

bool encode_2d(EncodeTiledFn enc, CUtensorMap* map, CUtensorMapDataType dt, int esize, const void* ptr,
               uint64_t inner, uint64_t outer, uint32_t box_inner, uint32_t box_outer) {
    const cuuint64_t dims[2] = {inner, outer};
    const cuuint64_t strides[1] = {inner * esize};
    const cuuint32_t box[2] = {box_inner, box_outer};
    const cuuint32_t estr[2] = {1, 1};
    return enc(map, dt, 2, const_cast<void*>(ptr), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
               CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_bf16_2d(EncodeTiledFn enc, CUtensorMap* map, const void* ptr, uint64_t inner, uint64_t outer,
                    uint32_t box_inner, uint32_t box_outer) {
    return encode_2d(enc, map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, ptr, inner, outer, box_inner, box_outer);
}

template <int BLK>
void set_smem_attrs() {
    cudaFuncSetAttribute(k1_project<BLK, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, K1_SMEM);
    cudaFuncSetAttribute(k1_project<BLK, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, K1_SMEM);
    cudaFuncSetAttribute(k2_backproject<BLK>, cudaFuncAttributeMaxDynamicSharedMemorySize, K2_SMEM);
}

}  // namespace

struct TcState {
    int device = 0;
    int* d_status = nullptr;
    int sms = 148;
    EncodeTiledFn encode = nullptr;
    std::string err;
    std::vector<TcMod> mods;               // indexed by module id (unsupported ones left zero)
    std::vector<CUtensorMap> maps;         // 4 per module id
    TcMod* d_mods = nullptr;
    CUtensorMap* d_maps = nullptr;
    int cap = 0;
    bool dirty = false;
    // Per-CTA work lists of one launch (CSR: start offsets, then tiles).
    struct Tiles {
        void* mem = nullptr;
        const int* k1_start = nullptr; const TcTile* k1 = nullptr; int g1 = 0;
        const int* k2_start = nullptr; const TcTile* k2 = nullptr; int g2 = 0;
    };
    std::map<std::vector<int>, Tiles> tiles;
    bool attrs_set = false;
    K1Params p1;                           // parameter block of the next K1 launch
};

bool tc_supported(int m, int n, int r, int B, int dtype, int decompose) {
    if (dtype != MOARA_DTYPE_BF16) return false;
    if (m < 1 || n < 8 || r < 8) return false;
    if ((n % 8) != 0 || (r % 8) != 0) return false;
    if (decompose && !(B == 8 || B == 16 || B == 32 || B == 64 || B == 128)) return false;
    if (!decompose && !(B >= 1)) return false;
    return true;
}

TcState* tc_create(int device, int* d_status) {
    TcState* st = new TcState();
    st->device = device;
    st->d_status = d_status;
    cudaDeviceProp prop{};
    if (cudaGetDeviceProperties(&prop, device) == cudaSuccess) {
        st->sms = prop.multiProcessorCount;
        if (prop.major != 10 || prop.minor != 3) {   // these kernels are built for sm_103a only
            delete st;
            return nullptr;
        }
    }
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
            cudaSuccess || q != cudaDriverEntryPointSuccess || fn == nullptr) {
        delete st;
        return nullptr;
    }
    st->encode = reinterpret_cast<EncodeTiledFn>(fn);
    return st;
}

void tc_destroy(TcState* st) {
    if (st == nullptr) return;
    if (st->d_mods) cudaFree(st->d_mods);
    if (st->d_maps) cudaFree(st->d_maps);
    for (auto& kv : st->tiles)
        if (kv.second.mem) cudaFree(kv.second.mem);
    delete st;
}

int tc_register(TcState* st, int id, const ModDev& md, const moara_hparams& hp) {
    if (st == nullptr) return MOARA_OK;
    if (static_cast<int>(st->mods.size()) <= id) {
        st->mods.resize(id + 1, TcMod{});
        st->maps.resize(4 * (id + 1));
    }
    if (!tc_supported(md.m, md.n, md.r, hp.block_size, md.dtype, hp.decompose) || md.Pb == nullptr) return MOARA_OK;
    TcMod t{};
    t.m = md.m; t.n = md.n; t.r = md.r; t.kb = md.kb;
    t.W = md.W; t.exp_avg = md.exp_avg; t.exp_avg_sq = md.exp_avg_sq;
    t.mag_avg = md.mag_avg; t.mag_avg_sq = md.mag_avg_sq;
    t.Nb = reinterpret_cast<uint16_t*>(md.ws_N);
    t.dM = md.ws_dM;
    CUtensorMap* mp = &st->maps[4 * id];
    if (!encode_bf16_2d(st->encode, &mp[0], md.Pb, md.r, md.m, 64, 64) ||
        !encode_bf16_2d(st->encode, &mp[1], md.Pb, md.r, md.m, 64, 128) ||
        !encode_bf16_2d(st->encode, &mp[2], t.Nb, md.n, md.r, 64, 64) ||
        !encode_2d(st->encode, &mp[3], CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, md.W, md.n, md.m, K2_WCOLS, K2_BM)) {
        st->err = "cuTensorMapEncodeTiled failed";
        return MOARA_ERR_CUDA;
    }
    st->mods[id] = t;
    st->dirty = true;
    return MOARA_OK;
}

static int tc_upload(TcState* st) {
    if (!st->dirty) return MOARA_OK;
    const int n = static_cast<int>(st->mods.size());
    if (n > st->cap) {
        int ncap = std::max(64, st->cap);
        while (ncap < n) ncap *= 2;
        if (st->d_mods) cudaFree(st->d_mods);
        if (st->d_maps) cudaFree(st->d_maps);
        st->d_mods = nullptr;
        st->d_maps = nullptr;
        if (cudaMalloc(&st->d_mods, sizeof(TcMod) * ncap) != cudaSuccess ||
            cudaMalloc(&st->d_maps, sizeof(CUtensorMap) * 4 * ncap) != cudaSuccess) {
            st->err = "cudaMalloc of the tensor-core module table failed";
            return MOARA_ERR_CUDA;
        }
        st->cap = ncap;
    }
    if (cudaMemcpy(st->d_mods, st->mods.data(), sizeof(TcMod) * n, cudaMemcpyHostToDevice) != cudaSuccess ||
        cudaMemcpy(st->d_maps, st->maps.data(), sizeof(CUtensorMap) * 4 * n, cudaMemcpyHostToDevice) !=
            cudaSuccess) {
        st->err = "upload of the tensor-core module table failed";
        return MOARA_ERR_CUDA;
    }
    st->dirty = false;
    return MOARA_OK;
}

// Longest-processing-time assignment of weighted tiles to `grid` persistent
// CTAs: tiles in descending cost, each to the CTA with the least work so far;
// each CTA runs its tiles in that (descending) order.
static void lpt_assign(const std::vector<TcTile>& tiles, const std::vector<double>& cost, int grid,
                       std::vector<int>& start, std::vector<TcTile>& out) {
    std::vector<int> order(tiles.size());
    for (size_t i = 0; i < order.size(); ++i) order[i] = static_cast<int>(i);
    std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return cost[a] > cost[b]; });
    std::vector<std::vector<int>> per(grid);
    std::vector<std::pair<double, int>> heap;
    for (int c = 0; c < grid; ++c) heap.push_back({0.0, c});
    auto cmp = [](const std::pair<double, int>& a, const std::pair<double, int>& b) {
        return a.first > b.first || (a.first == b.first && a.second > b.second);
    };
    std::make_heap(heap.begin(), heap.end(), cmp);
    for (int i : order) {
        std::pop_heap(heap.begin(), heap.end(), cmp);
        auto& top = heap.back();
        per[top.second].push_back(i);
        top.first += cost[i];
        std::push_heap(heap.begin(), heap.end(), cmp);
    }
    start.assign(grid + 1, 0);
    out.clear();
    for (int c = 0; c < grid; ++c) {
        start[c] = static_cast<int>(out.size());
        for (int i : per[c]) out.push_back(tiles[i]);
    }
    start[grid] = static_cast<int>(out.size());
}

// Work lists of one launch: K1 tiles (256-rank x 128-column) and K2 tiles
// (128-row x 256-column), cost-weighted (MMA clocks vs. epilogue traffic).
static TcState::Tiles* tc_tiles(TcState* st, const std::vector<int>& ids) {
    auto it = st->tiles.find(ids);
    if (it != st->tiles.end()) return &it->second;
    std::vector<TcTile> k1, k2;
    std::vector<double> c1, c2;
    for (size_t slot = 0; slot < ids.size(); ++slot) {
        const TcMod& md = st->mods[ids[slot]];
        const int nt = (md.n + K1_BN - 1) / K1_BN, rt = (md.r + K1_BM - 1) / K1_BM;
        for (int j = 0; j < nt; ++j)
            for (int i = 0; i < rt; ++i) {
                const int rows = std::min(K1_BM, md.r - i * K1_BM);
                const int nh = rows > 128 ? 2 : 1;
                const double mma = 8.0 * nh * md.m;                       // clocks, with V_lo
                const double epi = 0.8 * rows * std::min(K1_BN, md.n - j * K1_BN);
                k1.push_back({ids[slot], static_cast<int>(slot), i, j});
                c1.push_back(std::max(mma, epi));
            }
        const int mt = (md.m + K2_BM - 1) / K2_BM, nt2 = (md.n + K2_BN - 1) / K2_BN;
        for (int i = 0; i < mt; ++i)
            for (int j = 0; j < nt2; ++j) {
                const double mma = 8.0 * md.r;
                const double epi = 0.36 * std::min(K2_BM, md.m - i * K2_BM) * std::min(K2_BN, md.n - j * K2_BN);
                k2.push_back({ids[slot], static_cast<int>(slot), i, j});
                c2.push_back(std::max(mma, epi));
            }
    }
    TcState::Tiles t;
    t.g1 = std::max(1, std::min(static_cast<int>(k1.size()), st->sms));
    t.g2 = std::max(1, std::min(static_cast<int>(k2.size()), st->sms));
    std::vector<int> s1, s2;
    std::vector<TcTile> o1, o2;
    lpt_assign(k1, c1, t.g1, s1, o1);
    lpt_assign(k2, c2, t.g2, s2, o2);
    auto pad = [](size_t b) { return (b + 255) / 256 * 256; };
    const size_t b_s1 = pad(sizeof(int) * s1.size()), b_o1 = pad(sizeof(TcTile) * std::max<size_t>(1, o1.size()));
    const size_t b_s2 = pad(sizeof(int) * s2.size()), b_o2 = pad(sizeof(TcTile) * std::max<size_t>(1, o2.size()));
    std::vector<char> host(b_s1 + b_o1 + b_s2 + b_o2, 0);
    std::memcpy(host.data(), s1.data(), sizeof(int) * s1.size());
    std::memcpy(host.data() + b_s1, o1.data(), sizeof(TcTile) * o1.size());
    std::memcpy(host.data() + b_s1 + b_o1, s2.data(), sizeof(int) * s2.size());
    std::memcpy(host.data() + b_s1 + b_o1 + b_s2, o2.data(), sizeof(TcTile) * o2.size());
    if (cudaMalloc(&t.mem, host.size()) != cudaSuccess) return nullptr;
    if (cudaMemcpy(t.mem, host.data(), host.size(), cudaMemcpyHostToDevice) != cudaSuccess) {
        cudaFree(t.mem);
        return nullptr;
    }
    char* base = static_cast<char*>(t.mem);
    t.k1_start = reinterpret_cast<const int*>(base);
    t.k1 = reinterpret_cast<const TcTile*>(base + b_s1);
    t.k2_start = reinterpret_cast<const int*>(base + b_s1 + b_o1);
    t.k2 = reinterpret_cast<const TcTile*>(base + b_s1 + b_o1 + b_s2);
    return &(st->tiles[ids] = t);
}

template <int BLK>
static cudaError_t launch_pair(TcState* st, const K1Params& p1, const K2Params& p2, int g1, int g2,
                               bool decomp, cudaStream_t s, int64_t* launches, const TcProfile& prof) {
    if (prof.on) prof.mark(prof.ctx, MOARA_PHASE_TC_PROJECT, s, true);
    if (decomp) k1_project<BLK, true><<<g1, K1_THREADS, K1_SMEM, s>>>(p1);
    else k1_project<BLK, false><<<g1, K1_THREADS, K1_SMEM, s>>>(p1);
    if (prof.on) prof.mark(prof.ctx, MOARA_PHASE_TC_PROJECT, s, false);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    ++*launches;
    if (prof.on) prof.mark(prof.ctx, MOARA_PHASE_TC_BACKPROJECT, s, true);
    k2_backproject<BLK><<<g2, K2_THREADS, K2_SMEM, s>>>(p2);
    if (prof.on) prof.mark(prof.ctx, MOARA_PHASE_TC_BACKPROJECT, s, false);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    ++*launches;
    return cudaSuccess;
}

int tc_step(TcState* st, const moara_hparams& hp, int n_mod, const int* ids, const void* const* G, float bc1,
            float bc2, float lr, int first_step, cudaStream_t s, int64_t* launches, const TcProfile& prof) {
    if (!st->attrs_set) {
        set_smem_attrs<8>(); set_smem_attrs<16>(); set_smem_attrs<32>(); set_smem_attrs<64>();
        set_smem_attrs<128>();
        st->attrs_set = true;
    }
    int rc = tc_upload(st);
    if (rc != MOARA_OK) return rc;
    const int B = hp.decompose ? hp.block_size : 128;
    for (int c0 = 0; c0 < n_mod; c0 += kTcGroup) {
        const int cnt = std::min(kTcGroup, n_mod - c0);
        std::vector<int> chunk(ids + c0, ids + c0 + cnt);
        TcState::Tiles* tl = tc_tiles(st, chunk);
        if (tl == nullptr) { st->err = "tile list allocation failed"; return MOARA_ERR_CUDA; }
        K1Params& p1 = st->p1;
        std::memset(&p1, 0, sizeof(p1));
        for (int q = 0; q < cnt; ++q) {
            const TcMod& md = st->mods[chunk[q]];
            if (!encode_bf16_2d(st->encode, &p1.gmap[q], G[c0 + q], md.n, md.m, 64, 64)) {
                st->err = "cuTensorMapEncodeTiled failed for a gradient";
                return MOARA_ERR_CUDA;
            }
        }
        p1.cta_start = tl->k1_start; p1.tiles = tl->k1;
        p1.mods = st->d_mods; p1.maps = st->d_maps; p1.status = st->d_status;
        p1.beta1 = hp.beta1; p1.beta2 = hp.beta2; p1.adam_eps = hp.adam_eps;
        p1.bc1 = bc1; p1.bc2 = bc2; p1.decomp_eps = hp.decomp_eps;
        p1.hilo = first_step ? 1 : 0;
        K2Params p2{};
        p2.cta_start = tl->k2_start; p2.tiles = tl->k2;
        p2.mods = st->d_mods; p2.maps = st->d_maps; p2.status = st->d_status;
        p2.step_scale = lr * hp.scale;
        p2.decompose = hp.decompose;
        const int g1 = tl->g1;
        const int g2 = tl->g2;
        const bool dec = hp.decompose != 0;
        cudaError_t e;
        switch (B) {
            case 8: e = launch_pair<8>(st, p1, p2, g1, g2, dec, s, launches, prof); break;
            case 16: e = launch_pair<16>(st, p1, p2, g1, g2, dec, s, launches, prof); break;
            case 32: e = launch_pair<32>(st, p1, p2, g1, g2, dec, s, launches, prof); break;
            case 64: e = launch_pair<64>(st, p1, p2, g1, g2, dec, s, launches, prof); break;
            default: e = launch_pair<128>(st, p1, p2, g1, g2, dec, s, launches, prof); break;
        }
        if (e != cudaSuccess) {
            st->err = cudaGetErrorString(e);
            return MOARA_ERR_CUDA;
        }
    }
    return MOARA_OK;
}

const char* tc_last_error(const TcState* st) { return st ? st->err.c_str() : "no tensor-core state"; }

}  // namespace moara
