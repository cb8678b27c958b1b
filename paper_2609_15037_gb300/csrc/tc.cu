// Tensor-core path of the optimizer step for bf16 gradients (sm_103a):
//
//  K0  Decompose(G, B) of §3.1 / Appendix B.1 as a memory-bound prepass: block
//      norms in fp32 and the direction matrix V written in bf16 (at the first
//      Adam step also the residual V - V_hi, so that the projection carries
//      ~16 bits there); a second, small pass runs Optimizer_M (Adam on the
//      block magnitudes).
//  K1  R = P^T V on tcgen05 (2-SM pairs: 256 ranks x 256 columns per CTA pair,
//      P exact in bf16), then Optimizer_V (Adam) on R in the epilogue; writes
//      the Adam update N as bf16.  (Algorithm 1.)
//  K2  dV = P N (2-SM pairs: 256 rows x 256 columns per CTA pair), then
//      W <- W - lr*alpha*(Rep_B(dM) (.) dV) in the epilogue, reading and
//      writing W once through TMA.  (Algorithm 1.)
//
// K1 and K2 are persistent and warp specialised: one warp issues TMA tile
// loads into a shared-memory ring, one thread of the even CTA of each pair
// issues tcgen05.mma (cta_group::2) into double-buffered TMEM accumulators,
// and epilogue warps drain TMEM while the next tile's MMAs run.  Every
// mbarrier wait is bounded; on expiry the kernel records
// MOARA_ERR_DEVICE_TIMEOUT in the context's status word, drains its own TMA
// copies and MMAs, frees TMEM and returns.
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
constexpr int kMaps = 9;                      // tensor maps per module

struct TcMod {
    int m, n, r, kb;
    int right;        // right projector Q (n x r): K1 computes R = V Q (m x r)
    int w3d;          // fp32 W with n % 64 == 0: K2 adds its update in 64 x 64 chunks (map 8)
    uint16_t* Qt;     // r x n bf16 transpose of a right projector (K2's B operand)
    uint16_t* Vhi;    // m x n bf16 direction matrix (written by K0)
    uint16_t* Vlo;    // m x n bf16 residual (first Adam step)
    float* W;
    float* exp_avg;
    float* exp_avg_sq;
    float* mag;       // m x kb block norms (K0 -> magnitude Adam)
    float* mag_avg;
    float* mag_avg_sq;
    uint16_t* Nb;     // r x n bf16 Adam update of the direction branch
    float* dM;        // m x kb Adam update of the magnitude branch
    uint16_t* Pb;     // m x r bf16 projector
};

struct TcTile {
    int mod, slot, t0, t1;
};

// ------------------------------------------------------------------- K0
struct K0Item {
    const uint16_t* G;
    uint16_t* Vhi;
    uint16_t* Vlo;
    float* mag;                        // m x kb block norms M (written when do_mag)
    float* mag_avg;
    float* mag_avg_sq;
    float* dM;
    int m, n, kb, segs;                // segs = ceil(n / 1024) row segments
};

struct K0Params {
    int count;
    int hilo;                          // also write V_lo = V - V_hi
    int do_mag;                        // run Optimizer_M (off when only V is wanted)
    float decomp_eps, beta1, beta2, adam_eps, bc1, bc2;
    const float* clip;                 // gradient clipping coefficient (device) for M, or null
    long long start[kTcGroup + 1];     // warp items (row, 1024-column segment) per module
    long long mstart[kTcGroup + 1];    // magnitude entries (m x kb) per module, prefix sums
    K0Item p[kTcGroup];
};

// ------------------------------------------------------------------- K1
constexpr int K1_BM = 128, K1_BN = 256, K1_BK = 64;
constexpr int K1_A_BYTES = K1_BM * K1_BK * 2;           // 16 KB: two 64-rank chunks of P^T (MN-major)
constexpr int K1_B_BYTES = K1_BK * (K1_BN / 2) * 2;     // 16 KB: this CTA's two 64-column chunks of V
// The Adam moments stream through a ring of slots, each one 32-column chunk
// of exp_avg and of exp_avg_sq (128 rank rows x 32 fp32, 16 KB each), loaded
// and stored by TMA.
constexpr int K1_MCOLS = 32;                            // fp32 moments: columns per chunk
constexpr int K1_MCHUNK = K1_BM * K1_MCOLS * 4;          // 16 KB (64 columns of bf16 moments)
// Chunk width in columns for fp32 (SB false) or bf16 (SB true) states: one
// 128-byte row of a 128-row chunk either way.
template <bool SB> struct StateCols { static constexpr int N = SB ? 64 : 32; };
template <bool HILO> struct K1Cfg {
    static constexpr int STAGES = HILO ? 3 : 5;
    static constexpr int STAGE_BYTES = K1_A_BYTES + (HILO ? 2 : 1) * K1_B_BYTES;
    static constexpr int MSLOTS = HILO ? 1 : 2;
    static constexpr int RING = STAGES * STAGE_BYTES;     // offset of the moment slots
    static constexpr int CTL = RING + MSLOTS * 2 * K1_MCHUNK;
};
constexpr int K1_WARPS = 12;                            // 0 TMA, 1 MMA, 2 moment loader, 3 moment storer, 4-11 epilogue
constexpr int K1_THREADS = K1_WARPS * 32;
constexpr int kCtlBytes = 512;                         // barrier block of K1 / K2
constexpr int K1_SMEM = 1024 + (K1Cfg<false>::CTL > K1Cfg<true>::CTL ? K1Cfg<false>::CTL : K1Cfg<true>::CTL) + kCtlBytes;

struct K1Params {
    CUtensorMap gmap[kTcGroup];        // G of each launch slot (decomposition off): {n, m}, box {64, 64}
    const int* cta_start;              // tiles of CTA c: tiles[cta_start[c] .. cta_start[c+1])
    const TcTile* tiles;
    const TcMod* mods;
    const CUtensorMap* maps;           // per module: P (K1), P (K2), N, W, V_hi, V_lo, exp_avg, exp_avg_sq
    int* status;
    float beta1, beta2, adam_eps, bc1, bc2;
    float inv_bc1, inv_bc2;            // 1 / bias corrections
    int decompose;
    const float* clip;                 // decomposition off: clipping coefficient (device) for R, or null
};

// ------------------------------------------------------------------- K2
constexpr int K2_BM = 128, K2_BN = 256, K2_BK = 64;
constexpr int K2_A_BYTES = K2_BM * K2_BK * 2;           // 16 KB: P rows, K-major
constexpr int K2_B_BYTES = K2_BK * (K2_BN / 2) * 2;     // 16 KB: this CTA's two 64-column chunks of N
constexpr int K2_STAGE_BYTES = K2_A_BYTES + K2_B_BYTES;
// W moves in 16 KB chunks: 128 rows x one 128-byte row (32 fp32 / 64 bf16
// columns), or for an fp32 W whose n is a multiple of 64, 64 rows x 64
// columns through a 3-D view of W (256 contiguous bytes per row).
// fp32 W (SB false): the epilogue writes the update dW = -lr*alpha*(Rep_B(dM)
// (.) dV) into a staging chunk and a TMA reduce-add applies it to W in L2, so
// W never enters the SM: two staging chunks, six operand stages.  bf16 W (SB
// true; the fp32 update is rounded once, which an L2 add of a bf16 dW would
// not reproduce): a four-chunk ring, TMA in and out, five operand stages.
constexpr int K2_WCOLS = 32;
constexpr int K2_WBYTES = K2_BM * K2_WCOLS * 4;         // 16 KB
template <bool SB> struct K2Cfg {
    static constexpr int STAGES = SB ? 5 : 6;
    static constexpr int WBUF = SB ? 4 : 2;
    static constexpr int BYTES = STAGES * K2_STAGE_BYTES + WBUF * K2_WBYTES;
};
constexpr int K2_WARPS = 12;                            // 0 TMA, 1 MMA, 2 W loader, 3 W storer, 4-11 epilogue
constexpr int K2_THREADS = K2_WARPS * 32;
constexpr int K2_SMEM = 1024 + (K2Cfg<true>::BYTES > K2Cfg<false>::BYTES ? K2Cfg<true>::BYTES : K2Cfg<false>::BYTES) +
                        kCtlBytes;

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
    uint64_t full[8];
    uint64_t empty[8];   // sized for up to eight stages
    uint64_t accf[2];
    uint64_t acce[2];
    uint64_t drain;
    uint64_t wfull[8];
    uint64_t wdone[8];
    uint64_t wempty[8];
    uint32_t tmem_base;
    int abort;
};
static_assert(sizeof(SmemCtl) <= kCtlBytes, "the barrier block fits the space K1 and K2 reserve for it");
// K1 and K2 leave room beside them for one K0 CTA (no shared memory of its
// own, 1 KB reserved by the hardware per CTA) out of the SM's 228 KB.
static_assert(K1_SMEM + 1024 + 1024 <= 228 * 1024 && K2_SMEM + 1024 + 1024 <= 228 * 1024,
              "a decomposition CTA fits beside a K1 or K2 CTA");

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
// K0: Decompose(G, B) (§3.1 / App. B.1) and Optimizer_M.  One warp per (row,
// 1024-column segment), taken as four 256-column sub-segments whose loads are
// all issued first; in a sub-segment lane l holds columns 8l..8l+7, so a block
// of B columns spans B/8 lanes, reduced with xor shuffles.  Columns past n (the
// right zero padding of the last block) contribute nothing; V is written for
// c < n only.
// ===========================================================================
constexpr int K0_SEG = 1024;

template <int BLK>
__global__ void __launch_bounds__(256, 3) k0_decompose(const __grid_constant__ K0Params p) {
    constexpr int LPB = BLK / 8;                       // lanes per block (1..16)
    const int lane = threadIdx.x & 31;
    const long long total = p.start[p.count];
    const long long nwarps = ((long long)gridDim.x * blockDim.x) >> 5;
    long long item = (blockIdx.x * (long long)blockDim.x + threadIdx.x) >> 5;
    int mod = 0;                                       // module of `item` (items only increase)
    // G of the next item is loaded before the current one is processed, so
    // each warp keeps a 1024-column row segment in flight
    auto locate = [&](long long x, int& row, int& seg) {
        while (mod + 1 < p.count && p.start[mod + 1] <= x) ++mod;
        const int local = static_cast<int>(x - p.start[mod]);
        row = local / p.p[mod].segs;
        seg = local - row * p.p[mod].segs;
    };
    auto load = [&](int md, int row, int seg, uint4 (&g)[4]) {
        const K0Item& it = p.p[md];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int c0 = seg * K0_SEG + u * 256 + lane * 8;
            g[u] = make_uint4(0u, 0u, 0u, 0u);
            if (c0 < it.n) g[u] = __ldcs(reinterpret_cast<const uint4*>(it.G + (long long)row * it.n + c0));
        }
    };
    if (item >= total) return;
    int row, seg;
    locate(item, row, seg);
    uint4 g[4];
    load(mod, row, seg, g);
    while (true) {
        const int cmod = mod, crow = row, cseg = seg;
        uint4 cg[4] = {g[0], g[1], g[2], g[3]};
        item += nwarps;
        const bool more = item < total;
        if (more) {
            locate(item, row, seg);
            load(mod, row, seg, g);
        }
        const K0Item& it = p.p[cmod];
        const int n = it.n;
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int cs = cseg * K0_SEG + u * 256;     // first column of the sub-segment
            if (cs >= n) break;                         // warp-uniform
            const int c0 = cs + lane * 8;
            const uint32_t w[4] = {cg[u].x, cg[u].y, cg[u].z, cg[u].w};
            float ss = 0.0f;
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const float a = bf_lo(w[e]), b = bf_hi(w[e]);
                ss = fmaf(a, a, ss);
                ss = fmaf(b, b, ss);
            }
#pragma unroll
            for (int o = 1; o < LPB; o <<= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
            const float mag = sqrtf(ss);
            const float sc = 1.0f / (mag + p.decomp_eps);
            if (p.do_mag && (lane & (LPB - 1)) == 0 && c0 < n)   // first lane of a block that starts before n
                it.mag[(long long)crow * it.kb + c0 / BLK] = mag;
            if (c0 < n) {
                const long long off = (long long)crow * n + c0;
                uint32_t vh[4], vl[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float v0 = bf_lo(w[e]) * sc, v1 = bf_hi(w[e]) * sc;
                    vh[e] = pack_bf16x2(v0, v1);
                    vl[e] = pack_bf16x2(v0 - bf_lo(vh[e]), v1 - bf_hi(vh[e]));
                }
                *reinterpret_cast<uint4*>(it.Vhi + off) = make_uint4(vh[0], vh[1], vh[2], vh[3]);
                if (p.hilo) *reinterpret_cast<uint4*>(it.Vlo + off) = make_uint4(vl[0], vl[1], vl[2], vl[3]);
            }
        }
        if (!more) break;
    }
}

// Optimizer_M (Algorithm 1) on the block norms K0 wrote: Adam on M, dM out.
// A separate pass over the m x kb entries keeps these dependent loads out of
// K0's streaming loop.
__global__ void __launch_bounds__(256) k0_mag_adam(const __grid_constant__ K0Params p) {
    const long long total = p.mstart[p.count];
    // a clipped gradient c G has block norms c M and the same direction V
    const float cf = p.clip != nullptr ? *p.clip : 1.0f;
    int mod = 0;
    for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
         e += (long long)gridDim.x * blockDim.x) {
        while (mod + 1 < p.count && p.mstart[mod + 1] <= e) ++mod;
        const K0Item& it = p.p[mod];
        const long long o = e - p.mstart[mod];
        const float mag = it.mag[o] * cf;
        const float ma = p.beta1 * it.mag_avg[o] + (1.0f - p.beta1) * mag;
        const float mas = p.beta2 * it.mag_avg_sq[o] + (1.0f - p.beta2) * mag * mag;
        it.mag_avg[o] = ma;
        it.mag_avg_sq[o] = mas;
        it.dM[o] = (ma / p.bc1) / (sqrtf(mas / p.bc2) + p.adam_eps);
    }
}

// Sum of the squared block norms K0 wrote (= ||G||_F^2 of the group, up to
// their rounding) for global-norm clipping: chunks of kNormChunk entries,
// chunk c on CTA c mod gridDim, fp32 per chunk and fp64 across chunks in a
// fixed order, one partial sum per CTA.
__global__ void __launch_bounds__(256) k0_mag_sq(const __grid_constant__ K0Params p, double* partials) {
    __shared__ double red[8];
    const long long total = p.mstart[p.count];
    const long long nchunks = (total + kNormChunk - 1) / kNormChunk;
    double acc = 0.0;
    int mod = 0;
    for (long long c = blockIdx.x; c < nchunks; c += gridDim.x) {
        const long long e0 = c * kNormChunk, e1 = min(e0 + (long long)kNormChunk, total);
        float ss = 0.0f;
        for (long long e = e0 + threadIdx.x; e < e1; e += blockDim.x) {
            while (mod + 1 < p.count && p.mstart[mod + 1] <= e) ++mod;
            while (mod > 0 && p.mstart[mod] > e) --mod;
            const float x = p.p[mod].mag[e - p.mstart[mod]];
            ss = fmaf(x, x, ss);
        }
        acc += static_cast<double>(ss);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        double t = 0.0;
        for (int w = 0; w < 8; ++w) t += red[w];
        partials[blockIdx.x] = t;
    }
}

// ===========================================================================
// K1: projection R = P^T V (tile 128 ranks x 256 columns x 64 rows, MN-major
// operands), Optimizer_V (Adam) in the epilogue, N written in bf16.  HILO
// adds the MMA with V_lo (first Adam step).
// ===========================================================================
// RT: the launch may hold modules with a right projector (per-tile operand
// roles); without it those branches are compiled out.
template <bool HILO, bool SB, bool RT>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(K1_THREADS, 1)
k1_project(const __grid_constant__ K1Params p) {
    constexpr int MC = StateCols<SB>::N;              // moment columns per chunk
    constexpr int HC = MC / 2;                        // columns per epilogue thread and chunk
    constexpr int STAGES = K1Cfg<HILO>::STAGES;
    constexpr int STAGE_BYTES = K1Cfg<HILO>::STAGE_BYTES;
    constexpr int MSLOTS = K1Cfg<HILO>::MSLOTS;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = align1024(smem_raw);
    uint8_t* mring = smem + K1Cfg<HILO>::RING;
    SmemCtl* ctl = reinterpret_cast<SmemCtl*>(smem + K1Cfg<HILO>::CTL);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int crank = static_cast<int>(ptx::cluster_ctarank());   // rank tile 2 t0 + crank of each pair tile
    const int cluster = blockIdx.x >> 1;
    volatile int* abort_flag = &ctl->abort;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            ptx::mbar_init(ptx::smem_u32(&ctl->full[s]), 1);
            ptx::mbar_init(ptx::smem_u32(&ctl->empty[s]), 1);    // the pair MMA consumed the stage
        }
        for (int b = 0; b < 2; ++b) {
            ptx::mbar_init(ptx::smem_u32(&ctl->accf[b]), 1);
            ptx::mbar_init(ptx::smem_u32(&ctl->acce[b]), 16);    // both CTAs' epilogue warps
        }
        for (int b = 0; b < MSLOTS; ++b) {
            ptx::mbar_init(ptx::smem_u32(&ctl->wfull[b]), 1);
            ptx::mbar_init(ptx::smem_u32(&ctl->wdone[b]), 8);
            ptx::mbar_init(ptx::smem_u32(&ctl->wempty[b]), 1);
        }
        ptx::mbar_init(ptx::smem_u32(&ctl->drain), 1);
        ctl->abort = 0;
        ptx::fence_barrier_init();
    }
    if (warp == 1) {                // collective: one warp of each CTA of the pair
        ptx::tmem_alloc2(ptx::smem_u32(&ctl->tmem_base), 512);
        ptx::tmem_relinquish2();
    }
    ptx::tc_fence_before();
    __syncwarp();
    ptx::cluster_sync();            // barriers of both CTAs initialised before any remote signal
    ptx::tc_fence_after();
    const uint32_t tmem = ctl->tmem_base;
    const int t_begin = p.cta_start[cluster], t_end = p.cta_start[cluster + 1];

    if (warp == 0) {
        // ------------------------------------------------------ TMA producer
        // P^T rows of this CTA's rank tile and this CTA's half (128 columns)
        // of the V tile: the pair MMA reads A rows and B columns from both.
        // Both CTAs' copies complete on the even CTA's full barrier, which
        // the even CTA arms with the bytes of both.
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            uint32_t issued = 0, last_par = 0;
            bool ok = true;
            for (int t = t_begin; t < t_end && ok; ++t) {
                const TcTile tl = p.tiles[t];
                const TcMod& md = p.mods[tl.mod];
                const CUtensorMap* pmap = &p.maps[tl.mod * kMaps + 0];
                const CUtensorMap* vmap = p.decompose ? &p.maps[tl.mod * kMaps + 4] : &p.gmap[tl.slot];
                const CUtensorMap* lmap = &p.maps[tl.mod * kMaps + 5];
                const int r0 = (2 * tl.t0 + crank) * K1_BM, n0 = tl.t1 * K1_BN;
                const bool right = RT && md.right != 0;
                const int nk = ((right ? md.n : md.m) + K1_BK - 1) / K1_BK;
                for (int kb = 0; kb < nk; ++kb) {
                    if (!ptx::mbar_wait(ptx::smem_u32(&ctl->empty[stage]), phase ^ 1, abort_flag, p.status,
                                        MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit)) { ok = false; break; }
                    const uint32_t own = ptx::smem_u32(&ctl->full[stage]);
                    const uint32_t fb = ptx::mapa(own, 0);
                    if (crank == 0) ptx::mbar_arrive_expect_tx(own, 2 * STAGE_BYTES);
                    const uint32_t a = ptx::smem_u32(smem + stage * STAGE_BYTES);
                    const uint32_t b = a + K1_A_BYTES;
                    if (!right) {
#pragma unroll
                        for (int c = 0; c < 2; ++c) ptx::tma_load_2d_pair(a + c * 8192, pmap, fb, r0 + 64 * c, kb * K1_BK);
#pragma unroll
                        for (int h = 0; h < 2; ++h) {
                            const int c = 2 * crank + h;
                            ptx::tma_load_2d_pair(b + h * 8192, vmap, fb, n0 + 64 * c, kb * K1_BK);
                            if (HILO) ptx::tma_load_2d_pair(b + K1_B_BYTES + h * 8192, lmap, fb, n0 + 64 * c, kb * K1_BK);
                        }
                    } else {
                        // A: this CTA's 128 rows of V (64 columns, K-major; V_lo
                        // in the third slot at the first step); B: this CTA's
                        // 128 ranks of Q, two 64-rank chunks (MN-major)
                        ptx::tma_load_2d_pair(a, vmap, fb, kb * K1_BK, r0);
                        if (HILO) ptx::tma_load_2d_pair(b + K1_B_BYTES, lmap, fb, kb * K1_BK, r0);
#pragma unroll
                        for (int h = 0; h < 2; ++h)
                            ptx::tma_load_2d_pair(b + h * 8192, pmap, fb, n0 + 64 * (2 * crank + h), kb * K1_BK);
                    }
                    issued |= 1u << stage;
                    last_par = (last_par & ~(1u << stage)) | (phase << stage);
                    if (++stage == STAGES) { stage = 0; phase ^= 1; }
                }
            }
            if (!ok && crank == 0) {   // let the copies already in flight land before the CTA exits
                for (int s = 0; s < STAGES; ++s)
                    if (issued & (1u << s)) wait_drain(ptx::smem_u32(&ctl->full[s]), (last_par >> s) & 1);
            }
        }
    } else if (warp == 1) {
        if (crank == 0) {
            // -------------------------------------------- MMA issuer (even CTA)
            // M = 256 (both CTAs' rank tiles), N = 256, K = 16 per MMA; the
            // full barrier of a stage counts both CTAs' copies
            if (lane == 0) {
                constexpr uint32_t idesc_l = ptx::idesc_bf16(256, K1_BN, 1, 1);   // A MN-major (P^T)
                constexpr uint32_t idesc_r = ptx::idesc_bf16(256, K1_BN, 0, 1);   // A K-major (V rows)
                int stage = 0;
                uint32_t phase = 0;
                int buf = 0;
                uint32_t acc_phase = 0;
                bool ok = true;
                for (int t = t_begin; t < t_end && ok; ++t) {
                    const TcTile tl = p.tiles[t];
                    const TcMod& md = p.mods[tl.mod];
                    const bool right = RT && md.right != 0;
                    const uint32_t idesc = right ? idesc_r : idesc_l;
                    const int nk = ((right ? md.n : md.m) + K1_BK - 1) / K1_BK;
                    if (!ptx::mbar_wait_cluster(ptx::smem_u32(&ctl->acce[buf]), acc_phase ^ 1, abort_flag, p.status,
                                                MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit)) { ok = false; break; }
                    ptx::tc_fence_after();
                    const uint32_t d0 = tmem + buf * 256;
                    for (int kb = 0; kb < nk; ++kb) {
                        if (!ptx::mbar_wait_cluster(ptx::smem_u32(&ctl->full[stage]), phase, abort_flag, p.status,
                                                    MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit)) { ok = false; break; }
                        ptx::tc_fence_after();
                        const uint32_t a = ptx::smem_u32(smem + stage * STAGE_BYTES);
                        const uint32_t b = a + K1_A_BYTES;
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk) {
                            const uint64_t bdesc = ptx::smem_desc_sw128(b + kk * 2048, 8192, 1024);
                            if (!right) {
                                const uint64_t adesc = ptx::smem_desc_sw128(a + kk * 2048, 8192, 1024);
                                ptx::mma2_f16(d0, adesc, bdesc, idesc, (kb | kk) != 0);
                                if (HILO) {   // P^T V_lo: the bf16 rounding residual of V
                                    const uint64_t ldesc = ptx::smem_desc_sw128(b + K1_B_BYTES + kk * 2048, 8192, 1024);
                                    ptx::mma2_f16(d0, adesc, ldesc, idesc, 1);
                                }
                            } else {
                                const uint64_t adesc = ptx::smem_desc_sw128(a + kk * 32, 16, 1024);
                                ptx::mma2_f16(d0, adesc, bdesc, idesc, (kb | kk) != 0);
                                if (HILO) {   // V_lo Q
                                    const uint64_t ldesc = ptx::smem_desc_sw128(b + K1_B_BYTES + kk * 32, 16, 1024);
                                    ptx::mma2_f16(d0, ldesc, bdesc, idesc, 1);
                                }
                            }
                        }
                        ptx::mma2_commit_mc(ptx::smem_u32(&ctl->empty[stage]), 0x3);
                        if (++stage == STAGES) { stage = 0; phase ^= 1; }
                    }
                    if (!ok) break;
                    ptx::mma2_commit_mc(ptx::smem_u32(&ctl->accf[buf]), 0x3);
                    if (++buf == 2) { buf = 0; acc_phase ^= 1; }
                }
                // wait for every MMA this thread issued before TMEM is released
                ptx::mma2_commit_mc(ptx::smem_u32(&ctl->drain), 0x1);
                wait_drain(ptx::smem_u32(&ctl->drain), 0);
            }
        }
    } else if (warp == 2) {
        // ------------------------------------- moment chunk loader (TMA in)
        if (lane == 0) {
            uint32_t g = 0;
            uint32_t issued = 0, last_par = 0;
            bool ok = true;
            for (int t = t_begin; t < t_end && ok; ++t) {
                const TcTile tl = p.tiles[t];
                const TcMod& md = p.mods[tl.mod];
                const CUtensorMap* amap = &p.maps[tl.mod * kMaps + 6];
                const CUtensorMap* smap = &p.maps[tl.mod * kMaps + 7];
                const int r0 = (2 * tl.t0 + crank) * K1_BM, n0 = tl.t1 * K1_BN;
                const int cols = (RT && md.right) ? md.r : md.n;    // R is r x n, or m x r (right projector)
                const int nc = min(K1_BN / MC, (cols - n0 + MC - 1) / MC);
                for (int c = 0; c < nc; ++c, ++g) {
                    const int b = g % MSLOTS;
                    const uint32_t ph = (g / MSLOTS) & 1;
                    if (!ptx::mbar_wait(ptx::smem_u32(&ctl->wempty[b]), ph ^ 1, abort_flag, p.status,
                                        MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit)) { ok = false; break; }
                    const uint32_t fb = ptx::smem_u32(&ctl->wfull[b]);
                    ptx::mbar_arrive_expect_tx(fb, 2 * K1_MCHUNK);
                    const uint32_t dst = ptx::smem_u32(mring + b * 2 * K1_MCHUNK);
                    ptx::tma_load_2d(dst, amap, fb, n0 + c * MC, r0);
                    ptx::tma_load_2d(dst + K1_MCHUNK, smap, fb, n0 + c * MC, r0);
                    issued |= 1u << b;
                    last_par = (last_par & ~(1u << b)) | (ph << b);
                }
            }
            if (!ok) {
                for (int b = 0; b < MSLOTS; ++b)
                    if (issued & (1u << b)) wait_drain(ptx::smem_u32(&ctl->wfull[b]), (last_par >> b) & 1);
            }
        }
    } else if (warp == 3) {
        // ------------------------------------ moment chunk storer (TMA out)
        if (lane == 0) {
            uint32_t g = 0;
            bool ok = true;
            for (int t = t_begin; t < t_end && ok; ++t) {
                const TcTile tl = p.tiles[t];
                const TcMod& md = p.mods[tl.mod];
                const CUtensorMap* amap = &p.maps[tl.mod * kMaps + 6];
                const CUtensorMap* smap = &p.maps[tl.mod * kMaps + 7];
                const int r0 = (2 * tl.t0 + crank) * K1_BM, n0 = tl.t1 * K1_BN;
                const int cols = (RT && md.right) ? md.r : md.n;    // R is r x n, or m x r (right projector)
                const int nc = min(K1_BN / MC, (cols - n0 + MC - 1) / MC);
                for (int c = 0; c < nc; ++c, ++g) {
                    const int b = g % MSLOTS;
                    const uint32_t ph = (g / MSLOTS) & 1;
                    if (!ptx::mbar_wait(ptx::smem_u32(&ctl->wdone[b]), ph, abort_flag, p.status,
                                        MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit)) { ok = false; break; }
                    const uint32_t src = ptx::smem_u32(mring + b * 2 * K1_MCHUNK);
                    ptx::tma_store_2d(amap, src, n0 + c * MC, r0);
                    ptx::tma_store_2d(smap, src + K1_MCHUNK, n0 + c * MC, r0);
                    ptx::bulk_commit_group();
                    ptx::bulk_wait_read_all();            // the slot may be refilled once read
                    ptx::mbar_arrive(ptx::smem_u32(&ctl->wempty[b]));
                }
            }
            ptx::bulk_wait_all();
        }
    } else {
        // ------------------------------------------------- epilogue warps
        // 8 warps: TMEM lane quarter q = warp % 4 (rank row), column half ch
        // of each 32-column chunk.  Optimizer_V (Adam) on R: each thread
        // updates 16 entries of both moments of its rank row in the swizzled
        // ring slot and writes the update N in bf16 to global memory.
        const int ew = warp - 4;                       // 0..7
        const int q = warp & 3;
        const int ch = ew >> 2;
        const int il = q * 32 + lane;                  // rank row within the tile
        // R of a clipped gradient (decomposition off; with it V is unchanged)
        const float cf = p.clip != nullptr ? *p.clip : 1.0f;
        int buf = 0;
        uint32_t acc_phase = 0;
        uint32_t g = 0;
        bool ok = true;
        for (int t = t_begin; t < t_end && ok; ++t) {
            const TcTile tl = p.tiles[t];
            const TcMod& md = p.mods[tl.mod];
            // R (and the moments, N) is r x n, or m x r with a right projector
            const int rr = (RT && md.right) ? md.m : md.r, nn = (RT && md.right) ? md.r : md.n;
            uint16_t* const nb_p = md.Nb;
            const int r0 = (2 * tl.t0 + crank) * K1_BM, n0 = tl.t1 * K1_BN;
            const int a = r0 + il;
            const bool row_ok = a < rr;
            const int nc = min(K1_BN / MC, (nn - n0 + MC - 1) / MC);
            const bool got = ptx::mbar_wait(ptx::smem_u32(&ctl->accf[buf]), acc_phase, abort_flag, p.status,
                                            MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit);
            if (!__all_sync(0xffffffffu, got)) { ok = false; break; }
            ptx::tc_fence_after();
            for (int c = 0; c < nc; ++c, ++g) {
                const int b = g % MSLOTS;
                const uint32_t ph = (g / MSLOTS) & 1;
                const int j0 = n0 + c * MC + ch * HC;
                // the thread's HC columns in passes of 16: four 16-byte units
                // of its row per chunk, 4 fp32 or 8 bf16 moments each
                constexpr int PU = HC / 4;                  // moments per unit
                constexpr int UPH = 16 / PU;                // units per pass
                const uint32_t tcol = tmem + (static_cast<uint32_t>(q * 32) << 16) + buf * 256 + c * MC + ch * HC;
                float v[16];
                __syncwarp();
                ptx::tmem_ld16(tcol, v);
                const bool gotm = ptx::mbar_wait(ptx::smem_u32(&ctl->wfull[b]), ph, abort_flag, p.status,
                                                 MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit);
                if (!__all_sync(0xffffffffu, gotm)) { ok = false; break; }
                uint8_t* arow = mring + b * 2 * K1_MCHUNK + il * 128;
                uint8_t* srow = arow + K1_MCHUNK;
                const uint32_t x = static_cast<uint32_t>(il & 7);
#pragma unroll
                for (int h = 0; h < HC / 16; ++h) {
                    if (h > 0) ptx::tmem_ld16(tcol + 16 * h, v);
                    float nv[16];
#pragma unroll
                    for (int uu = 0; uu < UPH; ++uu) {
                        const int u = h * UPH + uu;
                        const uint32_t off = ((ch * 4 + u) ^ x) << 4;
                        uint4* a4 = reinterpret_cast<uint4*>(arow + off);
                        uint4* s4 = reinterpret_cast<uint4*>(srow + off);
                        const uint4 av = *a4, sv = *s4;
                        const uint32_t aw[4] = {av.x, av.y, av.z, av.w}, sw[4] = {sv.x, sv.y, sv.z, sv.w};
                        float ea[PU], es[PU];
                        if constexpr (SB) {
#pragma unroll
                            for (int k = 0; k < 4; ++k) {
                                ea[2 * k] = bf_lo(aw[k]); ea[2 * k + 1] = bf_hi(aw[k]);
                                es[2 * k] = bf_lo(sw[k]); es[2 * k + 1] = bf_hi(sw[k]);
                            }
                        } else {
#pragma unroll
                            for (int k = 0; k < PU; ++k) { ea[k] = __uint_as_float(aw[k]); es[k] = __uint_as_float(sw[k]); }
                        }
#pragma unroll
                        for (int e = 0; e < PU; ++e) {
                            const float rv = v[PU * uu + e] * cf;
                            ea[e] = p.beta1 * ea[e] + (1.0f - p.beta1) * rv;
                            es[e] = p.beta2 * es[e] + (1.0f - p.beta2) * rv * rv;
                            // N goes to K2 in bf16: approximate sqrt / reciprocal
                            // (relative error ~2^-22) are far below its rounding
                            nv[PU * uu + e] = ea[e] * p.inv_bc1 *
                                              ptx::rcp_approx(ptx::sqrt_approx(es[e] * p.inv_bc2) + p.adam_eps);
                        }
                        if constexpr (SB) {   // the moments are stored rounded to bf16
                            *a4 = make_uint4(pack_bf16x2(ea[0], ea[1]), pack_bf16x2(ea[2], ea[3]),
                                             pack_bf16x2(ea[4], ea[5]), pack_bf16x2(ea[6], ea[7]));
                            *s4 = make_uint4(pack_bf16x2(es[0], es[1]), pack_bf16x2(es[2], es[3]),
                                             pack_bf16x2(es[4], es[5]), pack_bf16x2(es[6], es[7]));
                        } else {
                            *a4 = make_uint4(__float_as_uint(ea[0]), __float_as_uint(ea[1]),
                                             __float_as_uint(ea[2]), __float_as_uint(ea[3]));
                            *s4 = make_uint4(__float_as_uint(es[0]), __float_as_uint(es[1]),
                                             __float_as_uint(es[2]), __float_as_uint(es[3]));
                        }
                    }
                    const int jh = j0 + 16 * h;
                    if (row_ok && jh < nn) {
                        const long long o = (long long)a * nn + jh;
                        if (jh + 16 <= nn) {
                            uint4* n4 = reinterpret_cast<uint4*>(nb_p + o);
                            n4[0] = make_uint4(pack_bf16x2(nv[0], nv[1]), pack_bf16x2(nv[2], nv[3]),
                                               pack_bf16x2(nv[4], nv[5]), pack_bf16x2(nv[6], nv[7]));
                            n4[1] = make_uint4(pack_bf16x2(nv[8], nv[9]), pack_bf16x2(nv[10], nv[11]),
                                               pack_bf16x2(nv[12], nv[13]), pack_bf16x2(nv[14], nv[15]));
                        } else {
#pragma unroll
                            for (int e = 0; e < 16; ++e) {
                                if (jh + e >= nn) continue;
                                __nv_bfloat16 hb = __float2bfloat16_rn(nv[e]);
                                nb_p[o + e] = *reinterpret_cast<uint16_t*>(&hb);
                            }
                        }
                    }
                }
                ptx::fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive(ptx::smem_u32(&ctl->wdone[b]));
            }
            if (!ok) break;
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) {   // the even CTA's issuer waits for both CTAs' epilogues
                if (crank == 0) ptx::mbar_arrive(ptx::smem_u32(&ctl->acce[buf]));
                else ptx::mbar_arrive_remote(ptx::mapa(ptx::smem_u32(&ctl->acce[buf]), 0));
            }
            if (++buf == 2) { buf = 0; acc_phase ^= 1; }
        }
    }

    ptx::tc_fence_before();
    __syncwarp();
    ptx::cluster_sync();            // no CTA leaves while its peer may still signal or fill it
    if (warp == 1) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc2(tmem, 512);
    }
}

// ===========================================================================
// K2: back-projection dV = P N and the weight update in the epilogue.
// ===========================================================================
template <int BLK, bool SB>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(K2_THREADS, 1)
k2_backproject(const __grid_constant__ K2Params p) {
    constexpr int WC = StateCols<SB>::N;              // W columns per ring chunk
    constexpr int HC = WC / 2;                        // columns per epilogue thread and chunk
    // fp32 W, blocks of >= 32 columns: 64 x 64 update chunks through the 3-D
    // map where the module allows it (TcMod::w3d)
    constexpr bool W3D = !SB && BLK >= 32 && K2_BN % BLK == 0;
    static_assert(!SB || BLK >= 32, "bf16 states: a thread's 32 columns lie in one block");
    constexpr int K2_STAGES = K2Cfg<SB>::STAGES, K2_WBUF = K2Cfg<SB>::WBUF;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = align1024(smem_raw);
    uint8_t* wring = smem + K2_STAGES * K2_STAGE_BYTES;
    SmemCtl* ctl = reinterpret_cast<SmemCtl*>(wring + K2_WBUF * K2_WBYTES);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int crank = static_cast<int>(ptx::cluster_ctarank());   // row tile 2 t0 + crank of each pair tile
    const int cluster = blockIdx.x >> 1;
    volatile int* abort_flag = &ctl->abort;

    if (threadIdx.x == 0) {
        for (int s = 0; s < K2_STAGES; ++s) {
            ptx::mbar_init(ptx::smem_u32(&ctl->full[s]), 1);
            ptx::mbar_init(ptx::smem_u32(&ctl->empty[s]), 1);    // the pair MMA consumed the stage
        }
        for (int b = 0; b < 2; ++b) {
            ptx::mbar_init(ptx::smem_u32(&ctl->accf[b]), 1);
            ptx::mbar_init(ptx::smem_u32(&ctl->acce[b]), 16);    // both CTAs' epilogue warps
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
    if (warp == 1) {                // collective: one warp of each CTA of the pair
        ptx::tmem_alloc2(ptx::smem_u32(&ctl->tmem_base), 512);
        ptx::tmem_relinquish2();
    }
    ptx::tc_fence_before();
    __syncwarp();
    ptx::cluster_sync();            // barriers of both CTAs initialised before any remote signal
    ptx::tc_fence_after();
    const uint32_t tmem = ctl->tmem_base;
    const int t_begin = p.cta_start[cluster], t_end = p.cta_start[cluster + 1];

    if (warp == 0) {
        // ------------------------------------------------ operand TMA producer
        // P rows of this CTA's row tile and this CTA's half (128 columns) of
        // the N tile; both CTAs' copies complete on the even CTA's barrier.
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            uint32_t issued = 0, last_par = 0;
            bool ok = true;
            for (int t = t_begin; t < t_end && ok; ++t) {
                const TcTile tl = p.tiles[t];
                const TcMod& md = p.mods[tl.mod];
                const CUtensorMap* amap = &p.maps[tl.mod * kMaps + 1];
                const CUtensorMap* bmap = &p.maps[tl.mod * kMaps + 2];
                const int i0 = (2 * tl.t0 + crank) * K2_BM, n0 = tl.t1 * K2_BN;
                const int nk = (md.r + K2_BK - 1) / K2_BK;
                for (int kb = 0; kb < nk; ++kb) {
                    if (!ptx::mbar_wait(ptx::smem_u32(&ctl->empty[stage]), phase ^ 1, abort_flag, p.status,
                                        MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit)) { ok = false; break; }
                    const uint32_t own = ptx::smem_u32(&ctl->full[stage]);
                    const uint32_t fb = ptx::mapa(own, 0);
                    if (crank == 0) ptx::mbar_arrive_expect_tx(own, 2 * K2_STAGE_BYTES);
                    const uint32_t a = ptx::smem_u32(smem + stage * K2_STAGE_BYTES);
                    const uint32_t b = a + K2_A_BYTES;
                    ptx::tma_load_2d_pair(a, amap, fb, kb * K2_BK, i0);
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        const int c = 2 * crank + h;
                        ptx::tma_load_2d_pair(b + h * 8192, bmap, fb, n0 + 64 * c, kb * K2_BK);
                    }
                    issued |= 1u << stage;
                    last_par = (last_par & ~(1u << stage)) | (phase << stage);
                    if (++stage == K2_STAGES) { stage = 0; phase ^= 1; }
                }
            }
            if (!ok && crank == 0) {
                for (int s = 0; s < K2_STAGES; ++s)
                    if (issued & (1u << s)) wait_drain(ptx::smem_u32(&ctl->full[s]), (last_par >> s) & 1);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------ MMA issuer (even CTA)
        // M = 256 (both CTAs' row tiles), N = 256, K = 16 per MMA
        if (crank == 0 && lane == 0) {
            constexpr uint32_t idesc = ptx::idesc_bf16(256, K2_BN, 0, 1);
            int stage = 0;
            uint32_t phase = 0;
            int buf = 0;
            uint32_t acc_phase = 0;
            bool ok = true;
            for (int t = t_begin; t < t_end && ok; ++t) {
                const TcTile tl = p.tiles[t];
                const TcMod& md = p.mods[tl.mod];
                const int nk = (md.r + K2_BK - 1) / K2_BK;
                if (!ptx::mbar_wait_cluster(ptx::smem_u32(&ctl->acce[buf]), acc_phase ^ 1, abort_flag, p.status,
                                            MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit)) { ok = false; break; }
                ptx::tc_fence_after();
                const uint32_t d0 = tmem + buf * 256;
                for (int kb = 0; kb < nk; ++kb) {
                    if (!ptx::mbar_wait_cluster(ptx::smem_u32(&ctl->full[stage]), phase, abort_flag, p.status,
                                                MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit)) { ok = false; break; }
                    ptx::tc_fence_after();
                    const uint32_t a = ptx::smem_u32(smem + stage * K2_STAGE_BYTES);
                    const uint32_t b = a + K2_A_BYTES;
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk) {
                        const uint64_t adesc = ptx::smem_desc_sw128(a + kk * 32, 16, 1024);
                        const uint64_t bdesc = ptx::smem_desc_sw128(b + kk * 2048, 8192, 1024);
                        ptx::mma2_f16(d0, adesc, bdesc, idesc, (kb | kk) != 0);
                    }
                    ptx::mma2_commit_mc(ptx::smem_u32(&ctl->empty[stage]), 0x3);
                    if (++stage == K2_STAGES) { stage = 0; phase ^= 1; }
                }
                if (!ok) break;
                ptx::mma2_commit_mc(ptx::smem_u32(&ctl->accf[buf]), 0x3);
                if (++buf == 2) { buf = 0; acc_phase ^= 1; }
            }
            ptx::mma2_commit_mc(ptx::smem_u32(&ctl->drain), 0x1);
            wait_drain(ptx::smem_u32(&ctl->drain), 0);
        }
    } else if (warp == 2) {
        // ------------------------------------------- W chunk loader (TMA in)
        // (bf16 W only: an fp32 W is updated by reduce-add, never loaded)
        if (SB && lane == 0) {
            uint32_t g = 0;
            uint32_t issued = 0, last_par = 0;
            bool ok = true;
            for (int t = t_begin; t < t_end && ok; ++t) {
                const TcTile tl = p.tiles[t];
                const TcMod& md = p.mods[tl.mod];
                const CUtensorMap* wmap = &p.maps[tl.mod * kMaps + 3];
                const int i0 = (2 * tl.t0 + crank) * K2_BM, n0 = tl.t1 * K2_BN;
                const int nc = min(K2_BN / WC, (md.n - n0 + WC - 1) / WC);
                for (int c = 0; c < nc; ++c, ++g) {
                    const int b = g % K2_WBUF;
                    const uint32_t ph = (g / K2_WBUF) & 1;
                    if (!ptx::mbar_wait(ptx::smem_u32(&ctl->wempty[b]), ph ^ 1, abort_flag, p.status,
                                        MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit)) { ok = false; break; }
                    const uint32_t fb = ptx::smem_u32(&ctl->wfull[b]);
                    ptx::mbar_arrive_expect_tx(fb, K2_WBYTES);
                    ptx::tma_load_2d(ptx::smem_u32(wring + b * K2_WBYTES), wmap, fb, n0 + c * WC, i0);
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
        // ------------------------------ W chunk storer (TMA store / reduce-add)
        if (lane == 0) {
            uint32_t g = 0;
            bool ok = true;
            for (int t = t_begin; t < t_end && ok; ++t) {
                const TcTile tl = p.tiles[t];
                const TcMod& md = p.mods[tl.mod];
                const CUtensorMap* wmap = &p.maps[tl.mod * kMaps + 3];
                const int i0 = (2 * tl.t0 + crank) * K2_BM, n0 = tl.t1 * K2_BN;
                const bool w3 = W3D && md.w3d;
                const int nc = w3 ? 2 * min(K2_BN / 64, (md.n - n0) / 64) : min(K2_BN / WC, (md.n - n0 + WC - 1) / WC);
                for (int c = 0; c < nc; ++c, ++g) {
                    const int b = g % K2_WBUF;
                    const uint32_t ph = (g / K2_WBUF) & 1;
                    if (!ptx::mbar_wait(ptx::smem_u32(&ctl->wdone[b]), ph, abort_flag, p.status,
                                        MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit)) { ok = false; break; }
                    const uint32_t src = ptx::smem_u32(wring + b * K2_WBYTES);
                    if constexpr (SB) ptx::tma_store_2d(wmap, src, n0 + c * WC, i0);
                    else if (w3) ptx::tma_reduce_add_3d(&p.maps[tl.mod * kMaps + 8], src, 0,
                                                        (n0 + 64 * (c % (nc / 2))) / 32, i0 + 64 * (c / (nc / 2)));
                    else ptx::tma_reduce_add_2d(wmap, src, n0 + c * WC, i0);
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
        // chunk (32 fp32 / 64 bf16 columns); each thread handles 16 / 32
        // values of its W row in the swizzled shared-memory chunk: the update
        // dW = -lr * alpha * dM * (P N) for an fp32 W (added to W by the
        // storer's reduce), or W - lr * alpha * dM * (P N) rounded to bf16.
        const int ew = warp - 4;                        // 0..7
        const int q = warp & 3;
        const int ch = ew >> 2;
        const int il = q * 32 + lane;                   // row within the tile
        constexpr int NDM = BLK >= 16 ? 1 : 16 / BLK;   // dM values per thread and chunk
        constexpr bool HOIST = BLK >= 32 && K2_BN % BLK == 0;
        int buf = 0;
        uint32_t acc_phase = 0;
        uint32_t g = 0;
        bool ok = true;
        for (int t = t_begin; t < t_end && ok; ++t) {
            const TcTile tl = p.tiles[t];
            const TcMod& md = p.mods[tl.mod];
            const int mm = md.m, nn = md.n, mkb = md.kb;
            const float* const dMp = md.dM;
            const int i0 = (2 * tl.t0 + crank) * K2_BM, n0 = tl.t1 * K2_BN;
            const int i = i0 + il;
            const bool row_ok = i < mm;
            const bool w3 = W3D && md.w3d;
            const int nc = w3 ? 2 * min(K2_BN / 64, (nn - n0) / 64) : min(K2_BN / WC, (nn - n0 + WC - 1) / WC);
            // blocks of B >= 32 columns: the tile's dM values of this row are
            // loaded once, before the wait for the accumulator
            float dmt[HOIST ? K2_BN / BLK : 1];
            if (HOIST) {
#pragma unroll
                for (int d = 0; d < K2_BN / BLK; ++d) {
                    const int jb = n0 / BLK + d;
                    dmt[d] = (p.decompose && row_ok && jb < mkb) ? dMp[(long long)i * mkb + jb] : 1.0f;
                }
            }
            const bool got = ptx::mbar_wait(ptx::smem_u32(&ctl->accf[buf]), acc_phase, abort_flag, p.status,
                                            MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit);
            if (!__all_sync(0xffffffffu, got)) { ok = false; break; }
            ptx::tc_fence_after();
            for (int c = 0; c < nc; ++c, ++g) {
                const int b = g % K2_WBUF;
                const uint32_t ph = (g / K2_WBUF) & 1;
                if constexpr (W3D) {
                    if (w3) {
                        // chunk c: rows 64 hq .. + 63 and columns 64 cq .. + 63 of the
                        // tile, hq = c / (nc / 2), cq = c % (nc / 2): a row half's chunks
                        // go out one after the other, so the reduces of a tile's rows
                        // cover their whole width in turn (K2 per two 7B layers 0.701 ->
                        // 0.690 ms against alternating row halves).  The four warps of
                        // that row half write it (warp ch: the 32-column group ch, one
                        // 128-byte line per row; two lines of a warp's store share a
                        // bank group); the other four only pass the chunk's barriers
                        const int ncq = nc / 2;
                        const bool mine = (c / ncq) == (q >> 1);
                        const int cb = (c % ncq) * 64 + ch * 32;
                        float v[32];
                        if (mine) {
                            __syncwarp();
                            const uint32_t ta = tmem + (static_cast<uint32_t>(q * 32) << 16) + buf * 256 + cb;
                            ptx::tmem_ld16(ta, *reinterpret_cast<float(*)[16]>(v));
                            ptx::tmem_ld16(ta + 16, *reinterpret_cast<float(*)[16]>(v + 16));
                        }
                        const bool gotw = ptx::mbar_wait(ptx::smem_u32(&ctl->wempty[b]), ph ^ 1, abort_flag, p.status,
                                                         MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit);
                        if (!__all_sync(0xffffffffu, gotw)) { ok = false; break; }
                        if (mine) {
                            float d0 = dmt[0];
#pragma unroll
                            for (int d = 1; d < K2_BN / BLK; ++d) d0 = (cb >= d * BLK) ? dmt[d] : d0;
                            const float ms = -p.step_scale;
                            const int ln = (32 * (q & 1) + lane) * 2 + ch;    // box line: row * 2 + group
                            uint8_t* line = wring + b * K2_WBYTES + ln * 128;
                            const uint32_t x = static_cast<uint32_t>(ln & 7);
#pragma unroll
                            for (int u = 0; u < 8; ++u)
                                *reinterpret_cast<uint4*>(line + ((u ^ x) << 4)) =
                                    make_uint4(__float_as_uint(ms * (d0 * v[4 * u + 0])),
                                               __float_as_uint(ms * (d0 * v[4 * u + 1])),
                                               __float_as_uint(ms * (d0 * v[4 * u + 2])),
                                               __float_as_uint(ms * (d0 * v[4 * u + 3])));
                        }
                        ptx::fence_proxy_async_smem();
                        __syncwarp();
                        if (lane == 0) ptx::mbar_arrive(ptx::smem_u32(&ctl->wdone[b]));
                        continue;
                    }
                }
                const int j0 = n0 + c * WC + ch * HC;
                float dm[NDM];
                if (HOIST) {
                    // the thread's 16 (32) columns of the chunk lie in one block
                    const int cb = c * WC + ch * HC;
                    dm[0] = dmt[0];
#pragma unroll
                    for (int d = 1; d < K2_BN / BLK; ++d) dm[0] = (cb >= d * BLK) ? dmt[d] : dm[0];
                } else {
#pragma unroll
                    for (int d = 0; d < NDM; ++d) {
                        const int jb = (j0 + 8 * d) / BLK;
                        dm[d] = (p.decompose && row_ok && jb < mkb) ? dMp[(long long)i * mkb + jb] : 1.0f;
                    }
                }
                float v[HC];
                __syncwarp();
#pragma unroll
                for (int h = 0; h < HC / 16; ++h)
                    ptx::tmem_ld16(tmem + (static_cast<uint32_t>(q * 32) << 16) + buf * 256 + c * WC + ch * HC + 16 * h,
                                   *reinterpret_cast<float(*)[16]>(v + 16 * h));
                // bf16 W: the loaded chunk; fp32 W: a free staging chunk
                const bool gotw = SB ? ptx::mbar_wait(ptx::smem_u32(&ctl->wfull[b]), ph, abort_flag, p.status,
                                                      MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit)
                                     : ptx::mbar_wait(ptx::smem_u32(&ctl->wempty[b]), ph ^ 1, abort_flag, p.status,
                                                      MOARA_ERR_DEVICE_TIMEOUT, kWaitLimit);
                if (!__all_sync(0xffffffffu, gotw)) { ok = false; break; }
                uint8_t* wrow = wring + b * K2_WBYTES + il * 128;
                const uint32_t x = static_cast<uint32_t>(il & 7);
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    uint4* w4 = reinterpret_cast<uint4*>(wrow + (((ch * 4 + u) ^ x) << 4));
                    if constexpr (SB) {
                        const uint4 wv = *w4;
                        const float d0 = dm[0];
                        const uint32_t ww[4] = {wv.x, wv.y, wv.z, wv.w};
                        uint32_t out[4];
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            const float lo = bf_lo(ww[k]) - p.step_scale * (d0 * v[8 * u + 2 * k]);
                            const float hi = bf_hi(ww[k]) - p.step_scale * (d0 * v[8 * u + 2 * k + 1]);
                            out[k] = pack_bf16x2(lo, hi);
                        }
                        *w4 = make_uint4(out[0], out[1], out[2], out[3]);
                    } else {
                        const float d0 = dm[NDM == 1 ? 0 : (u * 4) / BLK];
                        const float ms = -p.step_scale;
                        *w4 = make_uint4(__float_as_uint(ms * (d0 * v[4 * u + 0])),
                                         __float_as_uint(ms * (d0 * v[4 * u + 1])),
                                         __float_as_uint(ms * (d0 * v[4 * u + 2])),
                                         __float_as_uint(ms * (d0 * v[4 * u + 3])));
                    }
                }
                ptx::fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive(ptx::smem_u32(&ctl->wdone[b]));
            }
            if (!ok) break;
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) {   // the even CTA's issuer waits for both CTAs' epilogues
                if (crank == 0) ptx::mbar_arrive(ptx::smem_u32(&ctl->acce[buf]));
                else ptx::mbar_arrive_remote(ptx::mapa(ptx::smem_u32(&ctl->acce[buf]), 0));
            }
            if (++buf == 2) { buf = 0; acc_phase ^= 1; }
        }
    }

    ptx::tc_fence_before();
    __syncwarp();
    ptx::cluster_sync();            // no CTA leaves while its peer may still signal or fill it
    if (warp == 1) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc2(tmem, 512);
    }
}

// ---------------------------------------------------------------- host side
// ===========================================================================
// KR: bf16 tensor-core GEMM of the projector refresh (the TruncatedSVD of
// Algorithm 1, computed by randomized subspace iteration after Halko,
// Martinsson and Tropp, 2011 -- this library's choice of method, not the
// paper's): out (M x N) = op(A) B with fp32 accumulation,
// written in fp32 and/or bf16.  A is read K-major (stored M x K) or MN-major
// (stored K x M), optionally as two planes A_hi + A_lo (two MMAs per k-step
// keep ~16 significant bits of A, used for V); B is stored K x N (MN-major).
// Used for V^T Q, V Z, the Gram matrices X^T X and the triangular factor
// products X R^-1.  Tile 256 x 256 (two 128-row accumulators in TMEM), BK =
// 64, one tile per CTA: the contractions are long enough that the epilogue
// need not overlap the next tile.  The last column tile issues the MMA with
// N = 64 * ceil(cols / 64), so a ragged N costs at most 48 columns; with
// `ktri` the K loop of column tile n0 stops at n0 + 256 (B upper triangular).
// ===========================================================================
constexpr int KR_BM = 256, KR_BN = 256, KR_BK = 64;
constexpr int KR_PLANE = KR_BM * KR_BK * 2;               // 32 KB: one A plane or the B tile
template <bool LO> struct KrCfg {
    static constexpr int STAGES = LO ? 2 : 3;
    static constexpr int STAGE_BYTES = (LO ? 3 : 2) * KR_PLANE;
};
constexpr int KR_WARPS = 10;                              // 0 TMA, 1 MMA, 2-9 epilogue
constexpr int KR_THREADS = KR_WARPS * 32;
constexpr int KR_SMEM = 1024 + 6 * KR_PLANE + 2048;
constexpr int kKrGroup = 64;                              // problems per launch (three maps each in the parameters)

struct KrParams {
    CUtensorMap amap[kKrGroup];        // A_hi, box {64, 64}
    CUtensorMap lmap[kKrGroup];        // A_lo (same geometry), unused without LO
    CUtensorMap bmap[kKrGroup];        // B ({N, K}), box {64, 64}
    float* out[kKrGroup];              // M x N fp32 or null
    uint16_t* out_bf[kKrGroup];        // M x N bf16 or null
    uint16_t* out_lo[kKrGroup];        // M x N bf16 residual (out - bf16(out)) or null
    // alignment reduction (ALIGN): element (j, i) of the product (al_tr) or
    // element (i, j), weighted by the block norm mag[i][j / al_B], is dotted
    // with G[i][j]; al_m is the number of valid product columns
    const uint16_t* al_G[kKrGroup];
    const float* al_mag[kKrGroup];
    double* al_acc[kKrGroup];          // 3 doubles: <G, a>, <a, a>, <G, G>
    int al_ld[kKrGroup], al_kb[kKrGroup], al_m[kKrGroup], al_tr[kKrGroup];
    int al_B, al_log2B;                // block size (a power of two) and its log2
    int M[kKrGroup], N[kKrGroup], K[kKrGroup];
    int ktri[kKrGroup];
    int lower[kKrGroup];               // tiles above the diagonal are skipped
    int tiles_n[kKrGroup];
    int tile_start[kKrGroup + 1];
    int count;
    int* status;
    long long wait_limit;              // clock cycles of a bounded wait before it gives up
};

static_assert(sizeof(KrParams) <= 32764, "KR's parameter block fits the kernel parameter space");

template <bool KMAJOR, bool LO, bool ALIGN = false>
__global__ void __launch_bounds__(KR_THREADS, 1) kr_product(const __grid_constant__ KrParams p) {
    constexpr int STAGES = KrCfg<LO>::STAGES;
    constexpr int STAGE_BYTES = KrCfg<LO>::STAGE_BYTES;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = align1024(smem_raw);
    SmemCtl* ctl = reinterpret_cast<SmemCtl*>(smem + 6 * KR_PLANE);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    volatile int* abort_flag = &ctl->abort;

    // locate (problem, tile)
    const int tile = blockIdx.x;
    int lo = 0, hi = p.count - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (p.tile_start[mid] <= tile) lo = mid; else hi = mid - 1;
    }
    const int pi = lo;
    const int local = tile - p.tile_start[pi];
    const int M = p.M[pi], N = p.N[pi], K = p.K[pi];
    const int i0 = (local / p.tiles_n[pi]) * KR_BM;
    const int n0 = (local % p.tiles_n[pi]) * KR_BN;
    if (p.lower[pi] && n0 >= i0 + KR_BM) return;     // whole CTA, before any barrier or TMEM
    const int nch = min(4, (N - n0 + 63) / 64);            // 64-column chunks of B in this tile
    const int halves = (M - i0) > 128 ? 2 : 1;
    const int kend = p.ktri[pi] ? min(K, n0 + KR_BN) : K;
    const int nk = (kend + KR_BK - 1) / KR_BK;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            ptx::mbar_init(ptx::smem_u32(&ctl->full[s]), 1);
            ptx::mbar_init(ptx::smem_u32(&ctl->empty[s]), 1);
        }
        ptx::mbar_init(ptx::smem_u32(&ctl->accf[0]), 1);
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
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            uint32_t issued = 0, last_par = 0;
            const uint32_t bytes = (LO ? 2 : 1) * KR_PLANE + nch * 8192;
            for (int kb = 0; kb < nk; ++kb) {
                if (!ptx::mbar_wait(ptx::smem_u32(&ctl->empty[stage]), phase ^ 1, abort_flag, p.status,
                                    MOARA_ERR_DEVICE_TIMEOUT, p.wait_limit))
                    break;
                const uint32_t fb = ptx::smem_u32(&ctl->full[stage]);
                ptx::mbar_arrive_expect_tx(fb, bytes);
                const uint32_t a = ptx::smem_u32(smem + stage * STAGE_BYTES);
                const uint32_t b = a + (LO ? 2 : 1) * KR_PLANE;
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    const int x = KMAJOR ? kb * KR_BK : i0 + 64 * c;
                    const int y = KMAJOR ? i0 + 64 * c : kb * KR_BK;
                    ptx::tma_load_2d(a + c * 8192, &p.amap[pi], fb, x, y);
                    if (LO) ptx::tma_load_2d(a + KR_PLANE + c * 8192, &p.lmap[pi], fb, x, y);
                }
                for (int c = 0; c < nch; ++c) ptx::tma_load_2d(b + c * 8192, &p.bmap[pi], fb, n0 + 64 * c, kb * KR_BK);
                issued |= 1u << stage;
                last_par = (last_par & ~(1u << stage)) | (phase << stage);
                if (++stage == STAGES) { stage = 0; phase ^= 1; }
            }
            // every copy issued has landed before the CTA may leave (after a
            // wait that gave up elsewhere the MMA may not have consumed them)
            for (int s = 0; s < STAGES; ++s)
                if (issued & (1u << s)) wait_drain(ptx::smem_u32(&ctl->full[s]), (last_par >> s) & 1);
        }
    } else if (warp == 1) {
        if (lane == 0) {
            const uint32_t idesc = ptx::idesc_bf16(128, nch * 64, KMAJOR ? 0 : 1, 1);
            int stage = 0;
            uint32_t phase = 0;
            for (int kb = 0; kb < nk; ++kb) {
                if (!ptx::mbar_wait(ptx::smem_u32(&ctl->full[stage]), phase, abort_flag, p.status,
                                    MOARA_ERR_DEVICE_TIMEOUT, p.wait_limit)) break;
                ptx::tc_fence_after();
                const uint32_t a = ptx::smem_u32(smem + stage * STAGE_BYTES);
                const uint32_t b = a + (LO ? 2 : 1) * KR_PLANE;
                for (int h = 0; h < halves; ++h) {
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk) {
                        const uint32_t ao = a + h * 16384 + (KMAJOR ? kk * 32 : kk * 2048);
                        const uint64_t adesc = KMAJOR ? ptx::smem_desc_sw128(ao, 16, 1024)
                                                      : ptx::smem_desc_sw128(ao, 8192, 1024);
                        const uint64_t bdesc = ptx::smem_desc_sw128(b + kk * 2048, 8192, 1024);
                        ptx::mma_f16(tmem + h * 256, adesc, bdesc, idesc, (kb | kk) != 0);
                        if (LO) {
                            const uint32_t lo_addr = ao + KR_PLANE;
                            const uint64_t ldesc = KMAJOR ? ptx::smem_desc_sw128(lo_addr, 16, 1024)
                                                          : ptx::smem_desc_sw128(lo_addr, 8192, 1024);
                            ptx::mma_f16(tmem + h * 256, ldesc, bdesc, idesc, 1);
                        }
                    }
                }
                ptx::mma_commit(ptx::smem_u32(&ctl->empty[stage]));
                if (++stage == STAGES) { stage = 0; phase ^= 1; }
            }
            ptx::mma_commit(ptx::smem_u32(&ctl->accf[0]));
            ptx::mma_commit(ptx::smem_u32(&ctl->drain));
            wait_drain(ptx::smem_u32(&ctl->drain), 0);
        }
    } else {
        // 8 epilogue warps: lane quarter q = warp % 4, accumulator half h.
        const int ew = warp - 2;
        const int q = warp & 3;
        const int h = ew >> 2;
        const bool got = ptx::mbar_wait(ptx::smem_u32(&ctl->accf[0]), 0, abort_flag, p.status,
                                        MOARA_ERR_DEVICE_TIMEOUT, p.wait_limit);
        if (ALIGN && __all_sync(0xffffffffu, got) && h < halves) {
            // S(W, t) of §3.2: this thread's row of the product -- row j of
            // (P P^T V)^T against column j of G, or row i of V Q Q^T against
            // row i of G -- weighted by Rep_B(M)
            ptx::tc_fence_after();
            const int row = i0 + h * 128 + q * 32 + lane;
            const uint16_t* const Gp = p.al_G[pi];
            const float* const mg = p.al_mag[pi];
            const int ldg = p.al_ld[pi], kbm = p.al_kb[pi], mm = p.al_m[pi];
            const bool tr = p.al_tr[pi] != 0;
            const int lgB = p.al_log2B;
            const int jb = row >> lgB;
            float dot = 0.0f, na = 0.0f, gg = 0.0f;
            for (int c = 0; c < nch * 4; ++c) {
                const int c0 = n0 + c * 16;
                if (c0 >= mm) break;                      // warp-uniform
                float v[16];
                __syncwarp();
                ptx::tmem_ld16(tmem + (static_cast<uint32_t>(q * 32) << 16) + h * 256 + c * 16, v);
                if (row >= M) continue;
                if (tr) {                                 // product entry (j, i): G[i][j], M[i][j / B]
#pragma unroll
                    for (int e = 0; e < 16; ++e) {
                        const int ci = c0 + e;
                        if (ci < mm) {
                            const float g = __bfloat162float(__ushort_as_bfloat16(Gp[(long long)ci * ldg + row]));
                            const float a = mg[(long long)ci * kbm + jb] * v[e];
                            dot = fmaf(g, a, dot);
                            na = fmaf(a, a, na);
                            gg = fmaf(g, g, gg);
                        }
                    }
                } else {                                  // product entry (i, j): G[i][j], M[i][j / B]
                    const uint16_t* grow = Gp + (long long)row * ldg;
                    const float* mrow = mg + (long long)row * kbm;
#pragma unroll
                    for (int e = 0; e < 16; ++e) {
                        const int ci = c0 + e;
                        if (ci < mm) {
                            const float g = __bfloat162float(__ushort_as_bfloat16(grow[ci]));
                            const float a = mrow[ci >> lgB] * v[e];
                            dot = fmaf(g, a, dot);
                            na = fmaf(a, a, na);
                            gg = fmaf(g, g, gg);
                        }
                    }
                }
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                dot += __shfl_xor_sync(0xffffffffu, dot, o);
                na += __shfl_xor_sync(0xffffffffu, na, o);
                gg += __shfl_xor_sync(0xffffffffu, gg, o);
            }
            if (lane == 0) {
                double* acc = p.al_acc[pi];
                atomicAdd(acc + 0, static_cast<double>(dot));
                atomicAdd(acc + 1, static_cast<double>(na));
                atomicAdd(acc + 2, static_cast<double>(gg));
            }
        } else if (!ALIGN && __all_sync(0xffffffffu, got) && h < halves) {
            ptx::tc_fence_after();
            const int row = i0 + h * 128 + q * 32 + lane;
            uint16_t* const ol = p.out_lo[pi];
            float* const of = p.out[pi];
            uint16_t* const ob = p.out_bf[pi];
            const long long ro = (long long)row * N;
            for (int c = 0; c < nch * 4; ++c) {
                const int j0 = n0 + c * 16;
                if (j0 >= N) break;                       // warp-uniform
                float v[16];
                __syncwarp();
                ptx::tmem_ld16(tmem + (static_cast<uint32_t>(q * 32) << 16) + h * 256 + c * 16, v);
                if (row >= M) continue;
                if (j0 + 16 <= N) {                       // N % 8 == 0: 16-byte aligned rows
                    if (of != nullptr) {
                        float4* o4 = reinterpret_cast<float4*>(of + ro + j0);
#pragma unroll
                        for (int e = 0; e < 4; ++e)
                            o4[e] = make_float4(v[4 * e], v[4 * e + 1], v[4 * e + 2], v[4 * e + 3]);
                    }
                    if (ob != nullptr) {
                        uint4* b4 = reinterpret_cast<uint4*>(ob + ro + j0);
                        b4[0] = make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]),
                                           pack_bf16x2(v[4], v[5]), pack_bf16x2(v[6], v[7]));
                        b4[1] = make_uint4(pack_bf16x2(v[8], v[9]), pack_bf16x2(v[10], v[11]),
                                           pack_bf16x2(v[12], v[13]), pack_bf16x2(v[14], v[15]));
                    }
                    if (ol != nullptr) {
                        float rl[16];
#pragma unroll
                        for (int e = 0; e < 16; ++e)
                            rl[e] = v[e] - __bfloat162float(__float2bfloat16_rn(v[e]));
                        uint4* l4 = reinterpret_cast<uint4*>(ol + ro + j0);
                        l4[0] = make_uint4(pack_bf16x2(rl[0], rl[1]), pack_bf16x2(rl[2], rl[3]),
                                           pack_bf16x2(rl[4], rl[5]), pack_bf16x2(rl[6], rl[7]));
                        l4[1] = make_uint4(pack_bf16x2(rl[8], rl[9]), pack_bf16x2(rl[10], rl[11]),
                                           pack_bf16x2(rl[12], rl[13]), pack_bf16x2(rl[14], rl[15]));
                    }
                } else {
#pragma unroll
                    for (int e = 0; e < 16; ++e) {
                        if (j0 + e >= N) continue;
                        if (of != nullptr) of[ro + j0 + e] = v[e];
                        const __nv_bfloat16 hb = __float2bfloat16_rn(v[e]);
                        if (ob != nullptr) ob[ro + j0 + e] = *reinterpret_cast<const uint16_t*>(&hb);
                        if (ol != nullptr) {
                            const __nv_bfloat16 lb = __float2bfloat16_rn(v[e] - __bfloat162float(hb));
                            ol[ro + j0 + e] = *reinterpret_cast<const uint16_t*>(&lb);
                        }
                    }
                }
            }
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
// KS: fp32-accurate GEMM of the Rayleigh-Ritz step on tensor cores.  Both
// operands arrive as three bf16 planes (x = hi + mid + lo, 24 significant
// bits); six MMAs per k-step (hi.hi, hi.mid, mid.hi, hi.lo, mid.mid, lo.hi)
// leave out terms of relative size 2^-24 and below.  out (M x N, fp32) =
// A B with A stored K x M and B stored K x N (both MN-major), tile 256 x 256
// (two 128-row accumulators in TMEM), BK = 32, two stages of 96 KB; `ktri`
// stops the K loop of column tile n0 at n0 + 256 (B upper triangular).
// ===========================================================================
constexpr int KS_BM = 256, KS_BN = 256, KS_BK = 32;
constexpr int KS_PLANE = KS_BM * KS_BK * 2;               // 16 KB: one plane of A (or B)
constexpr int KS_RING = 12 * KS_PLANE;                    // 192 KB of stages
constexpr int KS_SMEM = 1024 + KS_RING + 2048;
// NP = 3 planes: six products per k-step, two stages of 96 KB.  NP = 2
// (hi + mid, 16 significant bits; for iterates that a later fp32-accurate
// pass corrects): three products (hi.hi, hi.mid, mid.hi), three stages of 64 KB.
template <int NP> struct KsCfg {
    static constexpr int STAGE = 2 * NP * KS_PLANE;
    static constexpr int STAGES = KS_RING / STAGE;
    static constexpr int PRODUCTS = NP == 3 ? 6 : 3;
};
constexpr int kKsGroup = 38;                              // problems per launch (six maps each in the parameters)

struct KsParams {
    CUtensorMap amap[kKsGroup][3];     // A planes ({M, K}, box {64, 32})
    CUtensorMap bmap[kKsGroup][3];     // B planes ({N, K}, box {64, 32})
    float* out[kKsGroup];
    int M[kKsGroup], N[kKsGroup], K[kKsGroup];
    int ktri[kKsGroup];
    int ldo[kKsGroup];                 // row pitch of out
    int sub[kKsGroup];                 // out -= A B
    int lower[kKsGroup];               // tiles above the diagonal are skipped
    int tiles_n[kKsGroup];
    int tile_start[kKsGroup + 1];
    int count;
    int* status;
    long long wait_limit;              // clock cycles of a bounded wait before it gives up
};

static_assert(sizeof(KsParams) <= 32764, "KS's parameter block fits the kernel parameter space");

template <int NP>
__global__ void __launch_bounds__(KR_THREADS, 1) ks_product(const __grid_constant__ KsParams p) {
    constexpr int KS_STAGE = KsCfg<NP>::STAGE, KS_STAGES = KsCfg<NP>::STAGES;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = align1024(smem_raw);
    SmemCtl* ctl = reinterpret_cast<SmemCtl*>(smem + KS_RING);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    volatile int* abort_flag = &ctl->abort;

    const int tile = blockIdx.x;
    int lo = 0, hi = p.count - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (p.tile_start[mid] <= tile) lo = mid; else hi = mid - 1;
    }
    const int pi = lo;
    const int local = tile - p.tile_start[pi];
    const int M = p.M[pi], N = p.N[pi], K = p.K[pi];
    const int i0 = (local / p.tiles_n[pi]) * KS_BM;
    const int n0 = (local % p.tiles_n[pi]) * KS_BN;
    if (p.lower[pi] && n0 >= i0 + KS_BM) return;     // whole CTA, before any barrier or TMEM
    const int nch = min(4, (N - n0 + 63) / 64);
    const int halves = (M - i0) > 128 ? 2 : 1;
    const int kend = p.ktri[pi] ? min(K, n0 + KS_BN) : K;
    const int nk = (kend + KS_BK - 1) / KS_BK;

    if (threadIdx.x == 0) {
        for (int s = 0; s < KS_STAGES; ++s) {
            ptx::mbar_init(ptx::smem_u32(&ctl->full[s]), 1);
            ptx::mbar_init(ptx::smem_u32(&ctl->empty[s]), 1);
        }
        ptx::mbar_init(ptx::smem_u32(&ctl->accf[0]), 1);
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
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            uint32_t issued = 0, last_par = 0;
            const uint32_t bytes = NP * KS_PLANE + NP * nch * 4096;
            for (int kb = 0; kb < nk; ++kb) {
                if (!ptx::mbar_wait(ptx::smem_u32(&ctl->empty[stage]), phase ^ 1, abort_flag, p.status,
                                    MOARA_ERR_DEVICE_TIMEOUT, p.wait_limit))
                    break;
                const uint32_t fb = ptx::smem_u32(&ctl->full[stage]);
                ptx::mbar_arrive_expect_tx(fb, bytes);
                const uint32_t a = ptx::smem_u32(smem + stage * KS_STAGE);
                const uint32_t b = a + NP * KS_PLANE;
#pragma unroll
                for (int q = 0; q < NP; ++q) {
#pragma unroll
                    for (int c = 0; c < 4; ++c)
                        ptx::tma_load_2d(a + q * KS_PLANE + c * 4096, &p.amap[pi][q], fb, i0 + 64 * c, kb * KS_BK);
                    for (int c = 0; c < nch; ++c)
                        ptx::tma_load_2d(b + q * KS_PLANE + c * 4096, &p.bmap[pi][q], fb, n0 + 64 * c, kb * KS_BK);
                }
                issued |= 1u << stage;
                last_par = (last_par & ~(1u << stage)) | (phase << stage);
                if (++stage == KS_STAGES) { stage = 0; phase ^= 1; }
            }
            // every copy issued has landed before the CTA may leave (after a
            // wait that gave up elsewhere the MMA may not have consumed them)
            for (int s = 0; s < KS_STAGES; ++s)
                if (issued & (1u << s)) wait_drain(ptx::smem_u32(&ctl->full[s]), (last_par >> s) & 1);
        }
    } else if (warp == 1) {
        if (lane == 0) {
            const uint32_t idesc = ptx::idesc_bf16(128, nch * 64, 1, 1);
            // plane pairs (A, B) of the six products
            constexpr int PA[6] = {0, 0, 1, 0, 1, 2};
            constexpr int PB[6] = {0, 1, 0, 2, 1, 0};
            int stage = 0;
            uint32_t phase = 0;
            for (int kb = 0; kb < nk; ++kb) {
                if (!ptx::mbar_wait(ptx::smem_u32(&ctl->full[stage]), phase, abort_flag, p.status,
                                    MOARA_ERR_DEVICE_TIMEOUT, p.wait_limit)) break;
                ptx::tc_fence_after();
                const uint32_t a = ptx::smem_u32(smem + stage * KS_STAGE);
                const uint32_t b = a + NP * KS_PLANE;
#pragma unroll
                for (int kk = 0; kk < 2; ++kk) {
#pragma unroll
                    for (int e = 0; e < KsCfg<NP>::PRODUCTS; ++e) {
                        const uint64_t bdesc = ptx::smem_desc_sw128(b + PB[e] * KS_PLANE + kk * 2048, 4096, 1024);
                        for (int h = 0; h < halves; ++h) {
                            const uint64_t adesc =
                                ptx::smem_desc_sw128(a + PA[e] * KS_PLANE + h * 8192 + kk * 2048, 4096, 1024);
                            ptx::mma_f16(tmem + h * 256, adesc, bdesc, idesc, (kb | kk | e) != 0);
                        }
                    }
                }
                ptx::mma_commit(ptx::smem_u32(&ctl->empty[stage]));
                if (++stage == KS_STAGES) { stage = 0; phase ^= 1; }
            }
            ptx::mma_commit(ptx::smem_u32(&ctl->accf[0]));
            ptx::mma_commit(ptx::smem_u32(&ctl->drain));
            wait_drain(ptx::smem_u32(&ctl->drain), 0);
        }
    } else {
        const int ew = warp - 2;
        const int q = warp & 3;
        const int h = ew >> 2;
        const bool got = ptx::mbar_wait(ptx::smem_u32(&ctl->accf[0]), 0, abort_flag, p.status,
                                        MOARA_ERR_DEVICE_TIMEOUT, p.wait_limit);
        if (__all_sync(0xffffffffu, got) && h < halves) {
            ptx::tc_fence_after();
            const int row = i0 + h * 128 + q * 32 + lane;
            float* const of = p.out[pi];
            const long long ro = (long long)row * p.ldo[pi];
            const bool sub = p.sub[pi] != 0;
            for (int c = 0; c < nch * 4; ++c) {
                const int j0 = n0 + c * 16;
                if (j0 >= N) break;                       // warp-uniform
                float v[16];
                __syncwarp();
                ptx::tmem_ld16(tmem + (static_cast<uint32_t>(q * 32) << 16) + h * 256 + c * 16, v);
                if (row >= M) continue;
                if (j0 + 16 <= N) {
                    float4* o4 = reinterpret_cast<float4*>(of + ro + j0);
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        float4 w = make_float4(v[4 * e], v[4 * e + 1], v[4 * e + 2], v[4 * e + 3]);
                        if (sub) {
                            const float4 o = o4[e];
                            w = make_float4(o.x - w.x, o.y - w.y, o.z - w.z, o.w - w.w);
                        }
                        o4[e] = w;
                    }
                } else {
#pragma unroll
                    for (int e = 0; e < 16; ++e)
                        if (j0 + e < N) of[ro + j0 + e] = sub ? of[ro + j0 + e] - v[e] : v[e];
                }
            }
        }
    }

    ptx::tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, 512);
    }
}

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

// Largest number of 2-CTA clusters of `fn` resident at once (at most `cap`).
int max_clusters(const void* fn, int threads, int smem, int cap) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(2 * cap, 1, 1);
    cfg.blockDim = dim3(threads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, fn, &cfg) != cudaSuccess || n < 1) {
        cudaGetLastError();
        return cap;
    }
    return std::min(n, cap);
}

template <int BLK>
void set_smem_attrs() {
    cudaFuncSetAttribute(k2_backproject<BLK, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, K2_SMEM);
    if constexpr (BLK >= 32)
        cudaFuncSetAttribute(k2_backproject<BLK, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, K2_SMEM);
}

}  // namespace

struct TcState {
    int device = 0;
    int* d_status = nullptr;
    int sms = 148;
    EncodeTiledFn encode = nullptr;
    std::string err;
    std::vector<TcMod> mods;               // indexed by module id (unsupported ones left zero)
    std::vector<CUtensorMap> maps;         // kMaps per module id
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
    int k1_clusters = 1, k2_clusters = 1;  // co-resident 2-CTA clusters of K1 / K2
    K1Params p1;                           // parameter block of the next K1 launch
    K0Params p0;                           // parameter block of the next K0 launch
    KrParams pr;                           // parameter block of the next refresh GEMM launch
    bool kr_attrs = false;
    KsParams ps;                           // parameter block of the next split-precision GEMM launch
    bool ks_attrs = false;
    // decomposition of later module parts, overlapped with K1 / K2 of earlier ones
    cudaStream_t aux = nullptr;
    cudaEvent_t ev_start = nullptr;
    cudaEvent_t ev_part[32] = {};          // decomposition of part q done (auxiliary stream)
    cudaEvent_t ev_k1[32] = {};            // K1 of part q about to start (launching stream)
    long long wait_limit = kWaitLimit;     // bounded waits of the refresh / alignment products (KR, KS)
};

bool tc_supported(int m, int n, int r, int B, int dtype, int decompose, int state_dtype) {
    if (state_dtype == MOARA_DTYPE_BF16 && decompose && B < 32) return false;
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
    if (st->aux) cudaStreamDestroy(st->aux);
    if (st->ev_start) cudaEventDestroy(st->ev_start);
    for (cudaEvent_t e : st->ev_part)
        if (e) cudaEventDestroy(e);
    for (cudaEvent_t e : st->ev_k1)
        if (e) cudaEventDestroy(e);
    delete st;
}

int tc_register(TcState* st, int id, const ModDev& md, const moara_hparams& hp) {
    if (st == nullptr) return MOARA_OK;
    if (static_cast<int>(st->mods.size()) <= id) {
        st->mods.resize(id + 1, TcMod{});
        st->maps.resize(kMaps * (id + 1));
    }
    if (!tc_supported(md.m, md.n, md.r, hp.block_size, md.dtype, hp.decompose, hp.state_dtype) || md.Pb == nullptr)
        return MOARA_OK;
    // W and the direction moments: fp32, or bf16 (state_dtype); a ring chunk
    // is one 128-byte row wide either way
    const bool sb = hp.state_dtype == MOARA_DTYPE_BF16;
    const CUtensorMapDataType sdt = sb ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32;
    const int ses = sb ? 2 : 4, scols = sb ? StateCols<true>::N : StateCols<false>::N;
    TcMod t{};
    t.m = md.m; t.n = md.n; t.r = md.r; t.kb = md.kb;
    t.Vhi = md.ws_Vhi; t.Vlo = md.ws_Vlo;
    t.W = md.W; t.exp_avg = md.exp_avg; t.exp_avg_sq = md.exp_avg_sq;
    t.mag = md.ws_inv;     // the block-scale buffer of the fp32 path holds the norms here
    t.mag_avg = md.mag_avg; t.mag_avg_sq = md.mag_avg_sq;
    t.Nb = reinterpret_cast<uint16_t*>(md.ws_N);
    t.dM = md.ws_dM;
    t.Pb = md.Pb;
    t.right = md.right;
    t.Qt = md.ws_Qt;
    CUtensorMap* mp = &st->maps[kMaps * id];
    bool ok;
    if (!md.right) {
        // K1: A = P^T (MN-major chunks of P), B = V (MN-major), moments r x n;
        // K2: A = P rows (K-major), B = N (MN-major)
        ok = encode_bf16_2d(st->encode, &mp[0], md.Pb, md.r, md.m, 64, 64) &&
             encode_bf16_2d(st->encode, &mp[1], md.Pb, md.r, md.m, 64, 128) &&
             encode_bf16_2d(st->encode, &mp[2], t.Nb, md.n, md.r, 64, 64) &&
             encode_bf16_2d(st->encode, &mp[4], t.Vhi, md.n, md.m, 64, 64) &&
             encode_bf16_2d(st->encode, &mp[5], t.Vlo, md.n, md.m, 64, 64) &&
             encode_2d(st->encode, &mp[6], sdt, ses, md.exp_avg, md.n, md.r, scols, K1_BM) &&
             encode_2d(st->encode, &mp[7], sdt, ses, md.exp_avg_sq, md.n, md.r, scols, K1_BM);
    } else {
        // right projector Q (n x r): K1 computes R = V Q with A = V rows
        // (K-major, 128 rows x 64 columns) and B = Q (MN-major chunks), moments
        // m x r; K2 computes dV = N Q^T with A = N rows (K-major) and
        // B = Q^T (r x n, MN-major)
        ok = md.ws_Qt != nullptr &&
             encode_bf16_2d(st->encode, &mp[0], md.Pb, md.r, md.n, 64, 64) &&
             encode_bf16_2d(st->encode, &mp[1], t.Nb, md.r, md.m, 64, 128) &&
             encode_bf16_2d(st->encode, &mp[2], md.ws_Qt, md.n, md.r, 64, 64) &&
             encode_bf16_2d(st->encode, &mp[4], t.Vhi, md.n, md.m, 64, 128) &&
             encode_bf16_2d(st->encode, &mp[5], t.Vlo, md.n, md.m, 64, 128) &&
             encode_2d(st->encode, &mp[6], sdt, ses, md.exp_avg, md.r, md.m, scols, K1_BM) &&
             encode_2d(st->encode, &mp[7], sdt, ses, md.exp_avg_sq, md.r, md.m, scols, K1_BM);
    }
    ok = ok && encode_2d(st->encode, &mp[3], sdt, ses, md.W, md.n, md.m, scols, K2_BM);
    if (!ok) {
        st->err = "cuTensorMapEncodeTiled failed";
        return MOARA_ERR_CUDA;
    }
    // An fp32 W whose rows split into 64-column pairs of 128-byte groups is
    // also viewed as (32 columns, n / 32 groups, m rows): a box of 32 x 2 x 64
    // adds 64 rows x 256 contiguous bytes per row with one reduce, traversed
    // row by row, while each 128-byte group stays one swizzled line of the
    // staging chunk (line = row * 2 + group).  The wider contiguous pieces per
    // row keep HBM pages open longer than the 128-byte pieces of the 2-D map
    // (K2 per two 7B layers 0.74 -> 0.70 ms; the group-outer box order, whose
    // lines are free of bank conflicts, gave 0.72 ms).
    t.w3d = 0;
    if (!sb && md.n % 64 == 0) {
        const cuuint64_t dims[3] = {32, static_cast<cuuint64_t>(md.n / 32), static_cast<cuuint64_t>(md.m)};
        const cuuint64_t strides[2] = {128, static_cast<cuuint64_t>(md.n) * 4};
        const cuuint32_t box[3] = {32, 2, 64};
        const cuuint32_t estr[3] = {1, 1, 1};
        t.w3d = st->encode(&mp[8], CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, md.W, dims, strides, box, estr,
                           CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                           CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
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
            cudaMalloc(&st->d_maps, sizeof(CUtensorMap) * kMaps * ncap) != cudaSuccess) {
            st->err = "cudaMalloc of the tensor-core module table failed";
            return MOARA_ERR_CUDA;
        }
        st->cap = ncap;
    }
    if (cudaMemcpy(st->d_mods, st->mods.data(), sizeof(TcMod) * n, cudaMemcpyHostToDevice) != cudaSuccess ||
        cudaMemcpy(st->d_maps, st->maps.data(), sizeof(CUtensorMap) * kMaps * n, cudaMemcpyHostToDevice) !=
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

// Work lists of one launch: K1 tiles (128-rank x 256-column) and K2 tiles
// (128-row x 256-column), cost-weighted in SM clocks: MMA time (8 clocks per
// K row of a 128 x 256 tile) against the epilogue's HBM traffic (K1: the two
// moments read and written and N stored, 18 bytes per entry; K2: W read and
// written, 8 bytes per entry; about 27 bytes per clock per SM).
static TcState::Tiles* tc_tiles(TcState* st, const std::vector<int>& ids) {
    auto it = st->tiles.find(ids);
    if (it != st->tiles.end()) return &it->second;
    // Work units are pair tiles: the two CTAs of a cluster take rank (K1) or
    // row (K2) tiles 2 t0 and 2 t0 + 1 of the same column tile t1.
    std::vector<TcTile> k1, k2;
    std::vector<double> c1, c2;
    for (size_t slot = 0; slot < ids.size(); ++slot) {
        const TcMod& md = st->mods[ids[slot]];
        // column tiles outer, rank pairs inner: clusters that start together
        // share the V panel of one column tile in L2
        // R: r x n (K = m), or m x r (K = n) with a right projector
        const int Rr = md.right ? md.m : md.r, Rc = md.right ? md.r : md.n, Rk = md.right ? md.n : md.m;
        const int nt = (Rc + K1_BN - 1) / K1_BN, rt = (Rr + K1_BM - 1) / K1_BM;
        for (int j = 0; j < nt; ++j)
            for (int i = 0; i < (rt + 1) / 2; ++i) {
                const int rows = std::min(K1_BM, Rr - 2 * i * K1_BM);
                const double mma = 8.0 * Rk;
                const double epi = 0.66 * rows * std::min(K1_BN, Rc - j * K1_BN);
                k1.push_back({ids[slot], static_cast<int>(slot), i, j});
                c1.push_back(std::max(mma, epi));
            }
        const int mt = (md.m + K2_BM - 1) / K2_BM, nt2 = (md.n + K2_BN - 1) / K2_BN;
        for (int i = 0; i < (mt + 1) / 2; ++i)
            for (int j = 0; j < nt2; ++j) {
                const double mma = 8.0 * md.r;
                const double epi = 0.3 * std::min(K2_BM, md.m - 2 * i * K2_BM) * std::min(K2_BN, md.n - j * K2_BN);
                k2.push_back({ids[slot], static_cast<int>(slot), i, j});
                c2.push_back(std::max(mma, epi));
            }
    }
    TcState::Tiles t;
    t.g1 = std::max(1, std::min(static_cast<int>(k1.size()), st->k1_clusters));   // clusters
    t.g2 = std::max(1, std::min(static_cast<int>(k2.size()), st->k2_clusters));
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

// K0 and Optimizer_M of one module part.  `background`: a grid of short
// CTAs (about four row segments per warp) that fills the room K1 / K2 leave
// on each SM instead of a persistent grid that would hold SMs they need.
template <int BLK>
static cudaError_t launch_k0(TcState* st, const K0Params& p0, bool background, cudaStream_t s,
                             int64_t* launches, const TcProfile& prof, bool mag_adam = true) {
    const int phase = background ? MOARA_PHASE_TC_DECOMPOSE_OVERLAP : MOARA_PHASE_TC_DECOMPOSE;
    if (prof.on) prof.mark(prof.ctx, phase, s, true);
    const long long items = p0.start[p0.count];
    const int g0 = background ? static_cast<int>(std::max<long long>(1, std::min<long long>((items + 31) / 32, 1 << 30)))
                              : st->sms * 3;
    k0_decompose<BLK><<<g0, 256, 0, s>>>(p0);
    if (mag_adam) k0_mag_adam<<<background ? st->sms : st->sms * 4, 256, 0, s>>>(p0);
    if (prof.on) prof.mark(prof.ctx, phase, s, false);
    *launches += mag_adam ? 2 : 1;
    return cudaGetLastError();
}

// which: 1 = K1 only, 2 = K2 only, 3 = both
template <int BLK, bool SB>
static cudaError_t launch_k12(TcState* st, const K1Params& p1, const K2Params& p2, int g1, int g2, bool hilo,
                              cudaStream_t s, int64_t* launches, const TcProfile& prof, int which, bool rt) {
    cudaError_t e;
    if (which & 1) {
        if (prof.on) prof.mark(prof.ctx, MOARA_PHASE_TC_PROJECT, s, true);
        if (rt) {
            if (hilo) k1_project<true, SB, true><<<2 * g1, K1_THREADS, K1_SMEM, s>>>(p1);
            else k1_project<false, SB, true><<<2 * g1, K1_THREADS, K1_SMEM, s>>>(p1);
        } else {
            if (hilo) k1_project<true, SB, false><<<2 * g1, K1_THREADS, K1_SMEM, s>>>(p1);
            else k1_project<false, SB, false><<<2 * g1, K1_THREADS, K1_SMEM, s>>>(p1);
        }
        if (prof.on) prof.mark(prof.ctx, MOARA_PHASE_TC_PROJECT, s, false);
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
        ++*launches;
    }
    if (!(which & 2)) return cudaSuccess;
    if (prof.on) prof.mark(prof.ctx, MOARA_PHASE_TC_BACKPROJECT, s, true);
    k2_backproject<BLK, SB><<<2 * g2, K2_THREADS, K2_SMEM, s>>>(p2);
    if (prof.on) prof.mark(prof.ctx, MOARA_PHASE_TC_BACKPROJECT, s, false);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    ++*launches;
    return cudaSuccess;
}

static cudaError_t launch_k0_any(int B, TcState* st, const K0Params& p0, bool background, cudaStream_t s,
                                 int64_t* launches, const TcProfile& prof, bool mag_adam = true) {
    switch (B) {
        case 8: return launch_k0<8>(st, p0, background, s, launches, prof, mag_adam);
        case 16: return launch_k0<16>(st, p0, background, s, launches, prof, mag_adam);
        case 32: return launch_k0<32>(st, p0, background, s, launches, prof, mag_adam);
        case 64: return launch_k0<64>(st, p0, background, s, launches, prof, mag_adam);
        default: return launch_k0<128>(st, p0, background, s, launches, prof, mag_adam);
    }
}

static cudaError_t launch_k12_any(int B, bool sb, TcState* st, const K1Params& p1, const K2Params& p2, int g1,
                                  int g2, bool hilo, cudaStream_t s, int64_t* launches, const TcProfile& prof,
                                  int which = 3, bool rt = false) {
    if (sb) {   // bf16 states: B >= 32 (tc_supported)
        switch (B) {
            case 32: return launch_k12<32, true>(st, p1, p2, g1, g2, hilo, s, launches, prof, which, rt);
            case 64: return launch_k12<64, true>(st, p1, p2, g1, g2, hilo, s, launches, prof, which, rt);
            default: return launch_k12<128, true>(st, p1, p2, g1, g2, hilo, s, launches, prof, which, rt);
        }
    }
    switch (B) {
        case 8: return launch_k12<8, false>(st, p1, p2, g1, g2, hilo, s, launches, prof, which, rt);
        case 16: return launch_k12<16, false>(st, p1, p2, g1, g2, hilo, s, launches, prof, which, rt);
        case 32: return launch_k12<32, false>(st, p1, p2, g1, g2, hilo, s, launches, prof, which, rt);
        case 64: return launch_k12<64, false>(st, p1, p2, g1, g2, hilo, s, launches, prof, which, rt);
        default: return launch_k12<128, false>(st, p1, p2, g1, g2, hilo, s, launches, prof, which, rt);
    }
}

// Modules per launch group are split into this many parts (consecutive
// modules, about equal gradient bytes) when the group has at least
// kOverlapMin modules: the decomposition of part q + 1 runs on an auxiliary
// stream while K1 / K2 of part q run.
constexpr int kOverlapParts = 16;
constexpr int kOverlapMin = 32;
static_assert(kOverlapParts <= 32, "one event per part");

int tc_group_limit() { return kTcGroup; }

int tc_step(TcState* st, const moara_hparams& hp, int n_mod, const int* ids, const void* const* G, float bc1,
            float bc2, float lr, int first_step, const float* clip, const TcClipFuse* fuse, cudaStream_t s,
            int64_t* launches, const TcProfile& prof) {
    if (!st->attrs_set) {
        for (auto fn : {k1_project<true, false, false>, k1_project<false, false, false>, k1_project<true, true, false>,
                        k1_project<false, true, false>, k1_project<true, false, true>, k1_project<false, false, true>,
                        k1_project<true, true, true>, k1_project<false, true, true>})
            cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, K1_SMEM);
        set_smem_attrs<8>(); set_smem_attrs<16>(); set_smem_attrs<32>(); set_smem_attrs<64>();
        set_smem_attrs<128>();
        // clusters of two that fit on the GPU at once (persistent grids)
        st->k1_clusters = max_clusters(reinterpret_cast<const void*>(k1_project<false, false, false>), K1_THREADS,
                                       K1_SMEM,
                                       st->sms / 2);
        st->k2_clusters = max_clusters(reinterpret_cast<const void*>(k2_backproject<128, false>), K2_THREADS, K2_SMEM,
                                       st->sms / 2);
        st->attrs_set = true;
    }
    int rc = tc_upload(st);
    if (rc != MOARA_OK) return rc;
    const bool dec = hp.decompose != 0;
    const bool hilo = dec && first_step;
    const int B = dec ? hp.block_size : 128;
    auto fail = [&](const char* what) {
        st->err = what;
        return MOARA_ERR_CUDA;
    };
    // clipping from the block norms: Optimizer_M and K2 wait for the norm of
    // every module, so they run once after all decompositions and K1s
    const bool fused = fuse != nullptr && dec;
    if (fused && n_mod > kTcGroup) {
        st->err = "fused clipping takes at most tc_group_limit() modules";
        return MOARA_ERR_UNSUPPORTED;
    }
    for (int c0 = 0; c0 < n_mod; c0 += kTcGroup) {
        const int cnt = std::min(kTcGroup, n_mod - c0);
        // parts of the group (consecutive modules, about equal G bytes)
        const int nparts = (dec && cnt >= kOverlapMin) ? kOverlapParts : 1;
        std::vector<int> pstart{0};
        if (nparts > 1) {
            double tot = 0.0;
            for (int q = 0; q < cnt; ++q) tot += (double)st->mods[ids[c0 + q]].m * st->mods[ids[c0 + q]].n;
            double acc = 0.0;
            for (int q = 0; q < cnt; ++q) {
                acc += (double)st->mods[ids[c0 + q]].m * st->mods[ids[c0 + q]].n;
                if ((int)pstart.size() < nparts && acc >= tot * pstart.size() / nparts && q + 1 < cnt)
                    pstart.push_back(q + 1);
            }
        }
        pstart.push_back(cnt);
        const int np = static_cast<int>(pstart.size()) - 1;
        if (np > 1) {
            if (st->aux == nullptr) {
                cudaError_t e = cudaStreamCreateWithFlags(&st->aux, cudaStreamNonBlocking);
                if (e == cudaSuccess) e = cudaEventCreateWithFlags(&st->ev_start, cudaEventDisableTiming);
                for (int q = 0; q < 32 && e == cudaSuccess; ++q) {
                    e = cudaEventCreateWithFlags(&st->ev_part[q], cudaEventDisableTiming);
                    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&st->ev_k1[q], cudaEventDisableTiming);
                }
                if (e != cudaSuccess) return fail("auxiliary stream / events");
            }
            // the auxiliary stream starts after everything queued on s so far
            if (cudaEventRecord(st->ev_start, s) != cudaSuccess ||
                cudaStreamWaitEvent(st->aux, st->ev_start, 0) != cudaSuccess)
                return fail("auxiliary stream ordering");
        }
        auto build_p0 = [&](int a, int b) {
            K0Params& p0 = st->p0;
            std::memset(&p0, 0, sizeof(p0));
            p0.count = b - a;
            p0.hilo = hilo ? 1 : 0;
            p0.do_mag = 1;
            p0.decomp_eps = hp.decomp_eps;
            p0.beta1 = hp.beta1; p0.beta2 = hp.beta2; p0.adam_eps = hp.adam_eps;
            p0.bc1 = bc1; p0.bc2 = bc2;
            p0.clip = clip;
            long long acc = 0, macc = 0;
            for (int q = 0; q < b - a; ++q) {
                const TcMod& md = st->mods[ids[c0 + a + q]];
                const int segs = (md.n + K0_SEG - 1) / K0_SEG;
                p0.start[q] = acc;
                p0.mstart[q] = macc;
                p0.p[q] = K0Item{static_cast<const uint16_t*>(G[c0 + a + q]), md.Vhi, md.Vlo, md.mag, md.mag_avg,
                                 md.mag_avg_sq, md.dM, md.m, md.n, md.kb, segs};
                acc += static_cast<long long>(md.m) * segs;
                macc += static_cast<long long>(md.m) * md.kb;
            }
            p0.start[b - a] = acc;
            p0.mstart[b - a] = macc;
            return &p0;
        };
        // decomposition: part 0 on s with the full grid; part q + 1 in the
        // background on the auxiliary stream, launched after K1 / K2 of part q
        // so that their persistent CTAs are placed first
        if (dec && launch_k0_any(B, st, *build_p0(pstart[0], pstart[1]), false, s, launches, prof, !fused) !=
                       cudaSuccess)
            return fail("decomposition launch failed");
        for (int q = 0; q < np; ++q) {
            const int a = pstart[q], b = pstart[q + 1];
            std::vector<int> chunk(ids + c0 + a, ids + c0 + b);
            TcState::Tiles* tl = tc_tiles(st, chunk);
            if (tl == nullptr) { st->err = "tile list allocation failed"; return MOARA_ERR_CUDA; }
            if (q > 0 && cudaStreamWaitEvent(s, st->ev_part[q], 0) != cudaSuccess) return fail("part wait");
            K1Params& p1 = st->p1;
            std::memset(&p1, 0, sizeof(p1));
            if (!dec) {
                for (int k = 0; k < b - a; ++k) {
                    const TcMod& md = st->mods[chunk[k]];
                    // G as K1's B operand (64 x 64 chunks), or as its A operand
                    // (128 rows x 64 columns) for a right projector
                    if (!encode_bf16_2d(st->encode, &p1.gmap[k], G[c0 + a + k], md.n, md.m, 64, md.right ? 128 : 64)) {
                        st->err = "cuTensorMapEncodeTiled failed for a gradient";
                        return MOARA_ERR_CUDA;
                    }
                }
            }
            p1.cta_start = tl->k1_start; p1.tiles = tl->k1;
            p1.mods = st->d_mods; p1.maps = st->d_maps; p1.status = st->d_status;
            p1.beta1 = hp.beta1; p1.beta2 = hp.beta2; p1.adam_eps = hp.adam_eps;
            p1.bc1 = bc1; p1.bc2 = bc2;
            p1.inv_bc1 = 1.0f / bc1; p1.inv_bc2 = 1.0f / bc2;
            p1.decompose = dec ? 1 : 0;
            p1.clip = dec ? nullptr : clip;
            K2Params p2{};
            p2.cta_start = tl->k2_start; p2.tiles = tl->k2;
            p2.mods = st->d_mods; p2.maps = st->d_maps; p2.status = st->d_status;
            p2.step_scale = lr * hp.scale;
            p2.decompose = hp.decompose;
            bool rt = false;
            for (int k = 0; k < b - a; ++k) rt = rt || st->mods[chunk[k]].right != 0;
            const bool sb = hp.state_dtype == MOARA_DTYPE_BF16;
            // The decomposition of part q + 1 starts when K1 of part q does:
            // K1 runs tensor-bound with HBM to spare, while K2, whose W
            // stream keeps HBM busy, loses most when it shares the memory
            // system.  (Also holding K2 back until the decomposition ends
            // left a gap after each K1 and was slower.)
            const bool bg = dec && q + 1 < np;
            if (bg && cudaEventRecord(st->ev_k1[q], s) != cudaSuccess) return fail("part event");
            cudaError_t e = launch_k12_any(B, sb, st, p1, p2, tl->g1, tl->g2, hilo, s, launches, prof, 1, rt);
            if (e != cudaSuccess) {
                st->err = cudaGetErrorString(e);
                return MOARA_ERR_CUDA;
            }
            if (bg) {
                if (cudaStreamWaitEvent(st->aux, st->ev_k1[q], 0) != cudaSuccess ||
                    launch_k0_any(B, st, *build_p0(pstart[q + 1], pstart[q + 2]), true, st->aux, launches, prof,
                                  !fused) != cudaSuccess ||
                    cudaEventRecord(st->ev_part[q + 1], st->aux) != cudaSuccess)
                    return fail("background decomposition launch failed");
            }
            if (!fused) {
                e = launch_k12_any(B, sb, st, p1, p2, tl->g1, tl->g2, hilo, s, launches, prof, 2, rt);
                if (e != cudaSuccess) {
                    st->err = cudaGetErrorString(e);
                    return MOARA_ERR_CUDA;
                }
            }
        }
        if (fused) {
            // total norm from every module's block norms, the coefficient,
            // Optimizer_M of the clipped magnitudes, then K2 over the group
            K0Params* pall = build_p0(0, cnt);
            pall->clip = fuse->state + 1;
            if (prof.on) prof.mark(prof.ctx, MOARA_PHASE_CLIP_NORM, s, true);
            k0_mag_sq<<<kNormParts, 256, 0, s>>>(*pall, fuse->partials);
            ++*launches;
            if (launch_clip_finish(fuse->partials, kNormParts, fuse->extra, fuse->max_norm, fuse->state, s,
                                   launches) != cudaSuccess)
                return fail("clipping coefficient launch failed");
            if (prof.on) prof.mark(prof.ctx, MOARA_PHASE_CLIP_NORM, s, false);
            if (prof.on) prof.mark(prof.ctx, MOARA_PHASE_TC_DECOMPOSE, s, true);
            k0_mag_adam<<<st->sms * 4, 256, 0, s>>>(*pall);
            ++*launches;
            if (prof.on) prof.mark(prof.ctx, MOARA_PHASE_TC_DECOMPOSE, s, false);
            std::vector<int> all(ids + c0, ids + c0 + cnt);
            TcState::Tiles* tl = tc_tiles(st, all);
            if (tl == nullptr) { st->err = "tile list allocation failed"; return MOARA_ERR_CUDA; }
            K2Params p2{};
            p2.cta_start = tl->k2_start; p2.tiles = tl->k2;
            p2.mods = st->d_mods; p2.maps = st->d_maps; p2.status = st->d_status;
            p2.step_scale = lr * hp.scale;
            p2.decompose = hp.decompose;
            const cudaError_t e = launch_k12_any(B, hp.state_dtype == MOARA_DTYPE_BF16, st, st->p1, p2, tl->g1, tl->g2,
                                                 hilo, s, launches, prof, 2);
            if (e != cudaSuccess) {
                st->err = cudaGetErrorString(e);
                return MOARA_ERR_CUDA;
            }
        }
    }
    return MOARA_OK;
}

const char* tc_last_error(const TcState* st) { return st ? st->err.c_str() : "no tensor-core state"; }

void tc_set_wait_limit(TcState* st, long long cycles) {
    if (st != nullptr) st->wait_limit = cycles > 0 ? cycles : kWaitLimit;
}

// Grouped KR launches; with align_B > 0 the alignment epilogue (A K-major
// with two planes only) replaces the stores.
static int kr_launch(TcState* st, int a_kmajor, const TcGemmItem* items, int count, int align_B,
                     const uint16_t* const* al_G, const float* const* al_mag, const int* al_ld, const int* al_kb,
                     const int* al_m, double* const* al_acc, cudaStream_t s, int64_t* launches,
                     const int* al_tr = nullptr) {
    if (!st->kr_attrs) {
        cudaFuncSetAttribute(kr_product<true, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, KR_SMEM);
        cudaFuncSetAttribute(kr_product<true, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, KR_SMEM);
        cudaFuncSetAttribute(kr_product<false, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, KR_SMEM);
        cudaFuncSetAttribute(kr_product<false, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, KR_SMEM);
        cudaFuncSetAttribute(kr_product<true, true, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, KR_SMEM);
        st->kr_attrs = true;
    }
    for (int i = 0; i < count; ++i) {
        const TcGemmItem& x = items[i];
        const int a_inner = a_kmajor ? x.K : x.M;
        if (x.M < 1 || x.N < 1 || x.K < 1 || (a_inner % 8) != 0 || (x.N % 8) != 0) {
            st->err = "tensor-core refresh GEMM: row pitches must be multiples of 16 bytes";
            return MOARA_ERR_UNSUPPORTED;
        }
        if (align_B > 0 && (!a_kmajor || x.A_lo == nullptr)) {
            st->err = "alignment product: A must be K-major with two planes";
            return MOARA_ERR_UNSUPPORTED;
        }
    }
    // two sub-launches: items with and without the A_lo plane
    for (int with_lo = 0; with_lo < 2; ++with_lo) {
        std::vector<int> sel;
        for (int i = 0; i < count; ++i)
            if ((items[i].A_lo != nullptr) == (with_lo == 1)) sel.push_back(i);
        for (size_t c0 = 0; c0 < sel.size(); c0 += kKrGroup) {
            const int cnt = static_cast<int>(std::min<size_t>(kKrGroup, sel.size() - c0));
            KrParams& kp = st->pr;
            std::memset(&kp, 0, sizeof(kp));
            int total = 0;
            for (int q = 0; q < cnt; ++q) {
                const int it = sel[c0 + q];
                const TcGemmItem& x = items[it];
                const uint64_t a_cols = a_kmajor ? x.K : x.M, a_rows = a_kmajor ? x.M : x.K;
                bool ok = encode_bf16_2d(st->encode, &kp.amap[q], x.A, a_cols, a_rows, 64, 64);
                if (with_lo) ok = ok && encode_bf16_2d(st->encode, &kp.lmap[q], x.A_lo, a_cols, a_rows, 64, 64);
                ok = ok && encode_bf16_2d(st->encode, &kp.bmap[q], x.B, x.N, x.K, 64, 64);
                if (!ok) {
                    st->err = "cuTensorMapEncodeTiled failed for a refresh operand";
                    return MOARA_ERR_CUDA;
                }
                kp.out[q] = x.out;
                kp.out_bf[q] = x.out_bf16;
                kp.out_lo[q] = x.out_lo;
                if (align_B > 0) {
                    kp.al_G[q] = al_G[it]; kp.al_mag[q] = al_mag[it]; kp.al_acc[q] = al_acc[it];
                    kp.al_ld[q] = al_ld[it]; kp.al_kb[q] = al_kb[it]; kp.al_m[q] = al_m[it];
                    kp.al_tr[q] = al_tr != nullptr ? al_tr[it] : 1;
                }
                kp.M[q] = x.M; kp.N[q] = x.N; kp.K[q] = x.K;
                kp.ktri[q] = x.ktri;
                kp.lower[q] = x.lower;
                kp.tiles_n[q] = (x.N + KR_BN - 1) / KR_BN;
                kp.tile_start[q] = total;
                total += ((x.M + KR_BM - 1) / KR_BM) * kp.tiles_n[q];
            }
            kp.tile_start[cnt] = total;
            kp.count = cnt;
            kp.status = st->d_status;
            kp.wait_limit = st->wait_limit;
            kp.al_B = align_B;
            kp.al_log2B = 0;
            while ((1 << kp.al_log2B) < align_B) ++kp.al_log2B;
            if (total == 0) continue;
            if (align_B > 0) {
                kr_product<true, true, true><<<total, KR_THREADS, KR_SMEM, s>>>(kp);
            } else if (!a_kmajor) {
                if (with_lo) kr_product<false, true><<<total, KR_THREADS, KR_SMEM, s>>>(kp);
                else kr_product<false, false><<<total, KR_THREADS, KR_SMEM, s>>>(kp);
            } else {
                if (with_lo) kr_product<true, true><<<total, KR_THREADS, KR_SMEM, s>>>(kp);
                else kr_product<true, false><<<total, KR_THREADS, KR_SMEM, s>>>(kp);
            }
            const cudaError_t e = cudaGetLastError();
            if (e != cudaSuccess) {
                st->err = cudaGetErrorString(e);
                return MOARA_ERR_CUDA;
            }
            ++*launches;
        }
    }
    return MOARA_OK;
}

int tc_gemm_bf16(TcState* st, int a_kmajor, const TcGemmItem* items, int count, cudaStream_t s,
                 int64_t* launches) {
    return kr_launch(st, a_kmajor, items, count, 0, nullptr, nullptr, nullptr, nullptr, nullptr, nullptr, s,
                     launches);
}

// out (cols x ld_out, bf16) = in^T for in (rows x cols, bf16, row pitch
// cols); columns rows..ld_out-1 of the output are zero.  32 x 32 tiles.
__global__ void __launch_bounds__(256) k_transpose_pad_bf16(const uint16_t* __restrict__ in, uint16_t* out,
                                                           int rows, int cols, int ld_out) {
    __shared__ uint16_t t[32][33];
    const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
    const int tr = (ld_out + 31) / 32, tc = (cols + 31) / 32;
    for (int tile = blockIdx.x; tile < tr * tc; tile += gridDim.x) {
        const int bi = tile / tc, bj = tile - bi * tc;      // input rows 32 bi.., columns 32 bj..
        for (int r = ty; r < 32; r += 8) {
            const int i = bi * 32 + r, j = bj * 32 + tx;
            t[r][tx] = (i < rows && j < cols) ? in[(long long)i * cols + j] : static_cast<uint16_t>(0);
        }
        __syncthreads();
        for (int r = ty; r < 32; r += 8) {
            const int j = bj * 32 + r, i = bi * 32 + tx;    // output row j, column i
            if (j < cols && i < ld_out) out[(long long)j * ld_out + i] = t[tx][r];
        }
        __syncthreads();
    }
}

cudaError_t tc_transpose_bf16(const uint16_t* in, uint16_t* out, int rows, int cols, cudaStream_t s,
                              int64_t* launches) {
    const int tiles = ((rows + 31) / 32) * ((cols + 31) / 32);
    k_transpose_pad_bf16<<<std::max(1, std::min(tiles, 152 * 8)), 256, 0, s>>>(in, out, rows, cols, rows);
    ++*launches;
    return cudaGetLastError();
}

__global__ void k_align_finish(const double* acc, float* S, int n) {
    const int q = blockIdx.x * blockDim.x + threadIdx.x;
    if (q >= n) return;
    const double dot = acc[3 * q], na = acc[3 * q + 1], gg = acc[3 * q + 2];
    const double den = sqrt(na) * sqrt(gg);
    S[q] = den > 0.0 ? static_cast<float>(dot / den) : 0.0f;
}

int tc_alignment(TcState* st, const moara_hparams& hp, int n_mod, const int* ids, const void* const* G,
                 float* S_out, double* acc, cudaStream_t s, int64_t* launches) {
    const int B = hp.block_size;
    if (!(B == 8 || B == 16 || B == 32 || B == 64 || B == 128)) {
        st->err = "alignment on tensor cores needs a block size in {8, 16, 32, 64, 128}";
        return MOARA_ERR_UNSUPPORTED;
    }
    for (int q = 0; q < n_mod; ++q) {
        const int id = ids[q];
        const TcMod* md = (id >= 0 && id < static_cast<int>(st->mods.size())) ? &st->mods[id] : nullptr;
        if (md == nullptr || md->Vhi == nullptr || md->Vlo == nullptr || md->Pb == nullptr) {
            st->err = "alignment: module is not on the tensor-core path";
            return MOARA_ERR_UNSUPPORTED;
        }
        const long long mp = (md->m + 7) / 8 * 8;
        if ((long long)md->r * mp > 2LL * md->m * md->n) {
            st->err = "alignment: workspace too small for the transposed projector";
            return MOARA_ERR_UNSUPPORTED;
        }
    }
    int rc = tc_upload(st);
    if (rc != MOARA_OK) return rc;
    // 1. block norms M (into the module's norm buffer) and V = V_hi + V_lo
    for (int c0 = 0; c0 < n_mod; c0 += kTcGroup) {
        const int cnt = std::min(kTcGroup, n_mod - c0);
        K0Params& p0 = st->p0;
        std::memset(&p0, 0, sizeof(p0));
        p0.count = cnt;
        p0.hilo = 1;
        p0.do_mag = 1;                   // writes the norms; Optimizer_M is not launched
        p0.decomp_eps = hp.decomp_eps;
        long long acc_items = 0;
        for (int q = 0; q < cnt; ++q) {
            const TcMod& md = st->mods[ids[c0 + q]];
            const int segs = (md.n + K0_SEG - 1) / K0_SEG;
            p0.start[q] = acc_items;
            p0.p[q] = K0Item{static_cast<const uint16_t*>(G[c0 + q]), md.Vhi, md.Vlo, md.mag, nullptr, nullptr,
                             nullptr, md.m, md.n, md.kb, segs};
            acc_items += static_cast<long long>(md.m) * segs;
        }
        p0.start[cnt] = acc_items;
        switch (B) {
            case 8: k0_decompose<8><<<st->sms * 3, 256, 0, s>>>(p0); break;
            case 16: k0_decompose<16><<<st->sms * 3, 256, 0, s>>>(p0); break;
            case 32: k0_decompose<32><<<st->sms * 3, 256, 0, s>>>(p0); break;
            case 64: k0_decompose<64><<<st->sms * 3, 256, 0, s>>>(p0); break;
            default: k0_decompose<128><<<st->sms * 3, 256, 0, s>>>(p0); break;
        }
        ++*launches;
        if (cudaGetLastError() != cudaSuccess) {
            st->err = "alignment decomposition launch failed";
            return MOARA_ERR_CUDA;
        }
    }
    // 2. left projector: R^T = V^T P (n x r); right projector: R = V Q
    //    (m x r); as two bf16 planes in the module's N buffer
    std::vector<TcGemmItem> g1[2];
    for (int q = 0; q < n_mod; ++q) {
        const TcMod& md = st->mods[ids[q]];
        if (!md.right)
            g1[0].push_back(TcGemmItem{md.Vhi, md.Vlo, md.Pb, nullptr, md.Nb, md.n, md.r, md.m, 0,
                                       md.Nb + (size_t)md.n * md.r});
        else
            g1[1].push_back(TcGemmItem{md.Vhi, md.Vlo, md.Pb, nullptr, md.Nb, md.m, md.r, md.n, 0,
                                       md.Nb + (size_t)md.m * md.r});
    }
    for (int side = 0; side < 2; ++side) {
        if (g1[side].empty()) continue;
        rc = kr_launch(st, side, g1[side].data(), static_cast<int>(g1[side].size()), 0, nullptr, nullptr, nullptr,
                       nullptr, nullptr, nullptr, s, launches);
        if (rc != MOARA_OK) return rc;
    }
    // 3. left projector: P^T (r x mp, zero-padded columns) over the V planes,
    //    now free (a right projector's Q^T is kept in the workspace)
    for (int q = 0; q < n_mod; ++q) {
        const TcMod& md = st->mods[ids[q]];
        if (md.right) continue;
        const int mp = (md.m + 7) / 8 * 8;
        const int tiles = ((mp + 31) / 32) * ((md.r + 31) / 32);
        k_transpose_pad_bf16<<<std::min(tiles, st->sms * 8), 256, 0, s>>>(md.Pb, md.Vhi, md.m, md.r, mp);
        ++*launches;
    }
    if (cudaMemsetAsync(acc, 0, sizeof(double) * 3 * (size_t)n_mod, s) != cudaSuccess) {
        st->err = "alignment accumulator reset failed";
        return MOARA_ERR_CUDA;
    }
    // 4. left: (P R)^T = R^T P^T (n x mp); right: V Q Q^T = R Q^T (m x n);
    //    reduced against G in the epilogue
    std::vector<TcGemmItem> g2(n_mod);
    std::vector<const uint16_t*> aG(n_mod);
    std::vector<const float*> aM(n_mod);
    std::vector<int> ald(n_mod), akb(n_mod), am(n_mod), atr(n_mod);
    std::vector<double*> aacc(n_mod);
    for (int q = 0; q < n_mod; ++q) {
        const TcMod& md = st->mods[ids[q]];
        if (!md.right) {
            const int mp = (md.m + 7) / 8 * 8;
            g2[q] = TcGemmItem{md.Nb, md.Nb + (size_t)md.n * md.r, md.Vhi, nullptr, nullptr, md.n, mp, md.r, 0, nullptr};
            am[q] = md.m;
            atr[q] = 1;
        } else {
            g2[q] = TcGemmItem{md.Nb, md.Nb + (size_t)md.m * md.r, md.Qt, nullptr, nullptr, md.m, md.n, md.r, 0, nullptr};
            am[q] = md.n;
            atr[q] = 0;
        }
        aG[q] = static_cast<const uint16_t*>(G[q]);
        aM[q] = md.mag;
        ald[q] = md.n; akb[q] = md.kb;
        aacc[q] = acc + 3 * q;
    }
    rc = kr_launch(st, 1, g2.data(), n_mod, B, aG.data(), aM.data(), ald.data(), akb.data(), am.data(),
                   aacc.data(), s, launches, atr.data());
    if (rc != MOARA_OK) return rc;
    k_align_finish<<<(n_mod + 127) / 128, 128, 0, s>>>(acc, S_out, n_mod);
    ++*launches;
    if (cudaGetLastError() != cudaSuccess) {
        st->err = "alignment finish launch failed";
        return MOARA_ERR_CUDA;
    }
    return MOARA_OK;
}

int tc_split_v(TcState* st, const TcSplitItem* items, int count, int B, float decomp_eps, cudaStream_t s,
               int64_t* launches) {
    for (int c0 = 0; c0 < count; c0 += kTcGroup) {
        const int cnt = std::min(kTcGroup, count - c0);
        K0Params& p0 = st->p0;
        std::memset(&p0, 0, sizeof(p0));
        p0.count = cnt;
        p0.hilo = 1;
        p0.do_mag = 0;
        p0.decomp_eps = decomp_eps;
        long long acc = 0;
        for (int q = 0; q < cnt; ++q) {
            const TcSplitItem& x = items[c0 + q];
            const int segs = (x.n + K0_SEG - 1) / K0_SEG;
            p0.start[q] = acc;
            p0.p[q] = K0Item{static_cast<const uint16_t*>(x.G), x.Vhi, x.Vlo, nullptr, nullptr, nullptr, nullptr,
                             x.m, x.n, (x.n + B - 1) / B, segs};
            acc += static_cast<long long>(x.m) * segs;
        }
        p0.start[cnt] = acc;
        switch (B) {
            case 8: k0_decompose<8><<<st->sms * 3, 256, 0, s>>>(p0); break;
            case 16: k0_decompose<16><<<st->sms * 3, 256, 0, s>>>(p0); break;
            case 32: k0_decompose<32><<<st->sms * 3, 256, 0, s>>>(p0); break;
            case 64: k0_decompose<64><<<st->sms * 3, 256, 0, s>>>(p0); break;
            case 128: k0_decompose<128><<<st->sms * 3, 256, 0, s>>>(p0); break;
            default: st->err = "block size not supported on the tensor-core path"; return MOARA_ERR_UNSUPPORTED;
        }
        const cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) {
            st->err = cudaGetErrorString(e);
            return MOARA_ERR_CUDA;
        }
        ++*launches;
    }
    return MOARA_OK;
}

int tc_gemm_split3(TcState* st, const TcSplitGemmItem* items, int count, int planes, cudaStream_t s,
                   int64_t* launches) {
    if (!st->ks_attrs) {
        cudaFuncSetAttribute(ks_product<3>, cudaFuncAttributeMaxDynamicSharedMemorySize, KS_SMEM);
        cudaFuncSetAttribute(ks_product<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, KS_SMEM);
        st->ks_attrs = true;
    }
    if (planes != 2 && planes != 3) {
        st->err = "split-precision GEMM: 2 or 3 planes";
        return MOARA_ERR_INVALID_ARG;
    }
    for (int i = 0; i < count; ++i) {
        const TcSplitGemmItem& x = items[i];
        if (x.M < 1 || x.N < 1 || x.K < 1 || (x.M % 8) != 0 || (x.N % 8) != 0) {
            st->err = "split-precision GEMM: M and N must be multiples of 8";
            return MOARA_ERR_UNSUPPORTED;
        }
        const int ldo = x.ldo > 0 ? x.ldo : x.N;
        if (ldo < x.N || (ldo % 4) != 0 || (reinterpret_cast<uintptr_t>(x.out) & 15) != 0) {
            st->err = "split-precision GEMM: out must be 16-byte aligned with a row pitch >= N, a multiple of 4";
            return MOARA_ERR_UNSUPPORTED;
        }
    }
    for (int c0 = 0; c0 < count; c0 += kKsGroup) {
        const int cnt = std::min(kKsGroup, count - c0);
        KsParams& kp = st->ps;
        std::memset(&kp, 0, sizeof(kp));
        int total = 0;
        for (int q = 0; q < cnt; ++q) {
            const TcSplitGemmItem& x = items[c0 + q];
            bool ok = true;
            for (int pl = 0; pl < 3; ++pl) {
                ok = ok && encode_bf16_2d(st->encode, &kp.amap[q][pl], x.A + (size_t)pl * x.a_plane, x.M, x.K, 64, 32);
                ok = ok && encode_bf16_2d(st->encode, &kp.bmap[q][pl], x.B + (size_t)pl * x.b_plane, x.N, x.K, 64, 32);
            }
            if (!ok) {
                st->err = "cuTensorMapEncodeTiled failed for a split-precision operand";
                return MOARA_ERR_CUDA;
            }
            kp.out[q] = x.out;
            kp.M[q] = x.M; kp.N[q] = x.N; kp.K[q] = x.K;
            kp.ktri[q] = x.ktri;
            kp.ldo[q] = x.ldo > 0 ? x.ldo : x.N;
            kp.sub[q] = x.sub;
            kp.lower[q] = x.lower;
            kp.tiles_n[q] = (x.N + KS_BN - 1) / KS_BN;
            kp.tile_start[q] = total;
            total += ((x.M + KS_BM - 1) / KS_BM) * kp.tiles_n[q];
        }
        kp.tile_start[cnt] = total;
        kp.count = cnt;
        kp.status = st->d_status;
        kp.wait_limit = st->wait_limit;
        if (total == 0) continue;
        if (planes == 3) ks_product<3><<<total, KR_THREADS, KS_SMEM, s>>>(kp);
        else ks_product<2><<<total, KR_THREADS, KS_SMEM, s>>>(kp);
        const cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) {
            st->err = cudaGetErrorString(e);
            return MOARA_ERR_CUDA;
        }
        ++*launches;
    }
    return MOARA_OK;
}

}  // namespace moara
