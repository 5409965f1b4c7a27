// bf16 tensor-core path of one TTL segment step (tcgen05 + TMEM + TMA, sm_103a).
//
// A segment step of the SiLU-MLP memory M(u) = SiLU(u W1^T) W2 (Eq. 3 form) on
// T tokens is four dense contractions (Eq. 10), done in two persistent kernels:
//
//   phase A, tile = (chain, 128 tokens, 128 hidden units), two TMEM accumulators
//       H = U W1^T            K = d_in      (memory forward)
//       R = Y W2^T            K = d_out     (Y = [K || V], the targets of Eq. 7)
//     fused epilogue: A = SiLU(H), dH = c_t R * SiLU'(H), At = c_t A with
//     c_t = -eta_t / T'.  Eq. 7's loss is linear in M, so dL/dO = -eta Y / T'
//     does not depend on W and the raw target tile is the right operand.
//     Writes dH and At row-major (bf16 [token][hidden]) and the loss partial
//     sum_t sum_h A_th R_th = sum_t y_t . M(u_t).
//
//   phase B, tile = (chain, 128 columns of [W1 | W2], 256 hidden units)
//       G1^T = U^T dH         K = T'        (gradient of W1, transposed)
//       G2^T = Y^T At         K = T'        (gradient of W2, transposed)
//     Both operands are read MN-major straight from the row-major buffers.
//     The accumulator is transposed (TMEM lane = weight column) so the fused
//     update epilogue (Eq. 8, App. A) walks the fp32 state row by row with
//     128-byte coalesced loads and stores: mu = beta mu + G; W = s W_raw - mu
//     (s = the previous segment's pending row renormalisation); it writes W,
//     mu, the bf16 operand copy and the new row sums of squares.
//
// Both kernels: one CTA per SM, persistent over a static tile schedule, 10 warps.
// Warp 0 lane 0 streams operand tiles with TMA into a shared-memory ring
// (128-byte swizzle), warp 1 lane 0 issues tcgen05.mma into one of two TMEM
// accumulator buffers, warps 2..9 drain the other buffer, so the epilogue of
// tile i overlaps the main loop of tile i+1.  Every mbarrier wait is bounded
// (kWaitLimitNs); a timeout latches DEV_TIMEOUT and the kernel winds down.
#include <mutex>

#include "mone_common.cuh"

namespace mone {

namespace {

constexpr int BK = 64;                    // 64 bf16 = one 128-byte swizzle row
constexpr int EPI_WARPS = 8;
constexpr int THREADS = 64 + EPI_WARPS * 32;
constexpr int EPI_THREADS = EPI_WARPS * 32;
constexpr uint32_t EPI_BAR = 1;           // named barrier among the epilogue warps

// phase A
constexpr int A_BM = 128, A_BN = 128, A_STAGES = 6;
constexpr int A_STAGE = (A_BM + A_BN) * BK * 2;           // 32 KB
// phase B
constexpr int B_BM = 128, B_BN = 256;
constexpr int B_STAGE = (B_BM + B_BN) * BK * 2;           // 48 KB
constexpr int BOX = 64 * BK * 2;                          // one 64 x 64 MN-major box, 8 KB

template <int STAGES, int STAGE, int TABLE>
struct Layout {
    static constexpr int RING = STAGES * STAGE;
    static constexpr int BARS = RING;                     // full[S], empty[S], tfull[2], tempty[2]
    static constexpr int SLOT = BARS + (2 * STAGES + 4) * 8;
    static constexpr int FLAG = SLOT + 16;
    static constexpr int TAB = FLAG + 16;
    static constexpr int END = TAB + TABLE * 4;
    static constexpr int DYN = END + 1024;                // + alignment slack
};
// phase A table: [2 parity][2 matrix][A_BN] scales; phase B: [2][B_BN] scales + [2][8] beta partials
using LA = Layout<A_STAGES, A_STAGE, 4 * A_BN>;
static_assert(LA::DYN <= 227 * 1024, "shared memory budget");

struct TcArgs {
    int d_in, d_out, d_hid, T, Tp, c0, nc, C, paper, momentum, renorm_pending, parity;
    int u_row0, u_chain0, y_row0;
    long long tok0;             // per-token tables: entry of token t of chain cs is [cs * win + tok0 + t]
    int win;
    float lr;
    const float* eta_in;        // plain-mode caller rates, offset to the segment start, or null
    long long eta_cstride;
    const float* eta;           // paper-mode rates [C][T]
    const float* dbeta;         // [C][T]
    const float* zinv;          // [C][T] 1/|z_t| (paper mode), or null
    const float* b_beta;        // [C]
    float *W1, *W2, *mu1, *mu2;
    bf16 *W1b, *W2b;
    const float *n1, *n2;
    float* sumsq;               // [2 parity][2 matrix][C][d_hid]
    bf16 *dH, *At;              // [C][T][d_hid]
    float* loss;                // [nc] or null
    float* step_sq;             // [nc] squared norm of this segment's Eq. 8 step (phase B), or null
    int* status;
    int r_only;                 // phase A pairs: At and c SiLU'(x) / |z| come from the squared-error
                                // pre-pass (the latter in dH); accumulate R only and form dH in place
    unsigned long long wait_ns; // limit of every mbarrier wait of the launch (kWaitLimitNs)
    int stall;                  // test knob (phase A): the producer issues no loads, so the first
                                // wait for a full stage runs out; nothing is in flight when it does
};

__device__ __forceinline__ float* ss_row(const TcArgs& a, int parity, int which, int cs) {
    return a.sumsq + ((size_t)(parity * 2 + which) * a.C + cs) * a.d_hid;
}

struct Ctl {
    uint8_t* base;
    uint32_t bars;
    __device__ uint32_t full(int s) const { return bars + 8 * s; }
    __device__ uint32_t empty(int s, int S) const { return bars + 8 * (S + s); }
    __device__ uint32_t tfull(int b, int S) const { return bars + 8 * (2 * S + b); }
    __device__ uint32_t tempty(int b, int S) const { return bars + 8 * (2 * S + 2 + b); }
};

template <class L, int STAGES>
__device__ __forceinline__ Ctl setup(uint8_t* raw) {
    Ctl c;
    c.base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(raw) + 1023) & ~uintptr_t(1023));
    c.bars = smem_u32(c.base + L::BARS);
    if (threadIdx.x == 0) {
        for (int i = 0; i < STAGES; ++i) {
            mbar_init(c.full(i), 1);
            mbar_init(c.empty(i, STAGES), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(c.tfull(b, STAGES), 1);
            mbar_init(c.tempty(b, STAGES), EPI_WARPS);
        }
        fence_mbar_init();
    }
    if (threadIdx.x / 32 == 0) {
        tmem_alloc(smem_u32(c.base + L::SLOT), 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    return c;
}


// ------------------------------------------------------------------ phase A

// Epilogue of one phase A tile (chain cs, token rows trow.., hidden columns h0..h0+BN)
// held in TMEM at `tmem` (H in columns [0, BN), R in [BN, 2 BN), one token per lane), run
// by the EPI_WARPS epilogue warps (warp = TMEM lane quarter x column half).  Builds the
// tile's renormalisation scales, zeroes the segment's row sums of squares when `zero_ss`,
// waits for the accumulators, then writes dH and At and adds the loss partial.
// `release` is called by every epilogue warp once its last TMEM read of the tile is
// done.  Returns false if the accumulator wait timed out.
template <int BN, class Release>
__device__ __forceinline__ bool phase_a_epilogue(const TcArgs& a, uint32_t tmem, uint32_t tfull_bar, int parity_bit,
                                                 float* tab, int* flag, int cz, int cs, int h0, int trow,
                                                 bool zero_ss, uint8_t* stg, Release&& release) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int e = warp - 2, q = warp & 3, ch = e >> 2, et = threadIdx.x - 64;
    static_assert(BN <= EPI_THREADS && BN % 64 == 0, "one scale per epilogue thread, 32-column chunks");
    // the tile's rows of dH / At lie inside the [C][T][d_hid] scratch (index check of MONE_DEBUG builds)
    const bool wr = MONE_DCHECK(cs < a.C && trow + 128 <= a.T && h0 + BN <= a.d_hid, a.status, DS_PHASE_A_TILE);
    if (et < BN) {
        const int h = h0 + et;
        float s1 = 1.f, s2 = 1.f;
        if (a.renorm_pending) {
            s1 = renorm_scale(a.n1[(size_t)cs * a.d_hid + h], ss_row(a, a.parity ^ 1, 0, cs)[h]);
            s2 = renorm_scale(a.n2[(size_t)cs * a.d_hid + h], ss_row(a, a.parity ^ 1, 1, cs)[h]);
        }
        tab[et] = s1;
        tab[BN + et] = s2;
        if (zero_ss) {
            ss_row(a, a.parity, 0, cs)[h] = 0.f;
            ss_row(a, a.parity, 1, cs)[h] = 0.f;
        }
    }
    if (et == 0) *flag = mbar_wait(tfull_bar, parity_bit, a.status, a.wait_ns) ? 1 : 0;
    __syncwarp();
    named_bar_sync(EPI_BAR, EPI_THREADS);
    if (!*flag) return false;
    tc_fence_after();
    const int row = q * 32 + lane;
    const int t = trow + row;
    float ct = 0.f, zi = 1.f;
    if (t < a.Tp) {
        const float ev = a.paper ? a.eta[(size_t)cs * a.win + a.tok0 + t]
                                 : (a.eta_in ? a.eta_in[cz * a.eta_cstride + t] : a.lr);
        ct = -ev / (float)a.Tp;
        if (a.zinv) zi = a.zinv[(size_t)cs * a.win + a.tok0 + t];
    }
    const float czi = ct * zi;
    const uint32_t lane_base = tmem + ((uint32_t)(q * 32) << 16);
    bf16* dHrow = a.dH + ((size_t)cs * a.T + t) * a.d_hid + h0;
    bf16* Arow = a.At + ((size_t)cs * a.T + t) * a.d_hid + h0;
    float lsum = 0.f;
    constexpr int CHUNKS = BN / 64;  // 32-column chunks per warp (each warp holds BN / 2 columns)
#pragma unroll 1
    for (int cc = 0; cc < CHUNKS; ++cc) {
        const int c0 = ch * (BN / 2) + cc * 32;
        float hv[32], rv[32];
        tmem_ld32(lane_base + c0, hv);
        tmem_ld32(lane_base + BN + c0, rv);
        if (cc == CHUNKS - 1) {
            tc_fence_before();
            __syncwarp();
            release();
        }
        uint32_t pd[16], pa[16];
#pragma unroll
        for (int j = 0; j < 32; j += 4) {
            const float4 s1v = *reinterpret_cast<const float4*>(tab + c0 + j);
            const float4 s2v = *reinterpret_cast<const float4*>(tab + BN + c0 + j);
            const float s1a[4] = {s1v.x, s1v.y, s1v.z, s1v.w};
            const float s2a[4] = {s2v.x, s2v.y, s2v.z, s2v.w};
            float dv[4], av4[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const float x = hv[j + u] * s1a[u] * zi;
                const float r = rv[j + u] * s2a[u];
                const float sg = sigmoid_tanh(x);
                const float av = x * sg;
                lsum = fmaf(av, r, lsum);
                dv[u] = czi * r * (sg * fmaf(x, 1.f - sg, 1.f));  // c_t (dL/dA) SiLU'(x), scaled by 1/|z_t|
                av4[u] = ct * av;
            }
            pd[j / 2] = pack_bf16(dv[0], dv[1]);
            pd[j / 2 + 1] = pack_bf16(dv[2], dv[3]);
            pa[j / 2] = pack_bf16(av4[0], av4[1]);
            pa[j / 2 + 1] = pack_bf16(av4[2], av4[3]);
        }
        if (!wr) {
        } else if (stg) {
            // rows trow + q*32 .. +31 of this warp, columns h0 + c0 .. +31
            const size_t r0 = ((size_t)cs * a.T + trow + q * 32) * a.d_hid + h0 + c0;
            store_rows_coalesced(stg, pd, a.dH + r0, a.d_hid, lane);
            store_rows_coalesced(stg, pa, a.At + r0, a.d_hid, lane);
        } else {
#pragma unroll
            for (int v = 0; v < 4; ++v) {
                *reinterpret_cast<uint4*>(dHrow + c0 + v * 8) =
                    make_uint4(pd[4 * v], pd[4 * v + 1], pd[4 * v + 2], pd[4 * v + 3]);
                *reinterpret_cast<uint4*>(Arow + c0 + v * 8) =
                    make_uint4(pa[4 * v], pa[4 * v + 1], pa[4 * v + 2], pa[4 * v + 3]);
            }
        }
    }
    if (a.loss) {
        lsum = warp_sum(lsum);
        if (lane == 0) atomicAdd(&a.loss[cz], -lsum / (float)a.Tp);
    }
    return true;
}

// The same epilogue split in two for a tile whose H accumulator (over d_in) completes before
// its R accumulator (over d_out), the order phase A issues them in.  At = c SiLU(x) needs only
// H, so once `hfull_bar` fires (H done, R still accumulating) the epilogue writes At and leaves
// s' = c (1/|z|) SiLU'(x) in H's TMEM columns; once `tfull_bar` fires it forms dH = R s2 s'.
// Only the second part runs after the main loop.  No loss partial (the caller uses
// phase_a_epilogue when a loss is requested).
template <int BN, class Release>
__device__ __forceinline__ bool phase_a_epilogue_split(const TcArgs& a, uint32_t tmem, uint32_t hfull_bar,
                                                       uint32_t tfull_bar, int parity_bit, float* tab, int* flag,
                                                       int cz, int cs, int h0, int trow, bool zero_ss, uint8_t* stg,
                                                       Release&& release) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int e = warp - 2, q = warp & 3, ch = e >> 2, et = threadIdx.x - 64;
    static_assert(BN <= EPI_THREADS && BN % 64 == 0, "one scale per epilogue thread, 32-column chunks");
    // the tile's rows of dH / At lie inside the [C][T][d_hid] scratch (index check of MONE_DEBUG builds)
    const bool wr = MONE_DCHECK(cs < a.C && trow + 128 <= a.T && h0 + BN <= a.d_hid, a.status, DS_PHASE_A_TILE);
    if (et < BN) {
        const int h = h0 + et;
        float s1 = 1.f, s2 = 1.f;
        if (a.renorm_pending) {
            s1 = renorm_scale(a.n1[(size_t)cs * a.d_hid + h], ss_row(a, a.parity ^ 1, 0, cs)[h]);
            s2 = renorm_scale(a.n2[(size_t)cs * a.d_hid + h], ss_row(a, a.parity ^ 1, 1, cs)[h]);
        }
        tab[et] = s1;
        tab[BN + et] = s2;
        if (zero_ss) {
            ss_row(a, a.parity, 0, cs)[h] = 0.f;
            ss_row(a, a.parity, 1, cs)[h] = 0.f;
        }
    }
    if (et == 0) *flag = mbar_wait(hfull_bar, parity_bit, a.status, a.wait_ns) ? 1 : 0;
    __syncwarp();
    named_bar_sync(EPI_BAR, EPI_THREADS);
    if (!*flag) return false;
    tc_fence_after();
    const int row = q * 32 + lane;
    const int t = trow + row;
    float ct = 0.f, zi = 1.f;
    if (t < a.Tp) {
        const float ev = a.paper ? a.eta[(size_t)cs * a.win + a.tok0 + t]
                                 : (a.eta_in ? a.eta_in[cz * a.eta_cstride + t] : a.lr);
        ct = -ev / (float)a.Tp;
        if (a.zinv) zi = a.zinv[(size_t)cs * a.win + a.tok0 + t];
    }
    const float czi = ct * zi;
    const uint32_t lane_base = tmem + ((uint32_t)(q * 32) << 16);
    const size_t r0 = ((size_t)cs * a.T + trow + q * 32) * a.d_hid + h0;  // this warp's first row
    constexpr int CHUNKS = BN / 64;  // 32-column chunks per warp (each warp holds BN / 2 columns)
    // ---- part 1, overlapping the R main loop: At, and s' into H's columns
#pragma unroll 1
    for (int cc = 0; cc < CHUNKS; ++cc) {
        const int c0 = ch * (BN / 2) + cc * 32;
        float hv[32];
        tmem_ld32(lane_base + c0, hv);
        uint32_t pa[16];
#pragma unroll
        for (int j = 0; j < 32; j += 4) {
            const float4 s1v = *reinterpret_cast<const float4*>(tab + c0 + j);
            const float s1a[4] = {s1v.x, s1v.y, s1v.z, s1v.w};
            float av4[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const float x = hv[j + u] * s1a[u] * zi;
                const float sg = sigmoid_tanh(x);
                av4[u] = ct * (x * sg);
                hv[j + u] = czi * (sg * fmaf(x, 1.f - sg, 1.f));  // c_t SiLU'(x), scaled by 1/|z_t|
            }
            pa[j / 2] = pack_bf16(av4[0], av4[1]);
            pa[j / 2 + 1] = pack_bf16(av4[2], av4[3]);
        }
        tmem_st32(lane_base + c0, hv);
        if (wr) store_rows_coalesced(stg, pa, a.At + r0 + c0, a.d_hid, lane);
    }
    tmem_wait_st();
    // ---- part 2, after the main loop: dH = R s2 s'
    if (et == 0) flag[2] = mbar_wait(tfull_bar, parity_bit, a.status, a.wait_ns) ? 1 : 0;
    __syncwarp();
    named_bar_sync(EPI_BAR, EPI_THREADS);
    if (!flag[2]) return false;
    tc_fence_after();
#pragma unroll 1
    for (int cc = 0; cc < CHUNKS; ++cc) {
        const int c0 = ch * (BN / 2) + cc * 32;
        float sp[32], rv[32];
        tmem_ld32(lane_base + c0, sp);
        tmem_ld32(lane_base + BN + c0, rv);
        if (cc == CHUNKS - 1) {
            tc_fence_before();
            __syncwarp();
            release();
        }
        uint32_t pd[16];
#pragma unroll
        for (int j = 0; j < 32; j += 4) {
            const float4 s2v = *reinterpret_cast<const float4*>(tab + BN + c0 + j);
            pd[j / 2] = pack_bf16(rv[j] * s2v.x * sp[j], rv[j + 1] * s2v.y * sp[j + 1]);
            pd[j / 2 + 1] = pack_bf16(rv[j + 2] * s2v.z * sp[j + 2], rv[j + 3] * s2v.w * sp[j + 3]);
        }
        if (wr) store_rows_coalesced(stg, pd, a.dH + r0 + c0, a.d_hid, lane);
    }
    return true;
}

// Epilogue of a phase A pair tile in the R-only form (squared-error loss): At and
// s' = c_t SiLU'(x) / |z_t| were written by the pre-pass (s' in dH), so dH = R s2 s' in place.
template <int BN, class Release>
__device__ __forceinline__ bool phase_a_epilogue_r_only(const TcArgs& a, uint32_t tmem, uint32_t tfull_bar,
                                                        int parity_bit, float* tab, int* flag, int cs, int h0,
                                                        int trow, bool zero_ss, uint8_t* stg, Release&& release) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int e = warp - 2, q = warp & 3, ch = e >> 2, et = threadIdx.x - 64;
    // the tile's rows of dH lie inside the [C][T][d_hid] scratch (index check of MONE_DEBUG builds)
    const bool wr = MONE_DCHECK(cs < a.C && trow + 128 <= a.T && h0 + BN <= a.d_hid, a.status, DS_PHASE_A_TILE);
    if (et < BN) {
        const int h = h0 + et;
        float s2 = 1.f;
        if (a.renorm_pending)
            s2 = renorm_scale(a.n2[(size_t)cs * a.d_hid + h], ss_row(a, a.parity ^ 1, 1, cs)[h]);
        tab[BN + et] = s2;
        if (zero_ss) {
            ss_row(a, a.parity, 0, cs)[h] = 0.f;
            ss_row(a, a.parity, 1, cs)[h] = 0.f;
        }
    }
    if (et == 0) *flag = mbar_wait(tfull_bar, parity_bit, a.status, a.wait_ns) ? 1 : 0;
    __syncwarp();
    named_bar_sync(EPI_BAR, EPI_THREADS);
    if (!*flag) return false;
    tc_fence_after();
    const int row = q * 32 + lane;
    const uint32_t lane_base = tmem + ((uint32_t)(q * 32) << 16);
    const size_t r0 = ((size_t)cs * a.T + trow + q * 32) * a.d_hid + h0;  // this warp's first row
    const bf16* sp_row = a.dH + ((size_t)cs * a.T + trow + row) * a.d_hid + h0;
    constexpr int CHUNKS = BN / 64;
#pragma unroll 1
    for (int cc = 0; cc < CHUNKS; ++cc) {
        const int c0 = ch * (BN / 2) + cc * 32;
        float rv[32];
        tmem_ld32(lane_base + BN + c0, rv);
        if (cc == CHUNKS - 1) {
            tc_fence_before();
            __syncwarp();
            release();
        }
        uint4 sv[4];
#pragma unroll
        for (int v = 0; v < 4; ++v) sv[v] = *reinterpret_cast<const uint4*>(sp_row + c0 + v * 8);
        uint32_t pd[16];
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            const __nv_bfloat162* sb = reinterpret_cast<const __nv_bfloat162*>(&sv[v]);
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const float2 sf = __bfloat1622float2(sb[u]);
                const int j = v * 8 + 2 * u;
                pd[j / 2] = pack_bf16(rv[j] * tab[BN + c0 + j] * sf.x, rv[j + 1] * tab[BN + c0 + j + 1] * sf.y);
            }
        }
        if (wr) store_rows_coalesced(stg, pd, a.dH + r0 + c0, a.d_hid, lane);  // in place: every lane has read its row
    }
    return true;
}

__global__ void __launch_bounds__(THREADS, 1)
tc_phase_a_kernel(const __grid_constant__ CUtensorMap tmU, const __grid_constant__ CUtensorMap tmK,
                  const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmW1,
                  const __grid_constant__ CUtensorMap tmW2, const TcArgs a) {
    extern __shared__ uint8_t smem_raw[];
    const Ctl c = setup<LA, A_STAGES>(smem_raw);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t tmem = *reinterpret_cast<uint32_t*>(c.base + LA::SLOT);
    const int n_tt = a.T / A_BM, n_ht = a.d_hid / A_BN;
    const int ntiles = a.nc * n_ht * n_tt;
    const int KB1 = a.d_in / BK, KB = KB1 + a.d_out / BK, half = (a.d_out / 2) / BK;

    if (warp == 0) {
        if (lane == 0) {
            tma_prefetch_map(&tmU);
            tma_prefetch_map(&tmK);
            tma_prefetch_map(&tmV);
            tma_prefetch_map(&tmW1);
            tma_prefetch_map(&tmW2);
            const uint64_t wpol = l2_evict_last_policy();  // the bf16 W copy phase B wrote
            uint32_t kc = 0;
            bool ok = true;
            for (int tile = blockIdx.x; tile < ntiles && ok && !a.stall; tile += gridDim.x) {
                const int cz = tile / (n_ht * n_tt), ht = (tile / n_tt) % n_ht, tt = tile % n_tt;
                const int cs = a.c0 + cz, h0 = ht * A_BN, trow = tt * A_BM;
                for (int kb = 0; kb < KB; ++kb, ++kc) {
                    const int s = kc % A_STAGES;
                    if (kc >= A_STAGES && !mbar_wait(c.empty(s, A_STAGES), ((kc / A_STAGES) - 1) & 1, a.status, a.wait_ns)) {
                        ok = false;
                        break;
                    }
                    const uint32_t sa = smem_u32(c.base + s * A_STAGE), sb = sa + A_BM * BK * 2, fb = c.full(s);
                    mbar_expect_tx(fb, A_STAGE);
                    if (kb < KB1) {
                        tma_load_3d(sa, &tmU, fb, kb * BK, a.u_row0 + trow, a.u_chain0 + cz);
                        tma_load_3d_hint(sb, &tmW1, fb, kb * BK, h0, cs, wpol);
                    } else {
                        const int k2 = kb - KB1;
                        if (k2 < half)
                            tma_load_3d(sa, &tmK, fb, k2 * BK, a.y_row0 + trow, cz);
                        else
                            tma_load_3d(sa, &tmV, fb, (k2 - half) * BK, a.y_row0 + trow, cz);
                        tma_load_3d_hint(sb, &tmW2, fb, k2 * BK, h0, cs, wpol);
                    }
                }
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16_f32(A_BM, A_BN, false, false);
            uint32_t kc = 0;
            int local = 0;
            bool ok = true;
            for (int tile = blockIdx.x; tile < ntiles && ok; tile += gridDim.x, ++local) {
                const int b = local & 1;
                if (local >= 2 && !mbar_wait(c.tempty(b, A_STAGES), ((local >> 1) - 1) & 1, a.status, a.wait_ns)) break;
                tc_fence_after();
                const uint32_t dH = tmem + b * 256, dR = dH + A_BN;
                for (int kb = 0; kb < KB; ++kb, ++kc) {
                    const int s = kc % A_STAGES;
                    if (!mbar_wait(c.full(s), (kc / A_STAGES) & 1, a.status, a.wait_ns)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t sa = smem_u32(c.base + s * A_STAGE), sb = sa + A_BM * BK * 2;
                    const bool first = (kb == 0 || kb == KB1);
#pragma unroll
                    for (int k = 0; k < BK / 16; ++k)
                        umma_bf16(kb < KB1 ? dH : dR, sdesc_sw128(sa + k * 32, 16), sdesc_sw128(sb + k * 32, 16),
                                  idesc, (first && k == 0) ? 0u : 1u);
                    umma_commit(c.empty(s, A_STAGES));
                }
                umma_commit(c.tfull(b, A_STAGES));
            }
        }
        __syncwarp();
    } else {
        float* table = reinterpret_cast<float*>(c.base + LA::TAB);
        int* flag = reinterpret_cast<int*>(c.base + LA::FLAG);
        int local = 0;
        for (int tile = blockIdx.x; tile < ntiles; tile += gridDim.x, ++local) {
            const int cz = tile / (n_ht * n_tt), ht = (tile / n_tt) % n_ht, tt = tile % n_tt;
            const int b = local & 1;
            const uint32_t tempty = c.tempty(b, A_STAGES);
            if (!phase_a_epilogue<A_BN>(a, tmem + b * 256, c.tfull(b, A_STAGES), (local >> 1) & 1, table + b * 2 * A_BN,
                                  flag + b, cz, a.c0 + cz, ht * A_BN, tt * A_BM, tt == 0, nullptr, [&] {
                                      if (lane == 0) mbar_arrive(tempty);
                                  }))
                break;
        }
    }
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, 512);
}

// ------------------------------------------------------------------ phase A on CTA pairs
//
// The same tile step on a cluster of two CTAs that share each tcgen05.mma
// (cta_group::2): M = 256 tokens, 128 in each CTA, x N = 256 hidden units, whose W
// rows are split between the pair (128 rows staged in each CTA).  Each CTA's TMEM
// holds the H and R rows of its own tokens (256 + 256 columns: one accumulator
// buffer).  A TMA tensor load costs the SM about the same whether its box has 64 or
// 128 rows, and phase A is bounded by those loads: here an SM issues two 128-row
// boxes per 64-deep k-block for a 128 x 256 accumulator, twice the work per load of
// the one-CTA kernel's 128 x 128 tile.  Rank 0 of the pair issues the MMAs: both
// CTAs' loads complete on rank 0's full barrier (a relay, with each CTA's loads on
// its own barrier and one remote arrive per stage, measured 1.7x slower), each MMA
// commit arrives on the empty and accumulator-full barriers of both CTAs, and all 16
// epilogue warps of the pair release the accumulator on rank 0's tempty barrier.  The
// epilogue stores dH and At through per-warp transpose buffers (coalesced rows).
constexpr int P_BN = 256;
constexpr int P_STAGES = 6;
constexpr int P_A = A_BM * BK * 2;                  // 16 KB: this CTA's 128 token rows
constexpr int P_STAGE = P_A + (P_BN / 2) * BK * 2;  // + 16 KB: this CTA's 128 W rows
struct LP {
    static constexpr int RING = P_STAGES * P_STAGE;
    static constexpr int BARS = RING;  // full[S] empty[S] tfull[2] tempty[2]
    static constexpr int NBARS = 2 * P_STAGES + 4;
    static constexpr int SLOT = BARS + NBARS * 8;
    static constexpr int FLAG = SLOT + 16;              // 2 tiles x 4 flags
    static constexpr int TAB = FLAG + 32;               // scale tables of two consecutive tiles
    static constexpr int STG = TAB + 4 * P_BN * 4;      // per epilogue warp: 32 x 64 B transpose buffer
    static constexpr int END = STG + EPI_WARPS * 2048;
    static constexpr int DYN = END + 1024;
};
static_assert(LP::DYN <= 227 * 1024, "shared memory budget");
static_assert(LP::STG % 16 == 0, "staging buffers hold 16-byte pieces");

// Spin for about `ns` nanoseconds (abort path: lets copies already issued land first).
__device__ __forceinline__ void pause_ns(uint64_t ns) {
    const uint64_t t0 = globaltimer_ns();
    while (globaltimer_ns() - t0 < ns) __nanosleep(1000);
}

__global__ void __launch_bounds__(THREADS, 1)
tc_phase_a_pair_kernel(const __grid_constant__ CUtensorMap tmU, const __grid_constant__ CUtensorMap tmK,
                       const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmW1,
                       const __grid_constant__ CUtensorMap tmW2, const TcArgs a) {
    extern __shared__ uint8_t smem_raw[];
    Ctl c;
    c.base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    c.bars = smem_u32(c.base + LP::BARS);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();
    if (threadIdx.x == 0) {
        for (int i = 0; i < P_STAGES; ++i) {
            mbar_init(c.full(i), 1);
            mbar_init(c.empty(i, P_STAGES), 1);
        }
        mbar_init(c.tfull(0, P_STAGES), 1);
        mbar_init(c.tfull(1, P_STAGES), 1);  // H accumulator complete (R still accumulating)
        mbar_init(c.tempty(0, P_STAGES), 2 * EPI_WARPS);
        fence_mbar_init();
    }
    if (warp == 0) {
        tmem_alloc_pair(smem_u32(c.base + LP::SLOT), 512);
        tmem_relinquish_pair();
    }
    tc_fence_before();
    cluster_sync();  // barriers of both CTAs initialised, TMEM of the pair allocated
    tc_fence_after();
    const uint32_t tmem = *reinterpret_cast<uint32_t*>(c.base + LP::SLOT);
    const int n_tp = a.T / (2 * A_BM), n_ht = a.d_hid / P_BN;
    const int npairs = a.nc * n_ht * n_tp;
    const int cluster = blockIdx.x >> 1, nclusters = gridDim.x >> 1;
    // the R-only form (squared-error loss) takes no H k-blocks
    const int KB1 = a.r_only ? 0 : a.d_in / BK, KB = KB1 + a.d_out / BK, half = (a.d_out / 2) / BK;

    if (warp == 0) {
        if (lane == 0) {
            tma_prefetch_map(&tmU);
            tma_prefetch_map(&tmK);
            tma_prefetch_map(&tmV);
            tma_prefetch_map(&tmW1);
            tma_prefetch_map(&tmW2);
            const uint64_t wpol = l2_evict_last_policy();  // the bf16 W copy phase B wrote
            uint32_t kc = 0;
            bool ok = true;
            for (int pt = cluster; pt < npairs && ok && !a.stall; pt += nclusters) {
                const int cz = pt / (n_ht * n_tp), ht = (pt / n_tp) % n_ht, tp = pt % n_tp;
                const int cs = a.c0 + cz, hrow = ht * P_BN + (int)rank * (P_BN / 2);
                const int trow = tp * 2 * A_BM + (int)rank * A_BM;
                for (int kb = 0; kb < KB; ++kb, ++kc) {
                    const int s = kc % P_STAGES;
                    if (kc >= P_STAGES && !mbar_wait(c.empty(s, P_STAGES), ((kc / P_STAGES) - 1) & 1, a.status, a.wait_ns)) {
                        ok = false;
                        break;
                    }
                    // both CTAs' loads complete on rank 0's full barrier
                    const uint32_t sa = smem_u32(c.base + s * P_STAGE), sb = sa + P_A;
                    const uint32_t fb = map_to_cta(c.full(s), 0);
                    if (rank == 0) mbar_expect_tx(c.full(s), 2 * P_STAGE);
                    if (kb < KB1) {
                        tma_load_3d_pair(sa, &tmU, fb, kb * BK, a.u_row0 + trow, a.u_chain0 + cz);
                        tma_load_3d_pair_hint(sb, &tmW1, fb, kb * BK, hrow, cs, wpol);
                    } else {
                        const int k2 = kb - KB1;
                        if (k2 < half)
                            tma_load_3d_pair(sa, &tmK, fb, k2 * BK, a.y_row0 + trow, cz);
                        else
                            tma_load_3d_pair(sa, &tmV, fb, (k2 - half) * BK, a.y_row0 + trow, cz);
                        tma_load_3d_pair_hint(sb, &tmW2, fb, k2 * BK, hrow, cs, wpol);
                    }
                }
            }
            if (!ok) pause_ns(200000);
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0 && rank == 0) {
            const uint32_t idesc = idesc_bf16_f32(2 * A_BM, P_BN, false, false);
            uint32_t kc = 0;
            int local = 0;
            bool ok = true;
            for (int pt = cluster; pt < npairs && ok; pt += nclusters, ++local) {
                // one accumulator buffer: wait until both CTAs' epilogues have read the last tile
                if (local >= 1 && !mbar_wait(c.tempty(0, P_STAGES), (local - 1) & 1, a.status, a.wait_ns)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t dH = tmem, dR = tmem + P_BN;
                for (int kb = 0; kb < KB; ++kb, ++kc) {
                    const int s = kc % P_STAGES;
                    if (!mbar_wait(c.full(s), (kc / P_STAGES) & 1, a.status, a.wait_ns)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t sa = smem_u32(c.base + s * P_STAGE), sb = sa + P_A;
                    const bool first = (kb == 0 || kb == KB1);
#pragma unroll
                    for (int k = 0; k < BK / 16; ++k)
                        umma_bf16_pair(kb < KB1 ? dH : dR, sdesc_sw128(sa + k * 32, 16),
                                       sdesc_sw128(sb + k * 32, 16), idesc, (first && k == 0) ? 0u : 1u);
                    umma_commit_pair(c.empty(s, P_STAGES), 0x3);
                    if (kb == KB1 - 1) umma_commit_pair(c.tfull(1, P_STAGES), 0x3);  // H complete
                }
                if (!ok) break;
                umma_commit_pair(c.tfull(0, P_STAGES), 0x3);
            }
            if (!ok) pause_ns(200000);
        }
        __syncwarp();
    } else {
        float* table = reinterpret_cast<float*>(c.base + LP::TAB);
        int* flag = reinterpret_cast<int*>(c.base + LP::FLAG);
        const uint32_t tempty0 = map_to_cta(c.tempty(0, P_STAGES), 0);
        int local = 0;
        for (int pt = cluster; pt < npairs; pt += nclusters, ++local) {
            const int cz = pt / (n_ht * n_tp), ht = (pt / n_tp) % n_ht, tp = pt % n_tp;
            const int tt = tp * 2 + (int)rank;
            // the scale table and flag alternate between tiles: a warp may start the next
            // tile while another still reads this one's table
            auto release = [&] {
                if (lane == 0) mbar_arrive_remote(tempty0);
            };
            float* tab = table + (local & 1) * 2 * P_BN;
            int* fl = flag + (local & 1) * 4;
            uint8_t* stg = c.base + LP::STG + (warp - 2) * 2048;
            const bool ok =
                a.r_only ? phase_a_epilogue_r_only<P_BN>(a, tmem, c.tfull(0, P_STAGES), local & 1, tab, fl, a.c0 + cz,
                                                         ht * P_BN, tt * A_BM, tt == 0, stg, release)
                : a.loss ? phase_a_epilogue<P_BN>(a, tmem, c.tfull(0, P_STAGES), local & 1, tab, fl, cz, a.c0 + cz,
                                                  ht * P_BN, tt * A_BM, tt == 0, stg, release)
                         : phase_a_epilogue_split<P_BN>(a, tmem, c.tfull(1, P_STAGES), c.tfull(0, P_STAGES), local & 1,
                                                        tab, fl, cz, a.c0 + cz, ht * P_BN, tt * A_BM, tt == 0, stg,
                                                        release);
            if (!ok) break;
        }
    }
    tc_fence_before();
    cluster_sync();  // every MMA of the pair has completed and every TMEM read is done
    tc_fence_after();
    if (warp == 0) tmem_dealloc_pair(tmem, 512);
}

// ------------------------------------------------------------------ phase B
//
// Warps: 0 operand producer (TMA), 1 MMA issuer, 2..9 epilogue in two groups of
// four (one warp per TMEM lane quarter; thread = one weight column), 10 state
// producer.  The fp32 state of a tile (256 rows x 128 columns of W and mu) moves
// in chunks of 32 rows through a 4-slot shared-memory ring: the state producer
// TMA-loads chunks ahead of time; the two epilogue groups take alternate chunks,
// update a chunk in place and TMA-store it back (the bf16 copy goes out with
// coalesced 64-byte warp stores), and hand the slot back once the store has read it.
//
// PAIR: clusters of 2 CTAs run tcgen05.mma.cta_group::2 over 256 weight columns x 256
// hidden rows.  CTA r stages its own 128 columns of U (or Y) and rows r*128 .. +127 of the
// tile's 256 rows of dH (or At) per 64-token k-block, so each SM takes in 32 KB of operands
// a k-block instead of 48 KB for the same 128 x 256 accumulator.  Both CTAs' loads complete
// on rank 0's full barrier, rank 0 issues the MMAs, each commit arrives on both CTAs'
// barriers, and the 16 epilogue warps of the pair release an accumulator buffer on rank 0's
// tempty barrier.  Each CTA updates the state of its own 128 columns exactly as the one-CTA
// kernel does.  A pair's 256 columns lie in one matrix (d_in and d_out multiples of 256).

constexpr int S_ROWS = 32;                                 // hidden rows per state chunk
constexpr int S_SLOTS = 4;
constexpr int S_F32 = S_ROWS * B_BM * 4;                   // 16 KB
constexpr int S_SLOT = 2 * S_F32;                          // W and mu: 32 KB
constexpr int B_THREADS = 12 * 32;
constexpr int B_EPI_THREADS = 4 * 32;     // per epilogue group
constexpr int B_STATE_WARP = 10;          // TMA loads of state chunks
constexpr int B_STORE_WARP = 11;          // TMA stores of updated chunks, slot release

template <bool PAIR>
struct LayoutBT {
    // operand stages: one CTA 48 KB (128 columns + 256 hidden rows); a pair member 32 KB
    // (128 columns + its 128 hidden rows), three of them in the same space as two
    static constexpr int STAGE = PAIR ? (B_BM + B_BN / 2) * BK * 2 : B_STAGE;
    static constexpr int STAGES = PAIR ? 3 : 2;
    static constexpr int RING = STAGES * STAGE;
    static constexpr int STATE = RING;
    static constexpr int BARS = STATE + S_SLOTS * S_SLOT;  // full[S] empty[S] tfull[2] tempty[2] sfull/sdone/sempty[N]
    static constexpr int NBARS = 2 * STAGES + 4 + 3 * S_SLOTS;
    static constexpr int SLOT = BARS + NBARS * 8;
    static constexpr int FLAG = SLOT + 16;
    static constexpr int TAB = FLAG + 16;                  // per group: [B_BN/2] renorm scales + [4] decay partials
    static constexpr int END = TAB + 2 * (B_BN / 2 + 4) * 4;
    static constexpr int DYN = END + 1024;
};
using LayoutB = LayoutBT<false>;
using LayoutB2 = LayoutBT<true>;
static_assert(LayoutB::DYN <= 227 * 1024 && LayoutB2::DYN <= 227 * 1024, "phase B shared memory budget");

// The tiles one CTA of phase B walks: t = first, first + step, ... < count, each giving
// (chain of the launch, first hidden row, first weight column of this CTA).
template <bool PAIR>
struct BTiles {
    int first, step, count, n_ht, n_ct, rank;
    __device__ BTiles(const TcArgs& a) {
        n_ht = a.d_hid / B_BN;
        n_ct = (a.d_in + a.d_out) / (PAIR ? 2 * B_BM : B_BM);
        count = a.nc * n_ht * n_ct;
        rank = PAIR ? (int)cluster_ctarank() : 0;
        first = PAIR ? (int)(blockIdx.x >> 1) : (int)blockIdx.x;
        step = PAIR ? (int)(gridDim.x >> 1) : (int)gridDim.x;
    }
    __device__ void decode(int t, int& cz, int& h0, int& col0) const {
        cz = t / (n_ht * n_ct);
        h0 = ((t / n_ct) % n_ht) * B_BN;
        col0 = (t % n_ct) * (PAIR ? 2 * B_BM : B_BM) + rank * B_BM;
    }
};

// STEP: also sum |mu_s|^2 per chain (the per-segment metrics); a separate instance, so the update
// loop of the ordinary one keeps its registers
template <bool PAIR, bool STEP>
__global__ void __launch_bounds__(B_THREADS, 1)
tc_phase_b_kernel(const __grid_constant__ CUtensorMap tmUb, const __grid_constant__ CUtensorMap tmKb,
                  const __grid_constant__ CUtensorMap tmVb, const __grid_constant__ CUtensorMap tmDH,
                  const __grid_constant__ CUtensorMap tmAT, const __grid_constant__ CUtensorMap tmW1s,
                  const __grid_constant__ CUtensorMap tmW2s, const __grid_constant__ CUtensorMap tmM1s,
                  const __grid_constant__ CUtensorMap tmM2s, const TcArgs a) {
    extern __shared__ uint8_t smem_raw[];
    using L = LayoutBT<PAIR>;
    constexpr int NS = L::STAGES;
    uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const uint32_t bars = smem_u32(base + L::BARS);
    auto full = [&](int s) { return bars + 8 * s; };
    auto empty = [&](int s) { return bars + 8 * (NS + s); };
    auto tfull = [&](int b) { return bars + 8 * (2 * NS + b); };
    auto tempty = [&](int b) { return bars + 8 * (2 * NS + 2 + b); };
    auto sfull = [&](int k) { return bars + 8 * (2 * NS + 4 + k); };
    auto sempty = [&](int k) { return bars + 8 * (2 * NS + 4 + S_SLOTS + k); };
    auto sdone = [&](int k) { return bars + 8 * (2 * NS + 4 + 2 * S_SLOTS + k); };
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const BTiles<PAIR> tl(a);
    if (threadIdx.x == 0) {
        for (int i = 0; i < NS; ++i) {
            mbar_init(full(i), 1);
            mbar_init(empty(i), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(tfull(b), 1);
            mbar_init(tempty(b), PAIR ? 16 : 8);  // every epilogue warp (of both CTAs of a pair)
        }
        for (int k = 0; k < S_SLOTS; ++k) {
            mbar_init(sfull(k), 1);
            mbar_init(sempty(k), 1);
            mbar_init(sdone(k), 4);  // the four warps of the epilogue group that updated the chunk
        }
        fence_mbar_init();
    }
    if (warp == 0) {
        if constexpr (PAIR) {
            tmem_alloc_pair(smem_u32(base + L::SLOT), 512);
            tmem_relinquish_pair();
        } else {
            tmem_alloc(smem_u32(base + L::SLOT), 512);
            tmem_relinquish();
        }
    }
    tc_fence_before();
    if constexpr (PAIR)
        cluster_sync();  // barriers of both CTAs initialised, TMEM of the pair allocated
    else
        __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *reinterpret_cast<uint32_t*>(base + L::SLOT);

    const int KB = (a.Tp + BK - 1) / BK;  // tokens beyond T' carry zero dH / At
    const int dhalf = a.d_out / 2;
    const int chunk_bytes = a.momentum ? 2 * S_F32 : S_F32;

    if (warp == 0) {
        if (lane == 0) {
            tma_prefetch_map(&tmUb);
            tma_prefetch_map(&tmKb);
            tma_prefetch_map(&tmVb);
            tma_prefetch_map(&tmDH);
            tma_prefetch_map(&tmAT);
            uint32_t kc = 0;
            bool ok = true;
            for (int t = tl.first; t < tl.count && ok; t += tl.step) {
                int cz, h0, col0;
                tl.decode(t, cz, h0, col0);
                const int cs = a.c0 + cz;
                const bool isW1 = col0 < a.d_in;
                // this CTA's share of the tile's hidden rows: all 256, or 128 of a pair
                const int hrow = h0 + (PAIR ? tl.rank * (B_BN / 2) : 0);
                constexpr int HB = (PAIR ? B_BN / 2 : B_BN) / 64;  // 64-row boxes of hidden rows
                for (int kb = 0; kb < KB; ++kb, ++kc) {
                    const int s = kc % NS;
                    if (kc >= NS && !mbar_wait(empty(s), ((kc / NS) - 1) & 1, a.status, a.wait_ns)) {
                        ok = false;
                        break;
                    }
                    const uint32_t sa = smem_u32(base + s * L::STAGE), sb = sa + B_BM * BK * 2;
                    uint32_t fb = full(s);
                    if constexpr (PAIR) {
                        fb = map_to_cta(full(s), 0);  // both CTAs' loads complete on rank 0's barrier
                        if (tl.rank == 0) mbar_expect_tx(full(s), 2 * L::STAGE);
                    } else {
                        mbar_expect_tx(fb, L::STAGE);
                    }
#pragma unroll
                    for (int bx = 0; bx < B_BM / 64; ++bx) {
                        const uint32_t dst = sa + bx * BOX;
                        const CUtensorMap* map;
                        int x, y, z;
                        if (isW1) {
                            map = &tmUb;
                            x = col0 + bx * 64;
                            y = a.u_row0 + kb * BK;
                            z = a.u_chain0 + cz;
                        } else {
                            const int o = col0 - a.d_in + bx * 64;
                            map = o < dhalf ? &tmKb : &tmVb;
                            x = o < dhalf ? o : o - dhalf;
                            y = a.y_row0 + kb * BK;
                            z = cz;
                        }
                        // a tiled copy's innermost coordinate must be 16-byte aligned (8 bf16)
                        if (!MONE_DCHECK((x & 7) == 0, a.status, DS_TMA_X)) continue;
                        if constexpr (PAIR)
                            tma_load_3d_pair(dst, map, fb, x, y, z);
                        else
                            tma_load_3d(dst, map, fb, x, y, z);
                    }
#pragma unroll
                    for (int bx = 0; bx < HB; ++bx) {
                        if constexpr (PAIR)
                            tma_load_3d_pair(sb + bx * BOX, isW1 ? &tmDH : &tmAT, fb, hrow + bx * 64, kb * BK, cs);
                        else
                            tma_load_3d(sb + bx * BOX, isW1 ? &tmDH : &tmAT, fb, hrow + bx * 64, kb * BK, cs);
                    }
                }
            }
            if (PAIR && !ok) pause_ns(200000);
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0 && (!PAIR || tl.rank == 0)) {
            const uint32_t idesc = idesc_bf16_f32(PAIR ? 2 * B_BM : B_BM, B_BN, true, true);
            uint32_t kc = 0;
            int local = 0;
            bool ok = true;
            for (int t = tl.first; t < tl.count && ok; t += tl.step, ++local) {
                const int b = local & 1;
                if (local >= 2 && !mbar_wait(tempty(b), ((local >> 1) - 1) & 1, a.status, a.wait_ns)) break;
                tc_fence_after();
                const uint32_t d = tmem + b * 256;
                for (int kb = 0; kb < KB; ++kb, ++kc) {
                    const int s = kc % NS;
                    if (!mbar_wait(full(s), (kc / NS) & 1, a.status, a.wait_ns)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t sa = smem_u32(base + s * L::STAGE), sb = sa + B_BM * BK * 2;
#pragma unroll
                    for (int k = 0; k < BK / 16; ++k) {
                        if constexpr (PAIR)
                            umma_bf16_pair(d, sdesc_sw128(sa + k * 16 * 128, BOX), sdesc_sw128(sb + k * 16 * 128, BOX),
                                           idesc, (kb == 0 && k == 0) ? 0u : 1u);
                        else
                            umma_bf16(d, sdesc_sw128(sa + k * 16 * 128, BOX), sdesc_sw128(sb + k * 16 * 128, BOX), idesc,
                                      (kb == 0 && k == 0) ? 0u : 1u);
                    }
                    if constexpr (PAIR)
                        umma_commit_pair(empty(s), 0x3);
                    else
                        umma_commit(empty(s));
                }
                if (!ok) break;
                if constexpr (PAIR)
                    umma_commit_pair(tfull(b), 0x3);
                else
                    umma_commit(tfull(b));
            }
            if (PAIR && !ok) pause_ns(200000);
        }
        __syncwarp();
    } else if (warp == B_STATE_WARP) {
        // ---- state producer: W (and mu) chunks of every tile, in epilogue order
        if (lane == 0) {
            tma_prefetch_map(&tmW1s);
            tma_prefetch_map(&tmW2s);
            if (a.momentum) {
                tma_prefetch_map(&tmM1s);
                tma_prefetch_map(&tmM2s);
            }
            uint32_t seq = 0;
            bool ok = true;
            for (int t = tl.first; t < tl.count && ok; t += tl.step) {
                int cz, h0, col0;
                tl.decode(t, cz, h0, col0);
                const int cs = a.c0 + cz;
                const bool isW1 = col0 < a.d_in;
                const int cl = isW1 ? col0 : col0 - a.d_in;
                for (int g = 0; g < B_BN / S_ROWS; ++g, ++seq) {
                    const int k = seq % S_SLOTS;
                    if (seq >= S_SLOTS && !mbar_wait(sempty(k), ((seq / S_SLOTS) - 1) & 1, a.status, a.wait_ns)) {
                        ok = false;
                        break;
                    }
                    const uint32_t dst = smem_u32(base + L::STATE + k * S_SLOT);
                    mbar_expect_tx(sfull(k), chunk_bytes);
                    tma_load_3d(dst, isW1 ? &tmW1s : &tmW2s, sfull(k), cl, h0 + g * S_ROWS, cs);
                    if (a.momentum) tma_load_3d(dst + S_F32, isW1 ? &tmM1s : &tmM2s, sfull(k), cl, h0 + g * S_ROWS, cs);
                }
            }
        }
        __syncwarp();
    } else if (warp == B_STORE_WARP) {
        // ---- store warp: write every updated chunk back with TMA, then free its slot
        if (lane == 0) {
            uint32_t seq = 0;
            bool ok = true;
            for (int t = tl.first; t < tl.count && ok; t += tl.step) {
                int cz, h0, col0;
                tl.decode(t, cz, h0, col0);
                const int cs = a.c0 + cz;
                const bool isW1 = col0 < a.d_in;
                const int cl = isW1 ? col0 : col0 - a.d_in;
                for (int g = 0; g < B_BN / S_ROWS; ++g, ++seq) {
                    const int k = seq % S_SLOTS;
                    if (!mbar_wait(sdone(k), (seq / S_SLOTS) & 1, a.status, a.wait_ns)) {
                        ok = false;
                        break;
                    }
                    const uint32_t src = smem_u32(base + L::STATE + k * S_SLOT);
                    tma_store_3d(isW1 ? &tmW1s : &tmW2s, src, cl, h0 + g * S_ROWS, cs);
                    if (a.momentum) tma_store_3d(isW1 ? &tmM1s : &tmM2s, src + S_F32, cl, h0 + g * S_ROWS, cs);
                    bulk_commit();
                    bulk_wait_read_all();  // the store has read the slot: hand it back
                    mbar_arrive(sempty(k));
                }
            }
            bulk_wait_all();
        }
        __syncwarp();
    } else {
        // ---- epilogue warps 2..9: group grp takes the tile's chunks grp, grp+2, grp+4, grp+6;
        //      within a group, TMEM lane quarter q = 32 weight columns
        const int grp = (warp - 2) >> 2, q = warp & 3, et = threadIdx.x - 64 - grp * B_EPI_THREADS;
        const uint32_t bar_id = 1 + grp;
        // Single-buffered per-tile tables: a warp writes tile i+1's entries only after
        // every warp of its group has passed the last chunk barrier of tile i.
        float* tab = reinterpret_cast<float*>(base + L::TAB) + grp * (B_BN / 2 + 4);  // [B_BN/2]
        float* bred = tab + B_BN / 2;                                                  // [4]
        int* flag = reinterpret_cast<int*>(base + L::FLAG) + grp * 2;
        const uint32_t tempty_rank0 = PAIR ? map_to_cta(tempty(0), 0) : tempty(0);
        bool finite = true;
        float step = 0.f;        // sum of mu_s^2 over this thread's elements of the current tile
        uint32_t tile_seq0 = 0;  // chunk sequence number of the current tile's first chunk
        int local = 0;
        for (int t = tl.first; t < tl.count; t += tl.step, ++local, tile_seq0 += B_BN / S_ROWS) {
            int cz, h0, col0;
            tl.decode(t, cz, h0, col0);
            const int cs = a.c0 + cz;
            const bool isW1 = col0 < a.d_in;
            const int which = isW1 ? 0 : 1;
            const int cl = isW1 ? col0 : col0 - a.d_in;
            const int width = isW1 ? a.d_in : a.d_out;
            const int b = local & 1;
            // the tile's rows and columns lie inside the chain's W (index check of MONE_DEBUG builds)
            const bool wr = MONE_DCHECK(cs < a.C && h0 + B_BN <= a.d_hid && cl + B_BM <= width, a.status,
                                        DS_PHASE_B_TILE);
            const float* n0 = (isW1 ? a.n1 : a.n2) + (size_t)cs * a.d_hid;
            const float* prevss = ss_row(a, a.parity ^ 1, which, cs);
            {   // scales of this group's 4 chunks x 32 rows
                const int i = et >> 5, j = et & 31;
                const int row = h0 + (2 * i + grp) * S_ROWS + j;
                tab[et] = a.renorm_pending ? renorm_scale(n0[row], prevss[row]) : 1.f;
            }
            if (a.momentum) {
                float v = 0.f;
                for (int tk = et; tk < a.Tp; tk += B_EPI_THREADS) v += a.dbeta[(size_t)cs * a.win + a.tok0 + tk];
                v = warp_sum(v);
                if (lane == 0) bred[q] = v;
            }
            if (et == 0) flag[0] = mbar_wait(tfull(b), (local >> 1) & 1, a.status, a.wait_ns) ? 1 : 0;
            __syncwarp();
            named_bar_sync(bar_id, B_EPI_THREADS);
            if (!flag[0]) break;
            tc_fence_after();
            float beta = 0.f;
            if (a.momentum) beta = sigmoidf_((bred[0] + bred[1] + bred[2] + bred[3]) / (float)a.Tp + a.b_beta[cs]);
            float* cur = ss_row(a, a.parity, which, cs);
            const int col = q * 32 + lane;  // column within the tile (= TMEM lane)
            bf16* Wb = (isW1 ? a.W1b : a.W2b) + (size_t)cs * a.d_hid * width + cl + col;
            const uint64_t wpol = l2_evict_last_policy();  // phase A of the next segment reads the copy
            const uint32_t lane_base = tmem + ((uint32_t)(q * 32) << 16) + b * 256;
            bool ok = true;
#pragma unroll 1
            for (int i = 0; i < B_BN / S_ROWS / 2; ++i) {
                const int c = 2 * i + grp;
                const uint32_t seq = tile_seq0 + c;
                const int k = seq % S_SLOTS;
                const int r0 = h0 + c * S_ROWS;
                float gv[32];
                tmem_ld32(lane_base + c * S_ROWS, gv);
                if (i == B_BN / S_ROWS / 2 - 1) {
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) {
                        if constexpr (PAIR)
                            mbar_arrive_remote(tempty_rank0 + 8 * b);
                        else
                            mbar_arrive(tempty(b));
                    }
                }
                if (et == 0) flag[1] = mbar_wait(sfull(k), (seq / S_SLOTS) & 1, a.status, a.wait_ns) ? 1 : 0;
                __syncwarp();
                named_bar_sync(bar_id, B_EPI_THREADS);
                if (!flag[1]) {
                    ok = false;
                    break;
                }
                uint8_t* slot = base + L::STATE + k * S_SLOT;
                float* Ws = reinterpret_cast<float*>(slot);
                float* Ms = reinterpret_cast<float*>(slot + S_F32);
                bf16* bp = Wb + (size_t)r0 * width;
                float v[32];
#pragma unroll
                for (int j = 0; j < 32; ++j) {
                    const float sc = tab[i * S_ROWS + j];
                    const float m = a.momentum ? Ms[j * B_BM + col] : 0.f;
                    const float mn = fmaf(beta, m, gv[j]);
                    const float wn = fmaf(sc, Ws[j * B_BM + col], -mn);
                    Ws[j * B_BM + col] = wn;
                    if (a.momentum) Ms[j * B_BM + col] = mn;
                    if (wr) st_bf16_hint(bp + j * width, __float2bfloat16_rn(wn), wpol);
                    v[j] = wn * wn;  // a NaN or Inf weight makes its row's sum non-finite
                    if constexpr (STEP) step = fmaf(mn, mn, step);
                }
                // transpose-reduce: afterwards lane j holds this warp's 32-column partial of row j
#pragma unroll
                for (int sft = 16; sft >= 1; sft >>= 1) {
                    const bool upper = (lane & sft) != 0;
#pragma unroll
                    for (int u = 0; u < sft; ++u) {
                        const float send = upper ? v[u] : v[u + sft];
                        const float keep = upper ? v[u + sft] : v[u];
                        v[u] = keep + __shfl_xor_sync(0xffffffffu, send, sft);
                    }
                }
                finite = finite && isfinite(v[0]);
                if (wr) atomicAdd(&cur[r0 + lane], v[0]);
                // make this warp's shared-memory writes visible to the TMA store, then tell the store warp
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) mbar_arrive(sdone(k));
            }
            if (!ok) break;
            if constexpr (STEP) {  // per-segment metric: the tile's share of |mu_s|^2
                const float t = warp_sum(step);
                if (lane == 0) atomicAdd(&a.step_sq[cz], t);
                step = 0.f;
            }
        }
        if (!finite) atomicOr(a.status, DEV_NONFINITE);
    }
    tc_fence_before();
    if constexpr (PAIR)
        cluster_sync();  // every MMA of the pair has completed and every TMEM read is done
    else
        __syncthreads();
    tc_fence_after();
    if (warp == 0) {
        if constexpr (PAIR)
            tmem_dealloc_pair(tmem, 512);
        else
            tmem_dealloc(tmem, 512);
    }
}

TcArgs make_args(const DevState& s, const SegWork& w) {
    TcArgs a{};
    a.d_in = s.d_in; a.d_out = s.d_out; a.d_hid = s.d_hid; a.T = s.T; a.Tp = w.Tp; a.c0 = w.c0; a.nc = w.nc;
    a.C = s.C;
    a.paper = s.mode == 1; a.momentum = s.momentum; a.renorm_pending = w.renorm_pending; a.parity = w.parity;
    a.u_row0 = a.paper ? (int)w.u_off : (int)w.row0;
    a.tok0 = w.u_off;
    a.win = s.win_rows;
    a.u_chain0 = a.paper ? w.c0 : 0;
    a.y_row0 = w.y_scratch ? 0 : (int)w.row0;
    a.lr = s.lr;
    a.eta_in = w.eta_in ? w.eta_in + w.row0 : nullptr;
    a.eta_cstride = w.eta_cstride;
    a.eta = s.eta; a.dbeta = s.dbeta; a.b_beta = s.b_beta;
    a.zinv = a.paper ? s.zinv : nullptr;
    a.W1 = s.W1; a.W2 = s.W2; a.mu1 = s.mu1; a.mu2 = s.mu2; a.W1b = s.W1b; a.W2b = s.W2b;
    a.n1 = s.n1; a.n2 = s.n2; a.sumsq = s.sumsq;
    a.dH = reinterpret_cast<bf16*>(s.dHt); a.At = reinterpret_cast<bf16*>(s.Att);
    a.loss = w.loss; a.step_sq = w.step_sq; a.status = s.status;
    a.wait_ns = kWaitLimitNs;
    return a;
}

// ------------------------------------------------------------------ memory read (Eq. 4)
//
// The read of generate_kv on the bf16 path, on the tensor cores, in two kernels:
//   hidden:  A_q = SiLU(U_q W1^T)    tile = (128 queries, 128 hidden units, chain), K = d_in
//   out:     O = A_q W2, then per output head h of width hd: g_h o_h / sqrt(mean(o_h^2) + eps)
//            written into the caller's K / V layout   tile = (128 queries, 128 outputs, chain), K = d_hid
// One tile per CTA: warp 0 streams the query rows and the bf16 weight copy with TMA,
// warp 1 issues tcgen05.mma into a 128-column TMEM accumulator, warps 2..5 (one per TMEM
// lane quarter, lane = query) run the epilogue.  Each weight tile is read by ceil(Q/128)
// CTAs; query rows >= Q arrive as TMA zero fill and are never stored.  W2 is [hidden][out],
// so in the out kernel the weight operand is MN-major (64-column boxes, as in phase B).
// A launch with more tiles than SMs runs two CTAs per SM (three 32 KB stages each), so one
// CTA's epilogue overlaps the other's loads; a launch that fits in one wave runs one CTA per
// SM with six stages, twice the operand bytes in flight for its single K loop.
constexpr int R_STAGE = 2 * 128 * BK * 2;  // 32 KB: 128 query rows + 128 weight rows / columns
constexpr int R_THREADS = 6 * 32;
constexpr uint32_t R_EPI_BAR = 1;
template <int NST>
struct LRT {
    static constexpr int STAGES = NST;
    static constexpr int CTAS_PER_SM = NST <= 3 ? 2 : 1;
    static constexpr int RING = NST * R_STAGE;
    static constexpr int BARS = RING;  // full[S] empty[S] tfull
    static constexpr int NBARS = 2 * NST + 1;
    static constexpr int SLOT = BARS + (NBARS * 8 + 15) / 16 * 16;
    static constexpr int FLAG = SLOT + 16;
    static constexpr int TAB = FLAG + 16;  // MSE_HIDDEN: renorm scales s1, s2 of the tile's rows
    static constexpr int STG = TAB + 256 * 4;  // 4 epilogue warps x 2 KB transpose buffers
    static constexpr int END = STG + 4 * 2048;
    static constexpr int DYN = END + 1024;
};
using LR = LRT<3>;   // several waves
using LR6 = LRT<6>;  // one wave
static_assert(LR::CTAS_PER_SM * (LR::DYN + 1024) <= 228 * 1024, "read kernel CTAs per SM");
static_assert(LR6::DYN <= 227 * 1024, "read kernel shared memory");
static_assert(LR::STG % 16 == 0, "staging buffers hold 16-byte pieces");

struct ReadArgs {
    int Q, d_in, d_hid, d_out, n_kv, L;
    float eps;
    const float* gate;     // [C][2 n_kv] per-head gates, or null (gate 1)
    bf16* Aq;              // [C][Q][d_hid]
    bf16 *Kout, *Vout;     // caller's K / V, element strides s0 (context), s1 (layer), s2 (head), s3 (query)
    long long s0, s1, s2, s3;
    int* status;
    // operand coordinates: A rows start at a_row0 + 128 * blockIdx.x of chain a_chain0 + blockIdx.z,
    // weights of chain b_chain0 + blockIdx.z
    int a_row0, a_chain0, b_chain0;
    // squared-error loss pre-pass (MSE_* modes): one segment of chains b_chain0 + blockIdx.z
    int C, T, Tp, win, parity, renorm_pending;
    long long tok0, row0, n_rows, y_cstride;
    const float *zinv, *n1, *n2, *sumsq;  // as in TcArgs
    const bf16 *K, *V;     // caller's targets of the group (chain z at z * y_cstride)
    bf16 *Kres, *Vres;     // [C][T][d_out/2] residual targets y - M(u)
    float* loss;           // [nc] or null
    // MSE_HIDDEN, when phase A runs in its R-only form: also write At = c_t SiLU(x) and
    // c_t SiLU'(x) / |z_t| (into dH), with c_t = -eta_t / T'
    bf16 *At, *Sp;         // [C][T][d_hid] or null
    int paper;
    float lr;
    const float *eta, *eta_in;
    long long eta_cstride;
    const float* qzinv;    // read with the weights as M: 1/|z| per query [C][Q] (paper mode), or null
};

enum { READ_HIDDEN = 0, MSE_HIDDEN = 1, MSE_OUT = 2 };  // other MODEs: read out with heads of width MODE

// MODE READ_HIDDEN: A_q = SiLU(U_q W1^T).  MODE 64 / 128: the read's out kernel with heads
// of that width.  MODE MSE_HIDDEN: A' = SiLU(s1 (1/|z_t|) H) s2, the segment's activations
// with the pending renorm scales (s2 folded in, so A' W2raw = A W2).  MODE MSE_OUT: the
// residual target y_t - M(u_t) = y_t - A'_t W2raw (and the segment's squared-error loss).
template <int MODE, int NST>
__global__ void __launch_bounds__(R_THREADS, LRT<NST>::CTAS_PER_SM)
tc_read_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, const ReadArgs a) {
    constexpr bool OUT = MODE != READ_HIDDEN && MODE != MSE_HIDDEN;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const uint32_t bars = smem_u32(base + LRT<NST>::BARS);
    auto full = [&](int s) { return bars + 8 * s; };
    auto empty = [&](int s) { return bars + 8 * (NST + s); };
    const uint32_t tfull = bars + 8 * (2 * NST);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int s = 0; s < NST; ++s) {
            mbar_init(full(s), 1);
            mbar_init(empty(s), 1);
        }
        mbar_init(tfull, 1);
        fence_mbar_init();
    }
    if (warp == 0) {
        tmem_alloc(smem_u32(base + LRT<NST>::SLOT), 128);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *reinterpret_cast<uint32_t*>(base + LRT<NST>::SLOT);
    const int q0 = blockIdx.x * 128, n0 = blockIdx.y * 128, c = blockIdx.z;
    const int KB = (OUT ? a.d_hid : a.d_in) / BK;
    float* table = reinterpret_cast<float*>(base + LRT<NST>::TAB);

    if (warp == 0) {
        if (lane == 0) {
            tma_prefetch_map(&tmA);
            tma_prefetch_map(&tmB);
            for (int kb = 0; kb < KB; ++kb) {
                const int s = kb % NST;
                if (kb >= NST && !mbar_wait(empty(s), ((kb / NST) - 1) & 1, a.status)) break;
                const uint32_t sa = smem_u32(base + s * R_STAGE), sb = sa + 128 * BK * 2, fb = full(s);
                mbar_expect_tx(fb, R_STAGE);
                tma_load_3d(sa, &tmA, fb, kb * BK, a.a_row0 + q0, a.a_chain0 + c);
                if (OUT) {
                    tma_load_3d(sb, &tmB, fb, n0, kb * BK, a.b_chain0 + c);
                    tma_load_3d(sb + BOX, &tmB, fb, n0 + 64, kb * BK, a.b_chain0 + c);
                } else {
                    tma_load_3d(sb, &tmB, fb, kb * BK, n0, a.b_chain0 + c);
                }
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16_f32(128, 128, false, OUT);
            bool ok = true;
            for (int kb = 0; kb < KB; ++kb) {
                const int s = kb % NST;
                if (!mbar_wait(full(s), (kb / NST) & 1, a.status)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t sa = smem_u32(base + s * R_STAGE), sb = sa + 128 * BK * 2;
#pragma unroll
                for (int k = 0; k < BK / 16; ++k)
                    umma_bf16(tmem, sdesc_sw128(sa + k * 32, 16),
                              OUT ? sdesc_sw128(sb + k * 16 * 128, BOX) : sdesc_sw128(sb + k * 32, 16), idesc,
                              (kb == 0 && k == 0) ? 0u : 1u);
                umma_commit(empty(s));
            }
            if (ok) umma_commit(tfull);
        }
        __syncwarp();
    } else {
        const int q = warp & 3;  // TMEM lane quarter of this warp
        int* flag = reinterpret_cast<int*>(base + LRT<NST>::FLAG);
        if constexpr (MODE == MSE_HIDDEN) {
            // renorm scales of this tile's 128 hidden rows (one per epilogue thread)
            const int h = n0 + (int)threadIdx.x - 64, cs = a.b_chain0 + c;
            float s1 = 1.f, s2 = 1.f;
            if (a.renorm_pending) {
                // row sums of squares of the last update: [2 parity][2 matrix][C][d_hid]
                const float* ss1 = a.sumsq + ((size_t)((a.parity ^ 1) * 2 + 0) * a.C + cs) * a.d_hid;
                const float* ss2 = a.sumsq + ((size_t)((a.parity ^ 1) * 2 + 1) * a.C + cs) * a.d_hid;
                s1 = renorm_scale(a.n1[(size_t)cs * a.d_hid + h], ss1[h]);
                s2 = renorm_scale(a.n2[(size_t)cs * a.d_hid + h], ss2[h]);
            }
            table[threadIdx.x - 64] = s1;
            table[128 + threadIdx.x - 64] = s2;
        }
        if (threadIdx.x == 64) *flag = mbar_wait(tfull, 0, a.status) ? 1 : 0;
        __syncwarp();
        named_bar_sync(R_EPI_BAR, 128);
        if (*flag) {
            tc_fence_after();
            const uint32_t lane_base = tmem + ((uint32_t)(q * 32) << 16);
            const int qw = q0 + q * 32;  // first query row of this warp
            if constexpr (MODE == MSE_HIDDEN) {
                const int cs = a.b_chain0 + c, t = qw + lane;
                const float zi = (t < a.Tp) ? (a.zinv ? a.zinv[(size_t)cs * a.win + a.tok0 + t] : 1.f) : 0.f;
                float ct = 0.f;  // c_t = -eta_t / T' (R-only outputs)
                if (a.At && t < a.Tp) {
                    const float ev = a.paper ? a.eta[(size_t)cs * a.win + a.tok0 + t]
                                             : (a.eta_in ? a.eta_in[c * a.eta_cstride + t] : a.lr);
                    ct = -ev / (float)a.Tp;
                }
                const float czi = ct * zi;
                uint8_t* stg = base + LRT<NST>::STG + (warp - 2) * 2048;
                const size_t roff = ((size_t)cs * a.T + qw) * a.d_hid + n0;
#pragma unroll 1
                for (int cc = 0; cc < 4; ++cc) {
                    float hv[32];
                    tmem_ld32(lane_base + cc * 32, hv);
                    uint32_t pk[16];
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        const int k0 = cc * 32 + 2 * j;
                        const float x0 = hv[2 * j] * table[k0] * zi, x1 = hv[2 * j + 1] * table[k0 + 1] * zi;
                        pk[j] = pack_bf16(x0 * sigmoidf_(x0) * table[128 + k0], x1 * sigmoidf_(x1) * table[128 + k0 + 1]);
                    }
                    store_rows_coalesced(stg, pk, a.Aq + roff + cc * 32, a.d_hid, lane);
                    if (a.At) {  // the R-only form of phase A takes At and c SiLU'(x) / |z| from here
                        uint32_t pa[16], ps[16];
#pragma unroll
                        for (int j = 0; j < 16; ++j) {
                            const int k0 = cc * 32 + 2 * j;
                            const float x0 = hv[2 * j] * table[k0] * zi, x1 = hv[2 * j + 1] * table[k0 + 1] * zi;
                            const float g0 = sigmoid_tanh(x0), g1 = sigmoid_tanh(x1);
                            pa[j] = pack_bf16(ct * x0 * g0, ct * x1 * g1);
                            ps[j] = pack_bf16(czi * (g0 * fmaf(x0, 1.f - g0, 1.f)), czi * (g1 * fmaf(x1, 1.f - g1, 1.f)));
                        }
                        store_rows_coalesced(stg, pa, a.At + roff + cc * 32, a.d_hid, lane);
                        store_rows_coalesced(stg, ps, a.Sp + roff + cc * 32, a.d_hid, lane);
                    }
                }
            } else if constexpr (MODE == MSE_OUT) {
                const int cs = a.b_chain0 + c, t = qw + lane, dh = a.d_out / 2;
                const bool kpart = n0 < dh;
                const int col0 = kpart ? n0 : n0 - dh;
                const bool live = t < a.Tp && a.row0 + t < a.n_rows;
                const bf16* yrow = (kpart ? a.K : a.V) + (size_t)c * a.y_cstride + (size_t)(a.row0 + t) * dh + col0;
                uint8_t* stg = base + LRT<NST>::STG + (warp - 2) * 2048;
                bf16* row0 = (kpart ? a.Kres : a.Vres) + ((size_t)cs * a.T + qw) * dh + col0;
                float lsum = 0.f;
#pragma unroll 1
                for (int cc = 0; cc < 4; ++cc) {
                    float ov[32];
                    tmem_ld32(lane_base + cc * 32, ov);
                    uint32_t pk[16];
#pragma unroll
                    for (int v = 0; v < 4; ++v) {
                        uint4 y = make_uint4(0, 0, 0, 0);
                        if (live) y = *reinterpret_cast<const uint4*>(yrow + cc * 32 + v * 8);
                        const __nv_bfloat162* yb = reinterpret_cast<const __nv_bfloat162*>(&y);
#pragma unroll
                        for (int u = 0; u < 4; ++u) {
                            const float2 yf = __bfloat1622float2(yb[u]);
                            const int j = v * 8 + 2 * u;
                            const float r0 = live ? yf.x - ov[j] : 0.f, r1 = live ? yf.y - ov[j + 1] : 0.f;
                            lsum = fmaf(r0, r0, fmaf(r1, r1, lsum));
                            pk[v * 4 + u] = pack_bf16(r0, r1);
                        }
                    }
                    store_rows_coalesced(stg, pk, row0 + cc * 32, dh, lane);
                }
                if (a.loss) {
                    lsum = warp_sum(lsum);
                    if (lane == 0) atomicAdd(&a.loss[c], 0.5f * lsum / (float)a.Tp);
                }
            } else if constexpr (!OUT) {
                uint8_t* stg = base + LRT<NST>::STG + (warp - 2) * 2048;
                bf16* row0 = a.Aq + ((size_t)c * a.Q + qw) * a.d_hid + n0;
                // the tile's columns of A_q lie inside [Q][d_hid] (index check of MONE_DEBUG builds)
                const bool wr = MONE_DCHECK(n0 + 128 <= a.d_hid, a.status, DS_READ_TILE);
#pragma unroll 1
                for (int cc = 0; cc < 4; ++cc) {
                    float hv[32];
                    tmem_ld32(lane_base + cc * 32, hv);
                    uint32_t pk[16];
#pragma unroll
                    for (int j = 0; j < 16; ++j)
                        pk[j] = pack_bf16(hv[2 * j] * sigmoidf_(hv[2 * j]), hv[2 * j + 1] * sigmoidf_(hv[2 * j + 1]));
                    if (wr) store_rows_coalesced(stg, pk, row0 + cc * 32, a.d_hid, lane, a.Q - qw);
                }
            } else {
                constexpr int HD = MODE;
                const int qi = qw + lane;
                const int nh = 2 * a.n_kv;
#pragma unroll 1
                for (int hh = 0; hh < 128 / HD; ++hh) {
                    float v[HD];
#pragma unroll
                    for (int cc = 0; cc < HD / 32; ++cc)
                        tmem_ld32(lane_base + hh * HD + cc * 32, *reinterpret_cast<float(*)[32]>(v + cc * 32));
                    float ss = 0.f;
#pragma unroll
                    for (int i = 0; i < HD; ++i) ss = fmaf(v[i], v[i], ss);
                    const int head = n0 / HD + hh;
                    const bool wr = MONE_DCHECK(head < nh, a.status, DS_READ_TILE);
                    const float g = a.gate && wr ? a.gate[(size_t)c * nh + head] : 1.f;
                    const float sc = g / sqrtf(ss / (float)HD + a.eps);
                    if (qi < a.Q && wr) {
                        const int kvh = head < a.n_kv ? head : head - a.n_kv;
                        bf16* out = (head < a.n_kv ? a.Kout : a.Vout) + (long long)(c / a.L) * a.s0 +
                                    (long long)(c % a.L) * a.s1 + (long long)kvh * a.s2 + (long long)qi * a.s3;
                        if ((reinterpret_cast<uintptr_t>(out) & 15u) == 0) {
#pragma unroll
                            for (int i = 0; i < HD; i += 8)
                                *reinterpret_cast<uint4*>(out + i) =
                                    make_uint4(pack_bf16(v[i] * sc, v[i + 1] * sc), pack_bf16(v[i + 2] * sc, v[i + 3] * sc),
                                               pack_bf16(v[i + 4] * sc, v[i + 5] * sc), pack_bf16(v[i + 6] * sc, v[i + 7] * sc));
                        } else {
#pragma unroll
                            for (int i = 0; i < HD; ++i) out[i] = __float2bfloat16_rn(v[i] * sc);
                        }
                    }
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, 128);
}

// ------------------------------------------------------------------ memory read, weights as the MMA rows
//
// For a query of Q <= 256 tokens the read runs with the operands the other way round: the
// weight tile is the tcgen05 A operand (M = 128 weight rows) and the queries are the B
// operand (N = NT = Q rounded up to 32), so neither an MMA row nor a staged query row is
// padding and each CTA takes in half the query bytes of the 128-query form.
//   hidden (HD = 0):  D[h][q] = W1[h] . z_q;  A_q[q][h] = SiLU(D[h][q] / |z_q|) (paper mode; the
//                     unnormalised z_q = SiLU(alpha x_q + gamma) comes from query_z_kernel, and
//                     the row scale commutes with the contraction), bf16 [C][Q][d_hid], stored
//                     through a per-warp 32 x 32 transpose so each row leaves as 64 contiguous bytes
//   out (HD = 64/128): D[o][q] = sum_h W2[h][o] A_q[q][h] (W2 MN-major); per head of HD
//                     features the RMS of each query's HD values is a reduction across the
//                     head's TMEM lanes (warp transpose-sums, then shared memory), then the
//                     gate, then the store into the caller's K / V (lanes = contiguous features)
// Warp 0 streams the weight tile and the query rows with TMA (2 to 8 stages), warp 1 issues
// the MMAs into one NT-column TMEM accumulator, warps 2..5 (one TMEM lane quarter each) run
// the epilogue.  Query rows >= Q arrive as TMA zero fill and are never stored.
// Both kernels are launched with programmatic stream serialisation: a CTA may start while the
// kernel before it (the query transform, or the hidden kernel) is still running, loads the
// weight tiles of its first stages, which that kernel does not write, and only then waits for
// that kernel's completion (griddepcontrol.wait) before it loads the query rows it produced.
constexpr int RT_THREADS = 6 * 32;
constexpr int RT_MAX_NT = 256;
constexpr int RT_A = 128 * BK * 2;  // 16 KB: the weight tile of one k-block
__host__ __device__ constexpr int rt_stage(int nt) { return RT_A + nt * BK * 2; }
// Ring budget: 192 KB (one CTA per SM) when the grid fits in one wave; 96 KB (two CTAs per SM,
// one's epilogue overlapping the other's loads) when it takes several.
constexpr int RT_RING_1 = 192 * 1024, RT_RING_2 = 96 * 1024;
__host__ __device__ constexpr int rt_stages(int nt, int ring = RT_RING_1) {
    return ring / rt_stage(nt) < 8 ? ring / rt_stage(nt) : 8;
}
// shared memory after the ring: barriers, TMEM slot and flag, then the epilogue's buffers:
// 4 warps x 2 KB transposes and the queries' 1/|z| (hidden), or 4 x NT column partial sums +
// 2 x NT scales (out)
__host__ __device__ constexpr int rt_bars(int nt, int ring = RT_RING_1) { return rt_stages(nt, ring) * rt_stage(nt); }
__host__ __device__ constexpr int rt_epi(int nt, int ring = RT_RING_1) { return rt_bars(nt, ring) + 256; }
__host__ __device__ constexpr int rt_dyn(int nt, int ring = RT_RING_1) {
    return rt_epi(nt, ring) + (4 * 2048 + RT_MAX_NT * 4 > 6 * nt * 4 ? 4 * 2048 + RT_MAX_NT * 4 : 6 * nt * 4) + 1024;
}
static_assert(rt_dyn(RT_MAX_NT) <= 227 * 1024 && rt_dyn(32) <= 227 * 1024, "read shared memory budget");
static_assert(rt_dyn(RT_MAX_NT, RT_RING_2) <= 113 * 1024 && rt_dyn(32, RT_RING_2) <= 113 * 1024,
              "two read CTAs per SM");
static_assert(rt_stages(RT_MAX_NT, RT_RING_2) >= 2, "read pipeline depth");

template <int HD>
__global__ void __launch_bounds__(RT_THREADS, 2)
tc_read_t_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmQ, const ReadArgs a,
                 int NT, int ring) {
    constexpr bool OUT = HD != 0;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int NST = rt_stages(NT, ring), STAGE = rt_stage(NT);
    const uint32_t bars = smem_u32(base + rt_bars(NT, ring));
    auto full = [&](int s) { return bars + 8 * s; };
    auto empty = [&](int s) { return bars + 8 * (8 + s); };
    const uint32_t tfull = bars + 8 * 16;
    uint32_t* slot = reinterpret_cast<uint32_t*>(base + rt_bars(NT, ring) + 8 * 17);
    int* flag = reinterpret_cast<int*>(base + rt_bars(NT, ring) + 8 * 17 + 8);
    uint8_t* epi = base + rt_epi(NT, ring);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int s = 0; s < NST; ++s) {
            mbar_init(full(s), 1);
            mbar_init(empty(s), 1);
        }
        mbar_init(tfull, 1);
        fence_mbar_init();
    }
    if (warp == 0) {
        tmem_alloc(smem_u32(slot), RT_MAX_NT);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *slot;
    const int q0 = blockIdx.x * NT, n0 = blockIdx.y * 128, c = blockIdx.z;
    const int KB = (OUT ? a.d_hid : a.d_in) / BK;
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");  // the out kernel may start

    if (warp == 0) {
        if (lane == 0) {
            tma_prefetch_map(&tmW);
            tma_prefetch_map(&tmQ);
            auto load_w = [&](int kb, uint32_t sa, uint32_t fb) {
                if (OUT) {  // W2 rows kb*64.. as [64 hidden][64 outputs] boxes: the MN-major A operand
                    tma_load_3d(sa, &tmW, fb, n0, kb * BK, a.b_chain0 + c);
                    tma_load_3d(sa + BOX, &tmW, fb, n0 + 64, kb * BK, a.b_chain0 + c);
                } else {
                    tma_load_3d(sa, &tmW, fb, kb * BK, n0, a.b_chain0 + c);
                }
            };
            // the first stages' weight tiles, then the wait for the kernel that writes the queries
            const int pre = KB < NST ? KB : NST;
            for (int kb = 0; kb < pre; ++kb) {
                const uint32_t sa = smem_u32(base + kb * STAGE), fb = full(kb);
                mbar_expect_tx(fb, STAGE);
                load_w(kb, sa, fb);
            }
            asm volatile("griddepcontrol.wait;" ::: "memory");
            for (int kb = 0; kb < KB; ++kb) {
                const int s = kb % NST;
                const uint32_t sa = smem_u32(base + s * STAGE), sb = sa + RT_A, fb = full(s);
                if (kb >= pre) {
                    if (!mbar_wait(empty(s), ((kb / NST) - 1) & 1, a.status)) break;
                    mbar_expect_tx(fb, STAGE);
                    load_w(kb, sa, fb);
                }
                tma_load_3d(sb, &tmQ, fb, kb * BK, a.a_row0 + q0, a.a_chain0 + c);
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16_f32(128, NT, OUT, false);
            bool ok = true;
            for (int kb = 0; kb < KB; ++kb) {
                const int s = kb % NST;
                if (!mbar_wait(full(s), (kb / NST) & 1, a.status)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t sa = smem_u32(base + s * STAGE), sb = sa + RT_A;
#pragma unroll
                for (int k = 0; k < BK / 16; ++k)
                    umma_bf16(tmem, OUT ? sdesc_sw128(sa + k * 16 * 128, BOX) : sdesc_sw128(sa + k * 32, 16),
                              sdesc_sw128(sb + k * 32, 16), idesc, (kb == 0 && k == 0) ? 0u : 1u);
                umma_commit(empty(s));
            }
            if (ok) umma_commit(tfull);
        }
        __syncwarp();
    } else {
        const int q = warp & 3;  // TMEM lane quarter: weight rows n0 + 32 q .. + 31
        const uint32_t lane_base = tmem + ((uint32_t)(q * 32) << 16);
        float* zs = reinterpret_cast<float*>(epi + 4 * 2048);  // hidden: 1/|z| of the tile's queries
        if constexpr (!OUT) {
            asm volatile("griddepcontrol.wait;" ::: "memory");  // zinv comes from the kernel before
            for (int j = threadIdx.x - 64; j < NT; j += 128)
                zs[j] = (a.qzinv && q0 + j < a.Q) ? a.qzinv[(size_t)c * a.Q + q0 + j] : 1.f;
        }
        if (threadIdx.x == 64) *flag = mbar_wait(tfull, 0, a.status) ? 1 : 0;
        __syncwarp();
        named_bar_sync(R_EPI_BAR, 128);
        if (*flag) {
            tc_fence_after();
            const int nch = NT / 32;
            if constexpr (!OUT) {
                // the tile's columns of A_q lie inside [Q][d_hid] (index check of MONE_DEBUG builds)
                const bool wr = MONE_DCHECK(n0 + 128 <= a.d_hid, a.status, DS_READ_TILE);
                uint16_t* stg = reinterpret_cast<uint16_t*>(epi + (warp - 2) * 2048);  // [32 queries][32 rows]
                const int h = n0 + q * 32;
#pragma unroll 1
                for (int cc = 0; cc < nch; ++cc) {
                    float v[32];
                    tmem_ld32(lane_base + cc * 32, v);
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        const float x = v[j] * zs[cc * 32 + j];
                        const bf16 b = __float2bfloat16_rn(x * sigmoidf_(x));
                        stg[j * 32 + lane] = *reinterpret_cast<const uint16_t*>(&b);
                    }
                    __syncwarp();
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        const int r = 8 * k + (lane >> 2), i = lane & 3;
                        const int qi = q0 + cc * 32 + r;
                        const uint4 val = *reinterpret_cast<const uint4*>(stg + r * 32 + i * 8);
                        if (qi < a.Q && wr)
                            *reinterpret_cast<uint4*>(a.Aq + ((size_t)c * a.Q + qi) * a.d_hid + h + i * 8) = val;
                    }
                    __syncwarp();
                }
            } else {
                // per-column sums of squares of this warp's 32 features, then the head's total
                float* part = reinterpret_cast<float*>(epi);  // [4 warps][NT]
                float* scl = part + 4 * NT;                   // [2 heads of the tile][NT]
                constexpr int HPT = 128 / HD;                 // heads per 128-feature tile
                constexpr int WPH = HD / 32;                  // warps per head
#pragma unroll 1
                for (int cc = 0; cc < nch; ++cc) {
                    float v[32];
                    tmem_ld32(lane_base + cc * 32, v);
#pragma unroll
                    for (int j = 0; j < 32; ++j) v[j] *= v[j];
                    // transpose-reduce: afterwards lane j holds the sum over the warp's lanes of column j
#pragma unroll
                    for (int sft = 16; sft >= 1; sft >>= 1) {
                        const bool upper = (lane & sft) != 0;
#pragma unroll
                        for (int u = 0; u < sft; ++u) {
                            const float send = upper ? v[u] : v[u + sft];
                            const float keep = upper ? v[u + sft] : v[u];
                            v[u] = keep + __shfl_xor_sync(0xffffffffu, send, sft);
                        }
                    }
                    part[q * NT + cc * 32 + lane] = v[0];
                }
                named_bar_sync(R_EPI_BAR, 128);
                const int nh = 2 * a.n_kv;
                for (int i = threadIdx.x - 64; i < HPT * NT; i += 128) {
                    const int hl = i / NT, j = i - hl * NT;
                    float ss = 0.f;
#pragma unroll
                    for (int w = 0; w < WPH; ++w) ss += part[(hl * WPH + w) * NT + j];
                    const int head = n0 / HD + hl;
                    const float g = a.gate && head < nh ? a.gate[(size_t)c * nh + head] : 1.f;
                    scl[hl * NT + j] = g / sqrtf(ss / (float)HD + a.eps);
                }
                named_bar_sync(R_EPI_BAR, 128);
                const int o = n0 + q * 32 + lane;  // this thread's output feature
                const int hl = (q * 32) / HD, head = n0 / HD + hl, d = o - head * HD;
                const bool wr = MONE_DCHECK(head < nh, a.status, DS_READ_TILE);
                const int kvh = head < a.n_kv ? head : head - a.n_kv;
                bf16* outp = (head < a.n_kv ? a.Kout : a.Vout) + (long long)(c / a.L) * a.s0 +
                             (long long)(c % a.L) * a.s1 + (long long)kvh * a.s2 + d;
#pragma unroll 1
                for (int cc = 0; cc < nch; ++cc) {
                    float v[32];
                    tmem_ld32(lane_base + cc * 32, v);
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        const int qi = q0 + cc * 32 + j;
                        if (qi < a.Q && wr)
                            outp[(long long)qi * a.s3] = __float2bfloat16_rn(v[j] * scl[hl * NT + cc * 32 + j]);
                    }
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, RT_MAX_NT);
}

std::once_flag g_attr_once;
cudaError_t g_attr_err = cudaSuccess;
int g_sms = 0;
int g_pair_clusters = 0;   // co-resident CTA pairs of the phase A pair kernel (0: use the one-CTA kernel)
int g_pairb_clusters = 0;  // the same for the phase B pair kernel

template <int MODE>
cudaError_t read_attrs() {
    cudaError_t e = cudaFuncSetAttribute(tc_read_kernel<MODE, 3>, cudaFuncAttributeMaxDynamicSharedMemorySize, LR::DYN);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(tc_read_kernel<MODE, 6>, cudaFuncAttributeMaxDynamicSharedMemorySize, LR6::DYN);
    return e;
}

// Launch a read-structured kernel with the stage count that suits its grid (see LRT).
template <int MODE>
cudaError_t launch_read_kernel(dim3 grid, const CUtensorMap& A, const CUtensorMap& B, const ReadArgs& a,
                               cudaStream_t st) {
    if ((long long)grid.x * grid.y * grid.z <= g_sms)
        tc_read_kernel<MODE, 6><<<grid, R_THREADS, LR6::DYN, st>>>(A, B, a);
    else
        tc_read_kernel<MODE, 3><<<grid, R_THREADS, LR::DYN, st>>>(A, B, a);
    return cudaGetLastError();
}

cudaError_t ensure_attrs() {
    std::call_once(g_attr_once, [] {
        int dev = 0;
        g_attr_err = cudaGetDevice(&dev);
        if (g_attr_err == cudaSuccess)
            g_attr_err = cudaDeviceGetAttribute(&g_sms, cudaDevAttrMultiProcessorCount, dev);
        if (g_attr_err == cudaSuccess)
            g_attr_err = cudaFuncSetAttribute(tc_phase_a_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, LA::DYN);
        if (g_attr_err == cudaSuccess)
            g_attr_err = cudaFuncSetAttribute(tc_phase_b_kernel<false, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                              LayoutB::DYN);
        if (g_attr_err == cudaSuccess)
            g_attr_err = cudaFuncSetAttribute(tc_phase_b_kernel<false, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                              LayoutB::DYN);
        if (g_attr_err == cudaSuccess)
            g_attr_err = cudaFuncSetAttribute(tc_phase_b_kernel<true, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                              LayoutB2::DYN);
        if (g_attr_err == cudaSuccess)
            g_attr_err = cudaFuncSetAttribute(tc_phase_b_kernel<true, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                              LayoutB2::DYN);
        if (g_attr_err == cudaSuccess)
            g_attr_err =
                cudaFuncSetAttribute(tc_phase_a_pair_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, LP::DYN);
        if (g_attr_err == cudaSuccess) g_attr_err = read_attrs<0>();
        if (g_attr_err == cudaSuccess) g_attr_err = read_attrs<64>();
        if (g_attr_err == cudaSuccess) g_attr_err = read_attrs<128>();
        if (g_attr_err == cudaSuccess) g_attr_err = read_attrs<MSE_HIDDEN>();
        if (g_attr_err == cudaSuccess) g_attr_err = read_attrs<MSE_OUT>();
        for (auto fn : {tc_read_t_kernel<0>, tc_read_t_kernel<64>, tc_read_t_kernel<128>})
            if (g_attr_err == cudaSuccess)
                g_attr_err = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, rt_dyn(RT_MAX_NT));
        if (g_attr_err == cudaSuccess) {
            cudaLaunchConfig_t cfg = {};
            cudaLaunchAttribute at[1];
            at[0].id = cudaLaunchAttributeClusterDimension;
            at[0].val.clusterDim.x = 2;
            at[0].val.clusterDim.y = 1;
            at[0].val.clusterDim.z = 1;
            cfg.gridDim = dim3(2 * (g_sms / 2));
            cfg.blockDim = dim3(THREADS);
            cfg.dynamicSmemBytes = LP::DYN;
            cfg.attrs = at;
            cfg.numAttrs = 1;
            if (cudaOccupancyMaxActiveClusters(&g_pair_clusters, tc_phase_a_pair_kernel, &cfg) != cudaSuccess) {
                cudaGetLastError();
                g_pair_clusters = 0;
            }
            cfg.blockDim = dim3(B_THREADS);
            cfg.dynamicSmemBytes = LayoutB2::DYN;
            if (cudaOccupancyMaxActiveClusters(&g_pairb_clusters, tc_phase_b_kernel<true, false>, &cfg) != cudaSuccess) {
                cudaGetLastError();
                g_pairb_clusters = 0;
            }
        }
    });
    return g_attr_err;
}

// Whether phase A runs on CTA pairs (256-token x 256-hidden tiles) for this handle's shape.
bool phase_a_pairs(const DevState& s) {
    return (s.T / A_BM) % 2 == 0 && s.d_hid % P_BN == 0 && g_pair_clusters > 0;
}

}  // namespace

cudaError_t launch_phase_a_tc(const DevState& s, const TcMaps& m, const TcInputMaps& in, const SegWork& w,
                              cudaStream_t st) {
    cudaError_t e = ensure_attrs();
    if (e != cudaSuccess) return e;
    TcArgs a = make_args(s, w);
    if (s.fault_stall > 0) {  // test knob: this launch's waits run out after 1 ms with nothing in flight
        --s.fault_stall;
        a.stall = 1;
        a.wait_ns = 1000000ull;
    }
    const CUtensorMap& U = s.mode == 1 ? m.Ua : in.Xa;
    if (phase_a_pairs(s)) {
        // squared-error segments: the pre-pass wrote At and c SiLU'(x) / |z|, only R is left
        a.r_only = (s.loss == 1) ? 1 : 0;  // 1: MONE_LOSS_MSE
        // CTA pairs over 256-token x 256-hidden tiles
        const int npairs = w.nc * (s.T / (2 * A_BM)) * (s.d_hid / P_BN);
        const int maxc = g_pair_clusters - (s.reserve_sms + 1) / 2;  // leave reserved SMs free
        const int clusters = npairs < maxc ? npairs : maxc;
        cudaLaunchConfig_t cfg = {};
        cudaLaunchAttribute at[1];
        at[0].id = cudaLaunchAttributeClusterDimension;
        at[0].val.clusterDim.x = 2;
        at[0].val.clusterDim.y = 1;
        at[0].val.clusterDim.z = 1;
        cfg.gridDim = dim3(2 * clusters);
        cfg.blockDim = dim3(THREADS);
        cfg.dynamicSmemBytes = LP::DYN;
        cfg.stream = st;
        cfg.attrs = at;
        cfg.numAttrs = 1;
        return cudaLaunchKernelEx(&cfg, tc_phase_a_pair_kernel, U, in.Ka, in.Va, m.W1b, m.W2b, a);
    }
    const int ntiles = w.nc * (s.T / A_BM) * (s.d_hid / A_BN);
    const int sms = g_sms - s.reserve_sms;
    const int grid = ntiles < sms ? ntiles : sms;
    tc_phase_a_kernel<<<grid, THREADS, LA::DYN, st>>>(U, in.Ka, in.Va, m.W1b, m.W2b, a);
    return cudaGetLastError();
}

cudaError_t launch_phase_b_tc(const DevState& s, const TcMaps& m, const TcInputMaps& in, const SegWork& w,
                              cudaStream_t st) {
    cudaError_t e = ensure_attrs();
    if (e != cudaSuccess) return e;
    const TcArgs a = make_args(s, w);
    const CUtensorMap& U = s.mode == 1 ? m.Ub : in.Xb;
    // CTA pairs over 256-column x 256-hidden tiles (a pair's columns lie in one matrix) from
    // T = 1024 on: there a tile's operand stream (768 KB a CTA) rivals its state stream, and the
    // pair halves the dH / At share of it.  At T = 512 the pair's coupled loads and accumulator
    // release cost more than they save (measured: 57.2 vs 54.8 ms a step on l16_d2048_128k).
    constexpr int PAIR_MIN_T = 1024;
    if (s.T >= PAIR_MIN_T && s.d_in % (2 * B_BM) == 0 && s.d_out % (2 * B_BM) == 0 && g_pairb_clusters > 0) {
        const int npairs = w.nc * ((s.d_in + s.d_out) / (2 * B_BM)) * (s.d_hid / B_BN);
        const int maxc = g_pairb_clusters - (s.reserve_sms + 1) / 2;
        const int clusters = npairs < maxc ? npairs : maxc;
        cudaLaunchConfig_t cfg = {};
        cudaLaunchAttribute at[1];
        at[0].id = cudaLaunchAttributeClusterDimension;
        at[0].val.clusterDim.x = 2;
        at[0].val.clusterDim.y = 1;
        at[0].val.clusterDim.z = 1;
        cfg.gridDim = dim3(2 * clusters);
        cfg.blockDim = dim3(B_THREADS);
        cfg.dynamicSmemBytes = LayoutB2::DYN;
        cfg.stream = st;
        cfg.attrs = at;
        cfg.numAttrs = 1;
        if (a.step_sq)
            return cudaLaunchKernelEx(&cfg, tc_phase_b_kernel<true, true>, U, in.Kb, in.Vb, m.dH, m.At, m.W1s, m.W2s,
                                      m.M1s, m.M2s, a);
        return cudaLaunchKernelEx(&cfg, tc_phase_b_kernel<true, false>, U, in.Kb, in.Vb, m.dH, m.At, m.W1s, m.W2s,
                                  m.M1s, m.M2s, a);
    }
    const int ntiles = w.nc * ((s.d_in + s.d_out) / B_BM) * (s.d_hid / B_BN);
    const int sms = g_sms - s.reserve_sms;
    const int grid = ntiles < sms ? ntiles : sms;
    if (a.step_sq)
        tc_phase_b_kernel<false, true><<<grid, B_THREADS, LayoutB::DYN, st>>>(U, in.Kb, in.Vb, m.dH, m.At, m.W1s,
                                                                              m.W2s, m.M1s, m.M2s, a);
    else
        tc_phase_b_kernel<false, false><<<grid, B_THREADS, LayoutB::DYN, st>>>(U, in.Kb, in.Vb, m.dH, m.At, m.W1s,
                                                                               m.W2s, m.M1s, m.M2s, a);
    return cudaGetLastError();
}

int tc_kernels_per_segment() { return 2; }

cudaError_t launch_mse_tc(const DevState& s, const TcMaps& m, const TcInputMaps& in, const SegWork& w,
                          cudaStream_t st) {
    cudaError_t e = ensure_attrs();
    if (e != cudaSuccess) return e;
    const bool paper = s.mode == 1;
    ReadArgs a{};
    a.d_in = s.d_in; a.d_hid = s.d_hid; a.d_out = s.d_out; a.n_kv = s.n_kv;
    a.status = s.status;
    a.C = s.C; a.T = s.T; a.Tp = w.Tp; a.win = s.win_rows; a.parity = w.parity; a.renorm_pending = w.renorm_pending;
    a.tok0 = w.u_off; a.row0 = w.row0; a.n_rows = w.n_rows; a.y_cstride = w.y_cstride;
    a.zinv = paper ? s.zinv : nullptr;
    a.n1 = s.n1; a.n2 = s.n2; a.sumsq = s.sumsq;
    a.K = static_cast<const bf16*>(w.K); a.V = static_cast<const bf16*>(w.V);
    a.Kres = s.Kres; a.Vres = s.Vres;
    a.loss = w.loss;
    a.Aq = s.Amse;
    if (phase_a_pairs(s)) {  // phase A runs in its R-only form: write At and c SiLU'(x) / |z| here
        a.At = reinterpret_cast<bf16*>(s.Att);
        a.Sp = reinterpret_cast<bf16*>(s.dHt);
        a.paper = paper ? 1 : 0;
        a.lr = s.lr;
        a.eta = s.eta;
        a.eta_in = w.eta_in ? w.eta_in + w.row0 : nullptr;
        a.eta_cstride = w.eta_cstride;
    }
    // hidden: U rows of the segment (paper: the transformed window, absolute chain; plain: the
    // caller's X of the group), W1 of chain c0 + z
    a.a_row0 = paper ? (int)w.u_off : (int)w.row0;
    a.a_chain0 = paper ? w.c0 : 0;
    a.b_chain0 = w.c0;
    e = launch_read_kernel<MSE_HIDDEN>(dim3(s.T / 128, s.d_hid / 128, w.nc), paper ? m.Ua : in.Xa, m.W1b, a, st);
    if (e != cudaSuccess) return e;
    // out: the activations of the same chains (absolute), W2 MN-major
    a.a_row0 = 0;
    a.a_chain0 = w.c0;
    return launch_read_kernel<MSE_OUT>(dim3(s.T / 128, s.d_out / 128, w.nc), m.Amse, m.W2m, a, st);
}

cudaError_t launch_read_tc(const DevState& s, const TcMaps& m, const void* Xq, void* Uq, void* Aq, float* zq, int Q,
                           int n_layers, void* K_out, void* V_out, const long long* strides, cudaStream_t st) {
    cudaError_t e = ensure_attrs();
    if (e != cudaSuccess) return e;
    if (s.hd != 64 && s.hd != 128) return cudaErrorInvalidValue;
    // the query side: unnormalised z and 1/|z| for the read with the weights as M (Q <= 256),
    // the normalised u for the 128-query form
    if (Q <= RT_MAX_NT)
        e = launch_query_z(s, Xq, Q, Uq, zq, st);
    else
        e = launch_query_transform(s, Xq, Q, Uq, true, st);
    if (e != cudaSuccess) return e;
    CUtensorMap mu, ma;
    if (!encode_map_bf16_3d(&mu, Uq, s.d_in, Q, s.C, 64, 128) || !encode_map_bf16_3d(&ma, Aq, s.d_hid, Q, s.C, 64, 128))
        return cudaErrorInvalidValue;
    ReadArgs a{};
    a.Q = Q; a.d_in = s.d_in; a.d_hid = s.d_hid; a.d_out = s.d_out; a.n_kv = s.n_kv; a.L = n_layers;
    a.eps = s.rms_eps;
    a.gate = s.gate;
    a.Aq = static_cast<bf16*>(Aq);
    a.Kout = static_cast<bf16*>(K_out);
    a.Vout = static_cast<bf16*>(V_out);
    a.s0 = strides[0]; a.s1 = strides[1]; a.s2 = strides[2]; a.s3 = strides[3];
    a.status = s.status;
    if (Q <= RT_MAX_NT) {  // weights as the 128-row operand, the queries as N
        a.qzinv = s.mode == 1 ? zq : nullptr;
        const int NT = (Q + 31) / 32 * 32;
        CUtensorMap tu, ta;
        if (!encode_map_bf16_3d(&tu, Uq, s.d_in, Q, s.C, 64, NT) || !encode_map_bf16_3d(&ta, Aq, s.d_hid, Q, s.C, 64, NT))
            return cudaErrorInvalidValue;
        // programmatic stream serialisation: each kernel may start before the one it follows ends
        cudaLaunchConfig_t cfg = {};
        cudaLaunchAttribute at[1];
        at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        at[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.blockDim = dim3(RT_THREADS);
        cfg.stream = st;
        cfg.attrs = at;
        cfg.numAttrs = 1;
        // one CTA per SM with the deep ring when a kernel's tiles fit in one wave, else two
        const int ring1 = (long long)(s.d_hid / 128) * s.C <= g_sms ? RT_RING_1 : RT_RING_2;
        const int ring2 = (long long)(s.d_out / 128) * s.C <= g_sms ? RT_RING_1 : RT_RING_2;
        cfg.gridDim = dim3(1, s.d_hid / 128, s.C);
        cfg.dynamicSmemBytes = rt_dyn(NT, ring1);
        if ((e = cudaLaunchKernelEx(&cfg, tc_read_t_kernel<0>, m.W1b, tu, a, NT, ring1)) != cudaSuccess) return e;
        cfg.gridDim = dim3(1, s.d_out / 128, s.C);
        cfg.dynamicSmemBytes = rt_dyn(NT, ring2);
        if (s.hd == 64) return cudaLaunchKernelEx(&cfg, tc_read_t_kernel<64>, m.W2m, ta, a, NT, ring2);
        return cudaLaunchKernelEx(&cfg, tc_read_t_kernel<128>, m.W2m, ta, a, NT, ring2);
    }
    const int nq = (Q + 127) / 128;
    if ((e = launch_read_kernel<0>(dim3(nq, s.d_hid / 128, s.C), mu, m.W1b, a, st)) != cudaSuccess) return e;
    if (s.hd == 64) return launch_read_kernel<64>(dim3(nq, s.d_out / 128, s.C), ma, m.W2m, a, st);
    return launch_read_kernel<128>(dim3(nq, s.d_out / 128, s.C), ma, m.W2m, a, st);
}

// ------------------------------------------------------------------ tensor maps

namespace {
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn g_encode = nullptr;
std::once_flag g_encode_once;

EncodeTiledFn encoder() {
    std::call_once(g_encode_once, [] {
        void* fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            g_encode = reinterpret_cast<EncodeTiledFn>(fn);
    });
    return g_encode;
}
}  // namespace

bool encode_map_bf16_3d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t rows, uint64_t chains,
                        uint32_t box_inner, uint32_t box_rows) {
    if (!encoder() || !map) return false;
    const cuuint64_t dims[3] = {inner, rows, chains};
    const cuuint64_t strides[2] = {inner * 2, inner * rows * 2};
    const cuuint32_t box[3] = {box_inner, box_rows, 1};
    const cuuint32_t estr[3] = {1, 1, 1};
    return g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_map_bf16_4d(CUtensorMap* map, const void* base, const uint64_t dims[4], const uint64_t strides[3],
                        const uint32_t box[4]) {
    if (!encoder() || !map) return false;
    const cuuint64_t d[4] = {dims[0], dims[1], dims[2], dims[3]};
    const cuuint64_t st[3] = {strides[0], strides[1], strides[2]};
    const cuuint32_t b[4] = {box[0], box[1], box[2], box[3]};
    const cuuint32_t estr[4] = {1, 1, 1, 1};
    return g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), d, st, b, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_map_plain_3d(CUtensorMap* map, const void* base, bool f32, uint64_t inner, uint64_t rows,
                         uint64_t chains, uint32_t box_inner, uint32_t box_rows) {
    if (!encoder() || !map) return false;
    const uint64_t es = f32 ? 4 : 2;
    const cuuint64_t dims[3] = {inner, rows, chains};
    const cuuint64_t strides[2] = {inner * es, inner * rows * es};
    const cuuint32_t box[3] = {box_inner, box_rows, 1};
    const cuuint32_t estr[3] = {1, 1, 1};
    return g_encode(map, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3,
                    const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                    CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace mone
