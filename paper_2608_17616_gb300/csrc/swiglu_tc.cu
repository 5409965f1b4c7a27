// Per-head SwiGLU memory of Eq. 3 on the tensor cores (bf16 path, memory = MONE_MEM_SWIGLU).
//
// A chain (context, layer) splits its input u (width d = H * dh) into H heads.  Head h holds
// three matrices over its slice u_h, rows = hidden units as Eq. 3 stores them:
//     P = u_h Win^T,  G = u_h Wg^T   (F hidden units),   Z = SiLU(P) * G,   O_h = Z Wout,
// Win, Wg, Wout [F][dh]; the output is the concatenation of the heads' O_h (width d).  The
// state keeps W1 = [Win; Wg] ([C][H][2F][dh]) and W2 = Wout ([C][H][F][dh]).  With
// dL/dO = -eta Y / T' (Eq. 7; independent of W), R = Y_h Wout^T and c_t = -eta_t / T':
//     dP = c R * G * SiLU'(P),  dG = c R * SiLU(P),
//     grad Win = dP^T u_h,  grad Wg = dG^T u_h,  grad Wout = (c Z)^T Y_h,
// then the same update as the two-matrix memory (momentum, W -= mu, row renormalisation).
//
// Kernels, one tile per CTA (warp 0 TMA producer, warp 1 MMA issuer, warps 2..5 epilogue,
// one TMEM lane quarter each):
//   swiglu_a_kernel  tile (128 tokens, 128 hidden units, head).  One N = 256 MMA per k-step
//                    over [Win rows; Wg rows] gives P | G, then R over Y_h.  The epilogue applies
//                    the pending renorm scales and 1/|z_t| and writes (1/|z|) c dP, (1/|z|) c dG
//                    and c Z in bf16.
//   swiglu_b_kernel  tile (matrix, 128 weight columns, 128 hidden rows, head): the gradient with
//                    TMEM lane = weight column (both operands MN-major), then the fused update
//                    against global memory (coalesced rows), bf16 copy and row sums of squares.
//   swiglu_rh_kernel / swiglu_ro_kernel   the memory read: Z_q = SiLU(u Win^T) * (u Wg^T),
//                    O = Z_q Wout into fp32 scratch (the per-head RMS norm follows on the read's
//                    norm kernel, since an output head of width hd may straddle two memory heads).
// Head slices of [..][H * dh] rows are 4-D tensor maps (dh, heads, rows, chains): a box that
// runs past a head's dh columns, or past F hidden rows, reads zeros.
#include <mutex>

#include "mone_common.cuh"

namespace mone {

namespace {

constexpr int SW_THREADS = 6 * 32;
constexpr int SW_BOX = 64 * 64 * 2;      // one 64 x 64 MN-major box
constexpr uint32_t SW_EPI_BAR = 1;

// Shared memory of one CTA: a ring of STAGES operand stages, then barriers (full[S] empty[S]
// tfull tempty), the TMEM slot, a flag, scale tables and (with STG) 4 epilogue warps x 2 KB
// transpose buffers.
template <int STAGES, int STAGE_BYTES, bool STG_BUFS>
struct SwLayoutT {
    static constexpr int NSTAGES = STAGES;
    static constexpr int RING = STAGES * STAGE_BYTES;
    static constexpr int BARS = RING;
    static constexpr int SLOT = BARS + ((2 * STAGES + 2) * 8 + 15) / 16 * 16;
    static constexpr int FLAG = SLOT + 16;
    static constexpr int TAB = FLAG + 16;          // up to 3 x 128 scales (+ reduction scratch)
    static constexpr int STG = TAB + 512 * 4;
    static constexpr int END = STG + (STG_BUFS ? 4 * 2048 : 0);
    static constexpr int DYN = END + 1024;
};
// phase A and the read kernels: 4 stages of up to 48 KB (A tile 16 KB + up to 32 KB of B)
using SwLayout = SwLayoutT<4, 48 * 1024, true>;
static_assert(SwLayout::DYN <= 227 * 1024, "shared memory budget");

struct SwArgs {
    int H, Hk, dh, F, T, Tp, C, c0, paper, momentum, renorm_pending, parity, win;
    long long tok0;          // token table offset of the segment in the window scratch
    int u_row0, u_chain0, y_row0;
    float lr;
    const float *eta, *dbeta, *zinv, *b_beta, *eta_in;
    long long eta_cstride;
    float *W1, *W2, *mu1, *mu2;
    bf16 *W1b, *W2b;
    float *n1, *n2;          // renormalisation targets [C*H][2F], [C*H][F]
    float* sumsq;            // [2 parity][2 matrix][C*H][2F]
    bf16 *dPG, *Zt;          // [C*H][T][2F], [C*H][T][F]
    float* loss;             // [nc] or null
    float* step_sq;          // [nc] squared norm of this segment's Eq. 8 step (phase B), or null
    int* status;
    // memory read
    int Q, d_out;
    int nc_launch;           // chains of this launch (persistent phase A)
    bf16* Zq;                // [C*H][Q][F]
    float* Oq;               // [C][Q][d_out]
};

__device__ __forceinline__ float* sw_ss(const SwArgs& a, int parity, int which, int ch) {
    return a.sumsq + ((size_t)(parity * 2 + which) * a.C * a.H + ch) * (2 * a.F);
}

template <class L>
struct SwCtl {
    uint8_t* base;
    uint32_t bars;
    __device__ uint32_t full(int s) const { return bars + 8 * s; }
    __device__ uint32_t empty(int s) const { return bars + 8 * (L::NSTAGES + s); }
    __device__ uint32_t tfull() const { return bars + 8 * (2 * L::NSTAGES); }
    __device__ uint32_t tempty() const { return bars + 8 * (2 * L::NSTAGES + 1); }
};

template <class L = SwLayout>
__device__ __forceinline__ SwCtl<L> sw_setup(uint8_t* raw, uint32_t tmem_cols) {
    SwCtl<L> c;
    c.base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(raw) + 1023) & ~uintptr_t(1023));
    c.bars = smem_u32(c.base + L::BARS);
    if (threadIdx.x == 0) {
        for (int s = 0; s < L::NSTAGES; ++s) {
            mbar_init(c.full(s), 1);
            mbar_init(c.empty(s), 1);
        }
        mbar_init(c.tfull(), 1);
        mbar_init(c.tempty(), 4);  // the four epilogue warps (persistent phase A)
        fence_mbar_init();
    }
    if (threadIdx.x / 32 == 0) {
        tmem_alloc(smem_u32(c.base + L::SLOT), tmem_cols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    return c;
}

__device__ __forceinline__ void sw_teardown(uint32_t tmem, uint32_t cols) {
    tc_fence_before();
    __syncthreads();
    if (threadIdx.x / 32 == 0) tmem_dealloc(tmem, cols);
}

// Epilogue entry: thread 64 waits for the accumulator, every epilogue warp learns the outcome.
template <class L>
__device__ __forceinline__ bool sw_wait_acc(const SwCtl<L>& c, int* status) {
    int* flag = reinterpret_cast<int*>(c.base + L::FLAG);
    if (threadIdx.x == 64) *flag = mbar_wait(c.tfull(), 0, status) ? 1 : 0;
    __syncwarp();
    named_bar_sync(SW_EPI_BAR, 128);
    const bool ok = *flag != 0;
    if (ok) tc_fence_after();
    return ok;
}

// ------------------------------------------------------------------ phase A (forward + backward epilogue)

// Persistent: at most one CTA per SM walks the tiles (128 tokens, 128 hidden units, head) of
// the launch.  The producer runs ahead into the next tile's operands while the epilogue
// drains the current one; the MMA warp waits for the epilogue to hand the accumulator back
// (tempty) before it starts the next tile.  (Two accumulator buffers would need 768 TMEM
// columns; 64-unit tiles that fit two buffers reload U and Y twice as often and measured
// slower.)
__global__ void __launch_bounds__(SW_THREADS, 1)
swiglu_a_kernel(const __grid_constant__ CUtensorMap tmU, const __grid_constant__ CUtensorMap tmK,
                const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmW1,
                const __grid_constant__ CUtensorMap tmW2, const SwArgs a) {
    extern __shared__ uint8_t smem_raw[];
    const auto c = sw_setup(smem_raw, 512);
    const uint32_t tmem = *reinterpret_cast<uint32_t*>(c.base + SwLayout::SLOT);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int KU = (a.dh + 63) / 64, KB = 2 * KU;
    const int n_tt = a.T / 128, n_ft = (a.F + 127) / 128;
    const int ntiles = n_tt * n_ft * a.nc_launch * a.H;
    // tile -> (token tile, hidden tile, chain-head of the launch)
    auto decode = [&](int tile, int& t0, int& f0, int& cz, int& h) {
        const int zh = tile / (n_tt * n_ft), r = tile % (n_tt * n_ft);
        f0 = (r / n_tt) * 128;
        t0 = (r % n_tt) * 128;
        cz = zh / a.H;
        h = zh % a.H;
    };

    if (warp == 0) {
        if (lane == 0) {
            uint32_t kc = 0;
            bool ok = true;
            for (int tile = blockIdx.x; tile < ntiles && ok; tile += gridDim.x) {
                int t0, f0, cz, h;
                decode(tile, t0, f0, cz, h);
                const int ch = (a.c0 + cz) * a.H + h;
                for (int kb = 0; kb < KB; ++kb, ++kc) {
                    const int s = kc % SwLayout::NSTAGES;
                    if (kc >= SwLayout::NSTAGES &&
                        !mbar_wait(c.empty(s), ((kc / SwLayout::NSTAGES) - 1) & 1, a.status)) {
                        ok = false;
                        break;
                    }
                    const uint32_t sa = smem_u32(c.base + s * (48 * 1024)), sb = sa + 128 * 128, fb = c.full(s);
                    if (kb < KU) {
                        mbar_expect_tx(fb, 3 * 128 * 128);
                        tma_load_4d(sa, &tmU, fb, kb * 64, h, a.u_row0 + t0, a.u_chain0 + cz);
                        tma_load_4d(sb, &tmW1, fb, kb * 64, f0, 0, ch);             // Win rows
                        tma_load_4d(sb + 128 * 128, &tmW1, fb, kb * 64, f0, 1, ch);  // Wg rows
                    } else {
                        const int k2 = kb - KU;
                        mbar_expect_tx(fb, 2 * 128 * 128);
                        if (h < a.Hk)
                            tma_load_4d(sa, &tmK, fb, k2 * 64, h, a.y_row0 + t0, cz);
                        else
                            tma_load_4d(sa, &tmV, fb, k2 * 64, h - a.Hk, a.y_row0 + t0, cz);
                        tma_load_3d(sb, &tmW2, fb, k2 * 64, f0, ch);                 // Wout rows
                    }
                }
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            const uint32_t id_pg = idesc_bf16_f32(128, 256, false, false), id_r = idesc_bf16_f32(128, 128, false, false);
            uint32_t kc = 0;
            int local = 0;
            bool ok = true;
            for (int tile = blockIdx.x; tile < ntiles && ok; tile += gridDim.x, ++local) {
                if (local >= 1 && !mbar_wait(c.tempty(), (local - 1) & 1, a.status)) break;
                tc_fence_after();
                for (int kb = 0; kb < KB; ++kb, ++kc) {
                    const int s = kc % SwLayout::NSTAGES;
                    if (!mbar_wait(c.full(s), (kc / SwLayout::NSTAGES) & 1, a.status)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t sa = smem_u32(c.base + s * (48 * 1024)), sb = sa + 128 * 128;
                    const bool u_part = kb < KU;
    #pragma unroll
                    for (int k = 0; k < 4; ++k)
                        umma_bf16(u_part ? tmem : tmem + 256, sdesc_sw128(sa + k * 32, 16), sdesc_sw128(sb + k * 32, 16),
                                  u_part ? id_pg : id_r, ((kb == 0 || kb == KU) && k == 0) ? 0u : 1u);
                    umma_commit(c.empty(s));
                }
                if (ok) umma_commit(c.tfull());
            }
        }
        __syncwarp();
    } else {
        const int q = warp & 3, et = threadIdx.x - 64;
        float* tab = reinterpret_cast<float*>(c.base + SwLayout::TAB);  // s_in[128] s_g[128] s_out[128]
        int* flag = reinterpret_cast<int*>(c.base + SwLayout::FLAG);
        int local = 0;
        for (int tile = blockIdx.x; tile < ntiles; tile += gridDim.x, ++local) {
            int t0, f0, cz, h;
            decode(tile, t0, f0, cz, h);
            const int cs = a.c0 + cz, ch = cs * a.H + h;
            {
                const int f = f0 + et;
                float si = 1.f, sg = 1.f, so = 1.f;
                if (f < a.F) {
                    if (a.renorm_pending) {
                        si = renorm_scale(a.n1[(size_t)ch * 2 * a.F + f], sw_ss(a, a.parity ^ 1, 0, ch)[f]);
                        sg = renorm_scale(a.n1[(size_t)ch * 2 * a.F + a.F + f], sw_ss(a, a.parity ^ 1, 0, ch)[a.F + f]);
                        so = renorm_scale(a.n2[(size_t)ch * a.F + f], sw_ss(a, a.parity ^ 1, 1, ch)[f]);
                    }
                    if (t0 == 0) {  // this segment's row sums of squares start from zero
                        sw_ss(a, a.parity, 0, ch)[f] = 0.f;
                        sw_ss(a, a.parity, 0, ch)[a.F + f] = 0.f;
                        sw_ss(a, a.parity, 1, ch)[f] = 0.f;
                    }
                }
                tab[et] = si;
                tab[128 + et] = sg;
                tab[256 + et] = so;
            }
            if (et == 0) *flag = mbar_wait(c.tfull(), local & 1, a.status) ? 1 : 0;
            __syncwarp();
            named_bar_sync(SW_EPI_BAR, 128);
            if (!*flag) break;
            tc_fence_after();
            {
                const int t = t0 + q * 32 + lane;
                float ct = 0.f, zi = 1.f;
                if (t < a.Tp) {
                    const float ev = a.paper ? a.eta[(size_t)cs * a.win + a.tok0 + t]
                                             : (a.eta_in ? a.eta_in[cz * a.eta_cstride + t] : a.lr);
                    ct = -ev / (float)a.Tp;
                    if (a.zinv) zi = a.zinv[(size_t)cs * a.win + a.tok0 + t];
                }
                const float czi = ct * zi;
                const uint32_t lane_base = tmem + ((uint32_t)(q * 32) << 16);
                uint8_t* stg = c.base + SwLayout::STG + (warp - 2) * 2048;
                const size_t rowoff = (size_t)ch * a.T + t0 + q * 32;  // first token row of this warp
                float lsum = 0.f;
    #pragma unroll 1
                for (int cc = 0; cc < 4 && f0 + cc * 32 < a.F; ++cc) {
                    const int fb = cc * 32;
                    float pv[32], gv[32], rv[32];
                    tmem_ld32(lane_base + fb, pv);
                    tmem_ld32(lane_base + 128 + fb, gv);
                    tmem_ld32(lane_base + 256 + fb, rv);
                    uint32_t pd[16], pg[16], pz[16];
    #pragma unroll
                    for (int j = 0; j < 32; j += 2) {
                        float d0[2], d1[2], d2[2];
    #pragma unroll
                        for (int u = 0; u < 2; ++u) {
                            const int k = fb + j + u;
                            const float x = pv[j + u] * tab[k] * zi;
                            const float g = gv[j + u] * tab[128 + k] * zi;
                            const float r = rv[j + u] * tab[256 + k];
                            const float sgm = sigmoid_tanh(x);
                            const float sl = x * sgm;
                            lsum = fmaf(sl * g, r, lsum);
                            d0[u] = czi * r * g * (sgm * fmaf(x, 1.f - sgm, 1.f));  // (1/|z|) c dP
                            d1[u] = czi * r * sl;                                   // (1/|z|) c dG
                            d2[u] = ct * sl * g;                                    // c Z
                        }
                        pd[j / 2] = pack_bf16(d0[0], d0[1]);
                        pg[j / 2] = pack_bf16(d1[0], d1[1]);
                        pz[j / 2] = pack_bf16(d2[0], d2[1]);
                    }
                    store_rows_coalesced(stg, pd, a.dPG + rowoff * 2 * a.F + f0 + fb, 2 * a.F, lane);
                    store_rows_coalesced(stg, pg, a.dPG + rowoff * 2 * a.F + a.F + f0 + fb, 2 * a.F, lane);
                    store_rows_coalesced(stg, pz, a.Zt + rowoff * a.F + f0 + fb, a.F, lane);
                }
                // every TMEM read of this tile is done: hand the accumulator back to the MMA warp
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(c.tempty());
                if (a.loss) {
                    lsum = warp_sum(lsum);
                    if (lane == 0) atomicAdd(&a.loss[cz], -lsum / (float)a.Tp);
                }
            }
            // the scale table and flag are rewritten for the next tile only after every warp is done
            named_bar_sync(SW_EPI_BAR, 128);
        }
    }
    sw_teardown(tmem, 512);
}

// ------------------------------------------------------------------ phase B (gradient + update)

// Persistent, one CTA per SM, over tiles (matrix m of W_in / W_gate / W_out, 256 hidden rows,
// 128 weight columns, head): the gradient with TMEM lane = weight column (both operands
// MN-major) into one of two TMEM accumulators, so the MMAs of tile i+1 run while tile i is
// updated.  Warps: 0 operand producer, 1 MMA issuer, 2..9 update in two groups of four (one warp
// per TMEM lane quarter), 10 state producer, 11 store warp.  The fp32 state of a tile moves in
// chunks of 32 rows x 128 columns (W and mu) through a 4-slot shared-memory ring: the state
// producer TMA-loads chunks ahead, the two groups update alternate chunks in place, the store
// warp TMA-stores them back and frees the slot.  Chunks whose rows lie past F are skipped
// (F is a multiple of 32); columns past dh load as zeros, are clipped from the stores and
// masked from the bf16 copy.
constexpr int SWB_ROWS = 32;                               // hidden rows per state chunk
constexpr int SWB_SLOTS = 4;
constexpr int SWB_F32 = SWB_ROWS * 128 * 4;                // 16 KB
constexpr int SWB_SLOT = 2 * SWB_F32;                      // W and mu: 32 KB
constexpr int SWB_N = 256;                                 // hidden rows per tile (all of F <= 256)
constexpr int SWB_STAGES = 2;
constexpr int SWB_STAGE = (2 + SWB_N / 64) * SW_BOX;       // 48 KB: 128 columns + 256 hidden rows
constexpr int SWB_THREADS = 12 * 32;
constexpr int SWB_EPI_THREADS = 4 * 32;                    // per update group
constexpr int SWB_STATE_WARP = 10, SWB_STORE_WARP = 11;
struct SwLayoutB {
    static constexpr int RING = SWB_STAGES * SWB_STAGE;
    static constexpr int STATE = RING;
    static constexpr int BARS = STATE + SWB_SLOTS * SWB_SLOT;  // full[S] empty[S] tfull[2] tempty[2] sfull/sempty/sdone[N]
    static constexpr int NBARS = 2 * SWB_STAGES + 4 + 3 * SWB_SLOTS;
    static constexpr int SLOT = BARS + NBARS * 8;
    static constexpr int FLAG = SLOT + 16;
    static constexpr int TAB = FLAG + 16;                      // per group: [SWB_N/2] renorm scales + [4] decay partials
    static constexpr int END = TAB + 2 * (SWB_N / 2 + 4) * 4;
    static constexpr int DYN = END + 1024;
};
static_assert(SwLayoutB::DYN <= 227 * 1024, "phase B shared memory budget");

// The tiles of a launch: t -> (chain-head of the launch, matrix, first hidden row, first column).
struct SwBTiles {
    int NC, NR, count;
    __device__ SwBTiles(const SwArgs& a) {
        NC = (a.dh + 127) / 128;
        NR = (a.F + SWB_N - 1) / SWB_N;
        count = a.nc_launch * a.H * 3 * NR * NC;
    }
    __device__ void decode(int t, int& zh, int& m, int& f0, int& col0) const {
        col0 = (t % NC) * 128;
        t /= NC;
        f0 = (t % NR) * SWB_N;
        t /= NR;
        m = t % 3;
        zh = t / 3;
    }
};

// STEP: also sum |mu_s|^2 per chain (the per-segment metrics), in a separate instance
template <bool STEP>
__global__ void __launch_bounds__(SWB_THREADS, 1)
swiglu_b_kernel(const __grid_constant__ CUtensorMap tmUb, const __grid_constant__ CUtensorMap tmKb,
                const __grid_constant__ CUtensorMap tmVb, const __grid_constant__ CUtensorMap tmPG,
                const __grid_constant__ CUtensorMap tmZ, const __grid_constant__ CUtensorMap tmW1s,
                const __grid_constant__ CUtensorMap tmM1s, const __grid_constant__ CUtensorMap tmW2s,
                const __grid_constant__ CUtensorMap tmM2s, const SwArgs a) {
    using L = SwLayoutB;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const uint32_t bars = smem_u32(base + L::BARS);
    auto full = [&](int s) { return bars + 8 * s; };
    auto empty = [&](int s) { return bars + 8 * (SWB_STAGES + s); };
    auto tfull = [&](int b) { return bars + 8 * (2 * SWB_STAGES + b); };
    auto tempty = [&](int b) { return bars + 8 * (2 * SWB_STAGES + 2 + b); };
    auto sfull = [&](int k) { return bars + 8 * (2 * SWB_STAGES + 4 + k); };
    auto sempty = [&](int k) { return bars + 8 * (2 * SWB_STAGES + 4 + SWB_SLOTS + k); };
    auto sdone = [&](int k) { return bars + 8 * (2 * SWB_STAGES + 4 + 2 * SWB_SLOTS + k); };
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const SwBTiles tl(a);
    if (threadIdx.x == 0) {
        for (int i = 0; i < SWB_STAGES; ++i) {
            mbar_init(full(i), 1);
            mbar_init(empty(i), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(tfull(b), 1);
            mbar_init(tempty(b), 8);  // every update warp, once per tile
        }
        for (int k = 0; k < SWB_SLOTS; ++k) {
            mbar_init(sfull(k), 1);
            mbar_init(sempty(k), 1);
            mbar_init(sdone(k), 4);  // the four warps of the group that updated the chunk
        }
        fence_mbar_init();
    }
    if (warp == 0) {
        tmem_alloc(smem_u32(base + L::SLOT), 2 * SWB_N);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *reinterpret_cast<uint32_t*>(base + L::SLOT);
    const int KB = (a.Tp + 63) / 64;  // tokens beyond T' carry zero gradients
    const int chunk_bytes = a.momentum ? 2 * SWB_F32 : SWB_F32;
    // state chunks of a tile: the rows of f0 .. f0 + SWB_N - 1 that lie below F
    auto nchunks = [&](int f0) { return min(SWB_N, a.F - f0) / SWB_ROWS; };

    if (warp == 0) {
        if (lane == 0) {
            uint32_t kc = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < tl.count && ok; t += gridDim.x) {
                int zh, m, f0, col0;
                tl.decode(t, zh, m, f0, col0);
                const int cz = zh / a.H, h = zh % a.H, ch = (a.c0 + cz) * a.H + h;
                for (int kb = 0; kb < KB; ++kb, ++kc) {
                    const int s = kc % SWB_STAGES;
                    if (kc >= SWB_STAGES && !mbar_wait(empty(s), ((kc / SWB_STAGES) - 1) & 1, a.status)) {
                        ok = false;
                        break;
                    }
                    const uint32_t sa = smem_u32(base + s * SWB_STAGE), sb = sa + 2 * SW_BOX, fb = full(s);
                    mbar_expect_tx(fb, SWB_STAGE);
#pragma unroll
                    for (int bx = 0; bx < 2; ++bx) {
                        const uint32_t dst = sa + bx * SW_BOX;
                        if (m < 2)
                            tma_load_4d(dst, &tmUb, fb, col0 + bx * 64, h, a.u_row0 + kb * 64, a.u_chain0 + cz);
                        else if (h < a.Hk)
                            tma_load_4d(dst, &tmKb, fb, col0 + bx * 64, h, a.y_row0 + kb * 64, cz);
                        else
                            tma_load_4d(dst, &tmVb, fb, col0 + bx * 64, h - a.Hk, a.y_row0 + kb * 64, cz);
                    }
#pragma unroll
                    for (int bx = 0; bx < SWB_N / 64; ++bx) {  // hidden rows past F load as zeros
                        if (m < 2)
                            tma_load_4d(sb + bx * SW_BOX, &tmPG, fb, f0 + bx * 64, m, kb * 64, ch);
                        else
                            tma_load_3d(sb + bx * SW_BOX, &tmZ, fb, f0 + bx * 64, kb * 64, ch);
                    }
                }
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16_f32(128, SWB_N, true, true);
            uint32_t kc = 0;
            int local = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < tl.count && ok; t += gridDim.x, ++local) {
                const int b = local & 1;
                if (local >= 2 && !mbar_wait(tempty(b), ((local >> 1) - 1) & 1, a.status)) break;
                tc_fence_after();
                const uint32_t d = tmem + b * SWB_N;
                for (int kb = 0; kb < KB; ++kb, ++kc) {
                    const int s = kc % SWB_STAGES;
                    if (!mbar_wait(full(s), (kc / SWB_STAGES) & 1, a.status)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t sa = smem_u32(base + s * SWB_STAGE), sb = sa + 2 * SW_BOX;
#pragma unroll
                    for (int k = 0; k < 4; ++k)
                        umma_bf16(d, sdesc_sw128(sa + k * 16 * 128, SW_BOX), sdesc_sw128(sb + k * 16 * 128, SW_BOX),
                                  idesc, (kb == 0 && k == 0) ? 0u : 1u);
                    umma_commit(empty(s));
                }
                if (ok) umma_commit(tfull(b));
            }
        }
        __syncwarp();
    } else if (warp == SWB_STATE_WARP || warp == SWB_STORE_WARP) {
        // ---- state producer (W and mu chunks of every tile, in update order) and store warp
        //      (write each updated chunk back, then free its slot)
        if (lane == 0) {
            const bool producer = warp == SWB_STATE_WARP;
            if (producer) {
                tma_prefetch_map(&tmW1s);
                tma_prefetch_map(&tmW2s);
                if (a.momentum) {
                    tma_prefetch_map(&tmM1s);
                    tma_prefetch_map(&tmM2s);
                }
            }
            uint32_t seq = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < tl.count && ok; t += gridDim.x) {
                int zh, m, f0, col0;
                tl.decode(t, zh, m, f0, col0);
                const int ch = (a.c0 + zh / a.H) * a.H + zh % a.H;
                const CUtensorMap* wm = m < 2 ? &tmW1s : &tmW2s;
                const CUtensorMap* mm = m < 2 ? &tmM1s : &tmM2s;
                const int row0 = (m == 1 ? a.F : 0) + f0;  // first state row of the tile within the head
                const int nch = nchunks(f0);
                for (int g = 0; g < nch; ++g, ++seq) {
                    const int k = seq % SWB_SLOTS;
                    const uint32_t slot = smem_u32(base + L::STATE + k * SWB_SLOT);
                    if (producer) {
                        if (seq >= SWB_SLOTS && !mbar_wait(sempty(k), ((seq / SWB_SLOTS) - 1) & 1, a.status)) {
                            ok = false;
                            break;
                        }
                        mbar_expect_tx(sfull(k), chunk_bytes);
                        tma_load_3d(slot, wm, sfull(k), col0, row0 + g * SWB_ROWS, ch);
                        if (a.momentum) tma_load_3d(slot + SWB_F32, mm, sfull(k), col0, row0 + g * SWB_ROWS, ch);
                    } else {
                        if (!mbar_wait(sdone(k), (seq / SWB_SLOTS) & 1, a.status)) {
                            ok = false;
                            break;
                        }
                        tma_store_3d(wm, slot, col0, row0 + g * SWB_ROWS, ch);
                        if (a.momentum) tma_store_3d(mm, slot + SWB_F32, col0, row0 + g * SWB_ROWS, ch);
                        bulk_commit();
                        bulk_wait_read_all();  // the store has read the slot: hand it back
                        mbar_arrive(sempty(k));
                    }
                }
            }
            if (!producer) bulk_wait_all();
        }
        __syncwarp();
    } else {
        // ---- update warps 2..9: group grp takes the tile's chunks grp, grp + 2; TMEM lane
        //      quarter q = 32 weight columns, thread = one column
        const int grp = (warp - 2) >> 2, q = warp & 3, et = threadIdx.x - 64 - grp * SWB_EPI_THREADS;
        const uint32_t bar_id = 1 + grp;
        float* tab = reinterpret_cast<float*>(base + L::TAB) + grp * (SWB_N / 2 + 4);  // [SWB_N/2] scales
        float* bred = tab + SWB_N / 2;                                                  // [4]
        int* flag = reinterpret_cast<int*>(base + L::FLAG) + grp * 2;
        bool finite = true;
        float step = 0.f;        // sum of mu_s^2 over this thread's live elements of the current tile
        uint32_t tile_seq0 = 0;  // state chunk sequence number of the current tile's first chunk
        int local = 0;
        for (int t = blockIdx.x; t < tl.count; t += gridDim.x, ++local) {
            int zh, m, f0, col0;
            tl.decode(t, zh, m, f0, col0);
            const int cz = zh / a.H, cs = a.c0 + cz, ch = cs * a.H + zh % a.H;
            const int which = m < 2 ? 0 : 1;
            const int row0 = (m == 1 ? a.F : 0) + f0;   // first state row of the tile within the head
            const int nch = nchunks(f0);
            const int mine = (nch - grp + 1) / 2;         // this group's chunks: grp, grp + 2
            const int b = local & 1;
            {   // renorm scales of this group's chunks (32 rows each)
                const int i = et >> 5, j = et & 31;
                float sc = 1.f;
                if (i < mine && a.renorm_pending) {
                    const int r = row0 + (2 * i + grp) * SWB_ROWS + j;  // row within the head's matrix
                    const float n = which ? a.n2[(size_t)ch * a.F + r] : a.n1[(size_t)ch * 2 * a.F + r];
                    sc = renorm_scale(n, sw_ss(a, a.parity ^ 1, which, ch)[r]);
                }
                tab[et] = sc;  // i < SWB_N / 64: four chunks of this group at most
            }
            if (a.momentum) {
                float v = 0.f;
                for (int tk = et; tk < a.Tp; tk += SWB_EPI_THREADS) v += a.dbeta[(size_t)cs * a.win + a.tok0 + tk];
                v = warp_sum(v);
                if (lane == 0) bred[q] = v;
            }
            if (et == 0) flag[0] = mbar_wait(tfull(b), (local >> 1) & 1, a.status) ? 1 : 0;
            __syncwarp();
            named_bar_sync(bar_id, SWB_EPI_THREADS);
            if (!flag[0]) break;
            tc_fence_after();
            float beta = 0.f;
            if (a.momentum) beta = sigmoidf_((bred[0] + bred[1] + bred[2] + bred[3]) / (float)a.Tp + a.b_beta[cs]);
            float* cur = sw_ss(a, a.parity, which, ch);
            const int col = q * 32 + lane;  // column within the tile (= TMEM lane)
            const bool live = col0 + col < a.dh;
            const size_t rows_head = which ? a.F : 2 * a.F;
            bf16* Wb = (which ? a.W2b : a.W1b) + (size_t)ch * rows_head * a.dh + col0 + col;
            const uint64_t wpol = l2_evict_last_policy();  // phase A of the next segment reads the copy
            const uint32_t lane_base = tmem + ((uint32_t)(q * 32) << 16) + b * SWB_N;
            if (mine == 0) {  // a group without chunks still hands the accumulator back
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(tempty(b));
            }
            bool ok = true;
#pragma unroll 1
            for (int i = 0; i < mine; ++i) {
                const int c = 2 * i + grp;
                const uint32_t seq = tile_seq0 + c;
                const int k = seq % SWB_SLOTS;
                const int r0 = row0 + c * SWB_ROWS;
                float gv[32];
                tmem_ld32(lane_base + c * SWB_ROWS, gv);
                if (i == mine - 1) {
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(tempty(b));
                }
                if (et == 0) flag[1] = mbar_wait(sfull(k), (seq / SWB_SLOTS) & 1, a.status) ? 1 : 0;
                __syncwarp();
                named_bar_sync(bar_id, SWB_EPI_THREADS);
                if (!flag[1]) {
                    ok = false;
                    break;
                }
                uint8_t* slot = base + L::STATE + k * SWB_SLOT;
                float* Ws = reinterpret_cast<float*>(slot);
                float* Ms = reinterpret_cast<float*>(slot + SWB_F32);
                bf16* bp = Wb + (size_t)r0 * a.dh;
                float v[32];
#pragma unroll
                for (int j = 0; j < 32; ++j) {
                    const float sc = tab[i * SWB_ROWS + j];
                    const float mo = a.momentum ? Ms[j * 128 + col] : 0.f;
                    const float mn = fmaf(beta, mo, gv[j]);
                    const float wn = fmaf(sc, Ws[j * 128 + col], -mn);
                    Ws[j * 128 + col] = wn;
                    if (a.momentum) Ms[j * 128 + col] = mn;
                    if (live) st_bf16_hint(bp + (size_t)j * a.dh, __float2bfloat16_rn(wn), wpol);
                    if constexpr (STEP) step = live ? fmaf(mn, mn, step) : step;
                    v[j] = wn * wn;  // columns past dh hold zeros; a NaN or Inf makes its row's sum non-finite
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
                atomicAdd(&cur[r0 + lane], v[0]);
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
            tile_seq0 += nch;
            // the scale table is rewritten for the next tile only after every warp of the group is done
            named_bar_sync(bar_id, SWB_EPI_THREADS);
        }
        if (!finite) atomicOr(a.status, DEV_NONFINITE);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tmem, 2 * SWB_N);
}

// ------------------------------------------------------------------ memory read

// Z_q = SiLU(u_h Win^T) * (u_h Wg^T): tile (128 queries, 128 hidden units, head).
__global__ void __launch_bounds__(SW_THREADS, 1)
swiglu_rh_kernel(const __grid_constant__ CUtensorMap tmU, const __grid_constant__ CUtensorMap tmW1, const SwArgs a) {
    extern __shared__ uint8_t smem_raw[];
    const auto c = sw_setup(smem_raw, 256);
    const uint32_t tmem = *reinterpret_cast<uint32_t*>(c.base + SwLayout::SLOT);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int q0 = blockIdx.x * 128, f0 = blockIdx.y * 128;
    const int cl = blockIdx.z / a.H, h = blockIdx.z % a.H, ch = blockIdx.z;
    const int KB = (a.dh + 63) / 64;
    if (warp == 0) {
        if (lane == 0) {
            for (int kb = 0; kb < KB; ++kb) {
                const int s = kb % SwLayout::NSTAGES;
                if (kb >= SwLayout::NSTAGES && !mbar_wait(c.empty(s), ((kb / SwLayout::NSTAGES) - 1) & 1, a.status)) break;
                const uint32_t sa = smem_u32(c.base + s * (48 * 1024)), sb = sa + 128 * 128, fb = c.full(s);
                mbar_expect_tx(fb, 3 * 128 * 128);
                tma_load_4d(sa, &tmU, fb, kb * 64, h, q0, cl);
                tma_load_4d(sb, &tmW1, fb, kb * 64, f0, 0, ch);
                tma_load_4d(sb + 128 * 128, &tmW1, fb, kb * 64, f0, 1, ch);
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16_f32(128, 256, false, false);
            bool ok = true;
            for (int kb = 0; kb < KB; ++kb) {
                const int s = kb % SwLayout::NSTAGES;
                if (!mbar_wait(c.full(s), (kb / SwLayout::NSTAGES) & 1, a.status)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t sa = smem_u32(c.base + s * (48 * 1024)), sb = sa + 128 * 128;
#pragma unroll
                for (int k = 0; k < 4; ++k)
                    umma_bf16(tmem, sdesc_sw128(sa + k * 32, 16), sdesc_sw128(sb + k * 32, 16), idesc,
                              (kb == 0 && k == 0) ? 0u : 1u);
                umma_commit(c.empty(s));
            }
            if (ok) umma_commit(c.tfull());
        }
        __syncwarp();
    } else {
        const int q = warp & 3;
        if (sw_wait_acc(c, a.status)) {
            const uint32_t lane_base = tmem + ((uint32_t)(q * 32) << 16);
            uint8_t* stg = c.base + SwLayout::STG + (warp - 2) * 2048;
            const int qw = q0 + q * 32;
#pragma unroll 1
            for (int cc = 0; cc < 4 && f0 + cc * 32 < a.F; ++cc) {
                float pv[32], gv[32];
                tmem_ld32(lane_base + cc * 32, pv);
                tmem_ld32(lane_base + 128 + cc * 32, gv);
                uint32_t pk[16];
#pragma unroll
                for (int j = 0; j < 16; ++j)
                    pk[j] = pack_bf16(pv[2 * j] * sigmoidf_(pv[2 * j]) * gv[2 * j],
                                      pv[2 * j + 1] * sigmoidf_(pv[2 * j + 1]) * gv[2 * j + 1]);
                store_rows_coalesced(stg, pk, a.Zq + ((size_t)ch * a.Q + qw) * a.F + f0 + cc * 32, a.F, lane, a.Q - qw);
            }
        }
    }
    sw_teardown(tmem, 256);
}

// O_h = Z_q Wout into the fp32 read scratch: tile (128 queries, 128 outputs of the head, head).
__global__ void __launch_bounds__(SW_THREADS, 1)
swiglu_ro_kernel(const __grid_constant__ CUtensorMap tmZ, const __grid_constant__ CUtensorMap tmW2m, const SwArgs a) {
    extern __shared__ uint8_t smem_raw[];
    const auto c = sw_setup(smem_raw, 128);
    const uint32_t tmem = *reinterpret_cast<uint32_t*>(c.base + SwLayout::SLOT);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int q0 = blockIdx.x * 128, o0 = blockIdx.y * 128;
    const int cl = blockIdx.z / a.H, h = blockIdx.z % a.H, ch = blockIdx.z;
    const int KB = (a.F + 63) / 64;
    if (warp == 0) {
        if (lane == 0) {
            for (int kb = 0; kb < KB; ++kb) {
                const int s = kb % SwLayout::NSTAGES;
                if (kb >= SwLayout::NSTAGES && !mbar_wait(c.empty(s), ((kb / SwLayout::NSTAGES) - 1) & 1, a.status)) break;
                const uint32_t sa = smem_u32(c.base + s * (48 * 1024)), sb = sa + 128 * 128, fb = c.full(s);
                mbar_expect_tx(fb, 128 * 128 + 2 * SW_BOX);
                tma_load_3d(sa, &tmZ, fb, kb * 64, q0, ch);
                tma_load_3d(sb, &tmW2m, fb, o0, kb * 64, ch);
                tma_load_3d(sb + SW_BOX, &tmW2m, fb, o0 + 64, kb * 64, ch);
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16_f32(128, 128, false, true);
            bool ok = true;
            for (int kb = 0; kb < KB; ++kb) {
                const int s = kb % SwLayout::NSTAGES;
                if (!mbar_wait(c.full(s), (kb / SwLayout::NSTAGES) & 1, a.status)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t sa = smem_u32(c.base + s * (48 * 1024)), sb = sa + 128 * 128;
#pragma unroll
                for (int k = 0; k < 4; ++k)
                    umma_bf16(tmem, sdesc_sw128(sa + k * 32, 16), sdesc_sw128(sb + k * 16 * 128, SW_BOX), idesc,
                              (kb == 0 && k == 0) ? 0u : 1u);
                umma_commit(c.empty(s));
            }
            if (ok) umma_commit(c.tfull());
        }
        __syncwarp();
    } else {
        const int q = warp & 3;
        if (sw_wait_acc(c, a.status)) {
            const uint32_t lane_base = tmem + ((uint32_t)(q * 32) << 16);
            const int qi = q0 + q * 32 + lane;
#pragma unroll 1
            for (int cc = 0; cc < 4 && o0 + cc * 32 < a.dh; ++cc) {
                float ov[32];
                tmem_ld32(lane_base + cc * 32, ov);
                if (qi < a.Q) {
                    float* out = a.Oq + ((size_t)cl * a.Q + qi) * a.d_out + (size_t)h * a.dh + o0 + cc * 32;
#pragma unroll
                    for (int j = 0; j < 32; j += 4) *reinterpret_cast<float4*>(out + j) = make_float4(ov[j], ov[j + 1], ov[j + 2], ov[j + 3]);
                }
            }
        }
    }
    sw_teardown(tmem, 128);
}

// ------------------------------------------------------------------ row upkeep (CUDA cores)

// One warp per state row (rows of W1 = [Win; Wg], then of W2 = Wout, per head), 8 rows a block.
// mode 0: renormalisation target n = |row| (init); 1: apply the pending row scale; 2: none.
// Every mode rewrites the row's bf16 operand copy.
__global__ void __launch_bounds__(256) swiglu_rows_kernel(SwArgs a, int mode, int parity) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int r = blockIdx.x * 8 + warp, ch = a.c0 * a.H + blockIdx.y, which = blockIdx.z;
    const int rows = which ? a.F : 2 * a.F;
    if (r >= rows) return;
    float* W = (which ? a.W2 : a.W1) + ((size_t)ch * rows + r) * a.dh;
    bf16* Wb = (which ? a.W2b : a.W1b) + ((size_t)ch * rows + r) * a.dh;
    float* n = which ? a.n2 + (size_t)ch * a.F + r : a.n1 + (size_t)ch * 2 * a.F + r;
    float sc = 1.f;
    if (mode == 0) {
        float v = 0.f;
        for (int i = lane; i < a.dh; i += 32) v = fmaf(W[i], W[i], v);
        v = warp_sum(v);
        if (lane == 0) *n = sqrtf(v);
    } else if (mode == 1) {
        sc = renorm_scale(*n, sw_ss(a, parity, which, ch)[r]);
    }
    for (int i = lane; i < a.dh; i += 32) {
        const float w = W[i] * sc;
        if (mode == 1) W[i] = w;
        Wb[i] = __float2bfloat16_rn(w);
    }
}

// SM count of the current device (grid of the persistent phase A).
int sw_sms() {
    static int n = 0;
    if (n == 0) {
        int dev = 0, v = 0;
        if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) !=
                                                      cudaSuccess || v <= 0)
            return 1;
        n = v;
    }
    return n;
}

std::once_flag g_sw_once;
cudaError_t g_sw_err = cudaSuccess;

cudaError_t sw_attrs() {
    std::call_once(g_sw_once, [] {
        const void* kb[] = {reinterpret_cast<const void*>(swiglu_b_kernel<false>),
                            reinterpret_cast<const void*>(swiglu_b_kernel<true>)};
        const void* ks[] = {reinterpret_cast<const void*>(swiglu_a_kernel), reinterpret_cast<const void*>(swiglu_rh_kernel),
                            reinterpret_cast<const void*>(swiglu_ro_kernel)};
        for (const void* k : kb)
            if (g_sw_err == cudaSuccess)
                g_sw_err = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, SwLayoutB::DYN);
        for (const void* k : ks)
            if (g_sw_err == cudaSuccess)
                g_sw_err = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, SwLayout::DYN);
    });
    return g_sw_err;
}

SwArgs sw_args(const DevState& s, const SegWork& w) {
    SwArgs a{};
    a.H = s.heads; a.dh = s.d_in / s.heads; a.Hk = (s.d_out / 2) / a.dh; a.F = s.d_hid; a.T = s.T; a.Tp = w.Tp;
    a.C = s.C; a.c0 = w.c0;
    a.paper = s.mode == 1; a.momentum = s.momentum; a.renorm_pending = w.renorm_pending; a.parity = w.parity;
    a.win = s.win_rows; a.tok0 = w.u_off;
    a.u_row0 = a.paper ? (int)w.u_off : (int)w.row0;
    a.u_chain0 = a.paper ? w.c0 : 0;
    a.y_row0 = (int)w.row0;
    a.lr = s.lr;
    a.eta = s.eta; a.dbeta = s.dbeta; a.zinv = a.paper ? s.zinv : nullptr; a.b_beta = s.b_beta;
    a.eta_in = w.eta_in ? w.eta_in + w.row0 : nullptr;
    a.eta_cstride = w.eta_cstride;
    a.W1 = s.W1; a.W2 = s.W2; a.mu1 = s.mu1; a.mu2 = s.mu2; a.W1b = s.W1b; a.W2b = s.W2b;
    a.n1 = s.n1; a.n2 = s.n2; a.sumsq = s.sumsq;
    a.dPG = static_cast<bf16*>(s.dHt); a.Zt = static_cast<bf16*>(s.Att);
    a.loss = w.loss; a.step_sq = w.step_sq; a.status = s.status;
    a.d_out = s.d_out;
    return a;
}

}  // namespace

cudaError_t launch_swiglu_phase_a(const DevState& s, const SwMaps& m, const SwInputMaps& in, const SegWork& w,
                                  cudaStream_t st) {
    cudaError_t e = sw_attrs();
    if (e != cudaSuccess) return e;
    SwArgs a = sw_args(s, w);
    a.nc_launch = w.nc;
    const int ntiles = (s.T / 128) * ((a.F + 127) / 128) * w.nc * a.H;
    const int sms = sw_sms() - s.reserve_sms;  // leave the host-input gather's SMs free
    const int grid = ntiles < sms ? ntiles : sms;
    swiglu_a_kernel<<<grid, SW_THREADS, SwLayout::DYN, st>>>(s.mode == 1 ? m.Ua : in.Xa, in.Ka, in.Va, m.W1a, m.W2a, a);
    return cudaGetLastError();
}

cudaError_t launch_swiglu_phase_b(const DevState& s, const SwMaps& m, const SwInputMaps& in, const SegWork& w,
                                  cudaStream_t st) {
    cudaError_t e = sw_attrs();
    if (e != cudaSuccess) return e;
    SwArgs a = sw_args(s, w);
    a.nc_launch = w.nc;
    const int ntiles = w.nc * a.H * 3 * ((a.F + SWB_N - 1) / SWB_N) * ((a.dh + 127) / 128);
    const int sms = sw_sms() - s.reserve_sms;  // leave the host-input gather's SMs free
    const int grid = ntiles < sms ? ntiles : sms;
    if (a.step_sq)
        swiglu_b_kernel<true><<<grid, SWB_THREADS, SwLayoutB::DYN, st>>>(s.mode == 1 ? m.Ub : in.Xb, in.Kb, in.Vb, m.PG,
                                                                         m.Z, m.W1s, m.M1s, m.W2s, m.M2s, a);
    else
        swiglu_b_kernel<false><<<grid, SWB_THREADS, SwLayoutB::DYN, st>>>(s.mode == 1 ? m.Ub : in.Xb, in.Kb, in.Vb, m.PG,
                                                                          m.Z, m.W1s, m.M1s, m.W2s, m.M2s, a);
    return cudaGetLastError();
}

cudaError_t launch_swiglu_rows(const DevState& s, int mode, int parity, int c0, int nc, cudaStream_t st) {
    SegWork w{};
    w.c0 = c0;
    w.nc = nc;
    SwArgs a = sw_args(s, w);
    swiglu_rows_kernel<<<dim3((2 * a.F + 7) / 8, nc * a.H, 2), 256, 0, st>>>(a, mode, parity);
    return cudaGetLastError();
}

cudaError_t launch_swiglu_read(const DevState& s, const SwMaps& m, const void* Uq, void* Zq, int Q, cudaStream_t st) {
    cudaError_t e = sw_attrs();
    if (e != cudaSuccess) return e;
    SegWork w{};
    w.c0 = 0;
    w.nc = s.C;
    SwArgs a = sw_args(s, w);
    a.Q = Q;
    a.Zq = static_cast<bf16*>(Zq);
    a.Oq = s.Oq;
    CUtensorMap mu, mz;
    const uint64_t H = a.H, dh = a.dh;
    const uint64_t du[4] = {dh, H, (uint64_t)Q, (uint64_t)s.C};
    const uint64_t su[3] = {dh * 2, H * dh * 2, (uint64_t)Q * H * dh * 2};
    const uint32_t bu[4] = {64, 1, 128, 1};
    if (!encode_map_bf16_4d(&mu, Uq, du, su, bu) || !encode_map_bf16_3d(&mz, Zq, a.F, Q, (uint64_t)s.C * H, 64, 128))
        return cudaErrorInvalidValue;
    const int nq = (Q + 127) / 128;
    swiglu_rh_kernel<<<dim3(nq, (a.F + 127) / 128, s.C * a.H), SW_THREADS, SwLayout::DYN, st>>>(mu, m.W1a, a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    swiglu_ro_kernel<<<dim3(nq, (a.dh + 127) / 128, s.C * a.H), SW_THREADS, SwLayout::DYN, st>>>(mz, m.W2m, a);
    return cudaGetLastError();
}

}  // namespace mone
