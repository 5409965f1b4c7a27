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
// phase B: 3 stages of 32 KB and no transpose buffers, so that two CTAs share an SM and
// one CTA's state update overlaps the others' operand loads and MMAs
constexpr int SWB_CTAS_PER_SM = 2;
using SwLayoutB = SwLayoutT<3, 4 * SW_BOX, false>;
static_assert(SwLayout::DYN <= 227 * 1024, "shared memory budget");
static_assert(SWB_CTAS_PER_SM * (SwLayoutB::DYN + 1024) <= 228 * 1024, "phase B CTAs per SM");

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

// One tile (matrix m, 128 weight columns, 128 hidden rows, head) per CTA; two CTAs per SM
// (three 32 KB operand stages each, 128 TMEM columns).  The update walks the tile's rows in
// chunks of 16: every chunk's W and mu loads are issued before its stores.
constexpr int SWB_ROWS = 16;

__global__ void __launch_bounds__(SW_THREADS, SWB_CTAS_PER_SM)
swiglu_b_kernel(const __grid_constant__ CUtensorMap tmUb, const __grid_constant__ CUtensorMap tmKb,
                const __grid_constant__ CUtensorMap tmVb, const __grid_constant__ CUtensorMap tmPG,
                const __grid_constant__ CUtensorMap tmZ, const SwArgs a) {
    using L = SwLayoutB;
    extern __shared__ uint8_t smem_raw[];
    const auto c = sw_setup<L>(smem_raw, 128);
    const uint32_t tmem = *reinterpret_cast<uint32_t*>(c.base + L::SLOT);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int NC = (a.dh + 127) / 128;
    const int m = blockIdx.x / NC, col0 = (blockIdx.x % NC) * 128, f0 = blockIdx.y * 128;
    const int cz = blockIdx.z / a.H, h = blockIdx.z % a.H;
    const int cs = a.c0 + cz, ch = cs * a.H + h;
    const int KB = (a.Tp + 63) / 64;  // tokens beyond T' carry zero gradients

    if (warp == 0) {
        if (lane == 0) {
            for (int kb = 0; kb < KB; ++kb) {
                const int s = kb % L::NSTAGES;
                if (kb >= L::NSTAGES && !mbar_wait(c.empty(s), ((kb / L::NSTAGES) - 1) & 1, a.status)) break;
                const uint32_t sa = smem_u32(c.base + s * (4 * SW_BOX)), sb = sa + 2 * SW_BOX, fb = c.full(s);
                mbar_expect_tx(fb, 4 * SW_BOX);
#pragma unroll
                for (int bx = 0; bx < 2; ++bx) {
                    const uint32_t dst = sa + bx * SW_BOX;
                    if (m < 2)
                        tma_load_4d(dst, &tmUb, fb, col0 + bx * 64, h, a.u_row0 + kb * 64, a.u_chain0 + cz);
                    else if (h < a.Hk)
                        tma_load_4d(dst, &tmKb, fb, col0 + bx * 64, h, a.y_row0 + kb * 64, cz);
                    else
                        tma_load_4d(dst, &tmVb, fb, col0 + bx * 64, h - a.Hk, a.y_row0 + kb * 64, cz);
                    if (m < 2)
                        tma_load_4d(sb + bx * SW_BOX, &tmPG, fb, f0 + bx * 64, m, kb * 64, ch);
                    else
                        tma_load_3d(sb + bx * SW_BOX, &tmZ, fb, f0 + bx * 64, kb * 64, ch);
                }
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16_f32(128, 128, true, true);
            bool ok = true;
            for (int kb = 0; kb < KB; ++kb) {
                const int s = kb % L::NSTAGES;
                if (!mbar_wait(c.full(s), (kb / L::NSTAGES) & 1, a.status)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t sa = smem_u32(c.base + s * (4 * SW_BOX)), sb = sa + 2 * SW_BOX;
#pragma unroll
                for (int k = 0; k < 4; ++k)
                    umma_bf16(tmem, sdesc_sw128(sa + k * 16 * 128, SW_BOX), sdesc_sw128(sb + k * 16 * 128, SW_BOX),
                              idesc, (kb == 0 && k == 0) ? 0u : 1u);
                umma_commit(c.empty(s));
            }
            if (ok) umma_commit(c.tfull());
        }
        __syncwarp();
    } else {
        const int q = warp & 3, et = threadIdx.x - 64;
        float* tab = reinterpret_cast<float*>(c.base + L::TAB);  // row scales [128], beta partials [4]
        const int which = m < 2 ? 0 : 1;
        const int rowbase = (m < 2 ? m * a.F : 0) + f0;  // first state row of the tile (within the head)
        {
            const int f = f0 + et;
            float sc = 1.f;
            if (a.renorm_pending && f < a.F) {
                const float n = which ? a.n2[(size_t)ch * a.F + f] : a.n1[(size_t)ch * 2 * a.F + rowbase + et];
                sc = renorm_scale(n, sw_ss(a, a.parity ^ 1, which, ch)[rowbase + et]);
            }
            tab[et] = sc;
            float v = 0.f;
            if (a.momentum)
                for (int t = et; t < a.Tp; t += 128) v += a.dbeta[(size_t)cs * a.win + a.tok0 + t];
            v = warp_sum(v);
            if (lane == 0) tab[128 + (warp - 2)] = v;
        }
        if (sw_wait_acc(c, a.status)) {
            float beta = 0.f;
            if (a.momentum) beta = sigmoidf_((tab[128] + tab[129] + tab[130] + tab[131]) / (float)a.Tp + a.b_beta[cs]);
            const int col = col0 + q * 32 + lane;
            const bool live = col < a.dh;
            float* W = which ? a.W2 : a.W1;
            float* M = which ? a.mu2 : a.mu1;
            bf16* Wb = which ? a.W2b : a.W1b;
            const size_t rows_head = which ? a.F : 2 * a.F;
            const size_t base = ((size_t)ch * rows_head + rowbase) * a.dh + col;
            const uint32_t lane_base = tmem + ((uint32_t)(q * 32) << 16);
            const uint64_t wpol = l2_evict_last_policy();  // phase A of the next segment reads the copy
            float* cur = sw_ss(a, a.parity, which, ch);
            bool finite = true;
            // F is a multiple of 32, so a chunk of 16 rows is either wholly live or past F.  The loads
            // of chunk cc + 1 are issued before chunk cc is updated and stored, so two chunks' loads
            // are in flight per thread (the stores could alias them as far as the compiler knows,
            // so it would not hoist them itself)
            int nchunks = 0;
            while (nchunks < 128 / SWB_ROWS && f0 + nchunks * SWB_ROWS < a.F) ++nchunks;
            float v[SWB_ROWS], mo[SWB_ROWS];
#pragma unroll
            for (int j = 0; j < SWB_ROWS; ++j) {
                const size_t idx = base + (size_t)j * a.dh;
                v[j] = (live && nchunks > 0) ? W[idx] : 0.f;
                mo[j] = (live && a.momentum && nchunks > 0) ? M[idx] : 0.f;
            }
#pragma unroll 1
            for (int cc = 0; cc < nchunks; ++cc) {
                float nv[SWB_ROWS], nmo[SWB_ROWS], gv[SWB_ROWS];
                const bool more = cc + 1 < nchunks;
#pragma unroll
                for (int j = 0; j < SWB_ROWS; ++j) {
                    const size_t idx = base + (size_t)((cc + 1) * SWB_ROWS + j) * a.dh;
                    nv[j] = (live && more) ? W[idx] : 0.f;
                    nmo[j] = (live && more && a.momentum) ? M[idx] : 0.f;
                }
                tmem_ld16(lane_base + cc * SWB_ROWS, gv);
#pragma unroll
                for (int j = 0; j < SWB_ROWS; ++j) {
                    const size_t idx = base + (size_t)(cc * SWB_ROWS + j) * a.dh;
                    const float mn = fmaf(beta, mo[j], gv[j]);
                    const float wn = fmaf(tab[cc * SWB_ROWS + j], v[j], -mn);
                    if (live) {
                        W[idx] = wn;
                        if (a.momentum) M[idx] = mn;
                        st_bf16_hint(Wb + idx, __float2bfloat16_rn(wn), wpol);
                    }
                    gv[j] = live ? wn * wn : 0.f;
                }
                // transpose-reduce over the 16 rows: afterwards lane l holds the partial of row
                // l & 15 over the 16 lanes that share bit 4 of l; the xor-16 exchange adds the rest
#pragma unroll
                for (int sft = SWB_ROWS / 2; sft >= 1; sft >>= 1) {
                    const bool upper = (lane & sft) != 0;
#pragma unroll
                    for (int u = 0; u < sft; ++u) {
                        const float send = upper ? gv[u] : gv[u + sft];
                        const float keep = upper ? gv[u + sft] : gv[u];
                        gv[u] = keep + __shfl_xor_sync(0xffffffffu, send, sft);
                    }
                }
                gv[0] += __shfl_xor_sync(0xffffffffu, gv[0], 16);
                finite = finite && isfinite(gv[0]);
                if (lane < SWB_ROWS) atomicAdd(&cur[rowbase + cc * SWB_ROWS + lane], gv[0]);
#pragma unroll
                for (int j = 0; j < SWB_ROWS; ++j) {
                    v[j] = nv[j];
                    mo[j] = nmo[j];
                }
            }
            if (!finite) atomicOr(a.status, DEV_NONFINITE);
        }
    }
    sw_teardown(tmem, 128);
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
        const void* ks[] = {reinterpret_cast<const void*>(swiglu_a_kernel), reinterpret_cast<const void*>(swiglu_b_kernel),
                            reinterpret_cast<const void*>(swiglu_rh_kernel), reinterpret_cast<const void*>(swiglu_ro_kernel)};
        for (const void* k : ks)
            if (g_sw_err == cudaSuccess)
                g_sw_err = cudaFuncSetAttribute(
                    k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                    k == reinterpret_cast<const void*>(swiglu_b_kernel) ? SwLayoutB::DYN : SwLayout::DYN);
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
    a.loss = w.loss; a.status = s.status;
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
    const int grid = ntiles < sw_sms() ? ntiles : sw_sms();
    swiglu_a_kernel<<<grid, SW_THREADS, SwLayout::DYN, st>>>(s.mode == 1 ? m.Ua : in.Xa, in.Ka, in.Va, m.W1a, m.W2a, a);
    return cudaGetLastError();
}

cudaError_t launch_swiglu_phase_b(const DevState& s, const SwMaps& m, const SwInputMaps& in, const SegWork& w,
                                  cudaStream_t st) {
    cudaError_t e = sw_attrs();
    if (e != cudaSuccess) return e;
    const SwArgs a = sw_args(s, w);
    dim3 grid(3 * ((a.dh + 127) / 128), (a.F + 127) / 128, w.nc * a.H);
    swiglu_b_kernel<<<grid, SW_THREADS, SwLayoutB::DYN, st>>>(s.mode == 1 ? m.Ub : in.Xb, in.Kb, in.Vb, m.PG, m.Z, a);
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
