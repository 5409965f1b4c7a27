// bf16 tensor-core path of one TTL segment step (tcgen05 + TMEM + TMA, sm_103a).
//
// A segment step of the SiLU-MLP memory M(u) = SiLU(u W1^T) W2 (Eq. 3 form) on
// T tokens is four dense contractions (Eq. 10):
//   phase A (per token tile x hidden tile, two TMEM accumulators)
//       H = U W1^T            K = d_in      (memory forward)
//       R = Y W2^T            K = d_out     (Y = [K || V] the targets of Eq. 7)
//     fused epilogue: A = SiLU(H), dH = c_t R * SiLU'(H), At = c_t A with
//     c_t = -eta_t / T' (Eq. 7's loss is linear in M, so dL/dO = -eta Y / T'
//     does not depend on W and the target tile can be multiplied directly);
//     writes dH^T and At^T (bf16, [hidden][token]) and the loss partial
//     sum_t sum_h A_th R_th = sum_t y_t . M(u_t).
//   phase B (per hidden tile x column tile of [W1 | W2])
//       G1 = dH^T U           K = T'        (gradient of W1)
//       G2 = At^T Y           K = T'        (gradient of W2)
//     fused epilogue (Eq. 8, App. A): mu = beta mu + G; W = s W_raw - mu with s
//     the previous segment's pending row renormalisation; stores W (fp32), mu,
//     the bf16 operand copy of W and the new row sums of squares.
//
// Each CTA: 4 warps.  Warp 0 lane 0 drives TMA into a 3-stage shared-memory ring
// (128-byte swizzle), warp 1 lane 0 issues tcgen05.mma (M = 128, N = 128,
// K = 16 per instruction) into TMEM, then all 4 warps drain TMEM (one TMEM lane
// quarter per warp).  ~98 KB of shared memory per CTA, so two CTAs share an SM
// and one CTA's memory-bound epilogue overlaps the other's MMA main loop.
// Every wait is bounded (kWaitLimitNs); a timeout latches DEV_TIMEOUT.
#include <mutex>

#include "mone_common.cuh"

namespace mone {

namespace {

constexpr int BM = 128;                 // MMA M (TMEM lanes)
constexpr int BN = 128;                 // MMA N
constexpr int BK = 64;                  // 64 bf16 = one 128-byte swizzle row
constexpr int STAGES = 3;
constexpr int A_TILE = BM * BK * 2;     // 16 KB
constexpr int B_TILE = BN * BK * 2;     // 16 KB
constexpr int STAGE_BYTES = A_TILE + B_TILE;
constexpr int RING_BYTES = STAGES * STAGE_BYTES;
constexpr int SMEM_BYTES = RING_BYTES + 1024 /*align slack*/ + 2048 /*barriers, scales*/;

static_assert(2 * BN * BM * 2 <= RING_BYTES, "phase A staging must fit in the ring");
static_assert(BM * BN * 4 <= RING_BYTES, "phase B staging must fit in the ring");

struct TcArgs {
    int d_in, d_out, d_hid, T, Tp, c0, C, paper, momentum, renorm_pending, parity;
    int u_row0, u_chain0, y_row0;
    float lr;
    const float* eta_in;        // plain-mode caller rates, offset to the segment start, or null
    long long eta_cstride;
    const float* eta;           // paper-mode rates [C][T]
    const float* dbeta;         // [C][T]
    const float* b_beta;        // [C]
    float *W1, *W2, *mu1, *mu2;
    bf16 *W1b, *W2b;
    const float *n1, *n2;
    float* sumsq;               // [2 parity][2 matrix][C][d_hid]
    bf16 *dHt, *Att;            // [C][d_hid][T]
    float* loss;                // [nc] or null
    int* status;
};

__device__ __forceinline__ float* ss_row(const TcArgs& a, int parity, int which, int cs) {
    return a.sumsq + ((size_t)(parity * 2 + which) * a.C + cs) * a.d_hid;
}

struct Smem {
    uint8_t* ring;
    uint32_t full0, empty0, accb;
    uint32_t* tmem_slot;
    float* scratch;             // 2*BN + 8 floats
};

__device__ __forceinline__ Smem carve(uint8_t* raw) {
    Smem s;
    s.ring = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(raw) + 1023) & ~uintptr_t(1023));
    uint64_t* bars = reinterpret_cast<uint64_t*>(s.ring + RING_BYTES);
    s.full0 = smem_u32(bars);
    s.empty0 = s.full0 + 8 * STAGES;
    s.accb = s.full0 + 16 * STAGES;
    s.tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * STAGES + 1);
    s.scratch = reinterpret_cast<float*>(s.tmem_slot + 4);
    return s;
}

__device__ __forceinline__ void init_barriers(const Smem& s) {
    for (int i = 0; i < STAGES; ++i) {
        mbar_init(s.full0 + 8 * i, 1);
        mbar_init(s.empty0 + 8 * i, 1);
    }
    mbar_init(s.accb, 1);
    fence_mbar_init();
}

// ------------------------------------------------------------------ phase A

__global__ void __launch_bounds__(128, 1)
tc_phase_a_kernel(const __grid_constant__ CUtensorMap tmU, const __grid_constant__ CUtensorMap tmK,
                  const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmW1,
                  const __grid_constant__ CUtensorMap tmW2, const TcArgs a) {
    extern __shared__ uint8_t smem_raw[];
    const Smem sm = carve(smem_raw);
    float* s_sc1 = sm.scratch;
    float* s_sc2 = sm.scratch + BN;
    float* s_red = sm.scratch + 2 * BN;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int ttile = blockIdx.x, h0 = blockIdx.y * BN, cz = blockIdx.z, cs = a.c0 + cz;

    if (tid == 0) {
        init_barriers(sm);
        tma_prefetch_map(&tmU);
        tma_prefetch_map(&tmK);
        tma_prefetch_map(&tmV);
        tma_prefetch_map(&tmW1);
        tma_prefetch_map(&tmW2);
    }
    if (warp == 0) {
        tmem_alloc(smem_u32(sm.tmem_slot), 2 * BN);
        tmem_relinquish();
    }
    {   // renorm scales of this hidden tile; zero this segment's row sums
        const int h = h0 + tid;
        float s1 = 1.f, s2 = 1.f;
        if (a.renorm_pending) {
            s1 = renorm_scale(a.n1[(size_t)cs * a.d_hid + h], ss_row(a, a.parity ^ 1, 0, cs)[h]);
            s2 = renorm_scale(a.n2[(size_t)cs * a.d_hid + h], ss_row(a, a.parity ^ 1, 1, cs)[h]);
        }
        s_sc1[tid] = s1;
        s_sc2[tid] = s2;
        if (ttile == 0) {
            ss_row(a, a.parity, 0, cs)[h] = 0.f;
            ss_row(a, a.parity, 1, cs)[h] = 0.f;
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *sm.tmem_slot;

    const int KB1 = a.d_in / BK, KB2 = a.d_out / BK, KB = KB1 + KB2, half = (a.d_out / 2) / BK;
    const int trow = ttile * BM;

    if (warp == 0) {
        if (lane == 0) {
            for (int kb = 0; kb < KB; ++kb) {
                const int s = kb % STAGES;
                const uint32_t it = kb / STAGES;
                if (kb >= STAGES && !mbar_wait(sm.empty0 + 8 * s, (it - 1) & 1, a.status)) break;
                const uint32_t sa = smem_u32(sm.ring + s * STAGE_BYTES), sb = sa + A_TILE, fb = sm.full0 + 8 * s;
                mbar_expect_tx(fb, STAGE_BYTES);
                if (kb < KB1) {
                    tma_load_3d(sa, &tmU, fb, kb * BK, a.u_row0 + trow, a.u_chain0 + cz);
                    tma_load_3d(sb, &tmW1, fb, kb * BK, h0, cs);
                } else {
                    const int k2 = kb - KB1;
                    if (k2 < half)
                        tma_load_3d(sa, &tmK, fb, k2 * BK, a.y_row0 + trow, cz);
                    else
                        tma_load_3d(sa, &tmV, fb, (k2 - half) * BK, a.y_row0 + trow, cz);
                    tma_load_3d(sb, &tmW2, fb, k2 * BK, h0, cs);
                }
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16_f32(BM, BN, false, false);
            for (int kb = 0; kb < KB; ++kb) {
                const int s = kb % STAGES;
                if (!mbar_wait(sm.full0 + 8 * s, (kb / STAGES) & 1, a.status)) break;
                tc_fence_after();
                const uint32_t sa = smem_u32(sm.ring + s * STAGE_BYTES), sb = sa + A_TILE;
                const uint32_t d = tmem + (kb < KB1 ? 0u : (uint32_t)BN);
                const bool first = (kb == 0 || kb == KB1);
#pragma unroll
                for (int k = 0; k < BK / 16; ++k)
                    umma_bf16(d, sdesc_sw128(sa + k * 32, 16), sdesc_sw128(sb + k * 32, 16), idesc,
                              (first && k == 0) ? 0u : 1u);
                umma_commit(sm.empty0 + 8 * s);
            }
            umma_commit(sm.accb);
        }
        __syncwarp();
    }

    // ---- epilogue: thread = token row of the tile
    mbar_wait(sm.accb, 0, a.status);
    tc_fence_after();
    const int row = warp * 32 + lane;
    const int t = trow + row;
    float ct = 0.f;
    if (t < a.Tp) {
        const float e = a.paper ? a.eta[(size_t)cs * a.T + t]
                                : (a.eta_in ? a.eta_in[cz * a.eta_cstride + t] : a.lr);
        ct = -e / (float)a.Tp;
    }
    bf16* sdH = reinterpret_cast<bf16*>(sm.ring);      // [BN][BM]
    bf16* sA = sdH + BN * BM;                          // [BN][BM]
    float lsum = 0.f;
    const uint32_t lane_base = tmem + ((uint32_t)(warp * 32) << 16);
#pragma unroll 1
    for (int j0 = 0; j0 < BN; j0 += 32) {
        float hv[32], rv[32];
        tmem_ld32(lane_base + j0, hv);
        tmem_ld32(lane_base + BN + j0, rv);
#pragma unroll
        for (int jj = 0; jj < 32; ++jj) {
            const int h = j0 + jj;
            const float x = hv[jj] * s_sc1[h];
            const float r = rv[jj] * s_sc2[h];
            const float sg = sigmoidf_(x);
            const float av = x * sg;
            const float ds = sg * (1.f + x * (1.f - sg));
            lsum = fmaf(av, r, lsum);
            sdH[h * BM + row] = __float2bfloat16_rn(ct * r * ds);
            sA[h * BM + row] = __float2bfloat16_rn(ct * av);
        }
    }
    tc_fence_before();
    __syncthreads();
    {
        constexpr int VPR = BM / 8;  // 16-byte vectors per hidden row
        const size_t base = ((size_t)cs * a.d_hid + h0) * a.T + trow;
        for (int v = tid; v < BN * VPR; v += 128) {
            const int h = v / VPR, q = v % VPR;
            const size_t off = base + (size_t)h * a.T + q * 8;
            *reinterpret_cast<uint4*>(a.dHt + off) = *reinterpret_cast<const uint4*>(sdH + h * BM + q * 8);
            *reinterpret_cast<uint4*>(a.Att + off) = *reinterpret_cast<const uint4*>(sA + h * BM + q * 8);
        }
    }
    if (a.loss) {
        lsum = warp_sum(lsum);
        if (lane == 0) s_red[warp] = lsum;
        __syncthreads();
        if (tid == 0) atomicAdd(&a.loss[cz], -(s_red[0] + s_red[1] + s_red[2] + s_red[3]) / (float)a.Tp);
    }
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, 2 * BN);
}

// ------------------------------------------------------------------ phase B

__global__ void __launch_bounds__(128, 1)
tc_phase_b_kernel(const __grid_constant__ CUtensorMap tmDH, const __grid_constant__ CUtensorMap tmAT,
                  const __grid_constant__ CUtensorMap tmUb, const __grid_constant__ CUtensorMap tmKb,
                  const __grid_constant__ CUtensorMap tmVb, const TcArgs a) {
    extern __shared__ uint8_t smem_raw[];
    const Smem sm = carve(smem_raw);
    float* s_red = sm.scratch;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int col0 = blockIdx.x * BN, h0 = blockIdx.y * BM, cz = blockIdx.z, cs = a.c0 + cz;
    const bool isW1 = col0 < a.d_in;
    const int dh = a.d_out / 2;

    if (tid == 0) {
        init_barriers(sm);
        tma_prefetch_map(isW1 ? &tmDH : &tmAT);
        tma_prefetch_map(isW1 ? &tmUb : &tmKb);
        if (!isW1) tma_prefetch_map(&tmVb);
    }
    if (warp == 0) {
        tmem_alloc(smem_u32(sm.tmem_slot), BN);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *sm.tmem_slot;

    const int KB = (a.Tp + BK - 1) / BK;  // tokens beyond T' carry zero dH / At
    if (warp == 0) {
        if (lane == 0) {
            for (int kb = 0; kb < KB; ++kb) {
                const int s = kb % STAGES;
                const uint32_t it = kb / STAGES;
                if (kb >= STAGES && !mbar_wait(sm.empty0 + 8 * s, (it - 1) & 1, a.status)) break;
                const uint32_t sa = smem_u32(sm.ring + s * STAGE_BYTES), sb = sa + A_TILE, fb = sm.full0 + 8 * s;
                mbar_expect_tx(fb, STAGE_BYTES);
                tma_load_3d(sa, isW1 ? &tmDH : &tmAT, fb, kb * BK, h0, cs);
#pragma unroll
                for (int b = 0; b < BN / 64; ++b) {
                    const uint32_t dst = sb + b * (64 * BK * 2);
                    if (isW1) {
                        tma_load_3d(dst, &tmUb, fb, col0 + b * 64, a.u_row0 + kb * BK, a.u_chain0 + cz);
                    } else {
                        const int o = col0 - a.d_in + b * 64;
                        if (o < dh)
                            tma_load_3d(dst, &tmKb, fb, o, a.y_row0 + kb * BK, cz);
                        else
                            tma_load_3d(dst, &tmVb, fb, o - dh, a.y_row0 + kb * BK, cz);
                    }
                }
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16_f32(BM, BN, false, true);
            for (int kb = 0; kb < KB; ++kb) {
                const int s = kb % STAGES;
                if (!mbar_wait(sm.full0 + 8 * s, (kb / STAGES) & 1, a.status)) break;
                tc_fence_after();
                const uint32_t sa = smem_u32(sm.ring + s * STAGE_BYTES), sb = sa + A_TILE;
#pragma unroll
                for (int k = 0; k < BK / 16; ++k)
                    umma_bf16(tmem, sdesc_sw128(sa + k * 32, 16), sdesc_sw128(sb + k * 16 * 128, 64 * BK * 2),
                              idesc, (kb == 0 && k == 0) ? 0u : 1u);
                umma_commit(sm.empty0 + 8 * s);
            }
            umma_commit(sm.accb);
        }
        __syncwarp();
    }

    // momentum decay beta_s = sigmoid(mean_t w_beta . x_t + b_beta) while the MMAs run
    float beta = 0.f;
    if (a.momentum) {
        float v = 0.f;
        for (int t = tid; t < a.Tp; t += 128) v += a.dbeta[(size_t)cs * a.T + t];
        v = warp_sum(v);
        if (lane == 0) s_red[warp] = v;
        __syncthreads();
        beta = sigmoidf_((s_red[0] + s_red[1] + s_red[2] + s_red[3]) / (float)a.Tp + a.b_beta[cs]);
    }

    // ---- epilogue part 1: TMEM -> shared staging (thread = hidden row)
    mbar_wait(sm.accb, 0, a.status);
    tc_fence_after();
    float4* stg = reinterpret_cast<float4*>(sm.ring);  // [BM rows][BN/4 float4], XOR-swizzled
    {
        const int r = warp * 32 + lane;
        const uint32_t lane_base = tmem + ((uint32_t)(warp * 32) << 16);
#pragma unroll 1
        for (int q = 0; q < BN / 32; ++q) {
            float g[32];
            tmem_ld32(lane_base + q * 32, g);
#pragma unroll
            for (int v = 0; v < 8; ++v) {
                const int f = q * 8 + v;
                stg[r * (BN / 4) + (f ^ (r & 31))] = make_float4(g[4 * v], g[4 * v + 1], g[4 * v + 2], g[4 * v + 3]);
            }
        }
    }
    tc_fence_before();
    __syncthreads();

    // ---- epilogue part 2: row-wise fused update, coalesced along columns
    const int which = isW1 ? 0 : 1;
    const int width = isW1 ? a.d_in : a.d_out;
    const int cl = isW1 ? col0 : col0 - a.d_in;
    float* W = (isW1 ? a.W1 : a.W2) + (size_t)cs * a.d_hid * width;
    float* M = a.momentum ? (isW1 ? a.mu1 : a.mu2) + (size_t)cs * a.d_hid * width : nullptr;
    bf16* Wb = (isW1 ? a.W1b : a.W2b) + (size_t)cs * a.d_hid * width;
    const float* n0 = (isW1 ? a.n1 : a.n2) + (size_t)cs * a.d_hid;
    const float* prev = ss_row(a, a.parity ^ 1, which, cs);
    float* cur = ss_row(a, a.parity, which, cs);
    bool finite = true;
    constexpr int RB = 8;  // rows in flight per warp
#pragma unroll 1
    for (int rb = 0; rb < 32; rb += RB) {
        float4 gv[RB], wv[RB], mv[RB];
#pragma unroll
        for (int u = 0; u < RB; ++u) {
            const int r = warp * 32 + rb + u;
            const size_t off = (size_t)(h0 + r) * width + cl + lane * 4;
            gv[u] = stg[r * (BN / 4) + (lane ^ (r & 31))];
            wv[u] = *reinterpret_cast<const float4*>(W + off);
            mv[u] = M ? *reinterpret_cast<const float4*>(M + off) : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int u = 0; u < RB; ++u) {
            const int r = warp * 32 + rb + u;
            const int h = h0 + r;
            const size_t off = (size_t)h * width + cl + lane * 4;
            const float s = a.renorm_pending ? renorm_scale(n0[h], prev[h]) : 1.f;
            float4 mn, wn;
            mn.x = fmaf(beta, mv[u].x, gv[u].x);
            mn.y = fmaf(beta, mv[u].y, gv[u].y);
            mn.z = fmaf(beta, mv[u].z, gv[u].z);
            mn.w = fmaf(beta, mv[u].w, gv[u].w);
            wn.x = s * wv[u].x - mn.x;
            wn.y = s * wv[u].y - mn.y;
            wn.z = s * wv[u].z - mn.z;
            wn.w = s * wv[u].w - mn.w;
            *reinterpret_cast<float4*>(W + off) = wn;
            if (M) *reinterpret_cast<float4*>(M + off) = mn;
            __nv_bfloat162 b01 = __floats2bfloat162_rn(wn.x, wn.y);
            __nv_bfloat162 b23 = __floats2bfloat162_rn(wn.z, wn.w);
            uint2 packed;
            packed.x = *reinterpret_cast<uint32_t*>(&b01);
            packed.y = *reinterpret_cast<uint32_t*>(&b23);
            *reinterpret_cast<uint2*>(Wb + off) = packed;
            float ss = wn.x * wn.x + wn.y * wn.y + wn.z * wn.z + wn.w * wn.w;
            finite = finite && isfinite(ss);
            ss = warp_sum(ss);
            if (lane == 0) atomicAdd(&cur[h], ss);
        }
    }
    if (!finite) atomicOr(a.status, DEV_NONFINITE);
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, BN);
}

TcArgs make_args(const DevState& s, const SegWork& w) {
    TcArgs a{};
    a.d_in = s.d_in; a.d_out = s.d_out; a.d_hid = s.d_hid; a.T = s.T; a.Tp = w.Tp; a.c0 = w.c0; a.C = s.C;
    a.paper = s.mode == 1; a.momentum = s.momentum; a.renorm_pending = w.renorm_pending; a.parity = w.parity;
    a.u_row0 = a.paper ? 0 : (int)w.row0;
    a.u_chain0 = a.paper ? w.c0 : 0;
    a.y_row0 = (int)w.row0;
    a.lr = s.lr;
    a.eta_in = w.eta_in ? w.eta_in + w.row0 : nullptr;
    a.eta_cstride = w.eta_cstride;
    a.eta = s.eta; a.dbeta = s.dbeta; a.b_beta = s.b_beta;
    a.W1 = s.W1; a.W2 = s.W2; a.mu1 = s.mu1; a.mu2 = s.mu2; a.W1b = s.W1b; a.W2b = s.W2b;
    a.n1 = s.n1; a.n2 = s.n2; a.sumsq = s.sumsq;
    a.dHt = reinterpret_cast<bf16*>(s.dHt); a.Att = reinterpret_cast<bf16*>(s.Att);
    a.loss = w.loss; a.status = s.status;
    return a;
}

std::once_flag g_attr_once;
cudaError_t g_attr_err = cudaSuccess;

cudaError_t ensure_attrs() {
    std::call_once(g_attr_once, [] {
        g_attr_err = cudaFuncSetAttribute(tc_phase_a_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
        if (g_attr_err == cudaSuccess)
            g_attr_err =
                cudaFuncSetAttribute(tc_phase_b_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
    });
    return g_attr_err;
}

}  // namespace

cudaError_t launch_phase_a_tc(const DevState& s, const TcMaps& m, const TcInputMaps& in, const SegWork& w,
                              cudaStream_t st) {
    cudaError_t e = ensure_attrs();
    if (e != cudaSuccess) return e;
    const TcArgs a = make_args(s, w);
    dim3 grid(s.T / BM, s.d_hid / BN, w.nc);
    tc_phase_a_kernel<<<grid, 128, SMEM_BYTES, st>>>(s.mode == 1 ? m.Ua : in.Xa, in.Ka, in.Va, m.W1b, m.W2b, a);
    return cudaGetLastError();
}

cudaError_t launch_phase_b_tc(const DevState& s, const TcMaps& m, const TcInputMaps& in, const SegWork& w,
                              cudaStream_t st) {
    cudaError_t e = ensure_attrs();
    if (e != cudaSuccess) return e;
    const TcArgs a = make_args(s, w);
    dim3 grid((s.d_in + s.d_out) / BN, s.d_hid / BM, w.nc);
    tc_phase_b_kernel<<<grid, 128, SMEM_BYTES, st>>>(m.dHt, m.Att, s.mode == 1 ? m.Ub : in.Xb, in.Kb, in.Vb, a);
    return cudaGetLastError();
}

int tc_kernels_per_segment() { return 2; }

// ------------------------------------------------------------------ tensor maps

namespace {
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn g_encode = nullptr;
std::once_flag g_encode_once;
}  // namespace

bool encode_map_bf16_3d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t rows, uint64_t chains,
                        uint32_t box_inner, uint32_t box_rows) {
    std::call_once(g_encode_once, [] {
        void* fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            g_encode = reinterpret_cast<EncodeTiledFn>(fn);
    });
    if (!g_encode) return false;
    const cuuint64_t dims[3] = {inner, rows, chains};
    const cuuint64_t strides[2] = {inner * 2, inner * rows * 2};
    const cuuint32_t box[3] = {box_inner, box_rows, 1};
    const cuuint32_t estr[3] = {1, 1, 1};
    return g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace mone
