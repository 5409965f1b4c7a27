// fp32 path of the TTL step, state upkeep kernels and the memory read.
//
// When d_in + d_out <= 512 the fp32 path runs every segment of a call in one launch with
// the rows resident on chip (ttl_resident_f32_kernel, below).  Otherwise it runs two
// kernels a segment (three with the squared-error pre-pass).  Those are latency-bound,
// so they use plain CUDA-core FFMA tiles (64 x 64 per CTA, 4 x 4 per thread, 64-deep K
// slabs so that each thread has 32 loads in flight per slab) in fp32 throughout, and
// compute the same two phases as the bf16 tensor-core path:
//   phase A  H = U W1^T, R = Y W2^T (Y = [K || V]); A = SiLU(H);
//            dH = c_t R * SiLU'(H), At = c_t A with c_t = -eta_t / T'   (Eq. 10)
//   phase B  G1 = dH^T U, G2 = At^T Y; mu = beta mu + G; W = s W_raw - mu  (Eq. 8)
// where s is the pending row renormalisation scale of the previous segment
// (App. A), applied lazily so that no extra pass over the weights is needed.
// The loss L_s = -(1/T') sum_t sum_h A_th R_th equals Eq. 7's segment mean
// because sum_h A_th R_th = y_t . (A_t W2) = y_t . M(u_t).
#include <mutex>

#include "mone_common.cuh"

namespace mone {

namespace {

constexpr int TM = 64, TN = 64, TK = 64;

// acc[i][j] += sum_k A(m0 + ty*MR + i, k) * B(n0 + tx*4 + j, k) for one (16 MR) x 64 tile.
// A(m, k) = A[m*sam + k*sak]; rows m >= m_valid and k >= k_valid read as 0.
template <int MR>
__device__ __forceinline__ void simt_tile(float (&acc)[MR][4], const float* A, long long sam, long long sak,
                                          const float* B, long long sbn, long long sbk, int K, int m_valid,
                                          int k_valid, float (*As)[16 * MR + 4], float (*Bs)[TN + 4]) {
    constexpr int TMR = 16 * MR;  // rows of the tile
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    for (int k0 = 0; k0 < K; k0 += TK) {
        // TMR x TK elements of A and 64 x TK of B, TK consecutive along the contiguous dimension
        float av[TMR * TK / 256], bv[TN * TK / 256];
#pragma unroll
        for (int r = 0; r < TMR * TK / 256; ++r) {
            const int e = tid + 256 * r;
            int m, k;
            if (sak == 1) { m = e / TK; k = e % TK; } else { m = e % TMR; k = e / TMR; }
            av[r] = (m < m_valid && k0 + k < k_valid) ? A[m * sam + (k0 + k) * sak] : 0.0f;
        }
#pragma unroll
        for (int r = 0; r < TN * TK / 256; ++r) {
            const int e = tid + 256 * r;
            int n, kb;
            if (sbk == 1) { n = e / TK; kb = e % TK; } else { n = e % TN; kb = e / TN; }
            bv[r] = (k0 + kb < k_valid) ? B[n * sbn + (k0 + kb) * sbk] : 0.0f;
        }
#pragma unroll
        for (int r = 0; r < TMR * TK / 256; ++r) {
            const int e = tid + 256 * r;
            int m, k;
            if (sak == 1) { m = e / TK; k = e % TK; } else { m = e % TMR; k = e / TMR; }
            As[k][m] = av[r];
        }
#pragma unroll
        for (int r = 0; r < TN * TK / 256; ++r) {
            const int e = tid + 256 * r;
            int n, kb;
            if (sbk == 1) { n = e / TK; kb = e % TK; } else { n = e % TN; kb = e / TN; }
            Bs[kb][n] = bv[r];
        }
        __syncthreads();
#pragma unroll
        for (int k = 0; k < TK; ++k) {
            float a[MR], b[4];
#pragma unroll
            for (int i = 0; i < MR; ++i) a[i] = As[k][ty * MR + i];
#pragma unroll
            for (int j = 0; j < 4; ++j) b[j] = Bs[k][tx * 4 + j];
#pragma unroll
            for (int i = 0; i < MR; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
        }
        __syncthreads();
    }
}

struct F32SegArgs {
    int d_in, d_hid, d_out, T, Tp, c0, paper, momentum, renorm_pending, parity, C;
    long long tok0;           // per-token tables: entry of token t of chain cs is [cs * win + tok0 + t]
    int win;
    float lr;
    const float *U;           // base of the memory input rows of this segment for chain cz (see below)
    long long u_cstride;      // element stride between chains of U
    const float *K, *V;
    long long y_cstride;
    long long row_avail;      // input rows available from the segment start
    const float* eta_in;      // plain mode caller rates (already offset to the segment) or null
    long long eta_cstride;
    const float* eta;         // paper mode rates [C][T] (state chain index)
    const float* dbeta;       // [C][T]
    const float* b_beta;
    float *W1, *W2, *mu1, *mu2;
    const float *n1, *n2;
    float* sumsq;             // [2][2][C][d_hid]
    float *dH, *At;           // [C][T][d_hid]
    float* loss;
    float* step_sq;           // [nc] squared norm of this segment's Eq. 8 step, or null
    int* status;
};

__device__ __forceinline__ const float* ss_ptr(const F32SegArgs& a, int parity, int which) {
    return a.sumsq + ((size_t)(parity * 2 + which) * a.C) * a.d_hid;
}

// Phase A takes tiles of 32 tokens x 64 hidden units (2 x 4 per thread): the fp32 workload has
// only T = 128 tokens a segment, so 64-row tiles would leave all but 16 SMs idle.
constexpr int A_MR = 2, A_TM = 16 * A_MR;

__global__ void __launch_bounds__(256) phase_a_f32_kernel(const F32SegArgs a) {
    __shared__ float As[TK][A_TM + 4], Bs[TK][TN + 4];
    __shared__ float red[8];
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const int t0 = blockIdx.x * A_TM, h0 = blockIdx.y * TN, cz = blockIdx.z, cs = a.c0 + cz;
    long long avail = a.row_avail - t0;
    int m_valid = (int)min((long long)min(A_TM, a.Tp - t0), avail);
    if (m_valid < 0) m_valid = 0;
    // zero this segment's row sums of squares (read by phase B of this segment)
    if (blockIdx.x == 0 && tid < TN) {
        float* cur = a.sumsq + ((size_t)(a.parity * 2) * a.C + cs) * a.d_hid + h0 + tid;
        cur[0] = 0.f;
        cur[(size_t)a.C * a.d_hid] = 0.f;
    }
    float accH[A_MR][4] = {}, accR[A_MR][4] = {};
    const float* U = a.U + cz * a.u_cstride + (long long)t0 * a.d_in;
    simt_tile(accH, U, a.d_in, 1, a.W1 + ((size_t)cs * a.d_hid + h0) * a.d_in, a.d_in, 1, a.d_in, m_valid,
              a.d_in, As, Bs);
    const int dh = a.d_out / 2;
    const float* W2 = a.W2 + ((size_t)cs * a.d_hid + h0) * a.d_out;
    simt_tile(accR, a.K + cz * a.y_cstride + (long long)t0 * dh, dh, 1, W2, a.d_out, 1, dh, m_valid, dh, As, Bs);
    simt_tile(accR, a.V + cz * a.y_cstride + (long long)t0 * dh, dh, 1, W2 + dh, a.d_out, 1, dh, m_valid, dh, As,
              Bs);

    const float* prev1 = ss_ptr(a, a.parity ^ 1, 0) + (size_t)cs * a.d_hid;
    const float* prev2 = ss_ptr(a, a.parity ^ 1, 1) + (size_t)cs * a.d_hid;
    float s1[4], s2[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const int h = h0 + tx * 4 + j;
        s1[j] = a.renorm_pending ? renorm_scale(a.n1[(size_t)cs * a.d_hid + h], prev1[h]) : 1.f;
        s2[j] = a.renorm_pending ? renorm_scale(a.n2[(size_t)cs * a.d_hid + h], prev2[h]) : 1.f;
    }
    float lsum = 0.f;
#pragma unroll
    for (int i = 0; i < A_MR; ++i) {
        const int t = t0 + ty * A_MR + i;
        float ct = 0.f;
        if (t < a.Tp && t - t0 < m_valid) {
            float e;
            if (a.paper)
                e = a.eta[(size_t)cs * a.win + a.tok0 + t];
            else
                e = a.eta_in ? a.eta_in[cz * a.eta_cstride + t] : a.lr;
            ct = -e / (float)a.Tp;
        }
        float* dHrow = a.dH + ((size_t)cs * a.T + t) * a.d_hid + h0 + tx * 4;
        float* Arow = a.At + ((size_t)cs * a.T + t) * a.d_hid + h0 + tx * 4;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float hv = accH[i][j] * s1[j];
            const float rv = accR[i][j] * s2[j];
            const float sg = sigmoidf_(hv);
            const float av = hv * sg;
            const float dsilu = sg * (1.f + hv * (1.f - sg));
            lsum += av * rv;
            dHrow[j] = ct * rv * dsilu;
            Arow[j] = ct * av;
        }
    }
    if (a.loss) {
        lsum = warp_sum(lsum);
        if ((tid & 31) == 0) red[tid >> 5] = lsum;
        __syncthreads();
        if (tid == 0) {
            float tot = 0.f;
            for (int w = 0; w < 8; ++w) tot += red[w];
            atomicAdd(&a.loss[cz], -tot / (float)a.Tp);
        }
    }
}

// Phase B takes tiles of 32 hidden rows x 64 weight columns (2 x 4 per thread), for the same reason.
constexpr int B_MR = 2, B_TM = 16 * B_MR;

__global__ void __launch_bounds__(256) phase_b_f32_kernel(const F32SegArgs a) {
    __shared__ float As[TK][B_TM + 4], Bs[TK][TN + 4];
    __shared__ float red[8];
    __shared__ float s_beta;
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const int col0 = blockIdx.x * TN, h0 = blockIdx.y * B_TM, cz = blockIdx.z, cs = a.c0 + cz;
    const bool isW1 = col0 < a.d_in;
    const int kv = (int)min((long long)a.Tp, a.row_avail);
    float acc[B_MR][4] = {};
    if (isW1) {
        const float* U = a.U + cz * a.u_cstride + col0;
        simt_tile(acc, a.dH + (size_t)cs * a.T * a.d_hid + h0, 1, a.d_hid, U, 1, a.d_in, a.Tp, B_TM, kv, As, Bs);
    } else {
        const int dh = a.d_out / 2;
        const int o0 = col0 - a.d_in;
        const float* Y = (o0 < dh ? a.K + o0 : a.V + (o0 - dh)) + cz * a.y_cstride;
        simt_tile(acc, a.At + (size_t)cs * a.T * a.d_hid + h0, 1, a.d_hid, Y, 1, dh, a.Tp, B_TM, kv, As, Bs);
    }
    // momentum decay beta_s = sigmoid(mean_t w_beta . x_t + b_beta)
    if (a.momentum) {
        float v = 0.f;
        for (int t = tid; t < a.Tp; t += 256) v += a.dbeta[(size_t)cs * a.win + a.tok0 + t];
        v = warp_sum(v);
        if ((tid & 31) == 0) red[tid >> 5] = v;
        __syncthreads();
        if (tid == 0) {
            float tot = 0.f;
            for (int w = 0; w < 8; ++w) tot += red[w];
            s_beta = sigmoidf_(tot / (float)a.Tp + a.b_beta[cs]);
        }
        __syncthreads();
    }
    const float beta = a.momentum ? s_beta : 0.f;
    const int which = isW1 ? 0 : 1;
    const int width = isW1 ? a.d_in : a.d_out;
    const int c_local = isW1 ? col0 : col0 - a.d_in;
    float* W = (isW1 ? a.W1 : a.W2) + (size_t)cs * a.d_hid * width;
    float* M = a.momentum ? (isW1 ? a.mu1 : a.mu2) + (size_t)cs * a.d_hid * width : nullptr;
    const float* n0 = (isW1 ? a.n1 : a.n2) + (size_t)cs * a.d_hid;
    const float* prev = ss_ptr(a, a.parity ^ 1, which) + (size_t)cs * a.d_hid;
    float* cur = a.sumsq + ((size_t)(a.parity * 2 + which) * a.C + cs) * a.d_hid;
    bool finite = true;
    float step = 0.f;  // sum of mu_s^2 over this thread's elements
#pragma unroll
    for (int i = 0; i < B_MR; ++i) {
        const int h = h0 + ty * B_MR + i;
        const float s = a.renorm_pending ? renorm_scale(n0[h], prev[h]) : 1.f;
        float* wrow = W + (size_t)h * width + c_local + tx * 4;
        float* mrow = M ? M + (size_t)h * width + c_local + tx * 4 : nullptr;
        float ss = 0.f;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float g = acc[i][j];
            const float mn = M ? fmaf(beta, mrow[j], g) : g;
            const float wn = s * wrow[j] - mn;
            wrow[j] = wn;
            if (M) mrow[j] = mn;
            ss = fmaf(wn, wn, ss);
            step = fmaf(mn, mn, step);
            finite = finite && isfinite(wn);
        }
        ss += __shfl_xor_sync(0xffffffffu, ss, 8);
        ss += __shfl_xor_sync(0xffffffffu, ss, 4);
        ss += __shfl_xor_sync(0xffffffffu, ss, 2);
        ss += __shfl_xor_sync(0xffffffffu, ss, 1);
        if (tx == 0) atomicAdd(&cur[h], ss);
    }
    if (a.step_sq) {
        step = warp_sum(step);
        if ((tid & 31) == 0) atomicAdd(&a.step_sq[cz], step);
    }
    if (!finite) atomicOr(a.status, DEV_NONFINITE);
}

F32SegArgs make_f32_args(const DevState& s, const SegWork& w) {
    F32SegArgs a{};
    a.d_in = s.d_in; a.d_hid = s.d_hid; a.d_out = s.d_out; a.T = s.T; a.Tp = w.Tp; a.c0 = w.c0;
    a.paper = s.mode == 1; a.momentum = s.momentum; a.renorm_pending = w.renorm_pending;
    a.tok0 = w.u_off; a.win = s.win_rows;
    a.parity = w.parity; a.C = s.C; a.lr = s.lr;
    const int dh = s.d_out / 2;
    if (a.paper) {
        a.U = reinterpret_cast<const float*>(s.U) + ((size_t)w.c0 * s.win_rows + w.u_off) * s.d_in;
        a.u_cstride = (long long)s.win_rows * s.d_in;
    } else {
        a.U = reinterpret_cast<const float*>(w.X) + w.row0 * s.d_in;
        a.u_cstride = w.x_cstride;
    }
    if (w.y_scratch) {  // squared error: the residual targets of this segment, rows from 0
        a.K = s.Kres32 + (size_t)w.c0 * s.T * dh;
        a.V = s.Vres32 + (size_t)w.c0 * s.T * dh;
        a.y_cstride = (long long)s.T * dh;
    } else {
        a.K = reinterpret_cast<const float*>(w.K) + w.row0 * dh;
        a.V = reinterpret_cast<const float*>(w.V) + w.row0 * dh;
        a.y_cstride = w.y_cstride;
    }
    a.row_avail = w.n_rows - w.row0;
    a.eta_in = w.eta_in ? w.eta_in + w.row0 : nullptr;
    a.eta_cstride = w.eta_cstride;
    a.eta = s.eta; a.dbeta = s.dbeta; a.b_beta = s.b_beta;
    a.W1 = s.W1; a.W2 = s.W2; a.mu1 = s.mu1; a.mu2 = s.mu2; a.n1 = s.n1; a.n2 = s.n2;
    a.sumsq = s.sumsq;
    a.dH = reinterpret_cast<float*>(s.dHt);
    a.At = reinterpret_cast<float*>(s.Att);
    a.loss = w.loss;
    a.step_sq = w.step_sq;
    a.status = s.status;
    return a;
}

// ------------------------------------------------------------------ squared-error pre-pass (fp32)
//
// Under the squared-error loss dL/dO = eta (M(u) - y) / T' = -eta (y - M(u)) / T', so the
// residual target y - M(u), with M(u) at the segment's starting weights, takes the place of
// y in both phases.  Two kernels: A' = SiLU(s1 H) s2 with the pending row scales folded in
// (so A' W2raw = A W2), written to the At scratch, which phase A overwrites only after
// the second kernel has read it; then the residual y - A' W2raw into the residual scratch
// and 1/2 |y - M(u)|^2 / T' into the loss.

__global__ void __launch_bounds__(256) mse_hidden_f32_kernel(const F32SegArgs a) {
    __shared__ float As[TK][A_TM + 4], Bs[TK][TN + 4];
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const int t0 = blockIdx.x * A_TM, h0 = blockIdx.y * TN, cz = blockIdx.z, cs = a.c0 + cz;
    int m_valid = (int)min((long long)min(A_TM, a.Tp - t0), a.row_avail - t0);
    if (m_valid < 0) m_valid = 0;
    float acc[A_MR][4] = {};
    simt_tile(acc, a.U + cz * a.u_cstride + (long long)t0 * a.d_in, a.d_in, 1,
              a.W1 + ((size_t)cs * a.d_hid + h0) * a.d_in, a.d_in, 1, a.d_in, m_valid, a.d_in, As, Bs);
    const float* prev1 = ss_ptr(a, a.parity ^ 1, 0) + (size_t)cs * a.d_hid;
    const float* prev2 = ss_ptr(a, a.parity ^ 1, 1) + (size_t)cs * a.d_hid;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const int h = h0 + tx * 4 + j;
        const float s1 = a.renorm_pending ? renorm_scale(a.n1[(size_t)cs * a.d_hid + h], prev1[h]) : 1.f;
        const float s2 = a.renorm_pending ? renorm_scale(a.n2[(size_t)cs * a.d_hid + h], prev2[h]) : 1.f;
#pragma unroll
        for (int i = 0; i < A_MR; ++i) {
            const int t = t0 + ty * A_MR + i;
            const float x = acc[i][j] * s1;
            a.At[((size_t)cs * a.T + t) * a.d_hid + h] = x * sigmoidf_(x) * s2;
        }
    }
}

__global__ void __launch_bounds__(256) mse_out_f32_kernel(const F32SegArgs a, float* Kres, float* Vres) {
    __shared__ float As[TK][A_TM + 4], Bs[TK][TN + 4];
    __shared__ float red[8];
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const int t0 = blockIdx.x * A_TM, o0 = blockIdx.y * TN, cz = blockIdx.z, cs = a.c0 + cz;
    const int dh = a.d_out / 2;
    float acc[A_MR][4] = {};
    simt_tile(acc, a.At + ((size_t)cs * a.T + t0) * a.d_hid, a.d_hid, 1, a.W2 + (size_t)cs * a.d_hid * a.d_out + o0,
              1, a.d_out, a.d_hid, min(A_TM, a.T - t0), a.d_hid, As, Bs);
    const bool kpart = o0 < dh;  // dh is a multiple of 64: a tile is all K or all V
    const int col0 = (kpart ? o0 : o0 - dh) + tx * 4;
    const float* Y = (kpart ? a.K : a.V) + cz * a.y_cstride + col0;
    float* R = (kpart ? Kres : Vres) + (size_t)cs * a.T * dh + col0;
    float lsum = 0.f;
#pragma unroll
    for (int i = 0; i < A_MR; ++i) {
        const int t = t0 + ty * A_MR + i;
        const bool live = t < a.Tp && t < a.row_avail;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float r = live ? Y[(long long)t * dh + j] - acc[i][j] : 0.f;
            R[(size_t)t * dh + j] = r;
            lsum = fmaf(r, r, lsum);
        }
    }
    if (a.loss) {
        lsum = warp_sum(lsum);
        if ((tid & 31) == 0) red[tid >> 5] = lsum;
        __syncthreads();
        if (tid == 0) {
            float tot = 0.f;
            for (int w = 0; w < 8; ++w) tot += red[w];
            atomicAdd(&a.loss[cz], 0.5f * tot / (float)a.Tp);
        }
    }
}

// ------------------------------------------------------------------ resident chains (fp32)
//
// When a chain's rows fit on chip, a whole call runs in one launch with the fast
// weights resident.  A CTA owns RB hidden units of one chain: their rows of W1 and
// W2, kept side by side as [W1 | W2] (width D = d_in + d_out) in shared memory, and
// their momentum and gradient in registers.  Hidden units do not interact within a
// step: H[:, r] = U W1[r]^T and R[:, r] = Y W2[r]^T use only row r, dL/dO does not
// depend on W (Eq. 10), the gradient rows dW1[r] = dH[:, r]^T U and dW2[r] =
// At[:, r]^T Y use only column r of dH and At, and Eq. 8's renormalisation is per
// row.  So a CTA takes its rows through every segment of the call without waiting
// for any other CTA, and the weights cross HBM once per call instead of once per
// segment.  Each segment streams its rows [U | K | V] once, RC tokens at a time,
// through a double-buffered cp.async stage: forward (H, R), the backward epilogue
// (dH, At), then the gradient accumulation from the same staged rows.  At the end
// of the segment the update (momentum, W -= mu) and the row renormalisation are
// applied in place.
//
// 512 threads (16 warps), so that shared-memory and FMA latencies are hidden.  Forward: half
// of the CTA contracts U with the W1 rows (H), the other half Y with the W2 rows (R); an
// output group is 2 tokens x 2 hidden units, its contraction split over KS = 32 / RB lanes
// (float4 steps over interleaved columns) and summed by shuffles; one thread per (token,
// hidden unit) then finishes the epilogue.  Backward: thread i owns column i of [W1 | W2]
// for all RB rows.
constexpr int RES_RC = 32;                                             // tokens per streamed chunk
__host__ __device__ constexpr int res_ld(int D) { return (D + 31) / 32 * 32 + 16; }  // row pitch, floats

struct ResArgs {
    int d_in, d_out, d_hid, T, c0, win, paper, momentum, renorm, n_seg;
    long long n_tok;             // tokens of this launch, from its first row
    const float* U;              // first row of the launch, chain cz at U + cz * u_cstride
    long long u_cstride;
    const float *K, *V;          // first row of the launch
    long long y_cstride;
    const float* eta;            // paper mode: rates [C][win] at the launch's first row (state chain index)
    const float* dbeta;          // paper mode: w_beta . x_t, same layout
    const float* eta_in;         // plain mode: caller rates at the launch's first row, or null
    long long eta_cstride;
    float lr;
    const float* b_beta;
    float *W1, *W2, *mu1, *mu2;
    const float *n1, *n2;
    float* loss;                 // loss of segment seg of chain cz at loss[seg * m_sstride + cz], or null
    float* step_sq;              // squared norm of the Eq. 8 step, same layout, or null
    long long m_sstride;         // stride between segments of loss and step_sq (0: one accumulator)
    int* status;
};

__device__ __forceinline__ void cp_async16(float* dst, const float* src, int src_bytes) {
    const unsigned d = (unsigned)__cvta_generic_to_shared(dst);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(d), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_async4(float* dst, const float* src, int src_bytes) {
    const unsigned d = (unsigned)__cvta_generic_to_shared(dst);
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(d), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N> __device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

__device__ __forceinline__ float dot4(const float4 a, const float4 b, float acc) {
    acc = fmaf(a.x, b.x, acc);
    acc = fmaf(a.y, b.y, acc);
    acc = fmaf(a.z, b.z, acc);
    return fmaf(a.w, b.w, acc);
}

constexpr int RES_NT = 512, RES_NW = RES_NT / 32;  // threads and warps of a resident CTA

// Sum of v over the CTA; every thread gets the total.  red: RES_NW floats.
__device__ __forceinline__ float block_sum_res(float v, float* red) {
    v = warp_sum(v);
    __syncthreads();
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
    __syncthreads();
    float t = 0.f;
#pragma unroll
    for (int w = 0; w < RES_NW; ++w) t += red[w];
    return t;
}

template <int RB>
__global__ void __launch_bounds__(RES_NT, 1) ttl_resident_f32_kernel(const ResArgs a) {
    constexpr int RC = RES_RC, KS = 32 / RB, RH = RB / 2, NW = RES_NW;
    static_assert(RB == 4 || RB == 8, "rows per CTA");
    extern __shared__ float4 res_smem[];
    const int D = a.d_in + a.d_out, LD = res_ld(D), dh = a.d_out / 2;
    float* Ws = reinterpret_cast<float*>(res_smem);  // [RB][LD]
    float* Xs = Ws + RB * LD;                        // [2][RC][LD]: rows [U | K | V] of a chunk
    float* Gs = Xs + 2 * RC * LD;                    // [RC][2][RB]: c dH, c A of the chunk
    float* HQ = Gs + RC * 2 * RB;                    // [2][RC][RB]: H and R of the chunk
    float* red = HQ + 2 * RC * RB;                   // [NW][2 RB]
    float* scl = red + NW * 2 * RB;                  // [2 RB] row scales, then beta
    float* etaS = scl + 2 * RB + 4;                  // [2][RC] rates of the chunk's tokens
    float* dbS = etaS + 2 * RC;                      // [2][RC] w_beta . x of the chunk's tokens
    float* nS = dbS + 2 * RC;                        // [2 RB] renormalisation targets
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int h0 = blockIdx.x * RB, cz = blockIdx.y, cs = a.c0 + cz;
    const float* Uc = a.U + cz * a.u_cstride;
    const float* Kc = a.K + cz * a.y_cstride;
    const float* Vc = a.V + cz * a.y_cstride;

    // stage RC token rows of segment seg, chunk ch into buffer b (a warp per row, lanes over
    // columns), with the tokens' rates and w_beta . x terms; rows past the segment read as 0
    auto issue = [&](int seg, int ch, int b) {
        const long long t_seg = (long long)seg * a.T;
        const int Tp = (int)min((long long)a.T, a.n_tok - t_seg);
        const int nvalid = min(RC, Tp - ch * RC);
        const long long r0 = t_seg + ch * RC;
        for (int t = warp; t < RC; t += NW) {
            const bool v = t < nvalid;
            const long long r = r0 + (v ? t : 0);
            const float* ur = Uc + r * a.d_in;
            const float* kr = Kc + r * dh;
            const float* vr = Vc + r * dh;
            float* dr = Xs + (b * RC + t) * LD;
            for (int c = 4 * lane; c < D; c += 128) {
                const float* src = c < a.d_in ? ur + c : c < a.d_in + dh ? kr + (c - a.d_in) : vr + (c - a.d_in - dh);
                cp_async16(dr + c, src, v ? 16 : 0);
            }
        }
        if (tid < 2 * RC) {
            const int t = tid & (RC - 1);
            const bool v = t < nvalid;
            const long long r = r0 + (v ? t : 0);
            if (tid < RC) {
                float* d = etaS + b * RC + t;
                if (a.paper)
                    cp_async4(d, a.eta + (size_t)cs * a.win + r, v ? 4 : 0);
                else if (a.eta_in)
                    cp_async4(d, a.eta_in + cz * a.eta_cstride + r, v ? 4 : 0);
                else
                    *d = v ? a.lr : 0.f;
            } else if (a.momentum) {
                cp_async4(dbS + b * RC + t, a.dbeta + (size_t)cs * a.win + r, v ? 4 : 0);
            }
        }
    };

    // resident rows, and the momentum of the thread's column (registers)
    for (int i = tid; i < RB * (D / 4); i += RES_NT) {
        const int r = i / (D / 4), c = 4 * (i - r * (D / 4));
        const size_t row = (size_t)cs * a.d_hid + h0 + r;
        const float* src = c < a.d_in ? a.W1 + row * a.d_in + c : a.W2 + row * a.d_out + (c - a.d_in);
        *reinterpret_cast<float4*>(Ws + r * LD + c) = *reinterpret_cast<const float4*>(src);
    }
    if (tid < 2 * RB) nS[tid] = (tid < RB ? a.n1 : a.n2)[(size_t)cs * a.d_hid + h0 + tid % RB];
    const float b_beta = a.momentum ? a.b_beta[cs] : 0.f;
    const int cb = tid;                          // owned column of [W1 | W2]
    const bool own = cb < D;
    const int kind = cb < a.d_in ? 0 : 1;
    float mu[RB], acc[RB];
#pragma unroll
    for (int r = 0; r < RB; ++r) {
        mu[r] = 0.f;
        acc[r] = 0.f;
        if (own && a.momentum) {
            const size_t row = (size_t)cs * a.d_hid + h0 + r;
            mu[r] = kind == 0 ? a.mu1[row * a.d_in + cb] : a.mu2[row * a.d_out + (cb - a.d_in)];
        }
    }

    // forward mapping: half 0 contracts U with W1 (H), half 1 Y with W2 (R); within a half an
    // output group og = (token pair tp, row pair rp) and a contraction lane ks
    const int half = tid >> 8, ht = tid & 255;
    const int ks = ht % KS, og = ht / KS, rp = og % RH, tp = og / RH;
    const int c_lo = half ? a.d_in : 0, c_hi = half ? D : a.d_in;
    bool finite = true;
    int buf = 0;
    issue(0, 0, 0);
    cp_async_commit();
    for (int seg = 0; seg < a.n_seg; ++seg) {
        const long long t_seg = (long long)seg * a.T;
        const int Tp = (int)min((long long)a.T, a.n_tok - t_seg);
        const int nch = (Tp + RC - 1) / RC;
        float lsum = 0.f, dbsum = 0.f;
        for (int ch = 0; ch < nch; ++ch) {
            if (ch + 1 < nch)
                issue(seg, ch + 1, buf ^ 1);
            else if (seg + 1 < a.n_seg)
                issue(seg + 1, 0, buf ^ 1);
            cp_async_commit();
            cp_async_wait<1>();
            __syncthreads();
            const float* Xb = Xs + buf * RC * LD;
            // tokens (tp, tp + 16) x rows (rp, rp + RH) of H (half 0) or R (half 1)
            float p[2][2] = {};
            {
                const float* x0 = Xb + tp * LD;
                const float* x1 = Xb + (tp + 16) * LD;
                const float* w0 = Ws + rp * LD;
                const float* w1 = Ws + (rp + RH) * LD;
#pragma unroll 2
                for (int c = c_lo + 4 * ks; c < c_hi; c += 4 * KS) {
                    const float4 u0 = *reinterpret_cast<const float4*>(x0 + c);
                    const float4 u1 = *reinterpret_cast<const float4*>(x1 + c);
                    const float4 b0 = *reinterpret_cast<const float4*>(w0 + c);
                    const float4 b1 = *reinterpret_cast<const float4*>(w1 + c);
                    p[0][0] = dot4(u0, b0, p[0][0]);
                    p[0][1] = dot4(u0, b1, p[0][1]);
                    p[1][0] = dot4(u1, b0, p[1][0]);
                    p[1][1] = dot4(u1, b1, p[1][1]);
                }
            }
#pragma unroll
            for (int o = 1; o < KS; o <<= 1)
#pragma unroll
                for (int i = 0; i < 2; ++i)
#pragma unroll
                    for (int j = 0; j < 2; ++j) p[i][j] += __shfl_xor_sync(0xffffffffu, p[i][j], o);
            if (ks == 0) {
#pragma unroll
                for (int i = 0; i < 2; ++i)
#pragma unroll
                    for (int j = 0; j < 2; ++j) HQ[(half * RC + tp + 16 * i) * RB + rp + RH * j] = p[i][j];
            }
            if (a.momentum && warp == 0) dbsum += warp_sum(lane < Tp - ch * RC ? dbS[buf * RC + lane] : 0.f);
            __syncthreads();
            if (tid < RC * RB) {
                // epilogue of output (t, r): c_t = -eta_t / T' (Eq. 10), A = SiLU(H)
                const int t = tid / RB, r = tid % RB;
                const float hv = HQ[t * RB + r], rv = HQ[(RC + t) * RB + r];
                const int ts = ch * RC + t;  // token within the segment
                const float ct = ts < Tp ? -etaS[buf * RC + t] / (float)Tp : 0.f;
                const float sg = sigmoidf_(hv);
                const float av = hv * sg;
                const float ds = sg * (1.f + hv * (1.f - sg));
                if (ts < Tp) lsum = fmaf(av, rv, lsum);
                Gs[(t * 2 + 0) * RB + r] = ct * rv * ds;
                Gs[(t * 2 + 1) * RB + r] = ct * av;
            }
            __syncthreads();
            // gradient rows: acc[r] += sum_t G[t][kind][r] * X[t][cb]
            if (own) {
                const int nv = min(RC, Tp - ch * RC);
                const float* gk = Gs + kind * RB;
#pragma unroll 4
                for (int t = 0; t < nv; ++t) {
                    const float x = Xb[t * LD + cb];
#pragma unroll
                    for (int r4 = 0; r4 < RB; r4 += 4) {
                        const float4 g4 = *reinterpret_cast<const float4*>(gk + t * 2 * RB + r4);
                        acc[r4] = fmaf(g4.x, x, acc[r4]);
                        acc[r4 + 1] = fmaf(g4.y, x, acc[r4 + 1]);
                        acc[r4 + 2] = fmaf(g4.z, x, acc[r4 + 2]);
                        acc[r4 + 3] = fmaf(g4.w, x, acc[r4 + 3]);
                    }
                }
            }
            __syncthreads();
            buf ^= 1;
        }
        // end of segment: Eq. 8 update, then the row renormalisation to the norms of W_0
        float beta = 0.f;
        if (a.momentum) {  // beta_s = sigmoid(mean_t w_beta . x_t + b_beta); warp 0 holds the sum
            if (tid == 0) scl[2 * RB] = sigmoidf_(dbsum / (float)Tp + b_beta);
            __syncthreads();
            beta = scl[2 * RB];
        }
        if (a.loss) {
            const float tot = block_sum_res(lsum, red);
            if (tid == 0) atomicAdd(&a.loss[seg * a.m_sstride + cz], -tot / (float)Tp);
        }
        float wn[RB], step = 0.f;
#pragma unroll
        for (int r = 0; r < RB; ++r) {
            const float mn = a.momentum ? fmaf(beta, mu[r], acc[r]) : acc[r];
            mu[r] = mn;
            acc[r] = 0.f;
            wn[r] = own ? Ws[r * LD + cb] - mn : 0.f;
            step = own ? fmaf(mn, mn, step) : step;
        }
        if (a.step_sq) {
            __syncthreads();  // red may still be read by block_sum_res above
            const float tot = block_sum_res(step, red);
            if (tid == 0) atomicAdd(&a.step_sq[seg * a.m_sstride + cz], tot);
        }
        if (a.renorm) {
            // row sums of squares per (matrix, row); a warp may hold columns of both matrices
            __syncthreads();  // red may still be read by block_sum_res above
#pragma unroll
            for (int k = 0; k < 2; ++k)
#pragma unroll
                for (int r = 0; r < RB; ++r) {
                    const float v = warp_sum(kind == k ? wn[r] * wn[r] : 0.f);
                    if (lane == 0) red[warp * 2 * RB + k * RB + r] = v;
                }
            __syncthreads();
            if (tid < 2 * RB) {
                float tot = 0.f;
                for (int w = 0; w < NW; ++w) tot += red[w * 2 * RB + tid];
                scl[tid] = renorm_scale(nS[tid], tot);
            }
            __syncthreads();
        }
        if (own) {
#pragma unroll
            for (int r = 0; r < RB; ++r) {
                const float wv = wn[r] * (a.renorm ? scl[kind * RB + r] : 1.f);
                finite = finite && isfinite(wv);
                Ws[r * LD + cb] = wv;
            }
        }
        __syncthreads();
    }
    cp_async_wait<0>();
    // write the rows and the momentum back (the CTA's rows lie inside the chain: index check of
    // MONE_DEBUG builds)
    if (!MONE_DCHECK(h0 + RB <= a.d_hid, a.status, DS_RESIDENT_ROWS)) return;
    for (int i = tid; i < RB * (D / 4); i += RES_NT) {
        const int r = i / (D / 4), c = 4 * (i - r * (D / 4));
        const size_t row = (size_t)cs * a.d_hid + h0 + r;
        float* dst = c < a.d_in ? a.W1 + row * a.d_in + c : a.W2 + row * a.d_out + (c - a.d_in);
        *reinterpret_cast<float4*>(dst) = *reinterpret_cast<const float4*>(Ws + r * LD + c);
    }
    if (own && a.momentum) {
#pragma unroll
        for (int r = 0; r < RB; ++r) {
            const size_t row = (size_t)cs * a.d_hid + h0 + r;
            (kind == 0 ? a.mu1[row * a.d_in + cb] : a.mu2[row * a.d_out + (cb - a.d_in)]) = mu[r];
        }
    }
    if (!finite) atomicOr(a.status, DEV_NONFINITE);
}

template <int RB> constexpr size_t res_smem_bytes(int D) {
    return sizeof(float) * ((size_t)(RB + 2 * RES_RC) * res_ld(D) + RES_RC * 2 * RB + 2 * RES_RC * RB +
                            RES_NW * 2 * RB + 2 * RB + 4 + 4 * RES_RC + 2 * RB);
}

// ------------------------------------------------------------------ state upkeep

// Apply the pending renormalisation of the last segment (when asked) and refresh
// the bf16 operand copies.  One warp per (row, chain, matrix), 8 rows a CTA; each lane
// moves 16-byte vectors, four of them in flight at a time (widths are multiples of 64).
__global__ void __launch_bounds__(256) finalize_kernel(DevState s, int c0, int parity, int apply_scale) {
    const int h = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
    const int cs = c0 + blockIdx.y, which = blockIdx.z;
    if (h >= s.d_hid) return;
    const int width = which ? s.d_out : s.d_in;
    float* w = (which ? s.W2 : s.W1) + ((size_t)cs * s.d_hid + h) * width;
    bf16* wb = s.dtype == 1 ? (which ? s.W2b : s.W1b) + ((size_t)cs * s.d_hid + h) * width : nullptr;
    float sc = 1.f;
    if (apply_scale) {
        const float* ss = s.sumsq + ((size_t)(parity * 2 + which) * s.C + cs) * s.d_hid;
        const float* n0 = (which ? s.n2 : s.n1) + (size_t)cs * s.d_hid;
        sc = renorm_scale(n0[h], ss[h]);
    }
    for (int base = lane * 4; base < width; base += 4 * 128) {
        float4 v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u)
            if (base + u * 128 < width) v[u] = *reinterpret_cast<const float4*>(w + base + u * 128);
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int i = base + u * 128;
            if (i >= width) break;
            const float4 x = make_float4(v[u].x * sc, v[u].y * sc, v[u].z * sc, v[u].w * sc);
            if (apply_scale) *reinterpret_cast<float4*>(w + i) = x;
            if (wb) {
                uint2 p;
                p.x = pack_bf16(x.x, x.y);
                p.y = pack_bf16(x.z, x.w);
                *reinterpret_cast<uint2*>(wb + i) = p;
            }
        }
    }
}

__global__ void __launch_bounds__(256) row_norms_kernel(DevState s) {
    const int h = blockIdx.x, cs = blockIdx.y, which = blockIdx.z;
    const int width = which ? s.d_out : s.d_in;
    const float* w = (which ? s.W2 : s.W1) + ((size_t)cs * s.d_hid + h) * width;
    __shared__ float red[8];
    float v = 0.f;
    for (int i = threadIdx.x; i < width; i += 256) v = fmaf(w[i], w[i], v);
    v = warp_sum(v);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
    __syncthreads();
    if (threadIdx.x == 0) {
        float tot = 0.f;
        for (int i = 0; i < 8; ++i) tot += red[i];
        (which ? s.n2 : s.n1)[(size_t)cs * s.d_hid + h] = sqrtf(tot);
    }
}

// ------------------------------------------------------------------ output-channel renormalisation
//
// The other reading of App. A's channel-wise renormalisation: a channel is an output
// channel of each matrix, so W1 keeps its rows (hidden units, renormalised inside the
// phase kernels) and every column of W2 (an output feature) is rescaled to its norm in
// W_0 after each update.  A column spans all hidden units, which the phase kernels tile
// apart, so this is a pass of its own over W2: partial column sums of squares over
// kColRowSlices row slices, then the rescale.  Warps cover 32 consecutive columns.

// 64 columns a CTA as 16 float4 column quads x 16 row groups: a warp reads 256 contiguous bytes
// of each of two rows.
__global__ void __launch_bounds__(256) col_partial_kernel(DevState s, int c0) {
    __shared__ float4 red[16][16];
    const int cq = threadIdx.x & 15, rg = threadIdx.x >> 4;
    const int col = blockIdx.x * 64 + 4 * cq, rs = blockIdx.y, cs = c0 + blockIdx.z;
    const int per = (s.d_hid + kColRowSlices - 1) / kColRowSlices;
    const int r1 = min(s.d_hid, (rs + 1) * per);
    const float* w = s.W2 + (size_t)cs * s.d_hid * s.d_out + col;
    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int r = rs * per + rg; r < r1; r += 16) {
        const float4 x = *reinterpret_cast<const float4*>(w + (size_t)r * s.d_out);
        v.x = fmaf(x.x, x.x, v.x);
        v.y = fmaf(x.y, x.y, v.y);
        v.z = fmaf(x.z, x.z, v.z);
        v.w = fmaf(x.w, x.w, v.w);
    }
    red[rg][cq] = v;
    __syncthreads();
    if (rg == 0) {
        float4 t = red[0][cq];
        for (int g = 1; g < 16; ++g) {
            t.x += red[g][cq].x; t.y += red[g][cq].y; t.z += red[g][cq].z; t.w += red[g][cq].w;
        }
        *reinterpret_cast<float4*>(s.colpart + ((size_t)rs * s.C + cs) * s.d_out + col) = t;
    }
}

__device__ __forceinline__ float col_sumsq(const DevState& s, int cs, int col) {
    float ss = 0.f;
    for (int rs = 0; rs < kColRowSlices; ++rs) ss += s.colpart[((size_t)rs * s.C + cs) * s.d_out + col];
    return ss;
}

// 64 rows x 64 columns a CTA (float4 column quads): W2[:, col] *= nc2[col] / |W2[:, col]|, and
// the bf16 copy.
__global__ void __launch_bounds__(256) col_scale_kernel(DevState s, int c0) {
    __shared__ float sc[64];
    const int cq = threadIdx.x & 15, rg = threadIdx.x >> 4;
    const int cs = c0 + blockIdx.z;
    if (threadIdx.x < 64) {
        const int col = blockIdx.x * 64 + threadIdx.x;
        sc[threadIdx.x] = renorm_scale(s.nc2[(size_t)cs * s.d_out + col], col_sumsq(s, cs, col));
    }
    __syncthreads();
    const float4 f = make_float4(sc[4 * cq], sc[4 * cq + 1], sc[4 * cq + 2], sc[4 * cq + 3]);
    const size_t base = (size_t)cs * s.d_hid * s.d_out + blockIdx.x * 64 + 4 * cq;
    const int r1 = min(s.d_hid, (int)blockIdx.y * 64 + 64);
    for (int r = blockIdx.y * 64 + rg; r < r1; r += 16) {
        const size_t i = base + (size_t)r * s.d_out;
        float4 x = *reinterpret_cast<const float4*>(s.W2 + i);
        x.x *= f.x; x.y *= f.y; x.z *= f.z; x.w *= f.w;
        *reinterpret_cast<float4*>(s.W2 + i) = x;
        if (s.dtype == 1) {
            uint2 p;
            p.x = pack_bf16(x.x, x.y);
            p.y = pack_bf16(x.z, x.w);
            *reinterpret_cast<uint2*>(s.W2b + i) = p;
        }
    }
}

__global__ void __launch_bounds__(256) col_targets_kernel(DevState s) {
    const int col = blockIdx.x * 256 + threadIdx.x, cs = blockIdx.y;
    if (col < s.d_out) s.nc2[(size_t)cs * s.d_out + col] = sqrtf(col_sumsq(s, cs, col));
    for (int h = col; h < s.d_hid; h += gridDim.x * 256) s.n2[(size_t)cs * s.d_hid + h] = -1.f;
}

__global__ void __launch_bounds__(256) gate_silu_kernel(float* g, size_t n, int from_one) {
    const size_t i = (size_t)blockIdx.x * 256 + threadIdx.x;
    if (i < n) {
        const float v = from_one ? 1.f : g[i];
        g[i] = v * sigmoidf_(v);
    }
}

// ------------------------------------------------------------------ memory read (Eq. 4)

__global__ void __launch_bounds__(256) read_hidden_kernel(DevState s, int Q) {
    __shared__ float As[TK][TM + 4], Bs[TK][TN + 4];
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const int q0 = blockIdx.x * TM, h0 = blockIdx.y * TN, c = blockIdx.z;
    float acc[4][4] = {};
    simt_tile(acc, s.Uq + ((size_t)c * Q + q0) * s.d_in, s.d_in, 1, s.W1 + ((size_t)c * s.d_hid + h0) * s.d_in,
              s.d_in, 1, s.d_in, min(TM, Q - q0), s.d_in, As, Bs);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int q = q0 + ty * 4 + i;
        if (q >= Q) continue;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float hv = acc[i][j];
            s.Aq[((size_t)c * Q + q) * s.d_hid + h0 + tx * 4 + j] = hv * sigmoidf_(hv);
        }
    }
}

__global__ void __launch_bounds__(256) read_out_kernel(DevState s, int Q) {
    __shared__ float As[TK][TM + 4], Bs[TK][TN + 4];
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const int q0 = blockIdx.x * TM, o0 = blockIdx.y * TN, c = blockIdx.z;
    float acc[4][4] = {};
    simt_tile(acc, s.Aq + ((size_t)c * Q + q0) * s.d_hid, s.d_hid, 1, s.W2 + (size_t)c * s.d_hid * s.d_out + o0, 1,
              s.d_out, s.d_hid, min(TM, Q - q0), s.d_hid, As, Bs);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int q = q0 + ty * 4 + i;
        if (q >= Q) continue;
#pragma unroll
        for (int j = 0; j < 4; ++j) s.Oq[((size_t)c * Q + q) * s.d_out + o0 + tx * 4 + j] = acc[i][j];
    }
}

// Per output head: gate_h * o_h / sqrt(mean(o_h^2) + eps), written with caller strides.
template <typename Tout>
__global__ void __launch_bounds__(256) read_norm_kernel(DevState s, int Q, Tout* Kout, Tout* Vout, long long s0,
                                                        long long s1, long long s2, long long s3, int L) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nh = 2 * s.n_kv;
    const long long job = (long long)blockIdx.x * 8 + warp;  // (c, q, head)
    if (job >= (long long)s.C * Q * nh) return;
    const int head = (int)(job % nh);
    const int q = (int)((job / nh) % Q);
    const int c = (int)(job / ((long long)nh * Q));
    const float* o = s.Oq + ((size_t)c * Q + q) * s.d_out + head * s.hd;
    float v = 0.f;
    for (int i = lane; i < s.hd; i += 32) v = fmaf(o[i], o[i], v);
    v = warp_sum(v);
    const float g = s.gate ? s.gate[(size_t)c * nh + head] : 1.f;
    const float sc = g / sqrtf(v / (float)s.hd + s.rms_eps);
    Tout* out = head < s.n_kv ? Kout : Vout;
    const int kvh = head < s.n_kv ? head : head - s.n_kv;
    out += (long long)(c / L) * s0 + (long long)(c % L) * s1 + (long long)kvh * s2 + (long long)q * s3;
    for (int i = lane; i < s.hd; i += 32) out[i] = from_f<Tout>(o[i] * sc);
}

}  // namespace

cudaError_t launch_phase_a_f32(const DevState& s, const SegWork& w, cudaStream_t st) {
    F32SegArgs a = make_f32_args(s, w);
    dim3 grid((s.T + A_TM - 1) / A_TM, s.d_hid / TN, w.nc);
    phase_a_f32_kernel<<<grid, 256, 0, st>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_phase_b_f32(const DevState& s, const SegWork& w, cudaStream_t st) {
    F32SegArgs a = make_f32_args(s, w);
    dim3 grid((s.d_in + s.d_out) / TN, s.d_hid / B_TM, w.nc);
    phase_b_f32_kernel<<<grid, 256, 0, st>>>(a);
    return cudaGetLastError();
}

bool resident_f32_fits(const DevState& s) {
    return s.dtype == 0 && s.memory == 0 && s.loss == 0 && !s.col_renorm && s.d_in + s.d_out <= 512 && s.d_in % 4 == 0 &&
           s.d_out % 8 == 0 && s.d_hid % 8 == 0;
}

cudaError_t launch_resident_f32(const DevState& s, const SegWork& w, long long n_tok, cudaStream_t st) {
    ResArgs a{};
    a.d_in = s.d_in; a.d_out = s.d_out; a.d_hid = s.d_hid; a.T = s.T; a.c0 = w.c0; a.win = s.win_rows;
    a.paper = s.mode == 1; a.momentum = s.momentum; a.renorm = s.renorm;
    a.n_tok = n_tok;
    a.n_seg = (int)((n_tok + s.T - 1) / s.T);
    const int dh = s.d_out / 2;
    if (a.paper) {
        a.U = reinterpret_cast<const float*>(s.U) + ((size_t)w.c0 * s.win_rows + w.u_off) * s.d_in;
        a.u_cstride = (long long)s.win_rows * s.d_in;
        a.eta = s.eta + w.u_off;
        a.dbeta = s.dbeta + w.u_off;
    } else {
        a.U = reinterpret_cast<const float*>(w.X) + w.row0 * s.d_in;
        a.u_cstride = w.x_cstride;
    }
    a.K = reinterpret_cast<const float*>(w.K) + w.row0 * dh;
    a.V = reinterpret_cast<const float*>(w.V) + w.row0 * dh;
    a.y_cstride = w.y_cstride;
    a.eta_in = w.eta_in ? w.eta_in + w.row0 : nullptr;
    a.eta_cstride = w.eta_cstride;
    a.lr = s.lr;
    a.b_beta = s.b_beta;
    a.W1 = s.W1; a.W2 = s.W2; a.mu1 = s.mu1; a.mu2 = s.mu2; a.n1 = s.n1; a.n2 = s.n2;
    a.loss = w.loss0 ? w.loss0 : w.loss;
    a.step_sq = w.step0;
    a.m_sstride = w.loss0 || w.step0 ? w.mstride : 0;
    a.status = s.status;
    int dev = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    // four rows a CTA while that still fits the chains in one wave, else eight (less re-streaming)
    const int D = s.d_in + s.d_out;
    if ((long long)w.nc * (s.d_hid / 4) <= sms) {
        const size_t bytes = res_smem_bytes<4>(D);
        e = cudaFuncSetAttribute(ttl_resident_f32_kernel<4>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
        if (e != cudaSuccess) return e;
        ttl_resident_f32_kernel<4><<<dim3(s.d_hid / 4, w.nc), RES_NT, bytes, st>>>(a);
    } else {
        const size_t bytes = res_smem_bytes<8>(D);
        e = cudaFuncSetAttribute(ttl_resident_f32_kernel<8>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
        if (e != cudaSuccess) return e;
        ttl_resident_f32_kernel<8><<<dim3(s.d_hid / 8, w.nc), RES_NT, bytes, st>>>(a);
    }
    return cudaGetLastError();
}

cudaError_t launch_mse_f32(const DevState& s, const SegWork& w, cudaStream_t st) {
    F32SegArgs a = make_f32_args(s, w);
    mse_hidden_f32_kernel<<<dim3((s.T + A_TM - 1) / A_TM, s.d_hid / TN, w.nc), 256, 0, st>>>(a);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    mse_out_f32_kernel<<<dim3((s.T + A_TM - 1) / A_TM, s.d_out / TN, w.nc), 256, 0, st>>>(a, s.Kres32, s.Vres32);
    return cudaGetLastError();
}

cudaError_t launch_finalize(const DevState& s, int c0, int nc, int parity, int apply_scale, cudaStream_t st) {
    finalize_kernel<<<dim3((s.d_hid + 7) / 8, nc, 2), 256, 0, st>>>(s, c0, parity, apply_scale);
    return cudaGetLastError();
}

cudaError_t launch_col_renorm(const DevState& s, int c0, int nc, cudaStream_t st) {
    col_partial_kernel<<<dim3(s.d_out / 64, kColRowSlices, nc), 256, 0, st>>>(s, c0);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    col_scale_kernel<<<dim3(s.d_out / 64, (s.d_hid + 63) / 64, nc), 256, 0, st>>>(s, c0);
    return cudaGetLastError();
}

cudaError_t launch_col_targets(const DevState& s, cudaStream_t st) {
    col_partial_kernel<<<dim3(s.d_out / 64, kColRowSlices, s.C), 256, 0, st>>>(s, 0);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    col_targets_kernel<<<dim3((s.d_out + 255) / 256, s.C), 256, 0, st>>>(s);
    return cudaGetLastError();
}

cudaError_t launch_gate_silu(float* gate, size_t n, int from_one, cudaStream_t st) {
    gate_silu_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(gate, n, from_one);
    return cudaGetLastError();
}

cudaError_t launch_row_norms(const DevState& s, cudaStream_t st) {
    row_norms_kernel<<<dim3(s.d_hid, s.C, 2), 256, 0, st>>>(s);
    return cudaGetLastError();
}

cudaError_t launch_read_norm(const DevState& s, int Q, int n_layers, void* K_out, void* V_out,
                             const long long* strides, cudaStream_t st) {
    const long long jobs = (long long)s.C * Q * 2 * s.n_kv;
    dim3 grid((unsigned)((jobs + 7) / 8));
    if (s.dtype == 0)
        read_norm_kernel<float><<<grid, 256, 0, st>>>(s, Q, (float*)K_out, (float*)V_out, strides[0], strides[1],
                                                      strides[2], strides[3], n_layers);
    else
        read_norm_kernel<bf16><<<grid, 256, 0, st>>>(s, Q, (bf16*)K_out, (bf16*)V_out, strides[0], strides[1],
                                                     strides[2], strides[3], n_layers);
    return cudaGetLastError();
}

cudaError_t launch_read(const DevState& s, int Q, int n_layers, void* K_out, void* V_out,
                        const long long* strides, cudaStream_t st) {
    read_hidden_kernel<<<dim3((Q + TM - 1) / TM, s.d_hid / TN, s.C), 256, 0, st>>>(s, Q);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    read_out_kernel<<<dim3((Q + TM - 1) / TM, s.d_out / TN, s.C), 256, 0, st>>>(s, Q);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    const long long jobs = (long long)s.C * Q * 2 * s.n_kv;
    dim3 grid((unsigned)((jobs + 7) / 8));
    if (s.dtype == 0)
        read_norm_kernel<float><<<grid, 256, 0, st>>>(s, Q, (float*)K_out, (float*)V_out, strides[0], strides[1],
                                                      strides[2], strides[3], n_layers);
    else
        read_norm_kernel<bf16><<<grid, 256, 0, st>>>(s, Q, (bf16*)K_out, (bf16*)V_out, strides[0], strides[1],
                                                     strides[2], strides[3], n_layers);
    return cudaGetLastError();
}

// ------------------------------------------------------------------ allocation-free memory read
//
// Scratch of mone_mem_generate_kv_noalloc: a fixed file-scope device array that
// every GPU loading the library holds until the process exits.  Host code cannot
// use the array's name as a device address (it is a host-side stand-in), so the
// address is resolved with cudaGetSymbolAddress, once per device, with that
// device current.

static __device__ __align__(256) float g_noalloc_scratch[kNoAllocScratchFloats];

namespace {
std::mutex g_noalloc_mu;
float* g_noalloc_ptr[64] = {};  // per device ordinal
}  // namespace

cudaError_t noalloc_scratch(float** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lk(g_noalloc_mu);
    if (!g_noalloc_ptr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) return e;
        g_noalloc_ptr[dev] = static_cast<float*>(p);
    }
    *out = g_noalloc_ptr[dev];
    return cudaSuccess;
}

cudaError_t launch_read_noalloc(const DevState& s, const TcMaps* tc, const void* Xq, int Q, int n_layers,
                                void* K_out, void* V_out, const long long* strides, cudaStream_t st) {
    float* base = nullptr;
    cudaError_t e = noalloc_scratch(&base);
    if (e != cudaSuccess) return e;
    // the same kernels as the allocating read, pointed at the fixed scratch; every
    // element of the regions is written before it is read, so nothing needs clearing
    // between calls
    DevState t = s;
    t.Uq = base;
    t.Aq = t.Uq + (size_t)s.C * Q * s.d_in;
    t.Oq = t.Aq + (size_t)s.C * Q * s.d_hid;
    if (tc) return launch_read_tc(t, *tc, Xq, t.Uq, t.Aq, t.Oq, Q, n_layers, K_out, V_out, strides, st);
    e = launch_query_transform(t, Xq, Q, t.Uq, false, st);
    return e != cudaSuccess ? e : launch_read(t, Q, n_layers, K_out, V_out, strides, st);
}

cudaError_t launch_zero_f32(float* p, size_t n, cudaStream_t st) {
    return cudaMemsetAsync(p, 0, n * sizeof(float), st);
}

}  // namespace mone
