// fp32 path of the TTL step, state upkeep kernels and the memory read.
//
// The fp32 path (the tiny fp32 workload: 256 -> 512 -> 256, T = 128) is
// latency-bound, so it uses plain CUDA-core FFMA tiles (64 x 64 per CTA, 4 x 4 per
// thread, 64-deep K slabs so that each thread has 32 loads in flight per slab) in fp32
// throughout.  It computes the same two phases as the bf16
// tensor-core path:
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
            finite = finite && isfinite(wn);
        }
        ss += __shfl_xor_sync(0xffffffffu, ss, 8);
        ss += __shfl_xor_sync(0xffffffffu, ss, 4);
        ss += __shfl_xor_sync(0xffffffffu, ss, 2);
        ss += __shfl_xor_sync(0xffffffffu, ss, 1);
        if (tx == 0) atomicAdd(&cur[h], ss);
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
    a.K = reinterpret_cast<const float*>(w.K) + w.row0 * dh;
    a.V = reinterpret_cast<const float*>(w.V) + w.row0 * dh;
    a.y_cstride = w.y_cstride;
    a.row_avail = w.n_rows - w.row0;
    a.eta_in = w.eta_in ? w.eta_in + w.row0 : nullptr;
    a.eta_cstride = w.eta_cstride;
    a.eta = s.eta; a.dbeta = s.dbeta; a.b_beta = s.b_beta;
    a.W1 = s.W1; a.W2 = s.W2; a.mu1 = s.mu1; a.mu2 = s.mu2; a.n1 = s.n1; a.n2 = s.n2;
    a.sumsq = s.sumsq;
    a.dH = reinterpret_cast<float*>(s.dHt);
    a.At = reinterpret_cast<float*>(s.Att);
    a.loss = w.loss;
    a.status = s.status;
    return a;
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

cudaError_t launch_finalize(const DevState& s, int c0, int nc, int parity, int apply_scale, cudaStream_t st) {
    finalize_kernel<<<dim3((s.d_hid + 7) / 8, nc, 2), 256, 0, st>>>(s, c0, parity, apply_scale);
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
    if (tc) {
        e = launch_query_transform(t, Xq, Q, t.Uq, true, st);
        return e != cudaSuccess ? e : launch_read_tc(t, *tc, t.Uq, t.Aq, Q, n_layers, K_out, V_out, strides, st);
    }
    e = launch_query_transform(t, Xq, Q, t.Uq, false, st);
    return e != cudaSuccess ? e : launch_read(t, Q, n_layers, K_out, V_out, strides, st);
}

cudaError_t launch_zero_f32(float* p, size_t n, cudaStream_t st) {
    return cudaMemsetAsync(p, 0, n * sizeof(float), st);
}

}  // namespace mone
