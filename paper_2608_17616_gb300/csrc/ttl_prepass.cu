// Input prepass of a segment (paper mode) and the query transform of the read.
//
// Paper mode (App. A): keys and queries go through an affine rescale, SiLU and a
// per-token L2 normalisation: u_j = z_j / sqrt(|z_j|^2 + 1e-12),
// z_j = SiLU(alpha * x_j + gamma).  The same pass produces the per-token learning
// rate eta_j = softplus(w_eta . x_j + b_eta) and the per-token term
// w_beta . x_j of the momentum decay beta_s = sigmoid(mean_j(w_beta . x_j) + b_beta).
//
// Streaming, HBM-bound: reads d_in elements and writes d_in elements per token.
#include "mone_common.cuh"

namespace mone {

namespace {

struct PrepassArgs {
    const void* X;
    long long x_cstride;  // elements between chains of X
    long long row0;       // first row of the segment in X
    long long n_rows;     // rows per chain in X (beyond: out of range)
    int Tp;               // tokens present
    int rows;             // rows to produce (segment size T, or Q for queries)
    int c0;               // state chain offset
    int d_in;
    int paper;            // transform on/off
    int query;            // query mode: fp32 output, no rates
    const float *alpha, *gamma, *w_eta, *b_eta, *w_beta;
    const float* eta_in;  // caller's rates (replace softplus) or null
    long long eta_cstride;
    void* U;              // [C][rows][d_in], type Tout
    float* eta;           // [C][rows]
    float* dbeta;         // [C][rows]
};

// 16-byte vector of inputs: 8 bf16 or 4 fp32 values, kept packed in registers.
template <typename T> struct Vec;
template <> struct Vec<bf16> {
    static constexpr int N = 8;
    __device__ static void unpack(const uint4& r, float (&v)[8]) {
        const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&r);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float2 f = __bfloat1622float2(h[i]);
            v[2 * i] = f.x;
            v[2 * i + 1] = f.y;
        }
    }
};
template <> struct Vec<float> {
    static constexpr int N = 4;
    __device__ static void unpack(const uint4& r, float (&v)[4]) {
        v[0] = __uint_as_float(r.x); v[1] = __uint_as_float(r.y);
        v[2] = __uint_as_float(r.z); v[3] = __uint_as_float(r.w);
    }
};

template <typename T, int N> __device__ __forceinline__ void store_vec(T* p, const float (&v)[N]);
template <> __device__ __forceinline__ void store_vec<bf16, 8>(bf16* p, const float (&v)[8]) {
    uint4 r;
    __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&r);
#pragma unroll
    for (int i = 0; i < 4; ++i) h[i] = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
    *reinterpret_cast<uint4*>(p) = r;
}
template <> __device__ __forceinline__ void store_vec<float, 4>(float* p, const float (&v)[4]) {
    *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
}
template <> __device__ __forceinline__ void store_vec<float, 8>(float* p, const float (&v)[8]) {
    *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
    *reinterpret_cast<float4*>(p + 4) = make_float4(v[4], v[5], v[6], v[7]);
}

template <int N>
__device__ __forceinline__ void load_f32(const float* p, float (&v)[N]) {
#pragma unroll
    for (int i = 0; i < N; i += 4) {
        const float4 r = *reinterpret_cast<const float4*>(p + i);
        v[i] = r.x; v[i + 1] = r.y; v[i + 2] = r.z; v[i + 3] = r.w;
    }
}

template <int N>
__device__ __forceinline__ void load_smem(const float* p, float (&v)[N]) {
#pragma unroll
    for (int i = 0; i < N; i += 4) {
        const float4 r = *reinterpret_cast<const float4*>(p + i);
        v[i] = r.x; v[i + 1] = r.y; v[i + 2] = r.z; v[i + 3] = r.w;
    }
}

// Logistic function: fast form for bf16 data (error far below bf16 rounding), the
// accurate one for the fp32 path.
template <typename T> __device__ __forceinline__ float sig(float z);
template <> __device__ __forceinline__ float sig<bf16>(float z) { return sigmoid_fast(z); }
template <> __device__ __forceinline__ float sig<float>(float z) { return sigmoidf_(z); }

constexpr int PRE_ROWS = 32;  // token rows per CTA (4 per warp)

// One warp per token row, 16-byte vector loads.  The chain's meta-parameters are
// staged once per CTA in shared memory ([4][d_in]: alpha, gamma, w_eta, w_beta).
// Statistics first; the output pass re-reads the row (an L1/L2 hit).
template <typename Tin, typename Tout>
__global__ void __launch_bounds__(256) prepass_kernel(const PrepassArgs a) {
    extern __shared__ float4 meta4[];
    float* meta = reinterpret_cast<float*>(meta4);
    constexpr int V = Vec<Tin>::N;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int cz = blockIdx.y;
    const int cs = a.c0 + cz;
    const int d = a.d_in;
    const int nmeta = a.paper ? (a.query ? 2 : 4) : 0;
    for (int m = 0; m < nmeta; ++m) {
        const float* src = (m == 0 ? a.alpha : m == 1 ? a.gamma : m == 2 ? a.w_eta : a.w_beta) + (size_t)cs * d;
        for (int i = threadIdx.x * 4; i < d; i += 256 * 4)
            *reinterpret_cast<float4*>(meta + m * d + i) = *reinterpret_cast<const float4*>(src + i);
    }
    __syncthreads();
    const float* al = meta;
    const float* ga = meta + d;
    const float* we = meta + 2 * d;
    const float* wb = meta + 3 * d;
    const int t_end = min(a.rows, (int)(blockIdx.x + 1) * PRE_ROWS);
    for (int t = blockIdx.x * PRE_ROWS + warp; t < t_end; t += 8) {
        Tout* u = reinterpret_cast<Tout*>(a.U) + ((size_t)cs * a.rows + t) * d;
        const bool present = t < a.Tp && (a.row0 + t) < a.n_rows;
        if (!present) {
            float z[V];
#pragma unroll
            for (int e = 0; e < V; ++e) z[e] = 0.f;
            for (int i0 = lane * V; i0 < d; i0 += 32 * V) store_vec<Tout, V>(u + i0, z);
            if (!a.query && lane == 0) {
                a.eta[(size_t)cs * a.rows + t] = 0.0f;
                a.dbeta[(size_t)cs * a.rows + t] = 0.0f;
            }
            continue;
        }
        const Tin* x = reinterpret_cast<const Tin*>(a.X) + cz * a.x_cstride + (a.row0 + t) * d;
        float ss = 0.f, de = 0.f, db = 0.f;
        if (a.paper) {
#pragma unroll 4
            for (int i0 = lane * V; i0 < d; i0 += 32 * V) {
                float xv[V], av[V], gv[V];
                Vec<Tin>::unpack(*reinterpret_cast<const uint4*>(x + i0), xv);
                load_smem<V>(al + i0, av);
                load_smem<V>(ga + i0, gv);
                if (!a.query) {
                    float wev[V], wbv[V];
                    load_smem<V>(we + i0, wev);
                    load_smem<V>(wb + i0, wbv);
#pragma unroll
                    for (int e = 0; e < V; ++e) {
                        de = fmaf(wev[e], xv[e], de);
                        db = fmaf(wbv[e], xv[e], db);
                    }
                }
#pragma unroll
                for (int e = 0; e < V; ++e) {
                    const float zp = fmaf(av[e], xv[e], gv[e]);
                    const float z = zp * sig<Tin>(zp);
                    ss = fmaf(z, z, ss);
                }
            }
            ss = warp_sum(ss);
            if (!a.query) {
                de = warp_sum(de);
                db = warp_sum(db);
            }
        }
        const float inv = a.paper ? 1.0f / sqrtf(ss + 1e-12f) : 1.0f;
#pragma unroll 4
        for (int i0 = lane * V; i0 < d; i0 += 32 * V) {
            float xv[V];
            Vec<Tin>::unpack(*reinterpret_cast<const uint4*>(x + i0), xv);
            if (a.paper) {
                float av[V], gv[V];
                load_smem<V>(al + i0, av);
                load_smem<V>(ga + i0, gv);
#pragma unroll
                for (int e = 0; e < V; ++e) {
                    const float zp = fmaf(av[e], xv[e], gv[e]);
                    xv[e] = zp * sig<Tin>(zp) * inv;
                }
            }
            store_vec<Tout, V>(u + i0, xv);
        }
        if (!a.query && lane == 0) {
            float e;
            if (a.eta_in)
                e = a.eta_in[cz * a.eta_cstride + a.row0 + t];
            else
                e = softplusf_(de + a.b_eta[cs]);
            a.eta[(size_t)cs * a.rows + t] = e;
            a.dbeta[(size_t)cs * a.rows + t] = db;
        }
    }
}

template <typename Tin, typename Tout>
cudaError_t launch_one(const PrepassArgs& a, int nchains, cudaStream_t st) {
    const size_t smem = (size_t)(a.paper ? (a.query ? 2 : 4) : 0) * a.d_in * sizeof(float);
    static bool attr_set = false;  // set once per process: the largest supported d_in needs 64 KB
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(prepass_kernel<Tin, Tout>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             4 * 4096 * (int)sizeof(float));
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    dim3 grid((a.rows + PRE_ROWS - 1) / PRE_ROWS, nchains);
    prepass_kernel<Tin, Tout><<<grid, 256, smem, st>>>(a);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_prepass(const DevState& s, const SegWork& w, cudaStream_t st) {
    PrepassArgs a{};
    a.X = w.X;
    a.x_cstride = w.x_cstride;
    a.row0 = w.row0;
    a.n_rows = w.n_rows;
    a.Tp = w.Tp;
    a.rows = s.T;
    a.c0 = w.c0;
    a.d_in = s.d_in;
    a.paper = 1;
    a.query = 0;
    a.alpha = s.alpha;
    a.gamma = s.gamma;
    a.w_eta = s.w_eta;
    a.b_eta = s.b_eta;
    a.w_beta = s.w_beta;
    a.eta_in = w.eta_in;
    a.eta_cstride = w.eta_cstride;
    a.U = s.U;
    a.eta = s.eta;
    a.dbeta = s.dbeta;
    return s.dtype == 0 ? launch_one<float, float>(a, w.nc, st) : launch_one<bf16, bf16>(a, w.nc, st);
}

cudaError_t launch_query_transform(const DevState& s, const void* Xq, int Q, cudaStream_t st) {
    PrepassArgs a{};
    a.X = Xq;
    a.x_cstride = (long long)Q * s.d_in;
    a.row0 = 0;
    a.n_rows = Q;
    a.Tp = Q;
    a.rows = Q;
    a.c0 = 0;
    a.d_in = s.d_in;
    a.paper = s.mode == 1;
    a.query = 1;
    a.alpha = s.alpha;
    a.gamma = s.gamma;
    a.U = s.Uq;
    return s.dtype == 0 ? launch_one<float, float>(a, s.C, st) : launch_one<bf16, float>(a, s.C, st);
}

}  // namespace mone
