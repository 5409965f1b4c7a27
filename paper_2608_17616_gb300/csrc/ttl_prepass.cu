// Input prepass of a segment (paper mode) and the query transform of the read.
// On the bf16 path the segment prepass writes the unnormalised z and 1/|z| per
// token in one pass; phase A applies the scale (H = diag(1/|z|) Z W1^T, and
// dH^T U = (diag(1/|z|) dH)^T Z), which is exact algebra, not an approximation.
//
// Paper mode (App. A): keys and queries go through an affine rescale, SiLU and a
// per-token L2 normalisation: u_j = z_j / sqrt(|z_j|^2 + 1e-12),
// z_j = SiLU(alpha * x_j + gamma).  The same pass produces the per-token learning
// rate eta_j = softplus(w_eta . x_j + b_eta) and the per-token term
// w_beta . x_j of the momentum decay beta_s = sigmoid(mean_j(w_beta . x_j) + b_beta).
//
// Streaming, HBM-bound: reads d_in elements and writes d_in elements per token.
#include <algorithm>

#include "mone_common.cuh"

namespace mone {

namespace {

struct PrepassArgs {
    const void* X;
    long long x_cstride;  // elements between chains of X
    long long row0;       // first row of the segment in X
    long long n_rows;     // rows per chain in X (beyond: out of range)
    int Tp;               // tokens present
    int rows;             // rows to produce (a window of tokens, or Q for queries)
    int row_stride;       // rows per chain in the output buffers
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
    float* zinv;          // [C][rows] 1/|z_t|; when set, U receives the unnormalised z (one pass)
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

// Logistic function: fast form for bf16 data (error far below bf16 rounding), the
// accurate one for the fp32 path.
template <typename T> __device__ __forceinline__ float sig(float z);
template <> __device__ __forceinline__ float sig<bf16>(float z) { return sigmoid_fast(z); }
template <> __device__ __forceinline__ float sig<float>(float z) { return sigmoidf_(z); }

constexpr int RPW = 2;                 // token rows per warp, processed together
constexpr int PRE_ROWS = 8 * RPW;      // token rows per CTA

// Each warp transforms RPW token rows at once with 16-byte vector loads, so every
// load of the chain's meta-parameters (alpha, gamma, w_eta, w_beta) serves RPW
// rows.  Statistics first; the output pass re-reads the rows (L1/L2 hits).
template <typename Tin, typename Tout>
__global__ void __launch_bounds__(256) prepass_kernel(const PrepassArgs a) {
    constexpr int V = Vec<Tin>::N;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int cz = blockIdx.y;
    const int cs = a.c0 + cz;
    const int d = a.d_in;
    const int t0 = blockIdx.x * PRE_ROWS + warp * RPW;
    const float* al = a.paper ? a.alpha + (size_t)cs * d : nullptr;
    const float* ga = a.paper ? a.gamma + (size_t)cs * d : nullptr;
    const float* we = (a.paper && !a.query) ? a.w_eta + (size_t)cs * d : nullptr;
    const float* wb = (a.paper && !a.query) ? a.w_beta + (size_t)cs * d : nullptr;
    bool live[RPW];
    const Tin* x[RPW];
    Tout* u[RPW];
#pragma unroll
    for (int r = 0; r < RPW; ++r) {
        const int t = t0 + r;
        live[r] = t < a.rows && t < a.Tp && (a.row0 + t) < a.n_rows;
        x[r] = reinterpret_cast<const Tin*>(a.X) + cz * a.x_cstride + (a.row0 + (live[r] ? t : 0)) * d;
        u[r] = reinterpret_cast<Tout*>(a.U) + ((size_t)cs * a.row_stride + (t < a.rows ? t : 0)) * d;
    }
    float ss[RPW], de[RPW], db[RPW];
#pragma unroll
    for (int r = 0; r < RPW; ++r) ss[r] = de[r] = db[r] = 0.f;
    if (a.paper && a.zinv) {
        // one pass: write z = SiLU(alpha x + gamma) unnormalised; the row scale 1/|z|
        // is applied by the consumer (it commutes with the contraction over d_in).
        // Loads of a 4-vector super-chunk are all issued before any arithmetic.
        constexpr int SC = 4;
        for (int base = lane * V; base < d; base += SC * 32 * V) {
            uint4 xr[RPW][SC];
#pragma unroll
            for (int r = 0; r < RPW; ++r)
#pragma unroll
                for (int q = 0; q < SC; ++q) {
                    const int i0 = base + q * 32 * V;
                    if (live[r] && i0 < d) xr[r][q] = __ldg(reinterpret_cast<const uint4*>(x[r] + i0));
                }
#pragma unroll
            for (int q = 0; q < SC; ++q) {
                const int i0 = base + q * 32 * V;
                if (i0 >= d) break;
                float av[V], gv[V], wev[V], wbv[V];
                load_f32<V>(al + i0, av);
                load_f32<V>(ga + i0, gv);
                load_f32<V>(we + i0, wev);
                load_f32<V>(wb + i0, wbv);
#pragma unroll
                for (int r = 0; r < RPW; ++r) {
                    if (t0 + r >= a.rows) continue;
                    float xv[V];
                    if (live[r]) {
                        Vec<Tin>::unpack(xr[r][q], xv);
#pragma unroll
                        for (int e = 0; e < V; ++e) {
                            de[r] = fmaf(wev[e], xv[e], de[r]);
                            db[r] = fmaf(wbv[e], xv[e], db[r]);
                            const float zp = fmaf(av[e], xv[e], gv[e]);
                            xv[e] = zp * sig<Tin>(zp);
                            ss[r] = fmaf(xv[e], xv[e], ss[r]);
                        }
                    } else {
#pragma unroll
                        for (int e = 0; e < V; ++e) xv[e] = 0.f;
                    }
                    store_vec<Tout, V>(u[r] + i0, xv);
                }
            }
        }
#pragma unroll
        for (int r = 0; r < RPW; ++r) {
            ss[r] = warp_sum(ss[r]);
            de[r] = warp_sum(de[r]);
            db[r] = warp_sum(db[r]);
            const int t = t0 + r;
            if (lane == 0 && t < a.rows)
                a.zinv[(size_t)cs * a.row_stride + t] = live[r] ? 1.0f / sqrtf(ss[r] + 1e-12f) : 0.f;
        }
    } else {
    if (a.paper) {
#pragma unroll 2
        for (int i0 = lane * V; i0 < d; i0 += 32 * V) {
            float av[V], gv[V];
            load_f32<V>(al + i0, av);
            load_f32<V>(ga + i0, gv);
            float wev[V], wbv[V];
            if (!a.query) {
                load_f32<V>(we + i0, wev);
                load_f32<V>(wb + i0, wbv);
            }
#pragma unroll
            for (int r = 0; r < RPW; ++r) {
                if (!live[r]) continue;
                float xv[V];
                Vec<Tin>::unpack(*reinterpret_cast<const uint4*>(x[r] + i0), xv);
#pragma unroll
                for (int e = 0; e < V; ++e) {
                    if (!a.query) {
                        de[r] = fmaf(wev[e], xv[e], de[r]);
                        db[r] = fmaf(wbv[e], xv[e], db[r]);
                    }
                    const float zp = fmaf(av[e], xv[e], gv[e]);
                    const float z = zp * sig<Tin>(zp);
                    ss[r] = fmaf(z, z, ss[r]);
                }
            }
        }
#pragma unroll
        for (int r = 0; r < RPW; ++r) {
            ss[r] = warp_sum(ss[r]);
            if (!a.query) {
                de[r] = warp_sum(de[r]);
                db[r] = warp_sum(db[r]);
            }
        }
    }
    float inv[RPW];
#pragma unroll
    for (int r = 0; r < RPW; ++r) inv[r] = a.paper ? 1.0f / sqrtf(ss[r] + 1e-12f) : 1.0f;
#pragma unroll 2
    for (int i0 = lane * V; i0 < d; i0 += 32 * V) {
        float av[V], gv[V];
        if (a.paper) {
            load_f32<V>(al + i0, av);
            load_f32<V>(ga + i0, gv);
        }
#pragma unroll
        for (int r = 0; r < RPW; ++r) {
            if (t0 + r >= a.rows) continue;
            float xv[V];
            if (live[r]) {
                Vec<Tin>::unpack(*reinterpret_cast<const uint4*>(x[r] + i0), xv);
                if (a.paper) {
#pragma unroll
                    for (int e = 0; e < V; ++e) {
                        const float zp = fmaf(av[e], xv[e], gv[e]);
                        xv[e] = zp * sig<Tin>(zp) * inv[r];
                    }
                }
            } else {
#pragma unroll
                for (int e = 0; e < V; ++e) xv[e] = 0.f;
            }
            store_vec<Tout, V>(u[r] + i0, xv);
        }
    }
    }
    if (!a.query && lane == 0) {
#pragma unroll
        for (int r = 0; r < RPW; ++r) {
            const int t = t0 + r;
            if (t >= a.rows) continue;
            float e = 0.f, dbv = 0.f;
            if (live[r]) {
                e = a.eta_in ? a.eta_in[cz * a.eta_cstride + a.row0 + t] : softplusf_(de[r] + a.b_eta[cs]);
                dbv = db[r];
            }
            a.eta[(size_t)cs * a.row_stride + t] = e;
            a.dbeta[(size_t)cs * a.row_stride + t] = dbv;
        }
    }
}

template <typename Tin, typename Tout>
cudaError_t launch_one(const PrepassArgs& a, int nchains, cudaStream_t st) {
    dim3 grid((a.rows + PRE_ROWS - 1) / PRE_ROWS, nchains);
    prepass_kernel<Tin, Tout><<<grid, 256, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_prepass(const DevState& s, const SegWork& w, cudaStream_t st) {
    PrepassArgs a{};
    a.X = w.X;
    a.x_cstride = w.x_cstride;
    a.row0 = w.row0;
    a.n_rows = w.n_rows;
    a.Tp = w.Tp;  // tokens present in the window
    // write whole segments: rows past the context end are zero, never stale scratch
    a.rows = (int)std::min<long long>(s.win_rows, ((long long)w.Tp + s.T - 1) / s.T * s.T);
    a.row_stride = s.win_rows;
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
    a.zinv = s.dtype == 1 ? s.zinv : nullptr;  // bf16 path: unnormalised z + row scale
    return s.dtype == 0 ? launch_one<float, float>(a, w.nc, st) : launch_one<bf16, bf16>(a, w.nc, st);
}

// Query side of the read on the bf16 path, in one pass: one warp per (chain, query token).
// Paper mode: z = SiLU(alpha x + gamma), stored in bf16 unnormalised, and 1/|z| per token into
// zinv (the read scales each query's pre-activation by it: the row scale commutes with the
// contraction over d_in, Sec. 3.3's L2 normalisation); plain mode: z = x.  A lane's x, alpha
// and gamma loads of a 4-vector group are all issued before any arithmetic.
__global__ void __launch_bounds__(256) query_z_kernel(const bf16* X, int Q, int d, int paper, const float* alpha,
                                                      const float* gamma, bf16* Z, float* zinv, int total) {
    // the read's hidden kernel, launched after this one with programmatic stream serialisation,
    // may start now; it waits for this grid's completion before it reads Z or zinv
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const int row = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
    if (row >= total) return;
    const int c = row / Q;
    const bf16* x = X + (size_t)row * d;
    bf16* z = Z + (size_t)row * d;
    const float* al = paper ? alpha + (size_t)c * d : nullptr;
    const float* ga = paper ? gamma + (size_t)c * d : nullptr;
    float ss = 0.f;
    constexpr int G = 4;  // 16-byte vectors of a group
    for (int base = lane * 8; base < d; base += G * 256) {
        uint4 xr[G];
        float4 av[G][2], gv[G][2];
#pragma unroll
        for (int q = 0; q < G; ++q) {
            const int i0 = base + q * 256;
            if (i0 < d) {
                xr[q] = __ldg(reinterpret_cast<const uint4*>(x + i0));
                if (paper) {
                    av[q][0] = __ldg(reinterpret_cast<const float4*>(al + i0));
                    av[q][1] = __ldg(reinterpret_cast<const float4*>(al + i0 + 4));
                    gv[q][0] = __ldg(reinterpret_cast<const float4*>(ga + i0));
                    gv[q][1] = __ldg(reinterpret_cast<const float4*>(ga + i0 + 4));
                }
            }
        }
#pragma unroll
        for (int q = 0; q < G; ++q) {
            const int i0 = base + q * 256;
            if (i0 >= d) break;
            if (!paper) {
                *reinterpret_cast<uint4*>(z + i0) = xr[q];
                continue;
            }
            float xv[8];
            Vec<bf16>::unpack(xr[q], xv);
            const float a8[8] = {av[q][0].x, av[q][0].y, av[q][0].z, av[q][0].w,
                                 av[q][1].x, av[q][1].y, av[q][1].z, av[q][1].w};
            const float g8[8] = {gv[q][0].x, gv[q][0].y, gv[q][0].z, gv[q][0].w,
                                 gv[q][1].x, gv[q][1].y, gv[q][1].z, gv[q][1].w};
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                const float zp = fmaf(a8[e], xv[e], g8[e]);
                xv[e] = zp * sig<bf16>(zp);
                ss = fmaf(xv[e], xv[e], ss);
            }
            store_vec<bf16, 8>(z + i0, xv);
        }
    }
    if (paper) {
        ss = warp_sum(ss);
        if (lane == 0) zinv[row] = 1.0f / sqrtf(ss + 1e-12f);
    }
}

cudaError_t launch_query_z(const DevState& s, const void* Xq, int Q, void* Z, float* zinv, cudaStream_t st) {
    const int total = s.C * Q;
    query_z_kernel<<<(total + 7) / 8, 256, 0, st>>>(static_cast<const bf16*>(Xq), Q, s.d_in, s.mode == 1, s.alpha,
                                                    s.gamma, static_cast<bf16*>(Z), zinv, total);
    return cudaGetLastError();
}

// Query side of the read, normalised (the SwiGLU read, the fp32 read and the 128-query form):
// one warp per (chain, query token), d_in <= 2048.  A lane keeps its z values in registers, so
// the row is read once: z = SiLU(alpha x + gamma), then u = z / sqrt(|z|^2 + 1e-12) (paper mode),
// u = x in plain mode.  The loads of a 4-vector group are issued before any arithmetic.
constexpr int QU_MAX_D = 2048;
template <typename Tin, typename Tout>
__global__ void __launch_bounds__(256) query_u_kernel(const Tin* X, int Q, int d, int paper, const float* alpha,
                                                      const float* gamma, Tout* U, int total) {
    constexpr int V = Vec<Tin>::N;                 // elements per 16-byte load
    constexpr int MAXV = QU_MAX_D / (32 * V);      // vectors per lane
    constexpr int G = 4;
    const int row = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
    if (row >= total) return;
    const int c = row / Q;
    const Tin* x = X + (size_t)row * d;
    Tout* u = U + (size_t)row * d;
    const float* al = paper ? alpha + (size_t)c * d : nullptr;
    const float* ga = paper ? gamma + (size_t)c * d : nullptr;
    float zv[MAXV][V];
    float ss = 0.f;
#pragma unroll
    for (int k0 = 0; k0 < MAXV; k0 += G) {
        uint4 xr[G];
        float av[G][V], gv[G][V];
#pragma unroll
        for (int k = 0; k < G; ++k) {
            const int i0 = (lane + 32 * (k0 + k)) * V;
            if (i0 < d) {
                xr[k] = __ldg(reinterpret_cast<const uint4*>(x + i0));
                if (paper) {
                    load_f32<V>(al + i0, av[k]);
                    load_f32<V>(ga + i0, gv[k]);
                }
            }
        }
#pragma unroll
        for (int k = 0; k < G; ++k) {
            const int i0 = (lane + 32 * (k0 + k)) * V;
            if (i0 < d) {
                Vec<Tin>::unpack(xr[k], zv[k0 + k]);
                if (paper) {
#pragma unroll
                    for (int e = 0; e < V; ++e) {
                        const float zp = fmaf(av[k][e], zv[k0 + k][e], gv[k][e]);
                        zv[k0 + k][e] = zp * sig<Tin>(zp);
                        ss = fmaf(zv[k0 + k][e], zv[k0 + k][e], ss);
                    }
                }
            }
        }
    }
    const float inv = paper ? 1.0f / sqrtf(warp_sum(ss) + 1e-12f) : 1.0f;
#pragma unroll
    for (int k = 0; k < MAXV; ++k) {
        const int i0 = (lane + 32 * k) * V;
        if (i0 < d) {
#pragma unroll
            for (int e = 0; e < V; ++e) zv[k][e] *= inv;
            store_vec<Tout, V>(u + i0, zv[k]);
        }
    }
}

template <typename Tin, typename Tout>
cudaError_t launch_query_u(const DevState& s, const void* Xq, int Q, void* U, cudaStream_t st) {
    const int total = s.C * Q;
    query_u_kernel<Tin, Tout><<<(total + 7) / 8, 256, 0, st>>>(static_cast<const Tin*>(Xq), Q, s.d_in, s.mode == 1,
                                                               s.alpha, s.gamma, static_cast<Tout*>(U), total);
    return cudaGetLastError();
}

cudaError_t launch_query_transform(const DevState& s, const void* Xq, int Q, void* U, bool bf16_out, cudaStream_t st) {
    if (s.d_in <= QU_MAX_D) {  // one warp per query row, its values kept in registers
        if (s.dtype == 0) return launch_query_u<float, float>(s, Xq, Q, U, st);
        return bf16_out ? launch_query_u<bf16, bf16>(s, Xq, Q, U, st) : launch_query_u<bf16, float>(s, Xq, Q, U, st);
    }
    PrepassArgs a{};
    a.X = Xq;
    a.x_cstride = (long long)Q * s.d_in;
    a.row0 = 0;
    a.n_rows = Q;
    a.Tp = Q;
    a.rows = Q;
    a.row_stride = Q;
    a.c0 = 0;
    a.d_in = s.d_in;
    a.paper = s.mode == 1;
    a.query = 1;
    a.alpha = s.alpha;
    a.gamma = s.gamma;
    a.U = U;
    if (s.dtype == 0) return launch_one<float, float>(a, s.C, st);
    return bf16_out ? launch_one<bf16, bf16>(a, s.C, st) : launch_one<bf16, float>(a, s.C, st);
}

}  // namespace mone
