// Input prepass of a segment (paper mode) and the query transform of the read.
//
// Paper mode (App. A): keys and queries go through an affine rescale, SiLU and a
// per-token L2 normalisation: u_j = z_j / sqrt(|z_j|^2 + 1e-12),
// z_j = SiLU(alpha * x_j + gamma).  The same pass produces the per-token learning
// rate eta_j = softplus(w_eta . x_j + b_eta) and the per-token term
// w_beta . x_j of the momentum decay beta_s = sigmoid(mean_j(w_beta . x_j) + b_beta).
//
// One warp per token row; the row is read twice (statistics, then output) and
// the second read hits L1/L2.  Streaming, HBM-bound: reads d_in elements and
// writes d_in elements per token.
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

template <typename Tin, typename Tout>
__global__ void __launch_bounds__(256) prepass_kernel(const PrepassArgs a) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int t = blockIdx.x * 8 + warp;
    const int cz = blockIdx.y;
    const int cs = a.c0 + cz;
    if (t >= a.rows) return;
    const int d = a.d_in;
    Tout* u = reinterpret_cast<Tout*>(a.U) + ((size_t)cs * a.rows + t) * d;
    const bool present = t < a.Tp && (a.row0 + t) < a.n_rows;
    if (!present) {
        for (int i = lane; i < d; i += 32) u[i] = from_f<Tout>(0.0f);
        if (!a.query && lane == 0) {
            a.eta[(size_t)cs * a.rows + t] = 0.0f;
            a.dbeta[(size_t)cs * a.rows + t] = 0.0f;
        }
        return;
    }
    const Tin* x = reinterpret_cast<const Tin*>(a.X) + cz * a.x_cstride + (a.row0 + t) * d;
    float ss = 0.f, de = 0.f, db = 0.f;
    if (a.paper) {
        const float* al = a.alpha + (size_t)cs * d;
        const float* ga = a.gamma + (size_t)cs * d;
        const float* we = a.w_eta + (size_t)cs * d;
        const float* wb = a.w_beta + (size_t)cs * d;
        for (int i = lane; i < d; i += 32) {
            const float xv = to_f<Tin>(x[i]);
            const float zp = al[i] * xv + ga[i];
            const float z = zp * sigmoidf_(zp);
            ss += z * z;
            if (!a.query) {
                de += we[i] * xv;
                db += wb[i] * xv;
            }
        }
        ss = warp_sum(ss);
        if (!a.query) {
            de = warp_sum(de);
            db = warp_sum(db);
        }
        const float inv = 1.0f / sqrtf(ss + 1e-12f);
        for (int i = lane; i < d; i += 32) {
            const float xv = to_f<Tin>(x[i]);
            const float zp = al[i] * xv + ga[i];
            u[i] = from_f<Tout>(zp * sigmoidf_(zp) * inv);
        }
    } else {
        for (int i = lane; i < d; i += 32) u[i] = from_f<Tout>(to_f<Tin>(x[i]));
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
    dim3 grid((s.T + 7) / 8, w.nc);
    if (s.dtype == 0)
        prepass_kernel<float, float><<<grid, 256, 0, st>>>(a);
    else
        prepass_kernel<bf16, bf16><<<grid, 256, 0, st>>>(a);
    return cudaGetLastError();
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
    dim3 grid((Q + 7) / 8, s.C);
    if (s.dtype == 0)
        prepass_kernel<float, float><<<grid, 256, 0, st>>>(a);
    else
        prepass_kernel<bf16, float><<<grid, 256, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace mone
