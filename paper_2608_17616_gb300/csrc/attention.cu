// Consumer attention of the read (Eq. 5, with Eq. 2 per head): the query tokens attend
// over [memory tokens || their own keys], softmax(q k^T / sqrt(hd)) v, with the memory
// tokens visible to every query token and the query tokens causal among themselves;
// query head h reads key/value head h / (n_q / n_kv) (grouped heads).
//
// A small, bandwidth-bound contraction, run on the CUDA cores in flash-decode form: a CTA
// takes one (chain, key/value head, tile of query tokens) and stages the cache rows its
// tokens can see through shared memory in chunks of KC = 64 positions (converted to fp32
// once, shared by every query head of the group).  Each warp owns up to MAXI (query
// head, token) items: per chunk, lane l scores keys l and l + 32 against every item
// (queries in shared memory), the chunk's max and sum are reduced once per item, and
// the probabilities pass through shared memory into the value accumulation, where a
// lane owns hd / 32 dimensions.
#include <algorithm>
#include <mutex>

#include "mone_common.cuh"

namespace mone {

namespace {

constexpr int ATT_WARPS = 8;
constexpr int ATT_ITEMS = 64;                 // (query head, token) items per CTA
constexpr int MAXI = ATT_ITEMS / ATT_WARPS;   // items per warp
constexpr int KC = 64;                        // cache positions per shared-memory chunk

struct AttnArgs {
    const void* Q;          // [C][n_q][Lq][hd]
    const void *K, *V;      // caches, element strides s0 (context), s1 (layer), s2 (head), s3 (position)
    void* out;              // [C][n_q][Lq][hd]
    long long s0, s1, s2, s3;
    int L, n_q, n_kv, group, Lq, n_mem, rows;  // rows: query tokens per CTA (group * rows <= ATT_ITEMS)
    float scale;            // 1 / sqrt(hd)
    int vec;                // caches 16-byte aligned (base and every stride): stage with 16-byte loads
};

// Stage cache positions [j0, j0 + nk) of one head into shared memory as fp32 rows of HD
// values, `pitch` floats apart.
template <typename T, int HD>
__device__ __forceinline__ void stage_rows(float* dst, const T* src, long long s3, int j0, int nk, bool vec,
                                           int pitch) {
    if (vec) {
        constexpr int PER = 16 / sizeof(T);   // elements per 16-byte load
        constexpr int VPR = HD / PER;         // loads per row
        const int nv = nk * VPR;
#pragma unroll 4
        for (int e = threadIdx.x; e < nv; e += ATT_WARPS * 32) {
            const int j = e / VPR, v = e % VPR;
            const uint4 r = *reinterpret_cast<const uint4*>(src + (long long)(j0 + j) * s3 + v * PER);
            float f[PER];
            if constexpr (sizeof(T) == 2) {
                const __nv_bfloat162* b = reinterpret_cast<const __nv_bfloat162*>(&r);
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const float2 x = __bfloat1622float2(b[u]);
                    f[2 * u] = x.x;
                    f[2 * u + 1] = x.y;
                }
            } else {
                f[0] = __uint_as_float(r.x); f[1] = __uint_as_float(r.y);
                f[2] = __uint_as_float(r.z); f[3] = __uint_as_float(r.w);
            }
#pragma unroll
            for (int u = 0; u < PER; ++u) dst[j * pitch + v * PER + u] = f[u];
        }
    } else {
        for (int e = threadIdx.x; e < nk * HD; e += ATT_WARPS * 32) {
            const int j = e / HD, d = e % HD;
            dst[j * pitch + d] = to_f<T>(src[(long long)(j0 + j) * s3 + d]);
        }
    }
}

template <typename T, int HD>
struct AttnSmem {
    // key rows padded by 4 floats: a lane reads its key row 16 bytes at a time, and the 8 lanes of a
    // quarter warp (one shared-memory wavefront of 128-bit loads) start 68 / 132 floats apart: 8 bank groups
    static constexpr int KP = HD + 4;
    static constexpr int K_OFF = 0;                          // [KC][KP] keys (fp32)
    static constexpr int V_OFF = K_OFF + KC * KP;            // [KC][HD] values
    static constexpr int Q_OFF = V_OFF + KC * HD;            // [warp][MAXI][HD] scaled queries
    static constexpr int P_OFF = Q_OFF + ATT_WARPS * MAXI * HD;  // [warp][MAXI][KC] probabilities of a chunk
    static constexpr int FLOATS = P_OFF + ATT_WARPS * MAXI * KC;
};

template <typename T, int HD>
__global__ void __launch_bounds__(ATT_WARPS * 32, 2) attention_kernel(const AttnArgs a) {
    using SM = AttnSmem<T, HD>;
    constexpr int D = HD / 32;  // value / accumulator dimensions per lane
    extern __shared__ float sh[];
    float* Ks = sh + SM::K_OFF;
    float* Vs = sh + SM::V_OFF;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    float* Qs = sh + SM::Q_OFF + warp * MAXI * HD;
    float* Ps = sh + SM::P_OFF + warp * MAXI * KC;
    const int c = blockIdx.z, g = blockIdx.y, r0 = blockIdx.x * a.rows;
    const long long kv_off = (long long)(c / a.L) * a.s0 + (long long)(c % a.L) * a.s1 + (long long)g * a.s2;
    const T* Kc = static_cast<const T*>(a.K) + kv_off;
    const T* Vc = static_cast<const T*>(a.V) + kv_off;

    // this warp's items: item = warp + ATT_WARPS * k -> (head in group, token row); the running
    // softmax (max, sum) is kept identical in every lane, the accumulator split over lanes by dimension
    float acc[MAXI][D], mx[MAXI], sum[MAXI];
    int vis[MAXI];  // keys item k sees (0: no item)
#pragma unroll
    for (int k = 0; k < MAXI; ++k) {
        const int it = warp + ATT_WARPS * k;
        const int hg = it / a.rows, i = r0 + it % a.rows;
        vis[k] = 0;
        mx[k] = -INFINITY;
        sum[k] = 0.f;
#pragma unroll
        for (int d = 0; d < D; ++d) acc[k][d] = 0.f;
        float qv[D];
#pragma unroll
        for (int d = 0; d < D; ++d) qv[d] = 0.f;
        if (hg < a.group && i < a.Lq) {
            vis[k] = a.n_mem + i + 1;
            const int h = g * a.group + hg;
            const T* qr = static_cast<const T*>(a.Q) + (((size_t)c * a.n_q + h) * a.Lq + i) * HD;
#pragma unroll
            for (int d = 0; d < D; ++d) qv[d] = to_f<T>(qr[lane + 32 * d]) * a.scale;
        }
#pragma unroll
        for (int d = 0; d < D; ++d) Qs[k * HD + lane + 32 * d] = qv[d];
    }
    const int last = min(a.Lq, r0 + a.rows) - 1;
    const int keys = a.n_mem + last + 1;  // positions the tile's last token sees
    for (int j0 = 0; j0 < keys; j0 += KC) {
        const int nk = min(KC, keys - j0);
        __syncthreads();
        stage_rows<T, HD>(Ks, Kc, a.s3, j0, nk, a.vec, SM::KP);
        stage_rows<T, HD>(Vs, Vc, a.s3, j0, nk, a.vec, HD);
        // value rows up to the next multiple of 4 are read with probability 0: make them finite
        for (int e = threadIdx.x; e < (((nk + 3) & ~3) - nk) * HD; e += ATT_WARPS * 32) Vs[nk * HD + e] = 0.f;
        __syncthreads();
        // scores: lane owns keys j0 + lane and j0 + lane + 32 of the chunk; keys and the (broadcast)
        // queries are read 4 dimensions at a time
        float z0[MAXI], z1[MAXI];
#pragma unroll
        for (int k = 0; k < MAXI; ++k) z0[k] = z1[k] = 0.f;
        const float4* k0 = reinterpret_cast<const float4*>(Ks + lane * SM::KP);
        const float4* k1 = reinterpret_cast<const float4*>(Ks + (lane + 32) * SM::KP);
        const float4* q4 = reinterpret_cast<const float4*>(Qs);
#pragma unroll 2
        for (int d4 = 0; d4 < HD / 4; ++d4) {
            const float4 a0 = k0[d4], a1 = k1[d4];
#pragma unroll
            for (int k = 0; k < MAXI; ++k) {
                const float4 qd = q4[k * (HD / 4) + d4];
                z0[k] = fmaf(qd.x, a0.x, fmaf(qd.y, a0.y, fmaf(qd.z, a0.z, fmaf(qd.w, a0.w, z0[k]))));
                z1[k] = fmaf(qd.x, a1.x, fmaf(qd.y, a1.y, fmaf(qd.z, a1.z, fmaf(qd.w, a1.w, z1[k]))));
            }
        }
#pragma unroll
        for (int k = 0; k < MAXI; ++k) {
            // causal / chunk masks; an item with no visible key in this chunk keeps its state
            const bool v0 = lane < nk && j0 + lane < vis[k], v1 = lane + 32 < nk && j0 + lane + 32 < vis[k];
            const float cm = warp_max(fmaxf(v0 ? z0[k] : -INFINITY, v1 ? z1[k] : -INFINITY));
            float p0 = 0.f, p1 = 0.f;
            if (cm != -INFINITY) {
                const float mn = fmaxf(mx[k], cm);
                const float corr = __expf(mx[k] - mn);
                p0 = v0 ? __expf(z0[k] - mn) : 0.f;
                p1 = v1 ? __expf(z1[k] - mn) : 0.f;
                sum[k] = fmaf(sum[k], corr, warp_sum(p0 + p1));
#pragma unroll
                for (int d = 0; d < D; ++d) acc[k][d] *= corr;
                mx[k] = mn;
            }
            Ps[k * KC + lane] = p0;
            Ps[k * KC + lane + 32] = p1;
        }
        __syncwarp();
        // values: lane owns dimensions lane + 32 d; the probabilities are read 4 keys at a time
        // (positions of the chunk past nk hold p = 0 and finite staged values)
        const float4* p4 = reinterpret_cast<const float4*>(Ps);
        for (int j = 0; j < nk; j += 4) {
            float vd[4][D];
#pragma unroll
            for (int u = 0; u < 4; ++u)
#pragma unroll
                for (int d = 0; d < D; ++d) vd[u][d] = Vs[(j + u) * HD + lane + 32 * d];
#pragma unroll
            for (int k = 0; k < MAXI; ++k) {
                const float4 p = p4[(k * KC + j) / 4];
#pragma unroll
                for (int d = 0; d < D; ++d)
                    acc[k][d] = fmaf(p.x, vd[0][d], fmaf(p.y, vd[1][d], fmaf(p.z, vd[2][d], fmaf(p.w, vd[3][d], acc[k][d]))));
            }
        }
        __syncwarp();
    }
#pragma unroll
    for (int k = 0; k < MAXI; ++k) {
        if (!vis[k]) continue;
        const int it = warp + ATT_WARPS * k;
        const int h = g * a.group + it / a.rows, i = r0 + it % a.rows;
        T* o = static_cast<T*>(a.out) + (((size_t)c * a.n_q + h) * a.Lq + i) * HD;
        const float inv = 1.f / sum[k];
#pragma unroll
        for (int d = 0; d < D; ++d) o[lane + 32 * d] = from_f<T>(acc[k][d] * inv);
    }
}

std::mutex g_attr_mu;

template <typename T, int HD>
cudaError_t launch_t(const AttnArgs& a, int C, cudaStream_t st) {
    const size_t smem = AttnSmem<T, HD>::FLOATS * sizeof(float);
    {
        // the shared-memory opt-in belongs to a device: set it once per device (a driver call
        // on every launch would cost more than the kernel)
        static bool done[64] = {};
        int dev = 0;
        cudaError_t e = cudaGetDevice(&dev);
        if (e != cudaSuccess) return e;
        if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
        std::lock_guard<std::mutex> lk(g_attr_mu);
        if (!done[dev]) {
            e = cudaFuncSetAttribute(attention_kernel<T, HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            if (e != cudaSuccess) return e;
            done[dev] = true;
        }
    }
    dim3 grid((a.Lq + a.rows - 1) / a.rows, a.n_kv, C);
    attention_kernel<T, HD><<<grid, ATT_WARPS * 32, smem, st>>>(a);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_attention(const DevState& s, int n_layers, const void* Q, int n_q, int Lq, const void* K,
                             const void* V, const long long* strides, int n_mem, void* out, cudaStream_t st) {
    AttnArgs a{};
    a.Q = Q; a.K = K; a.V = V; a.out = out;
    a.s0 = strides[0]; a.s1 = strides[1]; a.s2 = strides[2]; a.s3 = strides[3];
    a.L = n_layers; a.n_q = n_q; a.n_kv = s.n_kv; a.group = n_q / s.n_kv; a.Lq = Lq; a.n_mem = n_mem;
    a.rows = std::max(1, ATT_ITEMS / a.group);
    a.scale = 1.0f / sqrtf((float)s.hd);
    const long long el = s.dtype == 0 ? 4 : 2;
    a.vec = ((reinterpret_cast<uintptr_t>(K) | reinterpret_cast<uintptr_t>(V)) & 15u) == 0 && (a.s0 * el) % 16 == 0 &&
            (a.s1 * el) % 16 == 0 && (a.s2 * el) % 16 == 0 && (a.s3 * el) % 16 == 0;
    if (s.dtype == 0)
        return s.hd == 64 ? launch_t<float, 64>(a, s.C, st) : launch_t<float, 128>(a, s.C, st);
    return s.hd == 64 ? launch_t<bf16, 64>(a, s.C, st) : launch_t<bf16, 128>(a, s.C, st);
}

}  // namespace mone
