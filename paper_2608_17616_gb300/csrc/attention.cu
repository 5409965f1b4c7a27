// Consumer attention of the read (Eq. 5, with Eq. 2 per head): the query tokens attend
// over [memory tokens || their own keys], softmax(q k^T / sqrt(hd)) v, with the memory
// tokens visible to every query token and the query tokens causal among themselves;
// query head h reads key/value head h / (n_q / n_kv) (grouped heads).
//
// Two forms.  bf16 with 16-byte-aligned rows runs on the tensor cores
// (attention_tc_kernel: S = Q K^T and O = P V as tcgen05 MMAs with TMEM accumulators, the
// softmax one row per thread in between).  fp32, and bf16 caches with other strides, run
// on the CUDA cores in flash-decode form: a CTA takes one (chain, key/value head, tile of
// query tokens) and stages the cache rows its tokens can see through shared memory in
// chunks of KC = 64 positions (converted to fp32 once, shared by every query head of the
// group).  Each warp owns up to MAXI (query head, token) items: per chunk, lane l scores
// keys l and l + 32 against every item (queries in shared memory), the chunk's max and sum
// are reduced once per item, and the probabilities pass through shared memory into the
// value accumulation, where a lane owns hd / 32 dimensions.
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
    int* status;            // device status word (bounded waits of the tensor-core form)
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

// ---------------------------------------------------------------- tensor-core form (bf16)
// One CTA of 512 threads per (chain, key/value head, tile of query tokens).  Its 128 rows are
// (query head of the group, token) pairs, `rows` = 128 / group tokens of each of the group's
// heads, so the group's heads share every staged key and value row.  Keys are taken in chunks
// of up to AT_NC positions: S = Q K^T accumulates in TMEM columns [0, AT_NC).  Four threads
// share a row (TMEM lane): each reads its 32-key blocks of the row, the row max is exchanged
// through shared memory, and each writes its bf16 probabilities to shared memory and
// keeps its own part of the row sum.  O_c = P V accumulates in TMEM columns [AT_NC, AT_NC + HD),
// of which each of the four threads takes hd / 4; the running max rescales the output columns
// and the partial sums from one chunk to the next, and the partial sums meet once at the end.
// Q, K and V reach shared memory through 16-byte asynchronous copies (cp.async, zero-filled
// past the last key), all in flight at once, written in the 128-byte-swizzled layout the MMA
// descriptors read: Q, K and P as K-major operands, V as the MN-major B operand of P V (a value
// row holds 64 dimensions per 128-byte line, the same bytes as a key row).  S = Q K^T is issued
// once the queries and keys have landed, with the values still in flight.
constexpr int AT_THREADS = 512;
constexpr int AT_GROUPS = AT_THREADS / 128;  // threads per row, each with its own columns
constexpr int AT_NC = 256;     // key positions per chunk: S's MMA N and TMEM columns
constexpr int AT_TMEM = 512;   // S (AT_NC columns) + O (HD <= 128 columns), a power of two

template <int HD>
struct AtSmem {
    static constexpr int SLAB_Q = 128 * 128;    // one 64-dimension slab of the 128 query rows
    static constexpr int SLAB_K = AT_NC * 128;  // one 64-dimension slab of AT_NC key (or value) rows
    static constexpr int SLAB_P = 128 * 128;    // one 64-key slab of the 128 probability rows
    static constexpr int Q_OFF = 0;
    static constexpr int K_OFF = Q_OFF + (HD / 64) * SLAB_Q;
    static constexpr int V_OFF = K_OFF + (HD / 64) * SLAB_K;
    // hd 128: the probabilities take the key buffer (the same size; keys are dead once S is in TMEM)
    static constexpr int P_OFF = HD == 128 ? K_OFF : V_OFF + (HD / 64) * SLAB_K;
    static constexpr int RED_OFF = HD == 128 ? V_OFF + (HD / 64) * SLAB_K : P_OFF + (AT_NC / 64) * SLAB_P;
    static constexpr int BAR_OFF = RED_OFF + AT_GROUPS * 128 * 4;
    static constexpr int DYN = BAR_OFF + 64 + 1024;  // + barriers, TMEM slot, flag; + alignment slack
};
static_assert(AtSmem<128>::DYN <= 227 * 1024 && AtSmem<64>::DYN <= 227 * 1024, "attention tile exceeds shared memory");

// Issue the copies of n_pad rows of HD bf16 into 64-dimension slabs `slab` bytes apart; row r
// comes from row_ptr(r) (16-byte aligned) when r < n and row_ptr(r) is non-null, else it is
// zero-filled (from `any`, a valid global address of which no byte is read).  Nothing waits
// here: every copy of the tile is in flight at once.
template <int HD, typename RowPtr>
__device__ __forceinline__ void at_stage(uint8_t* dst, int slab, int n, int n_pad, const bf16* any, RowPtr row_ptr) {
    constexpr int VPR = HD / 8;  // 16-byte pieces per row
    const uint32_t d0 = smem_u32(dst);
    for (int e = threadIdx.x; e < n_pad * VPR; e += AT_THREADS) {
        const int r = e / VPR, v = e - r * VPR;
        const bf16* p = r < n ? row_ptr(r) : nullptr;
        cpa16(d0 + (v >> 3) * slab + sw128_off(r, v & 7), p ? p + v * 8 : any, p ? 16 : 0);
    }
}

// 2^x on the special-function unit (PTX ex2.approx), whose error is far below the bf16
// rounding of the probabilities it feeds (the parity tests bound the result at 1e-2).
__device__ __forceinline__ float at_exp2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

template <int HD>
__global__ void __launch_bounds__(AT_THREADS, 1) attention_tc_kernel(const AttnArgs a) {
    using SM = AtSmem<HD>;
    constexpr int OC = HD / AT_GROUPS;  // output columns per thread
    extern __shared__ uint8_t smem_raw[];
    uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* Qs = base + SM::Q_OFF;
    uint8_t* Ks = base + SM::K_OFF;
    uint8_t* Vs = base + SM::V_OFF;
    uint8_t* Ps = base + SM::P_OFF;
    float* red = reinterpret_cast<float*>(base + SM::RED_OFF);  // [AT_GROUPS][128] per-row partials
    const uint32_t bar_s = smem_u32(base + SM::BAR_OFF), bar_o = bar_s + 8;
    uint32_t* slot = reinterpret_cast<uint32_t*>(base + SM::BAR_OFF + 16);
    int* abort_flag = reinterpret_cast<int*>(base + SM::BAR_OFF + 24);
    const int tid = threadIdx.x, warp = tid >> 5;
    // thread -> (row, column group): a warp reaches TMEM lanes 32 (warp % 4) .. + 31, so the four
    // warps of a lane quarter share its 32 rows and split the columns
    const int row = (warp & 3) * 32 + (tid & 31), grp = warp >> 2;
    if (tid == 0) {
        mbar_init(bar_s, 1);
        mbar_init(bar_o, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 0) {
        tmem_alloc(smem_u32(slot), AT_TMEM);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *slot;
    const uint32_t t_row = tmem + ((uint32_t)((warp & 3) * 32) << 16);  // this thread's TMEM lane = its row

    const int c = blockIdx.z, g = blockIdx.y, rt = a.rows, r0 = blockIdx.x * rt;
    const bf16* Qb = static_cast<const bf16*>(a.Q);
    const long long kv_off = (long long)(c / a.L) * a.s0 + (long long)(c % a.L) * a.s1 + (long long)g * a.s2;
    const bf16* Kc = static_cast<const bf16*>(a.K) + kv_off;
    const bf16* Vc = static_cast<const bf16*>(a.V) + kv_off;
    // row r of the tile: query head g * group + r / rt of the group, token r0 + r % rt
    auto q_row = [&](int r) -> const bf16* {
        const int hr = r / rt, ir = r0 + r % rt;
        if (hr >= a.group || ir >= a.Lq) return nullptr;
        return Qb + (((size_t)c * a.n_q + g * a.group + hr) * a.Lq + ir) * HD;
    };
    const int hg = row / rt, i = r0 + row % rt;
    const bool live = hg < a.group && i < a.Lq;
    const int vis = live ? a.n_mem + i + 1 : 0;     // keys this row sees (causal among the query tokens)
    const int keys = a.n_mem + min(a.Lq, r0 + rt);  // keys the tile's last token sees
    const float k2 = a.scale * 1.4426950408889634f;  // softmax scale in base 2: exp(s x) = 2^(s log2(e) x)

    at_stage<HD>(Qs, SM::SLAB_Q, 128, 128, Qb, q_row);
    float o[OC];
#pragma unroll
    for (int d = 0; d < OC; ++d) o[d] = 0.f;
    float m_run = -INFINITY, l_part = 0.f;  // row max so far; this thread's share of the row sum
    bool ok = true;
    int chunk = 0;
    for (int j0 = 0; j0 < keys; j0 += AT_NC, ++chunk) {
        const int nk = min(AT_NC, keys - j0), nc = (nk + 15) & ~15;
        // copy groups: (the queries and) the keys, then the values, which S = Q K^T does not wait for
        at_stage<HD>(Ks, SM::SLAB_K, nk, nc, Kc, [&](int r) { return Kc + (long long)(j0 + r) * a.s3; });
        cpa_commit();
        at_stage<HD>(Vs, SM::SLAB_K, nk, nc, Vc, [&](int r) { return Vc + (long long)(j0 + r) * a.s3; });
        cpa_commit();
        cpa_wait(1);
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        if (tid == 0) {  // S = Q K^T over HD (K-major both)
            tc_fence_after();
            const uint32_t idesc = idesc_bf16_f32(128, nc, false, false);
#pragma unroll
            for (int kb = 0; kb < HD / 64; ++kb)
#pragma unroll
                for (int k = 0; k < 4; ++k)
                    umma_bf16(tmem, sdesc_sw128(smem_u32(Qs + kb * SM::SLAB_Q) + k * 32, 16),
                              sdesc_sw128(smem_u32(Ks + kb * SM::SLAB_K) + k * 32, 16), idesc, (kb | k) ? 1u : 0u);
            umma_commit(bar_s);
        }
        if (!mbar_wait(bar_s, chunk & 1, a.status)) atomicOr(abort_flag, 1);
        __syncthreads();
        if (*abort_flag) {
            ok = false;
            break;
        }
        tc_fence_after();
        // this thread's 32-key blocks of the chunk: cb = 32 (grp + AT_GROUPS k); its row sees keys [0, nv)
        const int nv = min(max(vis - j0, 0), nc);
        float cm = -INFINITY;
#pragma unroll
        for (int k = 0; k < AT_NC / (32 * AT_GROUPS); ++k) {
            const int cb = 32 * (grp + AT_GROUPS * k);
            if (cb < nc) {  // uniform over the warp
                float v[32];
                tmem_ld32(t_row + cb, v);
#pragma unroll
                for (int j = 0; j < 32; ++j)
                    if (cb + j < nv) cm = fmaxf(cm, v[j]);
            }
        }
        red[grp * 128 + row] = cm;
        __syncthreads();
#pragma unroll
        for (int q = 0; q < AT_GROUPS; ++q) cm = fmaxf(cm, red[q * 128 + row]);
        const float mn = fmaxf(m_run, cm);
        // rescale of what earlier chunks accumulated (none yet: m_run = -inf gives 0)
        const float corr = mn == -INFINITY ? 1.f : at_exp2((m_run - mn) * k2);
        const float moff = mn == -INFINITY ? 0.f : -mn * k2;
        float ps = 0.f;
#pragma unroll
        for (int k = 0; k < AT_NC / (32 * AT_GROUPS); ++k) {
            const int cb = 32 * (grp + AT_GROUPS * k);
            if (cb < nc) {
                float v[32];  // the scores again (a TMEM reload is cheaper than holding them over the exchange)
                tmem_ld32(t_row + cb, v);
                uint32_t pk[16];
#pragma unroll
                for (int j = 0; j < 32; j += 2) {
                    const float p0 = cb + j < nv ? at_exp2(fmaf(v[j], k2, moff)) : 0.f;
                    const float p1 = cb + j + 1 < nv ? at_exp2(fmaf(v[j + 1], k2, moff)) : 0.f;
                    const __nv_bfloat162 pb = __floats2bfloat162_rn(p0, p1);
                    const float2 pr = __bfloat1622float2(pb);  // the sum takes the probabilities the MMA sees
                    ps += pr.x + pr.y;
                    pk[j / 2] = *reinterpret_cast<const uint32_t*>(&pb);
                }
                uint8_t* prow = Ps + (cb >> 6) * SM::SLAB_P;
#pragma unroll
                for (int u = 0; u < 4; ++u)
                    *reinterpret_cast<uint4*>(prow + sw128_off(row, ((cb & 63) >> 3) + u)) =
                        make_uint4(pk[4 * u], pk[4 * u + 1], pk[4 * u + 2], pk[4 * u + 3]);
            }
        }
        l_part = fmaf(l_part, corr, ps);
        cpa_wait(0);  // this thread's value copies
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        if (tid == 0) {  // O_c = P V over the chunk's keys (P K-major, V MN-major)
            tc_fence_after();
            const uint32_t idesc = idesc_bf16_f32(128, HD, false, true);
            for (int kk = 0; kk < nc / 16; ++kk)
                umma_bf16(tmem + AT_NC, sdesc_sw128(smem_u32(Ps + (kk >> 2) * SM::SLAB_P) + (kk & 3) * 32, 16),
                          sdesc_sw128(smem_u32(Vs) + kk * 16 * 128, SM::SLAB_K), idesc, kk ? 1u : 0u);
            umma_commit(bar_o);
        }
        if (!mbar_wait(bar_o, chunk & 1, a.status)) atomicOr(abort_flag, 1);
        __syncthreads();
        if (*abort_flag) {
            ok = false;
            break;
        }
        tc_fence_after();
        {  // this thread's OC output columns
            float w[OC];
            if constexpr (OC == 32)
                tmem_ld32(t_row + AT_NC + grp * OC, w);
            else
                tmem_ld16(t_row + AT_NC + grp * OC, w);
#pragma unroll
            for (int d = 0; d < OC; ++d) o[d] = fmaf(o[d], corr, w[d]);
        }
        m_run = mn;
        // the next chunk restages K, V (and P) and rewrites red: the MMAs that read the buffers
        // have completed and every thread passed the barrier after its last read of red
    }
    red[grp * 128 + row] = l_part;
    __syncthreads();
    if (ok && live) {
        float l = 0.f;
#pragma unroll
        for (int q = 0; q < AT_GROUPS; ++q) l += red[q * 128 + row];
        const float inv = 1.f / l;
        bf16* orow = static_cast<bf16*>(a.out) + (((size_t)c * a.n_q + g * a.group + hg) * a.Lq + i) * HD + grp * OC;
#pragma unroll
        for (int v8 = 0; v8 < OC / 8; ++v8)
            *reinterpret_cast<uint4*>(orow + v8 * 8) =
                make_uint4(pack_bf16(o[8 * v8] * inv, o[8 * v8 + 1] * inv), pack_bf16(o[8 * v8 + 2] * inv, o[8 * v8 + 3] * inv),
                           pack_bf16(o[8 * v8 + 4] * inv, o[8 * v8 + 5] * inv),
                           pack_bf16(o[8 * v8 + 6] * inv, o[8 * v8 + 7] * inv));
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, AT_TMEM);
}

std::mutex g_attr_mu;

// The shared-memory opt-in belongs to a device: set it once per device and kernel (a driver
// call on every launch would cost more than the kernel).
template <typename K>
cudaError_t smem_opt_in(K kernel, size_t smem, bool (&done)[64]) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lk(g_attr_mu);
    if (!done[dev]) {
        e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        done[dev] = true;
    }
    return cudaSuccess;
}

template <typename T, int HD>
cudaError_t launch_t(const AttnArgs& a, int C, cudaStream_t st) {
    const size_t smem = AttnSmem<T, HD>::FLOATS * sizeof(float);
    static bool done[64] = {};
    cudaError_t e = smem_opt_in(attention_kernel<T, HD>, smem, done);
    if (e != cudaSuccess) return e;
    dim3 grid((a.Lq + a.rows - 1) / a.rows, a.n_kv, C);
    attention_kernel<T, HD><<<grid, ATT_WARPS * 32, smem, st>>>(a);
    return cudaGetLastError();
}

template <int HD>
cudaError_t launch_tc(AttnArgs a, int C, cudaStream_t st) {
    static bool done[64] = {};
    cudaError_t e = smem_opt_in(attention_tc_kernel<HD>, AtSmem<HD>::DYN, done);
    if (e != cudaSuccess) return e;
    a.rows = 128 / a.group;  // tokens per tile: the group's heads x rows fill the 128 MMA rows
    dim3 grid((a.Lq + a.rows - 1) / a.rows, a.n_kv, C);
    attention_tc_kernel<HD><<<grid, AT_THREADS, AtSmem<HD>::DYN, st>>>(a);
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
    a.status = s.status;
    if (s.dtype == 0)
        return s.hd == 64 ? launch_t<float, 64>(a, s.C, st) : launch_t<float, 128>(a, s.C, st);
    // bf16 on the tensor cores when every row it stages is 16-byte aligned (the queries and the
    // output are dense rows of hd elements); other cache layouts take the CUDA-core kernel
    if (a.vec && ((reinterpret_cast<uintptr_t>(Q) | reinterpret_cast<uintptr_t>(out)) & 15u) == 0)
        return s.hd == 64 ? launch_tc<64>(a, s.C, st) : launch_tc<128>(a, s.C, st);
    return s.hd == 64 ? launch_t<bf16, 64>(a, s.C, st) : launch_t<bf16, 128>(a, s.C, st);
}

}  // namespace mone
