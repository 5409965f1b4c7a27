// C-ABI front end of libmone.so: argument validation, state allocation, the
// segment loop of test-time learning (Eq. 9), and the memory read (Eq. 4).
// All arithmetic runs in the kernels of ttl_prepass.cu, ttl_simt.cu and ttl_tc.cu.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <new>
#include <set>
#include <vector>

#include "mone.h"
#include "mone_internal.h"

using namespace mone;

// Kernel kinds of the per-kernel timing (mone_mem_kernel_time).
enum { K_PREPASS = 0, K_PHASE_A = 1, K_PHASE_B = 2, K_FINALIZE = 3, K_READ = 4, K_MSE = 5, K_ATTN = 6,
       K_RESIDENT = 7, K_STAGE = 8, K_KINDS = 9 };

// Optional per-kernel device timing (mone_mem_set_timing).
struct KernelTiming {
    bool on = false;
    struct Pending {
        int kind;
        cudaEvent_t a, b;
    };
    std::vector<cudaEvent_t> pool;
    std::vector<Pending> pending;
    double ms[K_KINDS] = {};
    long long n[K_KINDS] = {};
    // start and end of every launch, in ms after `ref` (recorded before the first timed launch
    // since timing was enabled), for the busy time of a kernel kind (mone_mem_kernel_busy)
    cudaEvent_t ref = nullptr;
    bool ref_set = false;
    std::vector<std::pair<double, double>> iv[K_KINDS];

    void reset() {
        for (int k = 0; k < K_KINDS; ++k) {
            ms[k] = 0;
            n[k] = 0;
            iv[k].clear();
        }
        ref_set = false;
    }

    cudaEvent_t get() {
        if (!pool.empty()) {
            cudaEvent_t e = pool.back();
            pool.pop_back();
            return e;
        }
        cudaEvent_t e = nullptr;
        if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
        return e;
    }
    cudaError_t drain() {
        cudaError_t rc = cudaSuccess;
        for (auto& p : pending) {
            cudaError_t e = cudaEventSynchronize(p.b);
            float t = 0.f, t0 = 0.f;
            if (e == cudaSuccess) e = cudaEventElapsedTime(&t, p.a, p.b);
            if (e == cudaSuccess && ref_set) e = cudaEventElapsedTime(&t0, ref, p.a);
            if (e == cudaSuccess) {
                ms[p.kind] += t;
                n[p.kind] += 1;
                if (ref_set) iv[p.kind].push_back({t0, t0 + t});
            } else {
                rc = e;
            }
            pool.push_back(p.a);
            pool.push_back(p.b);
        }
        pending.clear();
        return rc;
    }
    ~KernelTiming() {
        drain();
        for (cudaEvent_t e : pool) cudaEventDestroy(e);
        if (ref) cudaEventDestroy(ref);
    }
};

// A captured memory read (mone_mem_generate_kv): the query transform and the read kernels as one
// CUDA graph, replayed while the call's buffers, Q and strides repeat, so that the GPU runs them
// back to back instead of waiting for each launch.  Captured from the second call with a key.
struct ReadGraph {
    cudaGraphExec_t exec = nullptr;
    const void *xq = nullptr, *ko = nullptr, *vo = nullptr, *uq = nullptr, *aq = nullptr, *oq = nullptr;
    int q = 0, seen = 0;
    long long strides[4] = {0, 0, 0, 0};
};

struct mone_mem {
    mone_config cfg;
    DevState s;
    TcMaps maps;
    SwMaps swmaps;   // SwiGLU memory
    long long launches;
    KernelTiming* timing;
    cudaStream_t side;               // second chain group's stream (bf16 path, >= 2 chains), or null
    cudaEvent_t ev_fork, ev_join;    // caller stream -> side stream, side stream -> caller stream
    cudaStream_t cap;                // capture stream of the read graph (created on first capture)
    ReadGraph* rg;                   // the captured read, or null
    // host-input pipeline (mone_ttl_context_host, created on first use): two device windows of
    // a chunk, the staging stream, and events: hstart (the caller's stream at the call), and per
    // window hstaged (its gather has finished) and hfree (the learning that last read it has)
    void* hwin[2];
    size_t hwin_bytes;
    cudaStream_t hstream;
    cudaEvent_t hstart, hstaged[2], hfree[2];
};

namespace {

std::mutex g_live_mu;
std::set<const mone_mem*> g_live;

bool is_live(const mone_mem* m) {
    std::lock_guard<std::mutex> lk(g_live_mu);
    return m && g_live.count(m);
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

mone_status validate_config(const mone_config* c) {
    if (!c) return MONE_ERR_INVALID_ARG;
    if (c->n_ctx < 1 || c->n_layers < 1 || c->d_in < 1 || c->d_hid < 1 || c->d_out < 2 || c->n_kv_heads < 1 ||
        c->head_dim < 1 || c->seg_T < 1)
        return MONE_ERR_INVALID_ARG;
    if (c->dtype != MONE_FP32 && c->dtype != MONE_BF16) return MONE_ERR_INVALID_ARG;
    if (c->mode != MONE_PLAIN && c->mode != MONE_PAPER) return MONE_ERR_INVALID_ARG;
    if (c->loss != MONE_LOSS_DOT && c->loss != MONE_LOSS_MSE) return MONE_ERR_INVALID_ARG;
    if (c->memory != MONE_MEM_MLP && c->memory != MONE_MEM_SWIGLU) return MONE_ERR_INVALID_ARG;
    if (c->renorm_axis != MONE_RENORM_ROWS && c->renorm_axis != MONE_RENORM_OUT) return MONE_ERR_INVALID_ARG;
    if (c->gate_act != MONE_GATE_LINEAR && c->gate_act != MONE_GATE_SILU) return MONE_ERR_INVALID_ARG;
    if (c->renorm_axis == MONE_RENORM_OUT && c->memory != MONE_MEM_MLP) return MONE_ERR_UNSUPPORTED;
    if (!std::isfinite(c->lr) || !(c->rms_eps >= 0.0f) || !std::isfinite(c->rms_eps)) return MONE_ERR_INVALID_ARG;
    if (c->memory == MONE_MEM_SWIGLU) {
        if (c->dtype != MONE_BF16 || c->loss != MONE_LOSS_DOT) return MONE_ERR_UNSUPPORTED;
        if (c->mem_heads < 1 || c->d_in % c->mem_heads) return MONE_ERR_INVALID_ARG;
        if (c->head_dim != 64 && c->head_dim != 128) return MONE_ERR_UNSUPPORTED_SHAPE;
        if (c->d_out != 2 * c->n_kv_heads * c->head_dim) return MONE_ERR_UNSUPPORTED_SHAPE;
        const int dh = c->d_in / c->mem_heads;
        if (c->d_out != c->d_in || dh % 32 || dh > 256 || (c->d_out / 2) % dh || c->d_hid % 32 || c->d_hid > 256 ||
            c->seg_T % 128 || c->seg_T > 4096 || (long long)c->n_ctx * c->n_layers * c->mem_heads > 65535)
            return MONE_ERR_UNSUPPORTED_SHAPE;
        return MONE_OK;
    }
    if (c->head_dim != 64 && c->head_dim != 128) return MONE_ERR_UNSUPPORTED_SHAPE;
    if (c->d_out != 2 * c->n_kv_heads * c->head_dim) return MONE_ERR_UNSUPPORTED_SHAPE;
    if (c->seg_T > 4096) return MONE_ERR_UNSUPPORTED_SHAPE;
    if ((long long)c->n_ctx * c->n_layers > 65535) return MONE_ERR_UNSUPPORTED_SHAPE;
    if (c->dtype == MONE_FP32) {
        if (c->d_in % 64 || c->d_hid % 64 || c->d_out % 64 || c->seg_T % 64) return MONE_ERR_UNSUPPORTED_SHAPE;
    } else {
        if (c->d_in % 128 || c->d_hid % 256 || (c->d_out / 2) % 128 || c->seg_T % 128)
            return MONE_ERR_UNSUPPORTED_SHAPE;
    }
    return MONE_OK;
}

thread_local char g_last_error[256] = "";

mone_status cuda_status(cudaError_t e) {
    if (e == cudaSuccess) return MONE_OK;
    std::snprintf(g_last_error, sizeof(g_last_error), "%s: %s", cudaGetErrorName(e), cudaGetErrorString(e));
    if (e == cudaErrorMemoryAllocation) return MONE_ERR_OOM;
    return MONE_ERR_CUDA;
}

template <typename T>
mone_status dalloc(T** p, size_t n) {
    *p = nullptr;
    if (n == 0) return MONE_OK;
    const char* f = std::getenv("MONE_FAULT_ALLOC");
    if (f && std::atoi(f) == 1) return MONE_ERR_OOM;  // host-side allocation-failure injection
    cudaError_t e = cudaMalloc(reinterpret_cast<void**>(p), n * sizeof(T));
    if (e != cudaSuccess) {
        cudaGetLastError();
        *p = nullptr;
        return e == cudaErrorMemoryAllocation ? MONE_ERR_OOM : MONE_ERR_CUDA;
    }
    return MONE_OK;
}

void free_state(DevState& s) {
    void* ptrs[] = {s.W1, s.W2, s.mu1, s.mu2, s.W1b, s.W2b, s.n1, s.n2, s.sumsq, s.status, s.alpha, s.gamma,
                    s.w_eta, s.b_eta, s.w_beta, s.b_beta, s.gate, s.U, s.eta, s.dbeta, s.zinv, s.dHt, s.Att, s.Uq, s.Aq,
                    s.Oq, s.Amse, s.Kres, s.Vres, s.Kres32, s.Vres32, s.nc2, s.colpart};
    for (void* p : ptrs)
        if (p) cudaFree(p);
    std::memset(&s, 0, sizeof(s));
}

size_t elsize(int dtype) { return dtype == MONE_FP32 ? 4 : 2; }

void destroy_host_pipeline(mone_mem* m) {
    for (int b = 0; b < 2; ++b) {
        if (m->hwin[b]) cudaFree(m->hwin[b]);
        if (m->hstaged[b]) cudaEventDestroy(m->hstaged[b]);
        if (m->hfree[b]) cudaEventDestroy(m->hfree[b]);
        m->hwin[b] = nullptr;
        m->hstaged[b] = m->hfree[b] = nullptr;
    }
    if (m->hstart) cudaEventDestroy(m->hstart);
    if (m->hstream) cudaStreamDestroy(m->hstream);
    m->hstart = nullptr;
    m->hstream = nullptr;
    m->hwin_bytes = 0;
}

void destroy_streams(mone_mem* m) {
    destroy_host_pipeline(m);
    if (m->rg) {
        if (m->rg->exec) cudaGraphExecDestroy(m->rg->exec);
        delete m->rg;
        m->rg = nullptr;
    }
    if (m->cap) cudaStreamDestroy(m->cap);
    m->cap = nullptr;
    if (m->ev_fork) cudaEventDestroy(m->ev_fork);
    if (m->ev_join) cudaEventDestroy(m->ev_join);
    if (m->side) cudaStreamDestroy(m->side);
    m->ev_fork = m->ev_join = nullptr;
    m->side = nullptr;
}

#define MONE_TRY(x)                           \
    do {                                      \
        mone_status _st = (x);                \
        if (_st != MONE_OK) return _st;       \
    } while (0)
#define MONE_CUDA(x)                              \
    do {                                          \
        cudaError_t _e = (x);                     \
        if (_e != cudaSuccess) return cuda_status(_e); \
    } while (0)

mone_status build_swiglu_maps(mone_mem* m) {
    DevState& s = m->s;
    SwMaps& w = m->swmaps;
    const uint64_t H = s.heads, dh = s.d_in / s.heads, F = s.d_hid, CH = (uint64_t)s.C * H, T = s.T;
    bool ok = true;
    {  // W1 = [Win; Wg] per head: (dh, F, 2, C*H)
        const uint64_t d[4] = {dh, F, 2, CH}, st[3] = {dh * 2, F * dh * 2, 2 * F * dh * 2};
        const uint32_t b[4] = {64, 128, 1, 1};
        ok = ok && encode_map_bf16_4d(&w.W1a, s.W1b, d, st, b);
    }
    ok = ok && encode_map_bf16_3d(&w.W2a, s.W2b, dh, F, CH, 64, 128) &&
         encode_map_bf16_3d(&w.W2m, s.W2b, dh, F, CH, 64, 64);
    {  // phase A outputs, MN-major: (1/|z|) c [dP | dG] as (F, 2, T, C*H) and c Z as (F, T, C*H)
        const uint64_t d[4] = {F, 2, T, CH}, st[3] = {F * 2, 2 * F * 2, T * 2 * F * 2};
        const uint32_t b[4] = {64, 1, 64, 1};
        ok = ok && encode_map_bf16_4d(&w.PG, s.dHt, d, st, b);
    }
    ok = ok && encode_map_bf16_3d(&w.Z, s.Att, F, T, CH, 64, 64);
    // fp32 state chunks of phase B (rows past a head's F hidden units or columns past dh are
    // never touched: the kernel skips such chunks and masks such columns)
    ok = ok && encode_map_plain_3d(&w.W1s, s.W1, true, dh, 2 * F, CH, 128, 32) &&
         encode_map_plain_3d(&w.W2s, s.W2, true, dh, F, CH, 128, 32);
    if (ok && s.mu1)
        ok = encode_map_plain_3d(&w.M1s, s.mu1, true, dh, 2 * F, CH, 128, 32) &&
             encode_map_plain_3d(&w.M2s, s.mu2, true, dh, F, CH, 128, 32);
    if (ok && s.U) {  // input-transform window as (dh, H, rows, C)
        const uint64_t d[4] = {dh, H, (uint64_t)s.win_rows, (uint64_t)s.C};
        const uint64_t st[3] = {dh * 2, H * dh * 2, (uint64_t)s.win_rows * H * dh * 2};
        const uint32_t ba[4] = {64, 1, 128, 1}, bb[4] = {64, 1, 64, 1};
        ok = encode_map_bf16_4d(&w.Ua, s.U, d, st, ba) && encode_map_bf16_4d(&w.Ub, s.U, d, st, bb);
    }
    return ok ? MONE_OK : MONE_ERR_CUDA;
}

// Inputs of one call for the SwiGLU memory: head slices of X (plain mode), K and V of `chains` chains.
mone_status build_swiglu_input_maps(const DevState& s, SwInputMaps* in, const void* X, const void* K, const void* V,
                                    long long rows, int chains) {
    const uint64_t H = s.heads, dh = s.d_in / s.heads, Hk = (s.d_out / 2) / dh;
    const uint32_t ba[4] = {64, 1, 128, 1}, bb[4] = {64, 1, 64, 1};
    const uint64_t dk[4] = {dh, Hk, (uint64_t)rows, (uint64_t)chains};
    const uint64_t sk[3] = {dh * 2, Hk * dh * 2, (uint64_t)rows * Hk * dh * 2};
    bool ok = encode_map_bf16_4d(&in->Ka, K, dk, sk, ba) && encode_map_bf16_4d(&in->Kb, K, dk, sk, bb) &&
              encode_map_bf16_4d(&in->Va, V, dk, sk, ba) && encode_map_bf16_4d(&in->Vb, V, dk, sk, bb);
    if (ok && s.mode == MONE_PLAIN) {
        const uint64_t dx[4] = {dh, H, (uint64_t)rows, (uint64_t)chains};
        const uint64_t sx[3] = {dh * 2, H * dh * 2, (uint64_t)rows * H * dh * 2};
        ok = encode_map_bf16_4d(&in->Xa, X, dx, sx, ba) && encode_map_bf16_4d(&in->Xb, X, dx, sx, bb);
    }
    return ok ? MONE_OK : MONE_ERR_CUDA;
}

mone_status build_state_maps(mone_mem* m) {
    DevState& s = m->s;
    if (s.dtype != MONE_BF16) return MONE_OK;
    if (s.memory == MONE_MEM_SWIGLU) return build_swiglu_maps(m);
    bool ok = encode_map_bf16_3d(&m->maps.W1b, s.W1b, s.d_in, s.d_hid, s.C, 64, 128) &&
              encode_map_bf16_3d(&m->maps.W2b, s.W2b, s.d_out, s.d_hid, s.C, 64, 128) &&
              encode_map_bf16_3d(&m->maps.W2m, s.W2b, s.d_out, s.d_hid, s.C, 64, 64) &&
              encode_map_bf16_3d(&m->maps.dH, s.dHt, s.d_hid, s.T, s.C, 64, 64) &&
              encode_map_bf16_3d(&m->maps.At, s.Att, s.d_hid, s.T, s.C, 64, 64);
    if (ok && s.Amse) ok = encode_map_bf16_3d(&m->maps.Amse, s.Amse, s.d_hid, s.T, s.C, 64, 128);
    if (ok && s.U)
        ok = encode_map_bf16_3d(&m->maps.Ua, s.U, s.d_in, s.win_rows, s.C, 64, 128) &&
             encode_map_bf16_3d(&m->maps.Ub, s.U, s.d_in, s.win_rows, s.C, 64, 64);
    if (ok)
        ok = encode_map_plain_3d(&m->maps.W1s, s.W1, true, s.d_in, s.d_hid, s.C, 128, 32) &&
             encode_map_plain_3d(&m->maps.W2s, s.W2, true, s.d_out, s.d_hid, s.C, 128, 32);
    if (ok && s.mu1)
        ok = encode_map_plain_3d(&m->maps.M1s, s.mu1, true, s.d_in, s.d_hid, s.C, 128, 32) &&
             encode_map_plain_3d(&m->maps.M2s, s.mu2, true, s.d_out, s.d_hid, s.C, 128, 32);
    return ok ? MONE_OK : MONE_ERR_CUDA;
}

// Inputs of one call: tensor maps over the caller's X, K, V ([chains][rows][width]).
mone_status build_input_maps(const DevState& s, TcInputMaps* in, const void* X, const void* K, const void* V,
                             long long rows, int chains) {
    const int dh = s.d_out / 2;
    bool ok = encode_map_bf16_3d(&in->Ka, K, dh, rows, chains, 64, 128) &&
              encode_map_bf16_3d(&in->Kb, K, dh, rows, chains, 64, 64) &&
              encode_map_bf16_3d(&in->Va, V, dh, rows, chains, 64, 128) &&
              encode_map_bf16_3d(&in->Vb, V, dh, rows, chains, 64, 64);
    if (ok && s.mode == MONE_PLAIN)
        ok = encode_map_bf16_3d(&in->Xa, X, s.d_in, rows, chains, 64, 128) &&
             encode_map_bf16_3d(&in->Xb, X, s.d_in, rows, chains, 64, 64);
    return ok ? MONE_OK : MONE_ERR_CUDA;
}


// Launch through `fn` (which returns a cudaError_t), bracketed by timing events
// when timing is on; `kernels` is the number of device kernels `fn` launches.
template <class F>
mone_status timed(mone_mem* m, int kind, cudaStream_t st, int kernels, F&& fn) {
    KernelTiming* T = m->timing;
    cudaEvent_t a = nullptr, b = nullptr;
    if (T && T->on) {
        if (!T->ref_set) {  // time origin of the launch intervals: before every later timed launch
            if (!T->ref && cudaEventCreate(&T->ref) != cudaSuccess) return MONE_ERR_CUDA;
            if (cudaEventRecord(T->ref, st) != cudaSuccess) return MONE_ERR_CUDA;
            T->ref_set = true;
        }
        a = T->get();
        b = T->get();
        if (!a || !b) return MONE_ERR_CUDA;
        if (cudaEventRecord(a, st) != cudaSuccess) return MONE_ERR_CUDA;
    }
    const cudaError_t e = fn();
    if (e != cudaSuccess) return cuda_status(e);
    if (a) {
        if (cudaEventRecord(b, st) != cudaSuccess) return MONE_ERR_CUDA;
        T->pending.push_back({kind, a, b});
    }
    m->launches += kernels;
    return MONE_OK;
}

// Run segments [0, S) of one call.  w carries chain range and input geometry.
//
// The chains of a call are independent (Eq. 11).  On the tensor-core path they
// run as two groups, one on the caller's stream and one on the handle's side
// stream, each group stepping through its segments in order.  Phase A (tensor
// and L2 bound) and phase B (HBM bound) of one group overlap the other group's
// kernels, which fills the SMs a single kernel leaves idle in its last wave and
// between launches.  The side stream forks from the caller's stream before the
// first phase launch and joins it before every input-transform window and at
// the end, so the call stays ordered on the caller's stream.
mone_status run_segment_loop(mone_mem* m, SegWork* gw, TcInputMaps* gin, TcInputMaps* rin, SwInputMaps* sin, int G,
                             const SegWork& w, long long N, cudaStream_t st, bool& forked) {
    DevState& s = m->s;
    const cudaStream_t gs[2] = {st, m->side};
    auto join = [&]() -> mone_status {
        if (forked) {
            forked = false;
            MONE_CUDA(cudaEventRecord(m->ev_join, m->side));
            MONE_CUDA(cudaStreamWaitEvent(st, m->ev_join, 0));
        }
        return MONE_OK;
    };
    if (resident_f32_fits(s)) {
        // fp32 chains that fit on chip: one launch per input window covers all of its segments
        const long long win = s.mode == MONE_PAPER ? s.win_rows : N;
        for (long long row0 = 0; row0 < N; row0 += win) {
            SegWork x = w;
            x.row0 = row0;
            x.u_off = 0;
            if (x.loss0) x.loss0 += (row0 / s.T) * x.mstride;  // per-segment metrics from the window's first
            if (x.step0) x.step0 += (row0 / s.T) * x.mstride;
            const long long n = std::min(win, N - row0);
            if (s.mode == MONE_PAPER) {
                x.Tp = (int)n;
                MONE_TRY(timed(m, K_PREPASS, st, 1, [&] { return launch_prepass(s, x, st); }));
            }
            MONE_TRY(timed(m, K_RESIDENT, st, 1, [&] { return launch_resident_f32(s, x, n, st); }));
        }
        return MONE_OK;
    }
    const long long S = (N + s.T - 1) / s.T;
    long long win0 = -1;  // first token of the current paper-mode input window
    for (long long i = 0; i < S; ++i) {
        const long long row0 = i * s.T;
        long long u_off = 0;
        if (s.mode == MONE_PAPER) {
            if (win0 < 0 || row0 >= win0 + s.win_rows) {
                // input transform of the next window of segments: depends on the inputs only,
                // and overwrites the previous window, so both groups must be done with it
                MONE_TRY(join());
                win0 = row0;
                SegWork pw = w;
                pw.row0 = row0;
                pw.Tp = (int)std::min<long long>(s.win_rows, N - win0);
                MONE_TRY(timed(m, K_PREPASS, st, 1, [&] { return launch_prepass(s, pw, st); }));
            }
            u_off = row0 - win0;
        }
        if (G > 1 && !forked) {
            MONE_CUDA(cudaEventRecord(m->ev_fork, st));
            MONE_CUDA(cudaStreamWaitEvent(m->side, m->ev_fork, 0));
            forked = true;
        }
        for (int g = 0; g < G; ++g) {
            SegWork& x = gw[g];
            const cudaStream_t sg = gs[g];
            x.row0 = row0;
            x.Tp = (int)std::min<long long>(s.T, N - row0);
            x.parity = (int)(i & 1);
            x.renorm_pending = (s.renorm && i > 0) ? 1 : 0;
            x.u_off = u_off;
            if (x.loss0) x.loss = x.loss0 + i * x.mstride;
            if (x.step0) x.step_sq = x.step0 + i * x.mstride;
            if (s.memory == MONE_MEM_SWIGLU) {
                MONE_TRY(timed(m, K_PHASE_A, sg, 1, [&] { return launch_swiglu_phase_a(s, m->swmaps, sin[g], x, sg); }));
                MONE_TRY(timed(m, K_PHASE_B, sg, 1, [&] { return launch_swiglu_phase_b(s, m->swmaps, sin[g], x, sg); }));
            } else if (s.dtype == MONE_BF16 && s.loss == MONE_LOSS_MSE) {
                // squared error: residual targets y - M(u) at the starting weights, then the
                // same two phases with them in place of y (dL/dO = eta (M(u) - y) / T')
                MONE_TRY(timed(m, K_MSE, sg, 2, [&] { return launch_mse_tc(s, m->maps, gin[g], x, sg); }));
                SegWork xr = x;
                xr.y_scratch = 1;
                xr.loss = nullptr;  // the pre-pass accumulated the squared-error loss
                MONE_TRY(timed(m, K_PHASE_A, sg, 1, [&] { return launch_phase_a_tc(s, m->maps, rin[g], xr, sg); }));
                MONE_TRY(timed(m, K_PHASE_B, sg, 1, [&] { return launch_phase_b_tc(s, m->maps, rin[g], xr, sg); }));
            } else if (s.dtype == MONE_BF16) {
                MONE_TRY(timed(m, K_PHASE_A, sg, 1, [&] { return launch_phase_a_tc(s, m->maps, gin[g], x, sg); }));
                MONE_TRY(timed(m, K_PHASE_B, sg, 1, [&] { return launch_phase_b_tc(s, m->maps, gin[g], x, sg); }));
            } else if (s.loss == MONE_LOSS_MSE) {  // fp32: the same scheme on the CUDA cores
                MONE_TRY(timed(m, K_MSE, sg, 2, [&] { return launch_mse_f32(s, x, sg); }));
                SegWork xr = x;
                xr.y_scratch = 1;
                xr.loss = nullptr;
                MONE_TRY(timed(m, K_PHASE_A, sg, 1, [&] { return launch_phase_a_f32(s, xr, sg); }));
                MONE_TRY(timed(m, K_PHASE_B, sg, 1, [&] { return launch_phase_b_f32(s, xr, sg); }));
            } else {
                MONE_TRY(timed(m, K_PHASE_A, sg, 1, [&] { return launch_phase_a_f32(s, x, sg); }));
                MONE_TRY(timed(m, K_PHASE_B, sg, 1, [&] { return launch_phase_b_f32(s, x, sg); }));
            }
            if (s.col_renorm)  // output channels: the columns of W2 back to their norms in W_0
                MONE_TRY(timed(m, K_FINALIZE, sg, 2, [&] { return launch_col_renorm(s, x.c0, x.nc, sg); }));
        }
    }
    MONE_TRY(join());
    if (s.renorm) {
        const int par = (int)((S - 1) & 1);
        if (s.memory == MONE_MEM_SWIGLU)
            MONE_TRY(timed(m, K_FINALIZE, st, 1, [&] { return launch_swiglu_rows(s, 1, par, w.c0, w.nc, st); }));
        else
            MONE_TRY(timed(m, K_FINALIZE, st, 1, [&] { return launch_finalize(s, w.c0, w.nc, par, 1, st); }));
    }
    return MONE_OK;
}

mone_status run_segments(mone_mem* m, SegWork w, long long N, cudaStream_t st) {
    DevState& s = m->s;
    const int G = (m->side && w.nc >= 2) ? 2 : 1;
    SegWork gw[2];
    TcInputMaps gin[2], rin[2];
    SwInputMaps sin[2];
    const size_t el = elsize(s.dtype);
    for (int g = 0, off = 0; g < G; ++g) {
        const int n = w.nc / G + (g < w.nc % G ? 1 : 0);
        gw[g] = w;
        gw[g].c0 = w.c0 + off;
        gw[g].nc = n;
        gw[g].X = static_cast<const uint8_t*>(w.X) + (size_t)off * w.x_cstride * el;
        gw[g].K = static_cast<const uint8_t*>(w.K) + (size_t)off * w.y_cstride * el;
        gw[g].V = static_cast<const uint8_t*>(w.V) + (size_t)off * w.y_cstride * el;
        if (w.eta_in) gw[g].eta_in = w.eta_in + (size_t)off * w.eta_cstride;
        if (w.loss) gw[g].loss = w.loss + off;
        if (w.loss0) gw[g].loss0 = w.loss0 + off;
        if (w.step0) gw[g].step0 = w.step0 + off;
        std::memset(&gin[g], 0, sizeof(TcInputMaps));
        std::memset(&rin[g], 0, sizeof(TcInputMaps));
        std::memset(&sin[g], 0, sizeof(SwInputMaps));
        if (s.memory == MONE_MEM_SWIGLU)
            MONE_TRY(build_swiglu_input_maps(s, &sin[g], gw[g].X, gw[g].K, gw[g].V, w.n_rows, n));
        else if (s.dtype == MONE_BF16)
            MONE_TRY(build_input_maps(s, &gin[g], gw[g].X, gw[g].K, gw[g].V, w.n_rows, n));
        if (s.dtype == MONE_BF16 && s.loss == MONE_LOSS_MSE) {
            // residual targets of this group's chains: [C][T][d_out/2] scratch, rows from 0
            const size_t o = (size_t)gw[g].c0 * s.T * (s.d_out / 2);
            MONE_TRY(build_input_maps(s, &rin[g], gw[g].X, s.Kres + o, s.Vres + o, s.T, n));
            if (s.mode == MONE_PLAIN) {  // U stays the caller's X
                rin[g].Xa = gin[g].Xa;
                rin[g].Xb = gin[g].Xb;
            }
        }
        off += n;
    }
    bool forked = false;
    const mone_status rc = run_segment_loop(m, gw, gin, rin, sin, G, w, N, st, forked);
    if (forked) {
        // error after the fork: still order the side stream's work before the caller's stream
        cudaEventRecord(m->ev_join, m->side);
        cudaStreamWaitEvent(st, m->ev_join, 0);
    }
    return rc;
}

// The device address of `bytes` of host memory the device can read: page-locked memory
// (cudaHostAlloc, cudaHostRegister), or any host memory where the device reads through the
// host's page tables (Grace).  Only the first and last bytes are checked (the caller
// guarantees the range between them).  Device and managed memory are refused:
// mone_ttl_context takes those.
mone_status host_device_view(const void* p, size_t bytes, const void** out) {
    cudaPointerAttributes a{}, b{};
    if (cudaPointerGetAttributes(&a, p) != cudaSuccess ||
        cudaPointerGetAttributes(&b, static_cast<const uint8_t*>(p) + bytes - 1) != cudaSuccess) {
        cudaGetLastError();
        return MONE_ERR_INVALID_ARG;
    }
    if (a.type == cudaMemoryTypeHost && b.type == cudaMemoryTypeHost && a.devicePointer &&
        static_cast<const uint8_t*>(b.devicePointer) == static_cast<const uint8_t*>(a.devicePointer) + bytes - 1) {
        *out = a.devicePointer;
        return MONE_OK;
    }
    if (a.type == cudaMemoryTypeUnregistered && b.type == cudaMemoryTypeUnregistered) {
        int dev = 0, via_host_tables = 0;
        if (cudaGetDevice(&dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&via_host_tables, cudaDevAttrPageableMemoryAccessUsesHostPageTables, dev) !=
                cudaSuccess)
            return MONE_ERR_CUDA;
        if (via_host_tables) {
            *out = p;
            return MONE_OK;
        }
    }
    return MONE_ERR_INVALID_ARG;
}

// Bytes of X, K and V per staged chunk when the caller leaves the chunk length to the library:
// large enough that a chunk's learning amortises the per-call setup, small enough that the
// first chunk's gather (not overlapped) stays short.
constexpr long long kHostChunkBytes = 512ll << 20;

}  // namespace

extern "C" {

int mone_abi_version(void) { return MONE_ABI_VERSION; }

const char* mone_last_error(void) { return g_last_error; }

const char* mone_status_string(mone_status st) {
    switch (st) {
        case MONE_OK: return "ok";
        case MONE_ERR_INVALID_ARG: return "invalid argument";
        case MONE_ERR_UNSUPPORTED_SHAPE: return "unsupported shape";
        case MONE_ERR_OOM: return "device out of memory";
        case MONE_ERR_CUDA: return "CUDA error";
        case MONE_ERR_TIMEOUT: return "device wait timed out";
        case MONE_ERR_NONFINITE: return "non-finite fast weight";
        case MONE_ERR_UNSUPPORTED: return "unsupported request";
        case MONE_ERR_CHECK: return "device index check failed";
    }
    return "unknown status";
}

mone_status mone_mem_init(const mone_config* cfg, const float* W1_0, const float* W2_0, const mone_meta* meta,
                          void* stream, mone_mem** out) {
    if (!out) return MONE_ERR_INVALID_ARG;
    *out = nullptr;
    MONE_TRY(validate_config(cfg));
    if (!W1_0 || !W2_0 || !aligned16(W1_0) || !aligned16(W2_0)) return MONE_ERR_INVALID_ARG;
    if (cfg->mode == MONE_PAPER &&
        (!meta || !meta->alpha || !meta->gamma || !meta->w_eta || !meta->b_eta || !meta->w_beta || !meta->b_beta))
        return MONE_ERR_INVALID_ARG;
    int ndev = 0;
    if (cudaGetDeviceCount(&ndev) != cudaSuccess || ndev < 1) {
        cudaGetLastError();
        return MONE_ERR_CUDA;
    }
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    mone_mem* m = new (std::nothrow) mone_mem;
    if (!m) return MONE_ERR_OOM;
    std::memset(m, 0, sizeof(*m));
    m->cfg = *cfg;
    DevState& s = m->s;
    s.C = cfg->n_ctx * cfg->n_layers;
    s.d_in = cfg->d_in; s.d_hid = cfg->d_hid; s.d_out = cfg->d_out;
    s.n_kv = cfg->n_kv_heads; s.hd = cfg->head_dim; s.T = cfg->seg_T;
    s.dtype = cfg->dtype; s.mode = cfg->mode;
    s.momentum = cfg->mode == MONE_PAPER; s.renorm = cfg->mode == MONE_PAPER;
    s.lr = cfg->lr; s.rms_eps = cfg->rms_eps;
    s.loss = cfg->loss;
    s.memory = cfg->memory;
    s.heads = cfg->memory == MONE_MEM_SWIGLU ? cfg->mem_heads : 1;
    s.col_renorm = (s.renorm && cfg->renorm_axis == MONE_RENORM_OUT) ? 1 : 0;
    if (s.mode == MONE_PAPER) {
        // the input transform covers a window of whole segments whose scratch stays within ~2 GiB
        const size_t row_bytes = (size_t)s.C * s.d_in * elsize(s.dtype);
        long long segs = (long long)((size_t(2) << 30) / (row_bytes * (size_t)s.T));
        segs = std::max(1ll, std::min(64ll, segs));
        s.win_rows = (int)(segs * s.T);
    }
    const size_t C = s.C, n1 = w1_elems(s), n2 = w2_elems(s);
    const size_t r1 = w1_rows(s);  // rows of W1 over all chains (and heads): sizes the row tables
    mone_status rc = MONE_OK;
    auto step = [&](mone_status r) { if (rc == MONE_OK) rc = r; };
    step(dalloc(&s.W1, n1));
    step(dalloc(&s.W2, n2));
    if (s.momentum) {
        step(dalloc(&s.mu1, n1));
        step(dalloc(&s.mu2, n2));
    }
    if (s.dtype == MONE_BF16) {
        step(dalloc(&s.W1b, n1));
        step(dalloc(&s.W2b, n2));
        if (s.loss == MONE_LOSS_MSE) {
            step(dalloc(&s.Amse, C * s.T * s.d_hid));
            step(dalloc(&s.Kres, C * s.T * (s.d_out / 2)));
            step(dalloc(&s.Vres, C * s.T * (s.d_out / 2)));
        }
    }
    if (s.dtype == MONE_FP32 && s.loss == MONE_LOSS_MSE) {
        step(dalloc(&s.Kres32, C * s.T * (s.d_out / 2)));
        step(dalloc(&s.Vres32, C * s.T * (s.d_out / 2)));
    }
    step(dalloc(&s.n1, r1));
    step(dalloc(&s.n2, w2_rows(s)));
    step(dalloc(&s.sumsq, 4 * r1));
    step(dalloc(&s.status, 2));  // flags, and the first failing check site (MONE_DEBUG builds)
    if (const char* f = std::getenv("MONE_FAULT_STALL"))  // test knob: see DevState::fault_stall
        s.fault_stall = std::atoi(f) > 0 ? std::atoi(f) : 0;
    if (s.mode == MONE_PAPER) {
        step(dalloc(&s.alpha, C * s.d_in));
        step(dalloc(&s.gamma, C * s.d_in));
        step(dalloc(&s.w_eta, C * s.d_in));
        step(dalloc(&s.w_beta, C * s.d_in));
        step(dalloc(&s.b_eta, C));
        step(dalloc(&s.b_beta, C));
        step(dalloc(reinterpret_cast<uint8_t**>(&s.U), C * s.win_rows * s.d_in * elsize(s.dtype)));
        step(dalloc(&s.eta, C * s.win_rows));
        step(dalloc(&s.dbeta, C * s.win_rows));
        step(dalloc(&s.zinv, C * s.win_rows));
    }
    const bool silu_gate = cfg->gate_act == MONE_GATE_SILU;
    if ((meta && meta->gate) || silu_gate) step(dalloc(&s.gate, C * 2 * s.n_kv));
    if (s.col_renorm) {
        step(dalloc(&s.nc2, C * s.d_out));
        step(dalloc(&s.colpart, (size_t)kColRowSlices * C * s.d_out));
    }
    const size_t elt = s.dtype == MONE_BF16 ? 2 : 4;
    // phase A outputs: c dH and c A ([C][T][d_hid]); SwiGLU: c [dP | dG] ([C*H][T][2 d_hid]) and c Z
    step(dalloc(reinterpret_cast<uint8_t**>(&s.dHt), r1 * s.T * elt));
    step(dalloc(reinterpret_cast<uint8_t**>(&s.Att), w2_rows(s) * s.T * elt));
    auto cp = [&](void* dst, const void* src, size_t bytes) {
        if (rc == MONE_OK) rc = cuda_status(cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDeviceToDevice, st));
    };
    cp(s.W1, W1_0, n1 * 4);
    cp(s.W2, W2_0, n2 * 4);
    if (s.mode == MONE_PAPER) {
        cp(s.alpha, meta->alpha, C * s.d_in * 4);
        cp(s.gamma, meta->gamma, C * s.d_in * 4);
        cp(s.w_eta, meta->w_eta, C * s.d_in * 4);
        cp(s.w_beta, meta->w_beta, C * s.d_in * 4);
        cp(s.b_eta, meta->b_eta, C * 4);
        cp(s.b_beta, meta->b_beta, C * 4);
    }
    const bool caller_gate = meta && meta->gate;
    if (caller_gate) cp(s.gate, meta->gate, C * 2 * s.n_kv * 4);
    if (silu_gate && rc == MONE_OK)  // the read scales head h by SiLU(g_h) (g_h = 1 when not given)
        step(cuda_status(launch_gate_silu(s.gate, C * 2 * s.n_kv, caller_gate ? 0 : 1, st)));
    if (rc == MONE_OK && s.momentum) {
        step(cuda_status(cudaMemsetAsync(s.mu1, 0, n1 * 4, st)));
        step(cuda_status(cudaMemsetAsync(s.mu2, 0, n2 * 4, st)));
    }
    if (rc == MONE_OK) step(cuda_status(cudaMemsetAsync(s.sumsq, 0, 4 * r1 * 4, st)));
    if (rc == MONE_OK) step(cuda_status(cudaMemsetAsync(s.status, 0, 2 * sizeof(int), st)));
    if (s.memory == MONE_MEM_SWIGLU) {
        if (rc == MONE_OK) step(cuda_status(launch_swiglu_rows(s, 0, 0, 0, s.C, st)));  // targets + bf16 copies
    } else {
        if (rc == MONE_OK) step(cuda_status(launch_row_norms(s, st)));
        if (rc == MONE_OK && s.col_renorm) step(cuda_status(launch_col_targets(s, st)));
        if (rc == MONE_OK && s.dtype == MONE_BF16) step(cuda_status(launch_finalize(s, 0, s.C, 0, 0, st)));
    }
    if (rc == MONE_OK) step(build_state_maps(m));
    if (rc == MONE_OK) step(cuda_status(cudaStreamSynchronize(st)));
    if (rc != MONE_OK) {
        cudaStreamSynchronize(st);
        cudaGetLastError();
        free_state(s);
        delete m;
        return rc;
    }
    if (s.dtype == MONE_BF16 && s.C >= 2) {
        // second chain group's stream and the fork/join events (see run_segments)
        cudaError_t e = cudaStreamCreateWithFlags(&m->side, cudaStreamNonBlocking);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&m->ev_fork, cudaEventDisableTiming);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&m->ev_join, cudaEventDisableTiming);
        if (e != cudaSuccess) {
            cudaGetLastError();
            destroy_streams(m);
            free_state(s);
            delete m;
            return cuda_status(e);
        }
    }
    m->launches = 1 + (s.dtype == MONE_BF16 ? 1 : 0);
    {
        std::lock_guard<std::mutex> lk(g_live_mu);
        g_live.insert(m);
    }
    *out = m;
    return MONE_OK;
}

mone_status mone_ttl_segment(mone_mem* m, int ctx, int layer, const void* X, const void* K, const void* V,
                             int n_tok, const float* eta, float* loss_out, void* stream) {
    if (!is_live(m)) return MONE_ERR_INVALID_ARG;
    const DevState& s = m->s;
    if (ctx < 0 || ctx >= m->cfg.n_ctx || layer < 0 || layer >= m->cfg.n_layers) return MONE_ERR_INVALID_ARG;
    if (n_tok < 1 || n_tok > s.T) return MONE_ERR_INVALID_ARG;
    if (!X || !K || !V || !aligned16(X) || !aligned16(K) || !aligned16(V)) return MONE_ERR_INVALID_ARG;
    if (eta && (reinterpret_cast<uintptr_t>(eta) & 3u)) return MONE_ERR_INVALID_ARG;
    if (loss_out && (reinterpret_cast<uintptr_t>(loss_out) & 3u)) return MONE_ERR_INVALID_ARG;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    SegWork w{};
    w.c0 = ctx * m->cfg.n_layers + layer;
    w.nc = 1;
    w.X = X; w.K = K; w.V = V;
    w.x_cstride = 0; w.y_cstride = 0;
    w.n_rows = n_tok;
    w.eta_in = eta;
    w.eta_cstride = 0;
    w.loss = loss_out;
    if (loss_out) MONE_CUDA(cudaMemsetAsync(loss_out, 0, sizeof(float), st));
    return run_segments(m, w, n_tok, st);
}

mone_status mone_ttl_context_metrics(mone_mem* m, const void* X, const void* K, const void* V, long long N,
                                     float* seg_loss, float* seg_step, void* stream) {
    if (!is_live(m)) return MONE_ERR_INVALID_ARG;
    const DevState& s = m->s;
    if (N < 1 || N > (1ll << 31) - 1) return MONE_ERR_INVALID_ARG;
    if (!X || !K || !V || !aligned16(X) || !aligned16(K) || !aligned16(V)) return MONE_ERR_INVALID_ARG;
    if ((seg_loss && (reinterpret_cast<uintptr_t>(seg_loss) & 3u)) ||
        (seg_step && (reinterpret_cast<uintptr_t>(seg_step) & 3u)))
        return MONE_ERR_INVALID_ARG;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const long long S = (N + s.T - 1) / s.T;
    if (seg_loss) MONE_CUDA(cudaMemsetAsync(seg_loss, 0, (size_t)S * s.C * sizeof(float), st));
    if (seg_step) MONE_CUDA(cudaMemsetAsync(seg_step, 0, (size_t)S * s.C * sizeof(float), st));
    SegWork w{};
    w.c0 = 0;
    w.nc = s.C;
    w.X = X; w.K = K; w.V = V;
    w.x_cstride = N * s.d_in;
    w.y_cstride = N * (s.d_out / 2);
    w.n_rows = N;
    w.loss0 = seg_loss;
    w.step0 = seg_step;
    w.mstride = s.C;
    return run_segments(m, w, N, st);
}

mone_status mone_ttl_context(mone_mem* m, const void* X, const void* K, const void* V, long long N, void* stream) {
    if (!is_live(m)) return MONE_ERR_INVALID_ARG;
    const DevState& s = m->s;
    if (N < 1 || N > (1ll << 31) - 1) return MONE_ERR_INVALID_ARG;
    if (!X || !K || !V || !aligned16(X) || !aligned16(K) || !aligned16(V)) return MONE_ERR_INVALID_ARG;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    SegWork w{};
    w.c0 = 0;
    w.nc = s.C;
    w.X = X; w.K = K; w.V = V;
    w.x_cstride = N * s.d_in;
    w.y_cstride = N * (s.d_out / 2);
    w.n_rows = N;
    w.eta_in = nullptr;
    w.loss = nullptr;
    return run_segments(m, w, N, st);
}

// Test-time learning of a context held in host memory: chunks of whole segments are gathered
// into two device windows on the staging stream while the previous chunk is learned on the
// caller's stream (the learning of each chunk is the call mone_ttl_context makes, continuing
// the state, so the chunks together equal one call on all N tokens).
mone_status mone_ttl_context_host(mone_mem* m, const void* X, const void* K, const void* V, long long N,
                                  long long chunk_tokens, void* stream) {
    if (!is_live(m)) return MONE_ERR_INVALID_ARG;
    const DevState& s = m->s;
    if (N < 1 || N > (1ll << 31) - 1) return MONE_ERR_INVALID_ARG;
    if (!X || !K || !V || !aligned16(X) || !aligned16(K) || !aligned16(V)) return MONE_ERR_INVALID_ARG;
    if (chunk_tokens < 0 || (chunk_tokens > 0 && chunk_tokens % s.T)) return MONE_ERR_INVALID_ARG;
    const long long el = (long long)elsize(s.dtype), C = s.C;
    const long long row_b[3] = {s.d_in * el, (s.d_out / 2) * el, (s.d_out / 2) * el};
    if (row_b[0] % 16 || row_b[1] % 16) return MONE_ERR_UNSUPPORTED_SHAPE;  // 16-byte units per row
    const void* hv[3];
    const void* hp[3] = {X, K, V};
    for (int t = 0; t < 3; ++t) MONE_TRY(host_device_view(hp[t], (size_t)(C * N * row_b[t]), &hv[t]));
    const long long tok_b = C * (row_b[0] + row_b[1] + row_b[2]);  // bytes of one token over all chains
    long long ct = chunk_tokens;
    if (ct == 0) ct = std::max<long long>(s.T, kHostChunkBytes / tok_b / s.T * s.T);
    ct = std::min(ct, (N + s.T - 1) / s.T * s.T);
    const size_t win_bytes = (size_t)(ct * tok_b);
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    if (!m->hstream) {
        MONE_CUDA(cudaStreamCreateWithFlags(&m->hstream, cudaStreamNonBlocking));
        MONE_CUDA(cudaEventCreateWithFlags(&m->hstart, cudaEventDisableTiming));
        for (int b = 0; b < 2; ++b) {
            MONE_CUDA(cudaEventCreateWithFlags(&m->hstaged[b], cudaEventDisableTiming));
            MONE_CUDA(cudaEventCreateWithFlags(&m->hfree[b], cudaEventDisableTiming));
        }
    }
    if (win_bytes > m->hwin_bytes) {  // grow the windows (not while earlier work may read them)
        MONE_CUDA(cudaStreamSynchronize(st));
        MONE_CUDA(cudaStreamSynchronize(m->hstream));
        for (int b = 0; b < 2; ++b) {
            if (m->hwin[b]) cudaFree(m->hwin[b]);
            m->hwin[b] = nullptr;
        }
        m->hwin_bytes = 0;
        for (int b = 0; b < 2; ++b)
            if (cudaMalloc(&m->hwin[b], win_bytes) != cudaSuccess) {
                cudaGetLastError();
                return MONE_ERR_OOM;
            }
        m->hwin_bytes = win_bytes;
    }
    // the gathers start after what the caller queued before this call
    MONE_CUDA(cudaEventRecord(m->hstart, st));
    MONE_CUDA(cudaStreamWaitEvent(m->hstream, m->hstart, 0));
    // the persistent learning kernels leave the gather's SMs free for the rest of this call
    struct Reserve {
        const DevState& s;
        explicit Reserve(const DevState& d) : s(d) { s.reserve_sms = stage_sms(); }
        ~Reserve() { s.reserve_sms = 0; }
    } reserve(s);
    for (long long r0 = 0, k = 0; r0 < N; r0 += ct, ++k) {
        const long long nr = std::min(ct, N - r0);
        const int b = (int)(k & 1);
        uint8_t* win = static_cast<uint8_t*>(m->hwin[b]);
        void* dst[3] = {win, win + C * nr * row_b[0], win + C * nr * (row_b[0] + row_b[1])};
        MONE_CUDA(cudaStreamWaitEvent(m->hstream, m->hfree[b], 0));  // never recorded: no wait
        MONE_TRY(timed(m, K_STAGE, m->hstream, 1,
                       [&] { return launch_stage_rows(hv, dst, row_b, N, r0, nr, s.C, m->hstream); }));
        MONE_CUDA(cudaEventRecord(m->hstaged[b], m->hstream));
        MONE_CUDA(cudaStreamWaitEvent(st, m->hstaged[b], 0));
        SegWork w{};
        w.c0 = 0;
        w.nc = s.C;
        w.X = dst[0]; w.K = dst[1]; w.V = dst[2];
        w.x_cstride = nr * s.d_in;
        w.y_cstride = nr * (s.d_out / 2);
        w.n_rows = nr;
        MONE_TRY(run_segments(m, w, nr, st));
        MONE_CUDA(cudaEventRecord(m->hfree[b], st));
    }
    return MONE_OK;
}

mone_status mone_mem_generate_kv(mone_mem* m, const void* Xq, int Q, void* K_out, void* V_out,
                                 const long long strides[4], void* stream) {
    if (!is_live(m)) return MONE_ERR_INVALID_ARG;
    if (Q < 1 || Q > 4096 || !Xq || !K_out || !V_out || !strides) return MONE_ERR_INVALID_ARG;
    for (int i = 0; i < 4; ++i)
        if (strides[i] < 0) return MONE_ERR_INVALID_ARG;
    DevState& s = m->s;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    if (Q > s.q_cap) {
        MONE_CUDA(cudaStreamSynchronize(st));
        if (s.Uq) cudaFree(s.Uq);
        if (s.Aq) cudaFree(s.Aq);
        if (s.Oq) cudaFree(s.Oq);
        s.Uq = s.Aq = s.Oq = nullptr;
        s.q_cap = 0;
        const size_t C = s.C;
        MONE_TRY(dalloc(&s.Uq, C * Q * s.d_in));
        MONE_TRY(dalloc(&s.Aq, C * Q * s.d_hid * s.heads));  // SwiGLU: bf16 Z_q of every head
        MONE_TRY(dalloc(&s.Oq, C * Q * s.d_out));
        s.q_cap = Q;
    }
    const int L = m->cfg.n_layers;
    auto launch = [&](cudaStream_t sx) -> cudaError_t {
        cudaError_t e;
        if (s.memory == MONE_MEM_SWIGLU) {
            e = launch_query_transform(s, Xq, Q, s.Uq, true, sx);
            if (e == cudaSuccess) e = launch_swiglu_read(s, m->swmaps, s.Uq, s.Aq, Q, sx);
            return e != cudaSuccess ? e : launch_read_norm(s, Q, L, K_out, V_out, strides, sx);
        }
        if (s.dtype == MONE_BF16) {  // tensor-core read: bf16 queries and hidden activations in the scratch
            return launch_read_tc(s, m->maps, Xq, s.Uq, s.Aq, s.Oq, Q, L, K_out, V_out, strides, sx);
        }
        e = launch_query_transform(s, Xq, Q, s.Uq, false, sx);
        return e != cudaSuccess ? e : launch_read(s, Q, L, K_out, V_out, strides, sx);
    };
    const int kernels = (s.memory == MONE_MEM_SWIGLU || s.dtype == MONE_FP32) ? 4 : 3;
    if (!m->rg) m->rg = new ReadGraph();
    ReadGraph& g = *m->rg;
    const bool same = g.xq == Xq && g.ko == K_out && g.vo == V_out && g.q == Q && g.uq == s.Uq && g.aq == s.Aq &&
                      g.oq == s.Oq && std::equal(strides, strides + 4, g.strides);
    if (!same) {  // a new key: drop the graph of the old one
        if (g.exec) cudaGraphExecDestroy(g.exec);
        g = ReadGraph();
        g.xq = Xq; g.ko = K_out; g.vo = V_out; g.q = Q; g.uq = s.Uq; g.aq = s.Aq; g.oq = s.Oq;
        std::copy(strides, strides + 4, g.strides);
    }
    if (!g.exec && ++g.seen >= 2) {
        // the key repeats: capture the launches on a private stream (nothing runs during capture)
        cudaError_t e = cudaSuccess;
        if (!m->cap) e = cudaStreamCreateWithFlags(&m->cap, cudaStreamNonBlocking);
        if (e == cudaSuccess) e = cudaStreamBeginCapture(m->cap, cudaStreamCaptureModeThreadLocal);
        if (e == cudaSuccess) {
            const cudaError_t le = launch(m->cap);
            cudaGraph_t graph = nullptr;
            e = cudaStreamEndCapture(m->cap, &graph);
            if (le != cudaSuccess) e = le;
            if (e == cudaSuccess) e = cudaGraphInstantiate(&g.exec, graph, 0);
            if (graph) cudaGraphDestroy(graph);
        }
        if (e != cudaSuccess) {
            g.exec = nullptr;
            return cuda_status(e);
        }
    }
    if (g.exec) return timed(m, K_READ, st, kernels, [&] { return cudaGraphLaunch(g.exec, st); });
    return timed(m, K_READ, st, kernels, [&] { return launch(st); });
}

mone_status mone_mem_generate_kv_noalloc(mone_mem* m, const void* Xq, int Q, void* K_out, void* V_out,
                                         const long long strides[4], void* stream) {
    if (!is_live(m)) return MONE_ERR_INVALID_ARG;
    if (Q < 1 || Q > 4096 || !Xq || !K_out || !V_out || !strides) return MONE_ERR_INVALID_ARG;
    for (int i = 0; i < 4; ++i)
        if (strides[i] < 0) return MONE_ERR_INVALID_ARG;
    const DevState& s = m->s;
    if (s.memory == MONE_MEM_SWIGLU) {
        std::snprintf(g_last_error, sizeof(g_last_error),
                      "mone_mem_generate_kv_noalloc: not available for the SwiGLU memory");
        return MONE_ERR_UNSUPPORTED;
    }
    const size_t need = (size_t)s.C * Q * ((size_t)s.d_in + s.d_hid + s.d_out);
    if (need > kNoAllocScratchFloats) {
        std::snprintf(g_last_error, sizeof(g_last_error),
                      "mone_mem_generate_kv_noalloc: chains*Q*(d_in+d_hid+d_out) = %zu floats exceeds the fixed "
                      "scratch of %zu floats (16 MiB)",
                      need, kNoAllocScratchFloats);
        return MONE_ERR_UNSUPPORTED_SHAPE;
    }
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const int L = m->cfg.n_layers;
    const TcMaps* tc = s.dtype == MONE_BF16 ? &m->maps : nullptr;
    return timed(m, K_READ, st, tc ? 3 : 4,
                 [&] { return launch_read_noalloc(s, tc, Xq, Q, L, K_out, V_out, strides, st); });
}

mone_status mone_attention(mone_mem* m, const void* Q, int n_q_heads, int Lq, const void* K, const void* V,
                           const long long kv_strides[4], int n_mem, void* out, void* stream) {
    if (!is_live(m)) return MONE_ERR_INVALID_ARG;
    const DevState& s = m->s;
    if (!Q || !K || !V || !out || !kv_strides) return MONE_ERR_INVALID_ARG;
    if (n_q_heads < s.n_kv || n_q_heads % s.n_kv || n_q_heads / s.n_kv > 64) return MONE_ERR_INVALID_ARG;
    if (Lq < 1 || n_mem < 0 || (long long)n_mem + Lq > (1ll << 20)) return MONE_ERR_INVALID_ARG;
    for (int i = 0; i < 4; ++i)
        if (kv_strides[i] < 0) return MONE_ERR_INVALID_ARG;
    if (kv_strides[3] < s.hd) return MONE_ERR_INVALID_ARG;  // positions hold head_dim contiguous elements
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const int L = m->cfg.n_layers;
    return timed(m, K_ATTN, st, 1, [&] {
        return launch_attention(s, L, Q, n_q_heads, Lq, K, V, kv_strides, n_mem, out, st);
    });
}

mone_status mone_mem_free(mone_mem* m) {
    {
        std::lock_guard<std::mutex> lk(g_live_mu);
        if (!m || !g_live.count(m)) return MONE_ERR_INVALID_ARG;
        g_live.erase(m);
    }
    cudaDeviceSynchronize();
    delete m->timing;
    destroy_streams(m);
    free_state(m->s);
    delete m;
    return MONE_OK;
}

mone_status mone_mem_read_state(const mone_mem* m, float* W1, float* W2, float* mu1, float* mu2, void* stream) {
    if (!is_live(m)) return MONE_ERR_INVALID_ARG;
    const DevState& s = m->s;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const size_t n1 = w1_elems(s) * 4, n2 = w2_elems(s) * 4;
    if (W1) MONE_CUDA(cudaMemcpyAsync(W1, s.W1, n1, cudaMemcpyDeviceToDevice, st));
    if (W2) MONE_CUDA(cudaMemcpyAsync(W2, s.W2, n2, cudaMemcpyDeviceToDevice, st));
    if (mu1) {
        if (s.mu1) MONE_CUDA(cudaMemcpyAsync(mu1, s.mu1, n1, cudaMemcpyDeviceToDevice, st));
        else MONE_CUDA(cudaMemsetAsync(mu1, 0, n1, st));
    }
    if (mu2) {
        if (s.mu2) MONE_CUDA(cudaMemcpyAsync(mu2, s.mu2, n2, cudaMemcpyDeviceToDevice, st));
        else MONE_CUDA(cudaMemsetAsync(mu2, 0, n2, st));
    }
    return MONE_OK;
}

mone_status mone_mem_write_state(mone_mem* m, const float* W1, const float* W2, const float* mu1, const float* mu2,
                                 void* stream) {
    if (!is_live(m)) return MONE_ERR_INVALID_ARG;
    DevState& s = m->s;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const size_t n1 = w1_elems(s) * 4, n2 = w2_elems(s) * 4;
    if ((mu1 || mu2) && !s.momentum) return MONE_ERR_INVALID_ARG;
    if (W1) MONE_CUDA(cudaMemcpyAsync(s.W1, W1, n1, cudaMemcpyDeviceToDevice, st));
    if (W2) MONE_CUDA(cudaMemcpyAsync(s.W2, W2, n2, cudaMemcpyDeviceToDevice, st));
    if (mu1) MONE_CUDA(cudaMemcpyAsync(s.mu1, mu1, n1, cudaMemcpyDeviceToDevice, st));
    if (mu2) MONE_CUDA(cudaMemcpyAsync(s.mu2, mu2, n2, cudaMemcpyDeviceToDevice, st));
    if (s.memory == MONE_MEM_SWIGLU && (W1 || W2))
        return timed(m, K_FINALIZE, st, 1, [&] { return launch_swiglu_rows(s, 2, 0, 0, s.C, st); });
    if (s.dtype == MONE_BF16 && (W1 || W2))
        return timed(m, K_FINALIZE, st, 1, [&] { return launch_finalize(s, 0, s.C, 0, 0, st); });
    return MONE_OK;
}

mone_status mone_mem_sync(mone_mem* m, void* stream) {
    if (!is_live(m)) return MONE_ERR_INVALID_ARG;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    MONE_CUDA(cudaStreamSynchronize(st));
    int flag = 0;
    int word[2] = {0, 0};
    MONE_CUDA(cudaMemcpy(word, m->s.status, sizeof(word), cudaMemcpyDeviceToHost));
    flag = word[0];
    if (flag) MONE_CUDA(cudaMemset(m->s.status, 0, sizeof(word)));
    if (flag & DEV_CHECK) {
        static const char* const sites[] = {"?", "phase A tile", "phase B tile", "read tile", "resident rows",
                                            "TMA x coordinate"};
        const int site = word[1] >= 1 && word[1] <= 5 ? word[1] : 0;
        std::snprintf(g_last_error, sizeof(g_last_error), "device index check failed: %s", sites[site]);
        return MONE_ERR_CHECK;
    }
    if (flag & DEV_TIMEOUT) return MONE_ERR_TIMEOUT;
    if (flag & DEV_NONFINITE) return MONE_ERR_NONFINITE;
    return MONE_OK;
}

long long mone_mem_launch_count(const mone_mem* m) { return is_live(m) ? m->launches : -1; }

mone_status mone_mem_set_timing(mone_mem* m, int enable) {
    if (!is_live(m)) return MONE_ERR_INVALID_ARG;
    if (!m->timing) {
        m->timing = new (std::nothrow) KernelTiming;
        if (!m->timing) return MONE_ERR_OOM;
    }
    KernelTiming* T = m->timing;
    const cudaError_t e = T->drain();
    T->on = enable != 0;
    if (enable) T->reset();
    return cuda_status(e);
}

mone_status mone_mem_kernel_time(mone_mem* m, int kind, double* ms, long long* launches) {
    if (!is_live(m) || kind < 0 || kind >= K_KINDS || !ms || !launches) return MONE_ERR_INVALID_ARG;
    *ms = 0;
    *launches = 0;
    if (!m->timing) return MONE_OK;
    MONE_CUDA(m->timing->drain());
    *ms = m->timing->ms[kind];
    *launches = m->timing->n[kind];
    return MONE_OK;
}

mone_status mone_mem_kernel_busy(mone_mem* m, int kind, double* busy_ms) {
    if (!is_live(m) || kind < 0 || kind >= K_KINDS || !busy_ms) return MONE_ERR_INVALID_ARG;
    *busy_ms = 0;
    if (!m->timing) return MONE_OK;
    MONE_CUDA(m->timing->drain());
    std::vector<std::pair<double, double>> v = m->timing->iv[kind];
    std::sort(v.begin(), v.end());
    double cur0 = 0, cur1 = -1;  // the union of the intervals, merged in start order
    for (const auto& x : v) {
        if (x.first > cur1) {
            if (cur1 > cur0) *busy_ms += cur1 - cur0;
            cur0 = x.first;
            cur1 = x.second;
        } else if (x.second > cur1) {
            cur1 = x.second;
        }
    }
    if (cur1 > cur0) *busy_ms += cur1 - cur0;
    return MONE_OK;
}

}  // extern "C"
