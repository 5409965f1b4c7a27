// Internal interface between the C-ABI front end (mone_api.cu) and the kernel
// translation units.  Host-side launchers only; no torch types anywhere.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace mone {

using bf16 = __nv_bfloat16;

// Bits of the device status word (latched until mone_mem_sync reads it).
enum : int { DEV_TIMEOUT = 1, DEV_NONFINITE = 2, DEV_CHECK = 4 };
// Sites of the device-side index checks of a MONE_DEBUG build; the first failing site is kept
// in status[1] (the word after the status flags) and named by mone_mem_sync's error text.
enum : int { DS_PHASE_A_TILE = 1, DS_PHASE_B_TILE = 2, DS_READ_TILE = 3, DS_RESIDENT_ROWS = 4,
             DS_TMA_X = 5 };

// Device-resident state of all chains (see mone_mem_init).
struct DevState {
    int C, d_in, d_hid, d_out, n_kv, hd, T, dtype, mode, momentum, renorm, loss;
    int memory, heads;            // MLP (heads 1) or per-head SwiGLU (d_hid = hidden units per head)
    float lr, rms_eps;
    float *W1, *W2, *mu1, *mu2;   // fp32 masters [C][d_hid][d_in|d_out]; mu only with momentum
    bf16 *W1b, *W2b;              // bf16 operand copies (bf16 path)
    float *n1, *n2;               // renormalisation targets [C][d_hid]; -1: row not renormalised
    int col_renorm;               // W2 columns renormalised instead of its rows (output channels)
    float* nc2;                   // [C][d_out] column norms of W2_0 (col_renorm)
    float* colpart;               // [kColRowSlices][C][d_out] partial column sums of squares
    float* sumsq;                 // [2 parity][2 matrix][C][d_hid] row sums of squares
    int* status;                  // device status word
    // test knob (MONE_FAULT_STALL=n at init): the next n tensor-core phase-A launches issue no
    // loads and wait 1 ms, so their bounded waits run out and latch DEV_TIMEOUT
    mutable int fault_stall;
    // SMs the persistent learning kernels leave free while mone_ttl_context_host runs: its
    // host-input gathers take them (one gather CTA an SM, never beside a learning CTA)
    mutable int reserve_sms;
    // meta-parameters (owned copies)
    float *alpha, *gamma, *w_eta, *b_eta, *w_beta, *b_beta, *gate;
    // paper-mode input scratch for a window of win_rows tokens (a multiple of T)
    int win_rows;
    void* U;                      // [C][win_rows][d_in] transformed inputs, dtype of X
    float* eta;                   // [C][win_rows] per-token rates
    float* dbeta;                 // [C][win_rows] w_beta . x_t
    float* zinv;                  // [C][win_rows] 1 / |z_t| (bf16 path: U holds unnormalised z)
    void* dHt;                    // [C][T][d_hid] c_t dH (bf16 or fp32 by path)
    void* Att;                    // [C][T][d_hid] c_t A
    // squared-error loss (bf16 path): the segment's activations with the W2 row scales folded
    // in, and the residual targets y - M(u) that phase A and phase B read in place of K, V
    bf16* Amse;                   // [C][T][d_hid]
    bf16 *Kres, *Vres;            // [C][T][d_out/2]
    float *Kres32, *Vres32;       // the same on the fp32 path
    // read scratch (grown on demand)
    int q_cap;
    float *Uq, *Aq, *Oq;          // [C][q_cap][d_in|d_hid|d_out]
};

// Row slices of the column sums of squares of W2 (output-channel renormalisation).
constexpr int kColRowSlices = 8;

// Elements of the state matrices and rows per chain.  MLP: W1 [d_hid][d_in], W2 [d_hid][d_out].
// SwiGLU: W1 [heads][2 d_hid][dh] (Win; Wg), W2 [heads][d_hid][dh] (Wout), dh = d_in / heads.
inline size_t w1_elems(const DevState& s) {
    return s.memory ? (size_t)s.C * s.heads * 2 * s.d_hid * (s.d_in / s.heads) : (size_t)s.C * s.d_hid * s.d_in;
}
inline size_t w2_elems(const DevState& s) {
    return s.memory ? (size_t)s.C * s.heads * s.d_hid * (s.d_in / s.heads) : (size_t)s.C * s.d_hid * s.d_out;
}
inline size_t w1_rows(const DevState& s) { return s.memory ? (size_t)s.C * s.heads * 2 * s.d_hid : (size_t)s.C * s.d_hid; }
inline size_t w2_rows(const DevState& s) { return s.memory ? (size_t)s.C * s.heads * s.d_hid : (size_t)s.C * s.d_hid; }

inline float* sumsq_ptr(const DevState& s, int parity, int which) {
    return s.sumsq + ((size_t)(parity * 2 + which) * s.C) * s.d_hid;
}

// One segment of work for chains [c0, c0+nc).
struct SegWork {
    int c0, nc;
    const void *X, *K, *V;       // inputs (caller's buffers)
    long long x_cstride, y_cstride;  // element stride between chains in X and in K/V
    long long n_rows;            // rows per chain in the caller's buffers
    long long row0;              // first token row of this segment
    long long u_off;             // row of the segment in the paper-mode input scratch window
    int Tp;                      // tokens present in this segment (<= T)
    const float* eta_in;         // caller per-token rates or null
    long long eta_cstride;
    int parity;                  // segment index parity within the call
    int renorm_pending;          // previous segment's renorm scale still to apply
    float* loss;                 // [C] loss accumulator of this segment or null
    float* step_sq;              // [C] squared norm of this segment's Eq. 8 step, or null
    // per-segment metrics of a whole call: segment i of chain c at [i * mstride + c], or null
    float *loss0, *step0;
    long long mstride;
    int y_scratch;               // targets are the residual scratch (rows from 0), not the caller's K, V
};

// ---- kernels in ttl_prepass.cu
cudaError_t launch_prepass(const DevState& s, const SegWork& w, cudaStream_t st);
// Query transform of the read into U ([C][Q][d_in]: fp32, or bf16 when bf16_out).
cudaError_t launch_query_transform(const DevState& s, const void* Xq, int Q, void* U, bool bf16_out, cudaStream_t st);
// The read's query side on the bf16 path in one pass: Z = SiLU(alpha x + gamma) unnormalised
// (bf16 [C][Q][d_in]) and zinv = 1/|z| per query ([C][Q]) in paper mode; Z = x in plain mode.
cudaError_t launch_query_z(const DevState& s, const void* Xq, int Q, void* Z, float* zinv, cudaStream_t st);

// ---- kernels in ttl_simt.cu (fp32 path, state upkeep, read path)
cudaError_t launch_phase_a_f32(const DevState& s, const SegWork& w, cudaStream_t st);
cudaError_t launch_phase_b_f32(const DevState& s, const SegWork& w, cudaStream_t st);
// Squared-error pre-pass of one segment on the fp32 path (two kernels): M(u) at the segment's
// starting weights, the residual targets y - M(u) into s.Kres32 / s.Vres32, the loss into w.loss.
cudaError_t launch_mse_f32(const DevState& s, const SegWork& w, cudaStream_t st);
// The whole call in one launch per input window, each CTA keeping RB hidden units of one chain
// on chip across the segments (fp32 MLP with the Eq. 7 loss, d_in + d_out <= 512).  Leaves the
// weights renormalised, so no finalize follows.  w: the call's chains, row0 / u_off of the window.
bool resident_f32_fits(const DevState& s);
cudaError_t launch_resident_f32(const DevState& s, const SegWork& w, long long n_tok, cudaStream_t st);
cudaError_t launch_finalize(const DevState& s, int c0, int nc, int parity, int apply_scale, cudaStream_t st);
cudaError_t launch_row_norms(const DevState& s, cudaStream_t st);
// Output-channel renormalisation: every column of W2 of chains [c0, c0 + nc) rescaled to its norm
// in W_0 (fp32 masters and, on the bf16 path, the operand copy).  Two kernels.
cudaError_t launch_col_renorm(const DevState& s, int c0, int nc, cudaStream_t st);
// At init: the column norms of W2_0 into s.nc2, and n2 = -1 (no row renormalisation of W2).
cudaError_t launch_col_targets(const DevState& s, cudaStream_t st);
// At init: gate[i] = SiLU(gate[i]) (from_one: SiLU(1)), n entries.
cudaError_t launch_gate_silu(float* gate, size_t n, int from_one, cudaStream_t st);
cudaError_t launch_read(const DevState& s, int Q, int n_layers, void* K_out, void* V_out,
                        const long long* strides, cudaStream_t st);
cudaError_t launch_zero_f32(float* p, size_t n, cudaStream_t st);

// Allocation-free read (mone_mem_generate_kv_noalloc): fixed device scratch of
// kNoAllocScratchFloats floats, shared by every call on a device.
constexpr size_t kNoAllocScratchFloats = (size_t(16) << 20) / sizeof(float);  // 16 MiB
struct TcMaps;
// tc: the handle's tensor maps on the bf16 path (tensor-core read), null on the fp32 path.
cudaError_t launch_read_noalloc(const DevState& s, const TcMaps* tc, const void* Xq, int Q, int n_layers,
                                void* K_out, void* V_out, const long long* strides, cudaStream_t st);

// ---- kernels in swiglu_tc.cu (per-head SwiGLU memory, bf16 tcgen05 path)
struct SwMaps {
    CUtensorMap Ua, Ub;        // U window as (dh, heads, rows, chains): K-major {64,1,128,1}, MN {64,1,64,1}
    CUtensorMap W1a;           // bf16 W1 as (dh, F, 2, chains*heads), K-major {64,128,1,1}
    CUtensorMap W2a, W2m;      // bf16 W2 (dh, F, chains*heads): K-major {64,128}, MN {64 outputs, 64 hidden}
    CUtensorMap PG, Z;         // phase A outputs, MN-major: (F, 2, T, chains*heads) {64,1,64,1}, (F, T, ..) {64,64}
    CUtensorMap W1s, M1s;      // fp32 W1 / mu1 as (dh, 2F, chains*heads), state chunks {128 cols, 32 rows}
    CUtensorMap W2s, M2s;      // fp32 W2 / mu2 as (dh, F, chains*heads), the same chunks
};
struct SwInputMaps {
    CUtensorMap Xa, Xb;        // caller's X of a group (dh, heads, rows, chains): K-major and MN boxes
    CUtensorMap Ka, Kb, Va, Vb;  // caller's K, V (dh, heads per half, rows, chains)
};
cudaError_t launch_swiglu_phase_a(const DevState& s, const SwMaps& m, const SwInputMaps& in, const SegWork& w,
                                  cudaStream_t st);
cudaError_t launch_swiglu_phase_b(const DevState& s, const SwMaps& m, const SwInputMaps& in, const SegWork& w,
                                  cudaStream_t st);
// Rows of chains [c0, c0 + nc): mode 0: renormalisation targets from W (init); 1: apply the
// pending row scales of `parity`; 2: none.  Every mode rewrites the bf16 operand copies.
cudaError_t launch_swiglu_rows(const DevState& s, int mode, int parity, int c0, int nc, cudaStream_t st);
// The read up to O (fp32, s.Oq): Uq bf16 [C][Q][d_in], Zq bf16 scratch [C*heads][Q][d_hid].
cudaError_t launch_swiglu_read(const DevState& s, const SwMaps& m, const void* Uq, void* Zq, int Q, cudaStream_t st);
// The read's per-head RMS norm and gate from s.Oq into the caller's K / V (ttl_simt.cu).
cudaError_t launch_read_norm(const DevState& s, int Q, int n_layers, void* K_out, void* V_out,
                             const long long* strides, cudaStream_t st);

// ---- kernels in host_stage.cu
// Gather rows [r0, r0 + nr) of every chain of three host tensors ([C][N][row_bytes[t]], device
// addresses of host memory) into device windows ([C][nr][row_bytes[t]]); row_bytes multiples of 16.
cudaError_t launch_stage_rows(const void* const src[3], void* const dst[3], const long long row_bytes[3], long long N,
                              long long r0, long long nr, int C, cudaStream_t st);
// SMs the gather occupies (one CTA on each); the learning kernels leave that many free.
int stage_sms();

// ---- kernels in attention.cu
cudaError_t launch_attention(const DevState& s, int n_layers, const void* Q, int n_q, int Lq, const void* K,
                             const void* V, const long long* strides, int n_mem, void* out, cudaStream_t st);

// ---- kernels in ttl_tc.cu (bf16 tcgen05 path)
struct TcMaps {
    CUtensorMap W1b, W2b;        // K-major boxes {64, 128}
    CUtensorMap dH, At;          // MN-major boxes {64, 64} over [C][T][d_hid]
    CUtensorMap Ua, Ub;          // scratch U: K-major {64,128} and MN {64,64}
    CUtensorMap W1s, W2s, M1s, M2s;  // fp32 state chunks {128 cols, 32 rows}, no swizzle
    CUtensorMap W2m;                 // bf16 W2 copy, MN-major boxes {64 outputs, 64 hidden} (memory read)
    CUtensorMap Amse;                // squared-error activations, K-major {64, 128}
};
struct TcInputMaps {
    CUtensorMap Xa, Xb, Ka, Kb, Va, Vb;  // per call: K-major {64,128} (a) and MN {64,64} (b)
};
cudaError_t launch_phase_a_tc(const DevState& s, const TcMaps& m, const TcInputMaps& in, const SegWork& w,
                              cudaStream_t st);
cudaError_t launch_phase_b_tc(const DevState& s, const TcMaps& m, const TcInputMaps& in, const SegWork& w,
                              cudaStream_t st);
int tc_kernels_per_segment();
// The whole memory read on the tensor cores (bf16 path), query side included: Xq bf16
// [C][Q][d_in]; Uq, Aq bf16 scratch [C][Q][d_in], [C][Q][d_hid]; zq fp32 scratch [C][Q]; writes
// K/V (bf16) with the caller's strides.
cudaError_t launch_read_tc(const DevState& s, const TcMaps& m, const void* Xq, void* Uq, void* Aq, float* zq, int Q,
                           int n_layers, void* K_out, void* V_out, const long long* strides, cudaStream_t st);
// Squared-error pre-pass of one segment (two kernels): M(u) at the segment's starting
// weights and the residual targets y - M(u) into s.Kres / s.Vres (plus the loss into w.loss).
cudaError_t launch_mse_tc(const DevState& s, const TcMaps& m, const TcInputMaps& in, const SegWork& w,
                          cudaStream_t st);

// Tensor-map encoders (driver entry point, resolved at run time).  3-D maps over
// [chains][rows][inner]; bf16 maps use 128-byte swizzle, the *_plain ones none.
bool encode_map_bf16_3d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t rows, uint64_t chains,
                        uint32_t box_inner, uint32_t box_rows);
bool encode_map_plain_3d(CUtensorMap* map, const void* base, bool f32, uint64_t inner, uint64_t rows,
                         uint64_t chains, uint32_t box_inner, uint32_t box_rows);
// 4-D bf16 map, 128-byte swizzle: dims[0] innermost, byte strides of dims 1..3.
bool encode_map_bf16_4d(CUtensorMap* map, const void* base, const uint64_t dims[4], const uint64_t strides[3],
                        const uint32_t box[4]);

}  // namespace mone
