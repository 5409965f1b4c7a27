// Host-input staging, the data path of mone_ttl_context_host: the rows [r0, r0 + nr) of every
// chain of a context held in host memory (X [C][N][d_in], K and V [C][N][d_out / 2]) are
// gathered into a device window ([C][nr][width] per tensor) by SM loads that read the host
// memory directly over the host link (NVLink-C2C on Grace).
//
// Why SM loads and not the copy engines: on this part both top out at the link's read rate
// (211 GB/s measured), but copy-engine transfers fell to 24-50 GB/s for stretches of a
// multi-GB pinned footprint, while SM loads held 211 GB/s on every chunk.
//
// Where the gather runs: on SMs of its own.  A gather CTA sharing an SM with a learning CTA
// slowed the learning far more than the gather's own work (a 128K-token step: 72 ms with 32
// shared SMs, 81-96 ms with 64-152), so the gather's CTAs ask for more shared memory than an
// SM has beside any learning CTA (at least 195 KB), and while mone_ttl_context_host runs the
// persistent learning kernels leave ST_GRID SMs free (DevState::reserve_sms).  8 CTAs of 512
// threads, 8 loads in flight each, reach 210 GB/s alone.
#include <mutex>

#include "mone_common.cuh"

namespace mone {

namespace {

constexpr int ST_THREADS = 512;
constexpr int ST_UNROLL = 8;  // 16-byte loads in flight per thread (64 KB per CTA)
constexpr int ST_GRID = 8;
constexpr int ST_SMEM = 120 * 1024;  // unused: one gather CTA an SM, none beside a learning CTA

struct StageArgs {
    const uint4* src[3];   // host tensors (device addresses) [C][N][row16[t]] in 16-byte units
    uint4* dst[3];         // device windows [C][nr][row16[t]]
    long long row16[3];    // 16-byte units per row
    long long N, r0, nr;
    int C;
};

// One tensor's rows; every index stays below its chain's `per_chain` units on both sides.
__device__ __forceinline__ void stage_tensor(const uint4* src0, uint4* dst0, long long row16, long long N, long long r0,
                                             long long nr, int C) {
    const long long step = (long long)gridDim.x * ST_THREADS * ST_UNROLL;
    const long long per_chain = nr * row16;  // units of one chain's rows: contiguous on both sides
#pragma unroll 1
    for (int c = 0; c < C; ++c) {
        const uint4* src = src0 + ((long long)c * N + r0) * row16;
        uint4* dst = dst0 + (long long)c * per_chain;
#pragma unroll 1
        for (long long i = (long long)blockIdx.x * ST_THREADS * ST_UNROLL + threadIdx.x; i < per_chain; i += step) {
            uint4 v[ST_UNROLL];
#pragma unroll
            for (int u = 0; u < ST_UNROLL; ++u) {
                const long long j = i + (long long)u * ST_THREADS;
                if (j < per_chain) v[u] = __ldcs(src + j);  // host memory, read once
            }
#pragma unroll
            for (int u = 0; u < ST_UNROLL; ++u) {
                const long long j = i + (long long)u * ST_THREADS;
                if (j < per_chain) dst[j] = v[u];
            }
        }
    }
}

__global__ void __launch_bounds__(ST_THREADS, 1) stage_rows_kernel(const StageArgs a) {
    stage_tensor(a.src[0], a.dst[0], a.row16[0], a.N, a.r0, a.nr, a.C);
    stage_tensor(a.src[1], a.dst[1], a.row16[1], a.N, a.r0, a.nr, a.C);
    stage_tensor(a.src[2], a.dst[2], a.row16[2], a.N, a.r0, a.nr, a.C);
}

}  // namespace

cudaError_t launch_stage_rows(const void* const src[3], void* const dst[3], const long long row_bytes[3], long long N,
                              long long r0, long long nr, int C, cudaStream_t st) {
    StageArgs a{};
    for (int t = 0; t < 3; ++t) {
        a.src[t] = static_cast<const uint4*>(src[t]);
        a.dst[t] = static_cast<uint4*>(dst[t]);
        a.row16[t] = row_bytes[t] / 16;
    }
    a.N = N;
    a.r0 = r0;
    a.nr = nr;
    a.C = C;
    static std::mutex mu;
    static bool opted_in[64] = {};  // the shared-memory opt-in belongs to a device
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lk(mu);
    if (!opted_in[dev]) {
        e = cudaFuncSetAttribute(stage_rows_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, ST_SMEM);
        if (e != cudaSuccess) return e;
        opted_in[dev] = true;
    }
    stage_rows_kernel<<<ST_GRID, ST_THREADS, ST_SMEM, st>>>(a);
    return cudaGetLastError();
}

int stage_sms() { return ST_GRID; }

}  // namespace mone
