// Window scores of one layer without any device allocation.
//
// Some callers cannot call cudaMalloc: a serving engine that reserves all of
// HBM for its KV cache up front and forbids side allocations, or code that
// must not pay the implicit device-wide synchronisation of cudaMalloc /
// cudaFree in the middle of prefill.  For them, bacon_window_scores_noalloc
// runs the same three window kernels as the context-based calls, but keeps
// their scratch (pass-1 partial statistics, the per-row normalisers and the
// two TMA descriptors) in one file-scope __device__ array instead of
// context-owned buffers.
//
// The call returns before its kernels run, so a device-side failure (a
// bounded pipeline wait that ran out) cannot come back as its status.  The
// same array holds an error word for that: each call clears it, the window
// kernels latch a timeout in it, and a last small kernel fills B, Q and E
// with NaN when it is set, so that a caller never reads partial scores as
// valid ones.
#include <atomic>
#include <cstdlib>
#include <cstring>
#include <mutex>

#include "bacon.h"
#include "common.cuh"
#include "window_tc.h"

using namespace bacon;

namespace {

constexpr int kMaxTotalRows = 4096;   // kv_heads * (q_heads / kv_heads) * window
constexpr int kMaxSeq = 16384;        // tokens per call
constexpr int kChunk = 1024;          // pass-1 token chunk, as in the context path
constexpr int kMaxChunks = kMaxSeq / kChunk;
constexpr int kMaxDevices = 64;

constexpr int kMapBytes = 2 * sizeof(CUtensorMap);  // K map, window-query map
constexpr int kErrSlots = 2;                        // 16 bytes holding the error word

// [units][chunks][rows] partial (max, sum) pairs, then [units][rows] fp32
// normalisers packed two per float2, then the two 128-byte TMA descriptors,
// then the device error word.  About 528 KiB, held by every GPU that loads
// the library until the process exits.
static __device__ __align__(256) float2
    g_scratch[kMaxTotalRows * kMaxChunks + kMaxTotalRows / 2 + kMapBytes / sizeof(float2) +
              kErrSlots];

std::mutex g_setup_mutex;
void* g_scratch_addr[kMaxDevices] = {};

// Test-only fault injection: when BACON_FAULT=missing_arrival is set at the
// first call of the process, that call's pass 1 withholds one K-tile load,
// so its bounded waits run out (nothing faults).  -1 = not read yet.
std::atomic<int> g_fault_pending{-1};

int take_fault()
{
    int s = g_fault_pending.load();
    if (s < 0) {
        const char* f = std::getenv("BACON_FAULT");
        g_fault_pending.compare_exchange_strong(s, (f && std::strcmp(f, "missing_arrival") == 0) ? 1 : 0);
    }
    int one = 1;
    return g_fault_pending.compare_exchange_strong(one, 0) ? 1 : 0;
}

// B, Q and E become NaN when a window kernel of this call latched an error.
__global__ void poison_on_error_kernel(const int* err, float* B, float* Q, float* E, size_t n)
{
    if (*reinterpret_cast<const volatile int*>(err) == 0) return;
    const float nan = __int_as_float(0x7fc00000);
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (size_t)gridDim.x * blockDim.x) {
        B[i] = nan;
        Q[i] = nan;
        E[i] = nan;
    }
}

}  // namespace

extern "C" {

bacon_status bacon_window_scores_noalloc(int kv_heads, int q_heads, int head_dim, int window,
                                         const void* q_win, const void* k, int seq_len,
                                         float* B_out, float* Q_out, float* E_out,
                                         bacon_stream stream)
{
    // malformed arguments
    if (kv_heads < 1 || q_heads < 1 || q_heads % kv_heads) return BACON_EINVAL;
    if (head_dim != 64 && head_dim != 128) return BACON_EINVAL;
    if (window < 1 || seq_len < window) return BACON_EINVAL;
    const void* ps[] = {q_win, k, B_out, Q_out, E_out};
    for (const void* p : ps)
        if (!p || (reinterpret_cast<uintptr_t>(p) & 15u)) return BACON_EINVAL;
    // sizes beyond what the static scratch (or the kernels) can hold
    const long long rows = (long long)(q_heads / kv_heads) * window;
    if (seq_len > kMaxSeq || rows * kv_heads > kMaxTotalRows || rows > window_tc_max_rows())
        return BACON_EUNSUPPORTED;

    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return BACON_ECUDA;
    float2* scratch = nullptr;
    {
        // one-time set-up per device, with that device current: the host-side
        // name of the array is not a device address, so look the address up
        std::lock_guard<std::mutex> lock(g_setup_mutex);
        if (!g_scratch_addr[dev]) {
            void* addr = nullptr;
            cudaError_t e = cudaGetSymbolAddress(&addr, g_scratch);
            if (e != cudaSuccess || !addr) return BACON_ECUDA;
            g_scratch_addr[dev] = addr;
        }
        scratch = static_cast<float2*>(g_scratch_addr[dev]);
    }

    Shape s;
    s.layers = 1;
    s.hkv = kv_heads;
    s.group = q_heads / kv_heads;
    s.d = head_dim;
    s.W = window;
    s.N = seq_len;
    s.units = kv_heads;
    s.rows = (int)rows;
    const int chunks = (seq_len + kChunk - 1) / kChunk;
    float2* partial = scratch;
    float* lse2 = reinterpret_cast<float*>(scratch + (size_t)kMaxTotalRows * kMaxChunks);
    CUtensorMap* maps =
        reinterpret_cast<CUtensorMap*>(scratch + (size_t)kMaxTotalRows * kMaxChunks + kMaxTotalRows / 2);
    int* err = reinterpret_cast<int*>(scratch + (size_t)kMaxTotalRows * kMaxChunks +
                                      kMaxTotalRows / 2 + kMapBytes / sizeof(float2));
    // descriptors are encoded on the host and copied from this stack buffer;
    // a copy from pageable memory is staged before cudaMemcpyAsync returns
    alignas(64) CUtensorMap host_maps[2];
    if (!encode_rows_map(&host_maps[0], k, head_dim, (long long)kv_heads * seq_len, kTcKBoxRows) ||
        !encode_rows_map(&host_maps[1], q_win, head_dim, (long long)q_heads * window, kTcQBoxRows))
        return BACON_ECUDA;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (cudaMemcpyAsync(maps, host_maps, sizeof host_maps, cudaMemcpyHostToDevice, st) != cudaSuccess)
        return BACON_ECUDA;
    // the error word must start at zero for this call
    if (cudaMemsetAsync(err, 0, sizeof(int), st) != cudaSuccess) return BACON_ECUDA;
    TcArgs a;
    a.kmaps = maps;
    a.qmaps = maps + 1;
    a.s = s;
    a.chunks = chunks;
    a.total_chunks = s.units * chunks;
    a.partial = partial;
    a.lse2 = lse2;
    a.B = B_out;
    a.Q = Q_out;
    a.E = E_out;
    a.err = err;
    TcArgs a1 = a;
    a1.fault = take_fault();
    cudaError_t e = launch_window_stats_tc(a1, st);
    if (e == cudaSuccess) e = launch_window_combine(s, chunks, partial, lse2, st);
    if (e == cudaSuccess) e = launch_window_scores_tc(a, st);
    if (e == cudaSuccess) {
        const size_t n = (size_t)kv_heads * seq_len;
        const size_t blocks = (n + 255) / 256;
        poison_on_error_kernel<<<(unsigned)(blocks < 1024 ? blocks : 1024), 256, 0, st>>>(
            err, B_out, Q_out, E_out, n);
        e = cudaGetLastError();
    }
    return e == cudaSuccess ? BACON_OK : BACON_ECUDA;
}

}  // extern "C"
