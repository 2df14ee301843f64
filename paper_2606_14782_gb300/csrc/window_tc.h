// Interface of the tcgen05 window-score kernels (window_tc.cu).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>

#include "common.cuh"

namespace bacon {

// One launch covers every (request, layer, kv-head) unit of a call.
struct TcArgs {
    const CUtensorMap* kmaps;  // [pairs] 2-D maps over each pair's K, [Hkv * N][d]
    const CUtensorMap* qmaps;  // [pairs] 2-D maps over each pair's window queries, [Hq * W][d]
    Shape s;
    int chunks;                // 1024-token chunks per unit
    int total_chunks;          // units * chunks
    float2* partial;           // pass 1 output [units][chunks][rows]
    const float* lse2;         // pass 2 input  [units][rows]
    float* B;                  // pass 2 outputs [units][N]
    float* Q;
    float* E;
    int* err;                  // device error word (timeouts)
    int fault = 0;             // test-only fault injection: 1 = CTA 0 of pass 1 never
                               // issues its first K-tile load (a missing arrival)
};

constexpr int kTcChunkTokens = 1024;

// Largest G * W the tcgen05 kernels take.
int window_tc_max_rows();

// Pass 1 / pass 2 on the tensor cores, and the merge between them.
cudaError_t launch_window_stats_tc(const TcArgs& a, cudaStream_t st);
cudaError_t launch_window_scores_tc(const TcArgs& a, cudaStream_t st);
cudaError_t launch_window_combine(const Shape& s, int chunks, const float2* partial, float* lse2,
                                  cudaStream_t st);

// One pass over K for units whose logits fit in tensor memory (at most 32
// window rows and 1024 tokens): B, Q and E as the two passes give them,
// without the partial statistics or the merge.
bool window_onepass_fits(const Shape& s);
cudaError_t launch_window_onepass(const TcArgs& a, cudaStream_t st);

// Per (request, layer) natural-log softmax normalisers of the window rows,
// [Hq][W] fp32, as a prefill attention kernel produces them.
struct LseTable {
    const float* lse[kMaxPairs];
};
cudaError_t launch_lse_from_prefill(const Shape& s, const LseTable& t, float* lse2,
                                    cudaStream_t st);

// 2-D tensor map over `rows` rows of d bf16 values at `base`: boxes of
// 64 columns x box_rows rows, 128-byte swizzle, zero fill out of bounds.
bool encode_rows_map(CUtensorMap* out, const void* base, int d, long long rows, int box_rows);

// Box heights of the K maps (one 128-token tile) and window-query maps.
constexpr int kTcKBoxRows = 128;
constexpr int kTcQBoxRows = 64;

}  // namespace bacon
