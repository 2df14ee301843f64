// Device helpers and launch interfaces shared by the BACON kernels (sm_103a).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace bacon {

// Upper bound on requests * layers of one call: the per-(request, layer)
// tensor pointers travel as kernel parameters.
constexpr int kMaxPairs = 256;

struct QKTable {
    const uint16_t* q[kMaxPairs];  // bf16 [Hq][W][d]
    const uint16_t* k[kMaxPairs];  // bf16 [Hkv][N][d]
};

struct GatherTable {
    const uint16_t* k[kMaxPairs];
    const uint16_t* v[kMaxPairs];
    uint16_t* ko[kMaxPairs];
    uint16_t* vo[kMaxPairs];
};

// Geometry of one call.  A "unit" is one (request, layer, kv-head); units
// are numbered ((request * layers) + layer) * kv_heads + head and the
// per-(request, layer) pointer index is unit / kv_heads.
struct Shape {
    int layers, hkv, group, d, W, N;
    int units;  // requests * layers * hkv
    int rows;   // group * W window rows per kv-head
};

// Calibration hyper-parameters (Sections 4.3-4.4).
struct Calib {
    int r, m, rho;
    float gamma, eps;
    int use_E, use_L, use_T;
    int keep_window;
    int pool;
};

// ---------------------------------------------------------------- PTX

__device__ __forceinline__ uint32_t smem_u32(const void* p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// 16-byte global -> shared copy; src_bytes = 0 fills the destination with 0.
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, int src_bytes)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src),
                 "r"(src_bytes));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N)); }

__device__ __forceinline__ void ldmatrix_x4(uint32_t addr, uint32_t& r0, uint32_t& r1,
                                            uint32_t& r2, uint32_t& r3)
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

// D = A * B + D, m16n8k16, bf16 inputs, fp32 accumulators.
__device__ __forceinline__ void mma_bf16(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1)
{
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
        "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// 2^x on the special-function unit (ex2.approx, flush-to-zero); 2^-inf = 0.
__device__ __forceinline__ float fast_exp2(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;\n" : "=f"(y) : "f"(x));
    return y;
}

// Order-preserving map of a float to an unsigned key (larger float ->
// larger key), used by the radix selections.
__device__ __forceinline__ uint32_t float_key(float f)
{
    uint32_t b = __float_as_uint(f);
    return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// ----------------------------------------------------------- launchers

// Pass 1 of the window softmax: per (unit, token chunk, window row) the
// running max and sum of 2^(logit * log2e / sqrt(d)).
cudaError_t launch_window_stats(const QKTable& tab, const Shape& s, int chunk_tokens,
                                float2* partial, cudaStream_t st);
// Per (unit, row) log2 of the softmax normaliser times G*W.
cudaError_t launch_window_combine(const Shape& s, int chunks, const float2* partial,
                                  float* lse2, cudaStream_t st);
// Pass 2: B, Q and E per token (Eqs. 1, 2, 4).
cudaError_t launch_window_scores(const QKTable& tab, const Shape& s, const float* lse2,
                                 float* B, float* Q, float* E, cudaStream_t st);

// Calibration + selection per unit (Eqs. 5-17).  The residual of layer j of
// request rq, kv-head h is read from
//     Ering + rq * ring_req_stride + (j % ring) * hkv * N + h * N,
// which covers both the whole-step path (ring = layers: every layer kept)
// and the layer-by-layer path (ring = m + 1 slots per request).  The
// absolute layer of unit u is layer0 + (u / hkv) % layers.
struct CalibArgs {
    const float* B;      // [units][N] window score
    const float* Ering;  // residual store (see above)
    int ring;
    long long ring_req_stride;
    int layer0;
    float* S;            // [units][N] final score (written when write_S)
    float* V;            // optional [units][N]
    float* Bp;           // optional [units][N]
    float* lambda;       // [units]
    int32_t* idx;        // [units][kept] (written when do_select)
    int budget;          // kept tokens per head (window included)
    int calib_budget;    // budget that sets K in Eq. 12
    int compute_scores;  // 1: V, B~, lambda, S from B and the residuals
    int do_select;       // 1: top-B selection into idx
    int write_S;
    int* err;
};
cudaError_t launch_calibrate_select(const Shape& s, const Calib& c, const CalibArgs& a,
                                    cudaStream_t st);

// Largest supported G*W for head dimension d (pass-2 shared memory).
int window_max_rows(int d);
// Dynamic shared memory of the calibration kernel for N tokens.
size_t calibrate_smem(int N);

// Gather of the kept K/V rows.
cudaError_t launch_gather(const GatherTable& tab, const Shape& s, const int32_t* idx, int kept,
                          int* err, cudaStream_t st);

}  // namespace bacon
