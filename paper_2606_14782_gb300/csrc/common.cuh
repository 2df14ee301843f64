// Device helpers and launch interfaces shared by the BACON kernels (sm_103a).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace bacon {

// Upper bound on requests * layers of one call: the per-(request, layer)
// tensor pointers travel as kernel parameters.
constexpr int kMaxPairs = 256;

struct GatherTable {
    const uint16_t* k[kMaxPairs];
    const uint16_t* v[kMaxPairs];
    uint16_t* ko[kMaxPairs];
    uint16_t* vo[kMaxPairs];
    const int32_t* idx[kMaxPairs];  // [Hkv][kept] kept positions of the pair
    int kept[kMaxPairs];             // rows kept per kv-head
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

// 2^x on the special-function unit (ex2.approx, flush-to-zero); 2^-inf = 0.
__device__ __forceinline__ float fast_exp2(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;\n" : "=f"(y) : "f"(x));
    return y;
}

// max(a, b, c) in one instruction.
__device__ __forceinline__ float max3f(float a, float b, float c)
{
    float d;
    asm("max.f32 %0, %1, %2, %3;\n" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}

// Order-preserving map of a float to an unsigned key (larger float ->
// larger key), used by the radix selections, and its inverse.
__device__ __forceinline__ uint32_t float_key(float f)
{
    uint32_t b = __float_as_uint(f);
    return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
__device__ __forceinline__ float key_float(uint32_t k)
{
    return __uint_as_float((k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k);
}

// ----------------------------------------------------------- launchers

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
    int32_t* idx[kMaxPairs];     // per (request, layer): [Hkv][kept] (written when do_select)
    int budget[kMaxPairs];       // kept tokens per head (window included)
    int calib_budget[kMaxPairs]; // budget that sets K in Eq. 12
    long long idx_variant_stride = 0;  // sweep only: elements between variants' indices
    int compute_scores;  // 1: V, B~, lambda, S from B and the residuals
    int do_select;       // 1: top-B selection into idx
    int write_S;
    int* err;
};
cudaError_t launch_calibrate_select(const Shape& s, const Calib& c, const CalibArgs& a,
                                    cudaStream_t st);

// Ablation / sensitivity sweep: every unit under each of `variants`
// hyper-parameter sets (compute_scores and do_select must be 1, write_S 0,
// V and Bp null).
constexpr int kMaxVariants = 32;
struct CalibTable {
    Calib c[kMaxVariants];
};
cudaError_t launch_calibrate_sweep(const Shape& s, const CalibTable& t, int variants,
                                   const CalibArgs& a, cudaStream_t st);

// AdaKV-style selection over the heads of each (request, layer).
struct AdaptArgs {
    const float* S;              // [units][N] final scores (0 off-candidates)
    int budget;                  // average per-head budget (window included)
    int guaranteed;              // g = floor(alpha K) candidates per head first
    int32_t* idx[kMaxPairs];     // per pair: flat [Hkv * kept] positions, heads in order
    int32_t* counts;             // [pairs][Hkv] kept per head (window included)
    int* err;
};
cudaError_t launch_adaptive_select(const Shape& s, int keep_window, const AdaptArgs& a,
                                   cudaStream_t st);
// Dynamic shared memory of the adaptive selection (one byte per candidate).
size_t adaptive_smem(int kv_heads, int n_cand);
// Gather into the flat per-layer layout of the adaptive selection.
cudaError_t launch_gather_flat(const GatherTable& tab, const Shape& s, const int32_t* counts,
                               int* err, cudaStream_t st);

// Gather of the kept K/V rows (kept counts may differ between pairs).
cudaError_t launch_gather(const GatherTable& tab, const Shape& s, int* err, cudaStream_t st);

}  // namespace bacon
