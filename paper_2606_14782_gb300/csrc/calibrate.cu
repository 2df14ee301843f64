// Calibration and selection, one CTA per (request, layer, kv-head):
//   V = E + L + T                (Sec. 4.3, Eqs. 5-11)
//   B~ = max-pool of B over the candidates
//   M = min(rho K, |I|), the M best candidates by B~, lambda =
//       gamma Std(B~) / (Std(V) + eps) over them      (Sec. 4.4, Eqs. 12-15)
//   S = B~ + lambda V                                 (Eq. 16)
//   the K best candidates by S, ascending, then the window (Eq. 17)
// Both "best k" sets use one order: larger value first, equal values ->
// lower position first (select.cuh: range-adaptive radix select, then
// index-ordered warp-segmented sweeps that resolve ties and emit ascending
// positions).  The two standard deviations come from one sweep that sums
// moments about fixed shifts in fp32 (the shifts keep the differences
// small, so no precision is lost to cancellation).
#include "common.cuh"
#include "select.cuh"

namespace bacon {
namespace {

using namespace sel;

// Threads per CTA and tokens per thread depend on the prompt length only
// (so that every call on the same shape reduces in the same order and gives
// the same bits): 256 threads of up to 8 tokens up to 2048 tokens, where
// several CTAs share an SM; 1024 threads of up to 16 tokens up to 16384
// tokens; 1024 threads of up to kMaxPer tokens above.
constexpr int kMaxPer = 24;
constexpr int kSmallPrompt = 2048;
constexpr int kMidPrompt = 16384;  // 1024 threads x 16 tokens

// Block-wide fp32 sum by a shuffle tree (pairwise, so the rounding error
// grows with log2 of the count).  FP64 is avoided: its rate on this part is
// a small fraction of fp32.
__device__ float block_sum(float v, float* red)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if (lane == 0) red[warp] = v;
    __syncthreads();
    if (warp == 0) {
        float t = lane < (int)(blockDim.x >> 5) ? red[lane] : 0.f;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
        if (lane == 0) red[32] = t;
    }
    __syncthreads();
    const float tot = red[32];
    __syncthreads();
    return tot;
}

// Four block-wide fp32 sums in one round (red holds 4 x 33 floats).
__device__ float4 block_sum4(float4 v, float* red)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        v.x += __shfl_xor_sync(0xffffffffu, v.x, o);
        v.y += __shfl_xor_sync(0xffffffffu, v.y, o);
        v.z += __shfl_xor_sync(0xffffffffu, v.z, o);
        v.w += __shfl_xor_sync(0xffffffffu, v.w, o);
    }
    if (lane == 0) {
        red[warp] = v.x;
        red[33 + warp] = v.y;
        red[66 + warp] = v.z;
        red[99 + warp] = v.w;
    }
    __syncthreads();
    if (warp < 4) {
        const int nw = (int)(blockDim.x >> 5);
        float t = lane < nw ? red[33 * warp + lane] : 0.f;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
        if (lane == 0) red[33 * warp + 32] = t;
    }
    __syncthreads();
    const float4 tot = make_float4(red[32], red[65], red[98], red[131]);
    __syncthreads();
    return tot;
}

// Ask L2 to fetch the n floats at p (one prefetch per 128-byte line, every
// address inside the array), so that later loads of them hit L2.
__device__ __forceinline__ void prefetch_l2(const float* p, int n)
{
    for (int i = (int)threadIdx.x * 32; i < n; i += (int)blockDim.x * 32)
        asm volatile("prefetch.global.L2 [%0];" ::"l"(p + i));
}

// dst[0, n) = src[0, n) with independent 16-byte loads (n % 4 == 0 and both
// 16-byte aligned), so the copy costs a few memory round trips, not one per
// element.
__device__ __forceinline__ void stage(float* dst, const float* src, int n)
{
    const float4* s4 = reinterpret_cast<const float4*>(src);
    float4* d4 = reinterpret_cast<float4*>(dst);
    const int n4 = n >> 2;
    for (int i = threadIdx.x; i < n4; i += 4 * blockDim.x) {
        float4 v[4];
#pragma unroll
        for (int k = 0; k < 4; ++k)
            if (i + k * (int)blockDim.x < n4) v[k] = __ldg(s4 + i + k * blockDim.x);
#pragma unroll
        for (int k = 0; k < 4; ++k)
            if (i + k * (int)blockDim.x < n4) d4[i + k * blockDim.x] = v[k];
    }
}

// One unit (request, layer, kv-head) u under hyper-parameters c.  lam_out
// (may be null) receives lambda; idx_pair is the pair's [Hkv][kept] output.
// PER bounds the tokens per thread (N <= PER blockDim.x).
template <int PER>
__device__ __forceinline__ void calibrate_unit(const Shape& s, const Calib& c, const CalibArgs& a,
                                               int u, float* lam_out, int32_t* idx_pair)
{
    extern __shared__ __align__(16) float sm[];
    const int N = s.N, W = s.W;
    float* Sb = sm;      // pooled backbone B~, then the final score S
    float* Vs = sm + N;  // calibrated evidence V
    __shared__ int hist[kSelHist];
    __shared__ int bcast[8];
    __shared__ int warp_sums[32];
    __shared__ float red[4 * 33];
    __shared__ int total_s;

    const int pair = u / s.hkv, h = u - pair * s.hkv;
    const int rq = pair / s.layers;
    const int layer = a.layer0 + (pair - rq * s.layers);
    const int win = c.keep_window ? W : 0;
    const int n_cand = N - win;
    const int kept_total = min(a.budget[pair], N);
    const int keep = kept_total - win;

    uint32_t skmin = 0xffffffffu, skmax = 0u;  // key range of S over the candidates
    auto Eof = [&](int j) -> const float* {
        return a.Ering + (long long)rq * a.ring_req_stride +
               (long long)(j % a.ring) * s.hkv * N + (long long)h * N;
    };

    if (a.compute_scores) {
        const float* Bu = a.B + (size_t)u * N;
        const float* Ec = Eof(layer);
        const int half = c.pool / 2;
        const int nprev = min(c.m, layer);
        const float inv_prev = nprev > 0 ? 1.f / (float)nprev : 0.f;
        // the residuals of this layer and of the preceding ones are read
        // only after the pooling: start bringing them into L2 now
        prefetch_l2(Ec, N);
        if (c.use_T)
            for (int j = layer - nprev; j < layer; ++j) prefetch_l2(Eof(j), N);
        // B -> Vs (staging), then the pooled backbone over the candidates -> Sb
        if ((N & 3) == 0)
            stage(Vs, Bu, N);
        else
            for (int i = threadIdx.x; i < N; i += blockDim.x) Vs[i] = Bu[i];
        __syncthreads();
        uint32_t kmin = 0xffffffffu, kmax = 0u;  // key range of B~ over the candidates
        for (int i = threadIdx.x; i < N; i += blockDim.x) {
            float mx = 0.f;
            if (i < n_cand) {
                mx = -INFINITY;
                const int lo = max(0, i - half), hi = min(n_cand - 1, i + half);
#pragma unroll 4
                for (int v = lo; v <= hi; ++v) mx = fmaxf(mx, Vs[v]);
                kmin = min(kmin, float_key(mx));
                kmax = max(kmax, float_key(mx));
            }
            Sb[i] = mx;
        }
        __syncthreads();
        // E -> Vs (staging); V is built in registers, then written over it
        if ((N & 3) == 0)
            stage(Vs, Ec, N);
        else
            for (int i = threadIdx.x; i < N; i += blockDim.x) Vs[i] = Ec[i];
        __syncthreads();
        float vreg[PER];
        // persistence: mean of E over the preceding min(m, l) layers (Eqs. 8-9)
#pragma unroll
        for (int k = 0; k < PER; ++k) vreg[k] = 0.f;
        if (c.use_T) {
            for (int j = layer - nprev; j < layer; ++j) {
                const float* Ej = Eof(j);
                // every load in flight at once: indices past the end are
                // clamped to the last token (in bounds) and their values
                // dropped
                float x[PER];
#pragma unroll
                for (int k = 0; k < PER; ++k) x[k] = Ej[min((int)threadIdx.x + k * (int)blockDim.x, N - 1)];
#pragma unroll
                for (int k = 0; k < PER; ++k)
                    if ((int)threadIdx.x + k * (int)blockDim.x < N) vreg[k] += x[k];
            }
        }
#pragma unroll
        for (int k = 0; k < PER; ++k) {
            const int i = threadIdx.x + k * blockDim.x;
            if (i < N) {
                // coherence: truncated radius-r box mean of E (Eqs. 5-7)
                const int lo = max(0, i - c.r), hi = min(N - 1, i + c.r);
                float sum = 0.f;
#pragma unroll 4
                for (int v = lo; v <= hi; ++v) sum += Vs[v];
                const float L = sum / (float)(hi - lo + 1);
                float V = 0.f;
                if (c.use_E) V += Vs[i];
                if (c.use_L) V += L;
                if (c.use_T) V += vreg[k] * inv_prev;
                vreg[k] = V;
            }
        }
        __syncthreads();
        float vsum = 0.f;  // over the candidates: the shift of the moments below
#pragma unroll
        for (int k = 0; k < PER; ++k) {
            const int i = threadIdx.x + k * blockDim.x;
            if (i < N) Vs[i] = vreg[k];
            if (i < n_cand) vsum += vreg[k];
        }
        __syncthreads();
        if (a.V) for (int i = threadIdx.x; i < N; i += blockDim.x) a.V[(size_t)u * N + i] = Vs[i];
        if (a.Bp) for (int i = threadIdx.x; i < N; i += blockDim.x) a.Bp[(size_t)u * N + i] = Sb[i];

        // Eqs. 12-15
        const int calib_keep = min(a.calib_budget[pair], N) - win;
        const long long Ml = (long long)c.rho * (long long)(calib_keep > 0 ? calib_keep : 0);
        const int M = (int)(Ml < n_cand ? Ml : n_cand);
        float lam = 0.f;
        if (M > 0) {
            const SelectResult sel =
                radix_select_range(n_cand, M, FloatKeys{Sb}, hist, bcast, kmin, kmax);
            const Segment sg = warp_segment(n_cand);
            const int eqb = eq_before_segment(Sb, sg, sel, warp_sums, &total_s);
            // moments about fixed shifts in one walk: B~ about its M-th value,
            // V about its mean over the candidates (both near the members'
            // means, so the fp32 differences keep their precision)
            const float pb = key_float(sel.tau);
            const float pv = block_sum(vsum, red) / (float)n_cand;
            float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
            walk_topk(Sb, sg, sel, eqb, [&](int i, bool, bool in) {
                if (in) {
                    const float db = Sb[i] - pb, dv = Vs[i] - pv;
                    acc.x += db;
                    acc.y = fmaf(db, db, acc.y);
                    acc.z += dv;
                    acc.w = fmaf(dv, dv, acc.w);
                }
            });
            const float4 tot = block_sum4(acc, red);
            const float inv_m = 1.f / (float)M;
            const float mb = tot.x * inv_m, mv = tot.z * inv_m;
            const float stdb = sqrtf(fmaxf(tot.y * inv_m - mb * mb, 0.f));
            const float stdv = sqrtf(fmaxf(tot.w * inv_m - mv * mv, 0.f));
            lam = c.gamma * stdb / (stdv + c.eps);
        }
        if (threadIdx.x == 0 && lam_out) *lam_out = lam;
        kmin = 0xffffffffu;
        kmax = 0u;
        for (int i = threadIdx.x; i < n_cand; i += blockDim.x) {
            const float sv = fmaf(lam, Vs[i], Sb[i]);
            Sb[i] = sv;
            kmin = min(kmin, float_key(sv));
            kmax = max(kmax, float_key(sv));
        }
        skmin = kmin;
        skmax = kmax;
        __syncthreads();
        if (a.write_S)
            for (int i = threadIdx.x; i < N; i += blockDim.x) a.S[(size_t)u * N + i] = Sb[i];
    } else {
        for (int i = threadIdx.x; i < N; i += blockDim.x) Sb[i] = a.S[(size_t)u * N + i];
        __syncthreads();
    }

    if (!a.do_select) return;
    if (!a.compute_scores)
        for (int i = threadIdx.x; i < n_cand; i += blockDim.x) {
            skmin = min(skmin, float_key(Sb[i]));
            skmax = max(skmax, float_key(Sb[i]));
        }
    int32_t* out = idx_pair + (size_t)h * kept_total;
    if (keep >= n_cand) {
        for (int i = threadIdx.x; i < n_cand; i += blockDim.x) out[i] = i;
    } else if (keep > 0) {
        const SelectResult sel =
            radix_select_range(n_cand, keep, FloatKeys{Sb}, hist, bcast, skmin, skmax);
        const Segment sg = warp_segment(n_cand);
        const int eqb = eq_before_segment(Sb, sg, sel, warp_sums, &total_s);
        const int lane = threadIdx.x & 31;
        const uint32_t lt = (1u << lane) - 1u;
        if constexpr (PER <= 16) {
            // membership ballots kept in registers for the emitting pass (a
            // warp segment is at most PER x 32 candidates: N <= PER blockDim)
            uint32_t masks[PER];
            const int mine = walk_topk_masks_by<PER>(sg, sel, eqb, FloatKeys{Sb}, masks);
            int pos = warp_exclusive_scan(mine, warp_sums, &total_s);
#pragma unroll
            for (int st = 0; st < PER; ++st) {
                const uint32_t m = masks[st];
                if ((m >> lane) & 1u) out[pos + __popc(m & lt)] = sg.lo + 32 * st + lane;
                pos += __popc(m);
            }
        } else {
            // longest prompts: no registers to spare, the keys are walked twice
            int mine = 0;
            walk_topk(Sb, sg, sel, eqb, [&](int, bool, bool in) { mine += in; });
            int pos = warp_exclusive_scan(warp_sum(mine), warp_sums, &total_s);
            walk_topk(Sb, sg, sel, eqb, [&](int i, bool, bool in) {
                const uint32_t ball = __ballot_sync(0xffffffffu, in);
                if (in) out[pos + __popc(ball & lt)] = i;
                pos += __popc(ball);
            });
        }
        if (threadIdx.x == 0 && total_s != keep && a.err) atomicCAS(a.err, 0, 2);
    }
    for (int w = threadIdx.x; w < win; w += blockDim.x) out[keep + w] = N - W + w;
}

template <int T, int PER>
__global__ void __launch_bounds__(T, 1024 / T)
calibrate_select_kernel(Shape s, Calib c, CalibArgs a)
{
    const int u = blockIdx.x;
    calibrate_unit<PER>(s, c, a, u, a.lambda + u, a.idx[u / s.hkv]);
}

// Several hyper-parameter sets over the same B and residuals: CTA (u, v)
// runs unit u under variant v; variant v's indices start v *
// idx_variant_stride elements after the single-variant layout and its
// lambdas v * units after a.lambda.
template <int T, int PER>
__global__ void __launch_bounds__(T, 1024 / T)
calibrate_sweep_kernel(Shape s, CalibTable t, CalibArgs a)
{
    const int u = blockIdx.x, v = blockIdx.y;
    float* lam = a.lambda ? a.lambda + (size_t)v * s.units + u : nullptr;
    calibrate_unit<PER>(s, t.c[v], a, u, lam, a.idx[u / s.hkv] + (size_t)v * a.idx_variant_stride);
}

}  // namespace

size_t calibrate_smem(int N) { return (size_t)2 * N * sizeof(float); }

namespace {

template <int T, int PER>
cudaError_t launch_select_t(const Shape& s, const Calib& c, const CalibArgs& a, cudaStream_t st)
{
    const size_t sm = calibrate_smem(s.N);
    cudaError_t e = cudaFuncSetAttribute(calibrate_select_kernel<T, PER>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e != cudaSuccess) return e;
    calibrate_select_kernel<T, PER><<<s.units, T, sm, st>>>(s, c, a);
    return cudaGetLastError();
}

template <int T, int PER>
cudaError_t launch_sweep_t(const Shape& s, const CalibTable& t, int variants, const CalibArgs& a,
                           cudaStream_t st)
{
    const size_t sm = calibrate_smem(s.N);
    cudaError_t e = cudaFuncSetAttribute(calibrate_sweep_kernel<T, PER>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e != cudaSuccess) return e;
    calibrate_sweep_kernel<T, PER><<<dim3(s.units, variants), T, sm, st>>>(s, t, a);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_calibrate_select(const Shape& s, const Calib& c, const CalibArgs& a,
                                    cudaStream_t st)
{
    if (s.N <= kSmallPrompt) return launch_select_t<256, kSmallPrompt / 256>(s, c, a, st);
    if (s.N <= kMidPrompt) return launch_select_t<1024, kMidPrompt / 1024>(s, c, a, st);
    return launch_select_t<1024, kMaxPer>(s, c, a, st);
}

cudaError_t launch_calibrate_sweep(const Shape& s, const CalibTable& t, int variants,
                                   const CalibArgs& a, cudaStream_t st)
{
    if (s.N <= kSmallPrompt) return launch_sweep_t<256, kSmallPrompt / 256>(s, t, variants, a, st);
    if (s.N <= kMidPrompt) return launch_sweep_t<1024, kMidPrompt / 1024>(s, t, variants, a, st);
    return launch_sweep_t<1024, kMaxPer>(s, t, variants, a, st);
}

}  // namespace bacon
