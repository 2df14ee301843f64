// Calibration and selection, one CTA per (request, layer, kv-head):
//   V = E + L + T                (Sec. 4.3, Eqs. 5-11)
//   B~ = max-pool of B over the candidates
//   M = min(rho K, |I|), the M best candidates by B~, lambda =
//       gamma Std(B~) / (Std(V) + eps) over them      (Sec. 4.4, Eqs. 12-15)
//   S = B~ + lambda V                                 (Eq. 16)
//   the K best candidates by S, ascending, then the window (Eq. 17)
// Both "best k" sets use one order: larger value first, equal values ->
// lower position first.  They are found by a 4 x 8-bit radix select on the
// order-preserving float keys, then an index-ordered block scan resolves the
// ties at the threshold and emits the kept positions in ascending order.
#include "common.cuh"

namespace bacon {
namespace {

constexpr int kThreads = 1024;

struct SelectResult {
    uint32_t tau;   // key of the k-th best element
    int need;       // how many elements with key == tau are taken
};

// Block-wide: k-th largest key over vals[0, n) (1 <= k <= n).  Every thread
// returns the same result.
__device__ SelectResult radix_select(const float* vals, int n, int k, int* hist, int* bcast)
{
    uint32_t prefix = 0, mask = 0;
    int remaining = k;
    for (int shift = 24; shift >= 0; shift -= 8) {
        for (int b = threadIdx.x; b < 256; b += blockDim.x) hist[b] = 0;
        __syncthreads();
        // warp-aggregated: lanes that fall into the same bin add once together
        const int n_round = (n + 31) & ~31;
        for (int i = threadIdx.x; i < n_round; i += blockDim.x) {
            const bool in = i < n;
            const uint32_t key = in ? float_key(vals[i]) : 0u;
            const bool hit = in && (key & mask) == prefix;
            const int bin = hit ? (int)((key >> shift) & 255u) : -1;
            const uint32_t peers = __match_any_sync(0xffffffffu, bin);
            if (hit && (threadIdx.x & 31) == __ffs(peers) - 1) atomicAdd(&hist[bin], __popc(peers));
        }
        __syncthreads();
        if (threadIdx.x < 32) {
            // warp 0: bins high to low; find the bin where the running count
            // from the top reaches `remaining`
            const int lane = threadIdx.x;
            int cum = 0, found_bin = -1, found_rem = 0;
            for (int base = 255; base >= 0 && found_bin < 0; base -= 32) {
                const int b = base - lane;
                const int c = hist[b];
                // inclusive scan from the top (lane 0 = highest bin)
                int incl = c;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const int y = __shfl_up_sync(0xffffffffu, incl, o);
                    if (lane >= o) incl += y;
                }
                const bool hit = cum + incl >= remaining;
                const uint32_t ballot = __ballot_sync(0xffffffffu, hit);
                if (ballot) {
                    const int first = __ffs(ballot) - 1;
                    const int excl = __shfl_sync(0xffffffffu, incl - c, first);
                    found_bin = base - first;
                    found_rem = remaining - (cum + excl);
                }
                cum += __shfl_sync(0xffffffffu, incl, 31);
            }
            if (lane == 0) {
                bcast[0] = found_bin;
                bcast[1] = found_rem;
            }
        }
        __syncthreads();
        prefix |= (uint32_t)bcast[0] << shift;
        mask |= 255u << shift;
        remaining = bcast[1];
        __syncthreads();
    }
    return {prefix, remaining};
}

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

// Index-ordered sweeps over vals[0, n): warp w owns the contiguous segment
// [lo, hi) and its lanes take consecutive elements, so shared-memory reads
// are conflict-free while ballots keep the index order inside a warp.
struct Segment {
    int lo, hi;
};

__device__ __forceinline__ Segment warp_segment(int n)
{
    const int nw = blockDim.x >> 5;
    const int per = ((n + nw - 1) / nw + 31) & ~31;
    const int lo = min(n, (int)(threadIdx.x >> 5) * per);
    return {lo, min(n, lo + per)};
}

__device__ __forceinline__ int warp_sum(int v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Exclusive scan of one value per warp (lane 0's `v`), returned to every lane.
__device__ int warp_exclusive_scan(int v, int* warp_sums, int* total)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (lane == 0) warp_sums[warp] = v;
    __syncthreads();
    if (warp == 0) {
        const int nw = blockDim.x >> 5;
        const int w = lane < nw ? warp_sums[lane] : 0;
        int incl = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += y;
        }
        if (lane < nw) warp_sums[lane] = incl - w;
        if (lane == 31) *total = incl;
    }
    __syncthreads();
    const int r = warp_sums[warp];
    __syncthreads();
    return r;
}

// Walks this warp's segment in index order; calls f(i, in) for every index
// with in = membership in the k best (key > tau, or key == tau among the
// first `need` equal keys).  eq_before = equal keys before the segment.
template <typename F>
__device__ __forceinline__ void walk_topk(const float* vals, Segment sg, SelectResult sel,
                                          int eq_before, F f)
{
    const int lane = threadIdx.x & 31;
    const uint32_t lt = (1u << lane) - 1u;
    int running = eq_before;
    for (int base = sg.lo; base < sg.hi; base += 32) {
        const int i = base + lane;
        const bool valid = i < sg.hi;
        const uint32_t key = valid ? float_key(vals[i]) : 0u;
        const bool eq = valid && key == sel.tau;
        const uint32_t ball = __ballot_sync(0xffffffffu, eq);
        const int rank = running + __popc(ball & lt);
        const bool in = valid && (key > sel.tau || (eq && rank < sel.need));
        f(i, valid, in);
        running += __popc(ball);
    }
}

// Equal-to-threshold keys before this warp's segment.
__device__ int eq_before_segment(const float* vals, Segment sg, uint32_t tau, int* warp_sums,
                                 int* total)
{
    int eq = 0;
    for (int i = sg.lo + (threadIdx.x & 31); i < sg.hi; i += 32) eq += float_key(vals[i]) == tau;
    return warp_exclusive_scan(warp_sum(eq), warp_sums, total);
}

__global__ void __launch_bounds__(kThreads)
calibrate_select_kernel(Shape s, Calib c, CalibArgs a)
{
    extern __shared__ __align__(16) float sm[];
    const int N = s.N, W = s.W;
    float* Sb = sm;      // pooled backbone B~, then the final score S
    float* Vs = sm + N;  // calibrated evidence V
    __shared__ int hist[256];
    __shared__ int bcast[4];
    __shared__ int warp_sums[32];
    __shared__ float red[33];
    __shared__ int total_s;

    const int u = blockIdx.x;
    const int pair = u / s.hkv, h = u - pair * s.hkv;
    const int rq = pair / s.layers;
    const int layer = a.layer0 + (pair - rq * s.layers);
    const int win = c.keep_window ? W : 0;
    const int n_cand = N - win;
    const int kept_total = min(a.budget[pair], N);
    const int keep = kept_total - win;

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
        // B -> Vs (staging), then the pooled backbone over the candidates -> Sb
        if ((N & 3) == 0)
            stage(Vs, Bu, N);
        else
            for (int i = threadIdx.x; i < N; i += blockDim.x) Vs[i] = Bu[i];
        __syncthreads();
        for (int i = threadIdx.x; i < N; i += blockDim.x) {
            float mx = 0.f;
            if (i < n_cand) {
                mx = -INFINITY;
                const int lo = max(0, i - half), hi = min(n_cand - 1, i + half);
                for (int v = lo; v <= hi; ++v) mx = fmaxf(mx, Vs[v]);
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
        constexpr int kMaxPer = 24;  // N <= 24576 with 1024 threads
        float vreg[kMaxPer];
        // persistence: mean of E over the preceding min(m, l) layers (Eqs. 8-9)
#pragma unroll
        for (int k = 0; k < kMaxPer; ++k) vreg[k] = 0.f;
        if (c.use_T) {
            for (int j = layer - nprev; j < layer; ++j) {
                const float* Ej = Eof(j);
#pragma unroll
                for (int k = 0; k < kMaxPer; ++k) {
                    const int i = threadIdx.x + k * blockDim.x;
                    if (i < N) vreg[k] += Ej[i];
                }
            }
        }
#pragma unroll
        for (int k = 0; k < kMaxPer; ++k) {
            const int i = threadIdx.x + k * blockDim.x;
            if (i < N) {
                // coherence: truncated radius-r box mean of E (Eqs. 5-7)
                const int lo = max(0, i - c.r), hi = min(N - 1, i + c.r);
                float sum = 0.f;
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
#pragma unroll
        for (int k = 0; k < kMaxPer; ++k) {
            const int i = threadIdx.x + k * blockDim.x;
            if (i < N) Vs[i] = vreg[k];
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
            const SelectResult sel = radix_select(Sb, n_cand, M, hist, bcast);
            const Segment sg = warp_segment(n_cand);
            const int eqb = eq_before_segment(Sb, sg, sel.tau, warp_sums, &total_s);
            float sb = 0.f, sv = 0.f;
            walk_topk(Sb, sg, sel, eqb, [&](int i, bool, bool in) {
                if (in) {
                    sb += Sb[i];
                    sv += Vs[i];
                }
            });
            const float mb = block_sum(sb, red) / (float)M;
            const float mv = block_sum(sv, red) / (float)M;
            float vb = 0.f, vv = 0.f;  // centred second moments (two-pass)
            walk_topk(Sb, sg, sel, eqb, [&](int i, bool, bool in) {
                if (in) {
                    const float db = Sb[i] - mb, dv = Vs[i] - mv;
                    vb = fmaf(db, db, vb);
                    vv = fmaf(dv, dv, vv);
                }
            });
            const float stdb = sqrtf(block_sum(vb, red) / (float)M);
            const float stdv = sqrtf(block_sum(vv, red) / (float)M);
            lam = c.gamma * stdb / (stdv + c.eps);
        }
        if (threadIdx.x == 0) a.lambda[u] = lam;
        for (int i = threadIdx.x; i < n_cand; i += blockDim.x) Sb[i] = fmaf(lam, Vs[i], Sb[i]);
        __syncthreads();
        if (a.write_S)
            for (int i = threadIdx.x; i < N; i += blockDim.x) a.S[(size_t)u * N + i] = Sb[i];
    } else {
        for (int i = threadIdx.x; i < N; i += blockDim.x) Sb[i] = a.S[(size_t)u * N + i];
        __syncthreads();
    }

    if (!a.do_select) return;
    int32_t* out = a.idx[pair] + (size_t)h * kept_total;
    if (keep >= n_cand) {
        for (int i = threadIdx.x; i < n_cand; i += blockDim.x) out[i] = i;
    } else if (keep > 0) {
        const SelectResult sel = radix_select(Sb, n_cand, keep, hist, bcast);
        const Segment sg = warp_segment(n_cand);
        const int eqb = eq_before_segment(Sb, sg, sel.tau, warp_sums, &total_s);
        int mine = 0;
        walk_topk(Sb, sg, sel, eqb, [&](int, bool, bool in) { mine += in; });
        const int base = warp_exclusive_scan(warp_sum(mine), warp_sums, &total_s);
        const int lane = threadIdx.x & 31;
        const uint32_t lt = (1u << lane) - 1u;
        int pos = base;
        walk_topk(Sb, sg, sel, eqb, [&](int i, bool, bool in) {
            const uint32_t ball = __ballot_sync(0xffffffffu, in);
            if (in) out[pos + __popc(ball & lt)] = i;
            pos += __popc(ball);
        });
        if (threadIdx.x == 0 && total_s != keep && a.err) atomicExch(a.err, 2);
    }
    for (int w = threadIdx.x; w < win; w += blockDim.x) out[keep + w] = N - W + w;
}

}  // namespace

size_t calibrate_smem(int N) { return (size_t)2 * N * sizeof(float); }

cudaError_t launch_calibrate_select(const Shape& s, const Calib& c, const CalibArgs& a,
                                    cudaStream_t st)
{
    const size_t sm = calibrate_smem(s.N);
    cudaError_t e = cudaFuncSetAttribute(calibrate_select_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e != cudaSuccess) return e;
    calibrate_select_kernel<<<s.units, kThreads, sm, st>>>(s, c, a);
    return cudaGetLastError();
}

}  // namespace bacon
