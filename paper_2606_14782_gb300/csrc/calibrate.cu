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
        for (int i = threadIdx.x; i < n; i += blockDim.x) {
            const uint32_t key = float_key(vals[i]);
            if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1);
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

// Block-wide exclusive scan of one int per thread; returns the exclusive
// prefix and writes the total to *total.
__device__ int block_exclusive_scan(int v, int* warp_sums, int* total)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
    }
    if (lane == 31) warp_sums[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        const int nw = blockDim.x >> 5;
        int w = lane < nw ? warp_sums[lane] : 0;
        int wi = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, wi, o);
            if (lane >= o) wi += y;
        }
        if (lane < nw) warp_sums[lane] = wi - w;
        if (lane == 31) *total = wi;
    }
    __syncthreads();
    const int res = warp_sums[warp] + incl - v;
    __syncthreads();
    return res;
}

// Block-wide double sum.
__device__ double block_sum(double v, double* red)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if (lane == 0) red[warp] = v;
    __syncthreads();
    double tot = 0.0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) tot += red[w];
    __syncthreads();
    return tot;
}

// Membership in the k best of vals[0, n): key > tau, or key == tau with fewer
// than `need` equal keys before it.  Each thread owns the contiguous index
// range [lo, hi); `eq_before` is the number of equal keys before lo.
struct RangeSel {
    int lo, hi;
};

__device__ __forceinline__ RangeSel my_range(int n)
{
    const int per = (n + blockDim.x - 1) / blockDim.x;
    const int lo = min(n, (int)threadIdx.x * per);
    return {lo, min(n, lo + per)};
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
    __shared__ double red[32];
    __shared__ int total_s;

    const int u = blockIdx.x;
    const int pair = u / s.hkv, h = u - pair * s.hkv;
    const int rq = pair / s.layers;
    const int layer = a.layer0 + (pair - rq * s.layers);
    const int win = c.keep_window ? W : 0;
    const int n_cand = N - win;
    const int kept_total = min(a.budget, N);
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
        for (int i = threadIdx.x; i < N; i += blockDim.x) {
            // pooled backbone over the candidates (positions outside ignored)
            if (i < n_cand) {
                float mx = -INFINITY;
                const int lo = max(0, i - half), hi = min(n_cand - 1, i + half);
                for (int v = lo; v <= hi; ++v) mx = fmaxf(mx, Bu[v]);
                Sb[i] = mx;
            } else {
                Sb[i] = 0.f;
            }
            // coherence: truncated radius-r box mean of E (Eqs. 5-7)
            const int lo = max(0, i - c.r), hi = min(N - 1, i + c.r);
            float sum = 0.f;
            for (int v = lo; v <= hi; ++v) sum += Ec[v];
            const float L = sum / (float)(hi - lo + 1);
            // persistence: mean of E over the preceding min(m, l) layers (Eqs. 8-9)
            float T = 0.f;
            for (int j = layer - nprev; j < layer; ++j) T += Eof(j)[i];
            T *= inv_prev;
            float V = 0.f;
            if (c.use_E) V += Ec[i];
            if (c.use_L) V += L;
            if (c.use_T) V += T;
            Vs[i] = V;
        }
        __syncthreads();
        if (a.V) for (int i = threadIdx.x; i < N; i += blockDim.x) a.V[(size_t)u * N + i] = Vs[i];
        if (a.Bp) for (int i = threadIdx.x; i < N; i += blockDim.x) a.Bp[(size_t)u * N + i] = Sb[i];

        // Eqs. 12-15
        const int calib_keep = min(a.calib_budget, N) - win;
        const long long Ml = (long long)c.rho * (long long)(calib_keep > 0 ? calib_keep : 0);
        const int M = (int)(Ml < n_cand ? Ml : n_cand);
        float lam = 0.f;
        if (M > 0) {
            const SelectResult sel = radix_select(Sb, n_cand, M, hist, bcast);
            const RangeSel rg = my_range(n_cand);
            int eq = 0;
            for (int i = rg.lo; i < rg.hi; ++i) eq += float_key(Sb[i]) == sel.tau;
            int eq_before = block_exclusive_scan(eq, warp_sums, &total_s);
            double sb = 0.0, sv = 0.0;
            {
                int e = eq_before;
                for (int i = rg.lo; i < rg.hi; ++i) {
                    const uint32_t key = float_key(Sb[i]);
                    bool in = key > sel.tau;
                    if (key == sel.tau) in = (e++ < sel.need);
                    if (in) {
                        sb += Sb[i];
                        sv += Vs[i];
                    }
                }
            }
            const double mb = block_sum(sb, red) / M;
            const double mv = block_sum(sv, red) / M;
            double vb = 0.0, vv = 0.0;
            {
                int e = eq_before;
                for (int i = rg.lo; i < rg.hi; ++i) {
                    const uint32_t key = float_key(Sb[i]);
                    bool in = key > sel.tau;
                    if (key == sel.tau) in = (e++ < sel.need);
                    if (in) {
                        const double db = Sb[i] - mb, dv = Vs[i] - mv;
                        vb += db * db;
                        vv += dv * dv;
                    }
                }
            }
            const double stdb = sqrt(block_sum(vb, red) / M);
            const double stdv = sqrt(block_sum(vv, red) / M);
            lam = (float)((double)c.gamma * stdb / (stdv + (double)c.eps));
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
    int32_t* out = a.idx + (size_t)u * kept_total;
    if (keep >= n_cand) {
        for (int i = threadIdx.x; i < n_cand; i += blockDim.x) out[i] = i;
    } else if (keep > 0) {
        const SelectResult sel = radix_select(Sb, n_cand, keep, hist, bcast);
        const RangeSel rg = my_range(n_cand);
        int eq = 0;
        for (int i = rg.lo; i < rg.hi; ++i) eq += float_key(Sb[i]) == sel.tau;
        const int eq_before = block_exclusive_scan(eq, warp_sums, &total_s);
        int mine = 0;
        {
            int e = eq_before;
            for (int i = rg.lo; i < rg.hi; ++i) {
                const uint32_t key = float_key(Sb[i]);
                bool in = key > sel.tau;
                if (key == sel.tau) in = (e++ < sel.need);
                mine += in;
            }
        }
        int pos = block_exclusive_scan(mine, warp_sums, &total_s);
        {
            int e = eq_before;
            for (int i = rg.lo; i < rg.hi; ++i) {
                const uint32_t key = float_key(Sb[i]);
                bool in = key > sel.tau;
                if (key == sel.tau) in = (e++ < sel.need);
                if (in) out[pos++] = i;
            }
        }
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
