// AdaKV-style adaptive head budgets (the base compressor of Sec. 5 / App. B
// that spreads a layer's budget over its kv-heads; BACON supplies the score,
// Eq. 16).  One CTA per (request, layer):
//   1. every head keeps its own top g = floor(alpha K) candidates;
//   2. the remaining Hkv K - Hkv g slots go to the best remaining candidates
//      of all heads together (larger S first; ties to the lower head, then
//      the lower position: the flattened index h * n_cand + i);
//   3. each head's kept positions are written in ascending order, followed
//      by the window, into one flat per-layer array (heads in order), and
//      the per-head counts are reported.
// The kept K/V rows are then gathered into the same flat layout.
#include "common.cuh"
#include "select.cuh"

namespace bacon {
namespace {

using namespace sel;

constexpr int kThreads = 1024;

__global__ void __launch_bounds__(kThreads)
adaptive_select_kernel(Shape s, int keep_window, AdaptArgs a)
{
    extern __shared__ uint8_t taken[];  // [Hkv][n_cand]
    __shared__ __align__(16) int hist[kSelHist];
    __shared__ int bcast[8];
    __shared__ int warp_sums[32];
    __shared__ int total_s;

    const int pair = blockIdx.x;
    const int H = s.hkv, N = s.N, W = s.W;
    const int win = keep_window ? W : 0;
    const int n_cand = N - win;
    const int kept_total = min(a.budget, N);
    const int keep = kept_total - win;
    const int g = min(a.guaranteed, keep);
    const float* Sp = a.S + (size_t)pair * H * N;
    const int total = H * n_cand;

    const uint8_t fill = keep >= n_cand ? 1 : 0;  // every candidate kept
    for (int i = threadIdx.x; i < total; i += blockDim.x) taken[i] = fill;
    __syncthreads();

    if (!fill) {
        // 1. each head's guaranteed share
        if (g > 0) {
            for (int h = 0; h < H; ++h) {
                const float* Sh = Sp + (size_t)h * N;
                const SelectResult r = radix_select(Sh, n_cand, g, hist, bcast);
                const Segment sg = warp_segment(n_cand);
                const int eqb = eq_before_segment(Sh, sg, r, warp_sums, &total_s);
                walk_topk(Sh, sg, r, eqb, [&](int i, bool, bool in) {
                    if (in) taken[h * n_cand + i] = 1;
                });
                __syncthreads();
            }
        }
        // 2. the rest, jointly over the heads (taken candidates excluded)
        const int rest = H * keep - H * g;
        if (rest > 0) {
            auto key_of = [&](int f, uint32_t& key) -> bool {
                if (taken[f]) return false;
                const int h = f / n_cand;
                key = float_key(Sp[(size_t)h * N + (f - h * n_cand)]);
                return true;
            };
            const SelectResult r = radix_select_by(total, rest, key_of, hist, bcast);
            const Segment sg = warp_segment(total);
            const int eqb = eq_before_segment_by(sg, r, key_of, warp_sums, &total_s);
            // a warp only marks its own segment, after evaluating each element
            walk_topk_by(sg, r, eqb, key_of, [&](int f, bool, bool in) {
                if (in) taken[f] = 1;
            });
            __syncthreads();
        }
    }

    // 3. per-head ascending compaction into the flat layout
    int32_t* out = a.idx[pair];
    const int lane = threadIdx.x & 31;
    const uint32_t lt = (1u << lane) - 1u;
    int off = 0;
    for (int h = 0; h < H; ++h) {
        const uint8_t* th = taken + h * n_cand;
        const Segment sg = warp_segment(n_cand);
        int mine = 0;
        for (int i = sg.lo + lane; i < sg.hi; i += 32) mine += th[i];
        const int base = warp_exclusive_scan(warp_sum(mine), warp_sums, &total_s);
        const int count = total_s;
        int pos = off + base;
        for (int b0 = sg.lo; b0 < sg.hi; b0 += 32) {
            const int i = b0 + lane;
            const bool in = i < sg.hi && th[i];
            const uint32_t ball = __ballot_sync(0xffffffffu, in);
            if (in) out[pos + __popc(ball & lt)] = i;
            pos += __popc(ball);
        }
        for (int w = threadIdx.x; w < win; w += blockDim.x) out[off + count + w] = N - W + w;
        if (threadIdx.x == 0) a.counts[(size_t)pair * H + h] = count + win;
        off += count + win;
        __syncthreads();
    }
    if (threadIdx.x == 0 && off != H * kept_total && a.err) atomicCAS(a.err, 0, 2);
}

// Flat per-layer gather: output row j of a pair belongs to the head whose
// segment (per-head counts, heads in order) contains it.
__global__ void __launch_bounds__(256)
gather_flat_kernel(GatherTable tab, Shape s, const int32_t* __restrict__ counts,
                   int* __restrict__ err)
{
    const int pair = blockIdx.y;
    const int total = tab.kept[pair];  // rows of the pair
    const int cpr = s.d / 8;
    const int e = blockIdx.x * blockDim.x + threadIdx.x;
    const int j = e / cpr, q = e - j * cpr;
    if (j >= total) return;
    int h = 0, start = 0;
    while (h < s.hkv - 1 && j >= start + counts[(size_t)pair * s.hkv + h]) {
        start += counts[(size_t)pair * s.hkv + h];
        ++h;
    }
    const int src = tab.idx[pair][j];
    if (src < 0 || src >= s.N) {
        if (err) atomicCAS(err, 0, 1);
        return;
    }
    const size_t in_off = ((size_t)h * s.N + src) * s.d;
    const size_t out_off = (size_t)j * s.d;
    const uint4 kv = __ldg(reinterpret_cast<const uint4*>(tab.k[pair] + in_off) + q);
    const uint4 vv = __ldg(reinterpret_cast<const uint4*>(tab.v[pair] + in_off) + q);
    reinterpret_cast<uint4*>(tab.ko[pair] + out_off)[q] = kv;
    reinterpret_cast<uint4*>(tab.vo[pair] + out_off)[q] = vv;
}

}  // namespace

size_t adaptive_smem(int kv_heads, int n_cand) { return (size_t)kv_heads * n_cand; }

cudaError_t launch_adaptive_select(const Shape& s, int keep_window, const AdaptArgs& a,
                                   cudaStream_t st)
{
    const int win = keep_window ? s.W : 0;
    const size_t sm = adaptive_smem(s.hkv, s.N - win);
    cudaError_t e = cudaFuncSetAttribute(adaptive_select_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e != cudaSuccess) return e;
    adaptive_select_kernel<<<s.units / s.hkv, kThreads, sm, st>>>(s, keep_window, a);
    return cudaGetLastError();
}

cudaError_t launch_gather_flat(const GatherTable& tab, const Shape& s, const int32_t* counts,
                               int* err, cudaStream_t st)
{
    const int pairs = s.units / s.hkv;
    int rows = 0;
    for (int p = 0; p < pairs; ++p) rows = tab.kept[p] > rows ? tab.kept[p] : rows;
    if (rows <= 0) return cudaSuccess;
    dim3 grid((rows * (s.d / 8) + 255) / 256, pairs);
    gather_flat_kernel<<<grid, 256, 0, st>>>(tab, s, counts, err);
    return cudaGetLastError();
}

}  // namespace bacon
