// Compacted cache construction (Sec. 4.4, after Eq. 17): the kept K and V
// rows of every (request, layer, kv-head) are copied bitwise into dense
// [kept][d] blocks.  One thread moves one 16-byte piece of a row of K and the
// same piece of V, so a row is read and written as contiguous, coalesced
// 16-byte accesses.
#include "common.cuh"

namespace bacon {
namespace {

__global__ void __launch_bounds__(256)
gather_kernel(GatherTable tab, Shape s, int* __restrict__ err)
{
    const int u = blockIdx.y;
    const int pair = u / s.hkv, h = u - pair * s.hkv;
    const int kept = tab.kept[pair];
    const int cpr = s.d / 8;
    const int e = blockIdx.x * blockDim.x + threadIdx.x;
    const int j = e / cpr, q = e - j * cpr;
    if (j >= kept) return;
    const int src = tab.idx[pair][(size_t)h * kept + j];
    if (src < 0 || src >= s.N) {
        if (err) atomicCAS(err, 0, 1);
        return;
    }
    const size_t in_off = ((size_t)h * s.N + src) * s.d;
    const size_t out_off = ((size_t)h * kept + j) * s.d;
    const uint4* ks = reinterpret_cast<const uint4*>(tab.k[pair] + in_off) + q;
    const uint4* vs = reinterpret_cast<const uint4*>(tab.v[pair] + in_off) + q;
    uint4* kd = reinterpret_cast<uint4*>(tab.ko[pair] + out_off) + q;
    uint4* vd = reinterpret_cast<uint4*>(tab.vo[pair] + out_off) + q;
    const uint4 kv = __ldg(ks);
    const uint4 vv = __ldg(vs);
    *kd = kv;
    *vd = vv;
}

}  // namespace

cudaError_t launch_gather(const GatherTable& tab, const Shape& s, int* err, cudaStream_t st)
{
    int kept = 0;
    for (int p = 0; p < s.units / s.hkv; ++p) kept = tab.kept[p] > kept ? tab.kept[p] : kept;
    if (kept <= 0) return cudaSuccess;
    const int pieces = kept * (s.d / 8);
    dim3 grid((pieces + 255) / 256, s.units);
    gather_kernel<<<grid, 256, 0, st>>>(tab, s, err);
    return cudaGetLastError();
}

}  // namespace bacon
