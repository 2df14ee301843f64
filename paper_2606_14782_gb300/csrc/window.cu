// Window-attention scores B (Eq. 1), last-query scores Q (Eq. 2) and the
// residual E (Eq. 4) for every (request, layer, kv-head) of a call.
//
// The softmax of each window row must be normalised over all N keys before
// any B_i is final, so the computation is two passes over K:
//   pass 1  logits -> per (row, token chunk) running max and sum of
//           2^(logit * log2 e / sqrt d)                     (window_stats)
//   merge   per row log2 of the normaliser, plus log2(G W)  (window_combine)
//   pass 2  logits again -> A_{q,i} / (G W) = 2^(logit' - lse2_q), summed
//           over the G W rows of the kv-head per token      (window_scores)
// Pass 1 puts window rows on the MMA M axis (a thread owns whole rows, so the
// row statistics are thread-local); pass 2 puts tokens on the M axis (a
// thread owns whole tokens, so the sum over rows is thread-local).  Both
// contract bf16 operands into fp32 on the tensor cores.
#include "common.cuh"

namespace bacon {
namespace {

constexpr int kTile = 128;    // tokens per shared-memory K tile
constexpr int kWarps = 8;     // warps per CTA in both passes
constexpr float kLog2e = 1.4426950408889634f;

template <int D>
struct Geo {
    static constexpr int LD = D + 8;   // padded shared row (elements): 16-B rows
                                       // land on distinct bank groups for ldmatrix
    static constexpr int KS = D / 16;  // k-steps of one row
    static constexpr int CPR = D / 8;  // 16-byte chunks per row
};

// rows [row0, row0 + nrows) of a row-major [total][D] bf16 matrix -> shared
// memory with row stride LD; rows >= total are zero-filled.
template <int D>
__device__ __forceinline__ void load_rows(uint16_t* sm, const uint16_t* g, int row0, int nrows,
                                          int total)
{
    constexpr int CPR = Geo<D>::CPR;
    for (int c = threadIdx.x; c < nrows * CPR; c += blockDim.x) {
        const int r = c / CPR, q = c - r * CPR;
        const int gr = row0 + r;
        const bool ok = gr < total;
        const uint16_t* src = g + (size_t)(ok ? gr : 0) * D + q * 8;
        cp_async16(smem_u32(sm + r * Geo<D>::LD + q * 8), src, ok ? 16 : 0);
    }
}

// ------------------------------------------------------------- pass 1

// CTA: 8 warps = row_warps x token_warps.  A warp owns 32 window rows (two
// m16 tiles, operands kept in registers) and a slice of each 128-token tile.
template <int D>
__global__ void __launch_bounds__(kWarps * 32)
window_stats_kernel(QKTable tab, Shape s, int chunk_tokens, int chunks, int row_warps,
                    float2* __restrict__ partial)
{
    constexpr int LD = Geo<D>::LD, KS = Geo<D>::KS;
    extern __shared__ __align__(16) uint16_t smem[];
    uint16_t* Qs = smem;                           // [row_warps * 32][LD]
    uint16_t* Ks = Qs + row_warps * 32 * LD;       // [2][kTile][LD]
    float2* red = reinterpret_cast<float2*>(Ks + 2 * kTile * LD);  // [kWarps][32]

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int g = lane >> 2, t = lane & 3;
    const int token_warps = kWarps / row_warps;
    const int rw = warp % row_warps, tw = warp / row_warps;
    const int chunk = blockIdx.y, u = blockIdx.z;
    const int pair = u / s.hkv, h = u - pair * s.hkv;
    const uint16_t* q = tab.q[pair] + (size_t)h * s.rows * D;
    const uint16_t* k = tab.k[pair] + (size_t)h * s.N * D;
    const int row_base = blockIdx.x * row_warps * 32;
    const int t_begin = chunk * chunk_tokens;
    const int t_end = min(s.N, t_begin + chunk_tokens);
    const int ntiles = (t_end - t_begin + kTile - 1) / kTile;

    load_rows<D>(Qs, q, row_base, row_warps * 32, s.rows);
    load_rows<D>(Ks, k, t_begin, kTile, t_end);
    cp_async_commit();
    cp_async_wait<0>();
    __syncthreads();

    uint32_t a[2][KS][4];
#pragma unroll
    for (int mt = 0; mt < 2; ++mt)
#pragma unroll
        for (int kt = 0; kt < KS; ++kt) {
            const int row = rw * 32 + mt * 16 + (lane & 15);
            const int col = kt * 16 + 8 * (lane >> 4);
            ldmatrix_x4(smem_u32(Qs + row * LD + col), a[mt][kt][0], a[mt][kt][1], a[mt][kt][2],
                        a[mt][kt][3]);
        }

    const float c = kLog2e * rsqrtf((float)D);
    float m_run[2][2], z_run[2][2];
    int last_vis[2][2];  // last key position the row's query may see
#pragma unroll
    for (int mt = 0; mt < 2; ++mt)
#pragma unroll
        for (int hr = 0; hr < 2; ++hr) {
            const int r = row_base + rw * 32 + mt * 16 + hr * 8 + g;
            m_run[mt][hr] = -INFINITY;
            z_run[mt][hr] = 0.f;
            last_vis[mt][hr] = s.N - s.W + (r % s.W);
        }

    const int tok_per_warp = kTile / token_warps;  // 128, 64, 32 or 16
    const int sub = tok_per_warp < 64 ? tok_per_warp : 64;

    for (int it = 0; it < ntiles; ++it) {
        const int buf = it & 1;
        if (it + 1 < ntiles)
            load_rows<D>(Ks + (buf ^ 1) * kTile * LD, k, t_begin + (it + 1) * kTile, kTile, t_end);
        cp_async_commit();
        const uint16_t* Kt = Ks + buf * kTile * LD;
        const int tile0 = t_begin + it * kTile;

        for (int s0 = tw * tok_per_warp; s0 < (tw + 1) * tok_per_warp; s0 += sub) {
            float acc[2][8][4];
#pragma unroll
            for (int mt = 0; mt < 2; ++mt)
#pragma unroll
                for (int nt = 0; nt < 8; ++nt)
#pragma unroll
                    for (int j = 0; j < 4; ++j) acc[mt][nt][j] = 0.f;
            const int npairs = sub / 16;
#pragma unroll
            for (int kt = 0; kt < KS; ++kt) {
#pragma unroll
                for (int np = 0; np < 4; ++np) {
                    if (np < npairs) {
                        const int row = s0 + np * 16 + (lane & 7) + 8 * (lane >> 4);
                        const int col = kt * 16 + 8 * ((lane >> 3) & 1);
                        uint32_t b0, b1, b2, b3;
                        ldmatrix_x4(smem_u32(Kt + row * LD + col), b0, b1, b2, b3);
#pragma unroll
                        for (int mt = 0; mt < 2; ++mt) {
                            mma_bf16(acc[mt][2 * np], a[mt][kt], b0, b1);
                            mma_bf16(acc[mt][2 * np + 1], a[mt][kt], b2, b3);
                        }
                    }
                }
            }
            const bool need_mask = (tile0 + s0 + sub - 1) > (s.N - s.W);
#pragma unroll
            for (int mt = 0; mt < 2; ++mt)
#pragma unroll
                for (int hr = 0; hr < 2; ++hr) {
                    float v[16];
                    float bm = -INFINITY;
#pragma unroll
                    for (int nt = 0; nt < 8; ++nt)
#pragma unroll
                        for (int j = 0; j < 2; ++j) {
                            float x = acc[mt][nt][2 * hr + j] * c;
                            const int tok = tile0 + s0 + nt * 8 + 2 * t + j;
                            if (nt >= 2 * npairs || (need_mask && tok > last_vis[mt][hr]))
                                x = -INFINITY;
                            v[nt * 2 + j] = x;
                            bm = fmaxf(bm, x);
                        }
                    bm = fmaxf(bm, __shfl_xor_sync(0xffffffffu, bm, 1));
                    bm = fmaxf(bm, __shfl_xor_sync(0xffffffffu, bm, 2));
                    const float m_new = fmaxf(m_run[mt][hr], bm);
                    if (m_new != -INFINITY) {
                        float zs = 0.f;
#pragma unroll
                        for (int e = 0; e < 16; ++e) zs += fast_exp2(v[e] - m_new);
                        z_run[mt][hr] = z_run[mt][hr] * fast_exp2(m_run[mt][hr] - m_new) + zs;
                        m_run[mt][hr] = m_new;
                    }
                }
        }
        cp_async_wait<0>();
        __syncthreads();
    }

    // the four lanes of a quad share m_run: their sums add
#pragma unroll
    for (int mt = 0; mt < 2; ++mt)
#pragma unroll
        for (int hr = 0; hr < 2; ++hr) {
            float z = z_run[mt][hr];
            z += __shfl_xor_sync(0xffffffffu, z, 1);
            z += __shfl_xor_sync(0xffffffffu, z, 2);
            if (t == 0) red[warp * 32 + mt * 16 + hr * 8 + g] = make_float2(m_run[mt][hr], z);
        }
    __syncthreads();
    if (tw == 0) {
        const int rl = lane;  // this warp's 32 rows
        const int r = row_base + rw * 32 + rl;
        float M = -INFINITY;
        for (int x = 0; x < token_warps; ++x) M = fmaxf(M, red[(rw + x * row_warps) * 32 + rl].x);
        float Z = 0.f;
        if (M != -INFINITY)
            for (int x = 0; x < token_warps; ++x) {
                const float2 p = red[(rw + x * row_warps) * 32 + rl];
                if (p.y > 0.f) Z += p.y * fast_exp2(p.x - M);
            }
        if (r < s.rows) partial[((size_t)u * chunks + chunk) * s.rows + r] = make_float2(M, Z);
    }
}

__global__ void window_combine_kernel(Shape s, int chunks, const float2* __restrict__ partial,
                                      float* __restrict__ lse2)
{
    const int u = blockIdx.x;
    const float log2_gw = log2f((float)s.rows);
    for (int r = threadIdx.x; r < s.rows; r += blockDim.x) {
        const float2* p = partial + (size_t)u * chunks * s.rows + r;
        float M = -INFINITY;
        for (int c = 0; c < chunks; ++c) M = fmaxf(M, p[(size_t)c * s.rows].x);
        float Z = 0.f;
        for (int c = 0; c < chunks; ++c) {
            const float2 v = p[(size_t)c * s.rows];
            if (v.y > 0.f) Z += v.y * exp2f(v.x - M);
        }
        lse2[(size_t)u * s.rows + r] = M + log2f(Z) + log2_gw;
    }
}

// ------------------------------------------------------------- pass 2

// CTA: 8 warps x 16 tokens = one 128-token tile at a time, looping over
// `tiles_per_cta` tiles of one unit; all G W window rows (zero-padded to a
// multiple of 16) stay in shared memory for the CTA's lifetime.
template <int D>
__global__ void __launch_bounds__(kWarps * 32)
window_scores_kernel(QKTable tab, Shape s, int tiles_per_cta, int rows_pad,
                     const float* __restrict__ lse2, float* __restrict__ Bo,
                     float* __restrict__ Qo, float* __restrict__ Eo)
{
    constexpr int LD = Geo<D>::LD, KS = Geo<D>::KS;
    extern __shared__ __align__(16) uint16_t smem[];
    uint16_t* Qs = smem;                             // [rows_pad][LD]
    uint16_t* Ks = Qs + rows_pad * LD;               // [2][kTile][LD]
    float* lse_s = reinterpret_cast<float*>(Ks + 2 * kTile * LD);  // [rows_pad]
    float* qw_s = lse_s + rows_pad;                  // W for last-position rows, else 0
    int* vis_s = reinterpret_cast<int*>(qw_s + rows_pad);  // last visible key per row

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int g = lane >> 2, t = lane & 3;
    const int u = blockIdx.y;
    const int pair = u / s.hkv, h = u - pair * s.hkv;
    const uint16_t* q = tab.q[pair] + (size_t)h * s.rows * D;
    const uint16_t* k = tab.k[pair] + (size_t)h * s.N * D;
    const int ntiles_all = (s.N + kTile - 1) / kTile;
    const int tile_lo = blockIdx.x * tiles_per_cta;
    const int tile_hi = min(ntiles_all, tile_lo + tiles_per_cta);
    if (tile_lo >= tile_hi) return;

    load_rows<D>(Qs, q, 0, rows_pad, s.rows);
    load_rows<D>(Ks, k, tile_lo * kTile, kTile, s.N);
    cp_async_commit();
    for (int r = threadIdx.x; r < rows_pad; r += blockDim.x) {
        const bool real = r < s.rows;
        lse_s[r] = real ? lse2[(size_t)u * s.rows + r] : INFINITY;
        qw_s[r] = (real && (r % s.W) == s.W - 1) ? (float)s.W : 0.f;
        vis_s[r] = s.N - s.W + (r % s.W);
    }
    cp_async_wait<0>();
    __syncthreads();

    const float c = kLog2e * rsqrtf((float)D);
    const int npairs_all = rows_pad / 16;

    for (int tile = tile_lo; tile < tile_hi; ++tile) {
        const int buf = (tile - tile_lo) & 1;
        if (tile + 1 < tile_hi)
            load_rows<D>(Ks + (buf ^ 1) * kTile * LD, k, (tile + 1) * kTile, kTile, s.N);
        cp_async_commit();
        const uint16_t* Kt = Ks + buf * kTile * LD;

        uint32_t a[KS][4];
#pragma unroll
        for (int kt = 0; kt < KS; ++kt) {
            const int row = warp * 16 + (lane & 15);
            const int col = kt * 16 + 8 * (lane >> 4);
            ldmatrix_x4(smem_u32(Kt + row * LD + col), a[kt][0], a[kt][1], a[kt][2], a[kt][3]);
        }
        const int tok0 = tile * kTile + warp * 16 + g;
        const int tok1 = tok0 + 8;
        const bool need_mask = (tile * kTile + warp * 16 + 15) > (s.N - s.W);
        float bsum0 = 0.f, bsum1 = 0.f, qsum0 = 0.f, qsum1 = 0.f;

        for (int p0 = 0; p0 < npairs_all; p0 += 4) {
            float acc[8][4];
#pragma unroll
            for (int nt = 0; nt < 8; ++nt)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[nt][j] = 0.f;
            const int npairs = min(4, npairs_all - p0);
#pragma unroll
            for (int kt = 0; kt < KS; ++kt)
#pragma unroll
                for (int np = 0; np < 4; ++np) {
                    if (np < npairs) {
                        const int row = (p0 + np) * 16 + (lane & 7) + 8 * (lane >> 4);
                        const int col = kt * 16 + 8 * ((lane >> 3) & 1);
                        uint32_t b0, b1, b2, b3;
                        ldmatrix_x4(smem_u32(Qs + row * LD + col), b0, b1, b2, b3);
                        mma_bf16(acc[2 * np], a[kt], b0, b1);
                        mma_bf16(acc[2 * np + 1], a[kt], b2, b3);
                    }
                }
#pragma unroll
            for (int nt = 0; nt < 8; ++nt) {
                if (nt < 2 * npairs) {
#pragma unroll
                    for (int j = 0; j < 2; ++j) {
                        const int r = p0 * 16 + nt * 8 + 2 * t + j;
                        const float L = lse_s[r];
                        float x0 = fast_exp2(fmaf(acc[nt][j], c, -L));
                        float x1 = fast_exp2(fmaf(acc[nt][2 + j], c, -L));
                        if (need_mask) {
                            const int vis = vis_s[r];
                            if (tok0 > vis) x0 = 0.f;
                            if (tok1 > vis) x1 = 0.f;
                        }
                        bsum0 += x0;
                        bsum1 += x1;
                        const float qw = qw_s[r];
                        qsum0 = fmaf(x0, qw, qsum0);
                        qsum1 = fmaf(x1, qw, qsum1);
                    }
                }
            }
        }
#pragma unroll
        for (int o = 1; o <= 2; o <<= 1) {
            bsum0 += __shfl_xor_sync(0xffffffffu, bsum0, o);
            bsum1 += __shfl_xor_sync(0xffffffffu, bsum1, o);
            qsum0 += __shfl_xor_sync(0xffffffffu, qsum0, o);
            qsum1 += __shfl_xor_sync(0xffffffffu, qsum1, o);
        }
        if (t == 0) {
            const size_t base = (size_t)u * s.N;
            if (tok0 < s.N) {
                Bo[base + tok0] = bsum0;
                Qo[base + tok0] = qsum0;
                Eo[base + tok0] = fmaxf(qsum0 - bsum0, 0.f);
            }
            if (tok1 < s.N) {
                Bo[base + tok1] = bsum1;
                Qo[base + tok1] = qsum1;
                Eo[base + tok1] = fmaxf(qsum1 - bsum1, 0.f);
            }
        }
        cp_async_wait<0>();
        __syncthreads();
    }
}

int stats_row_warps(int rows)
{
    const int need = (rows + 31) / 32;
    int rw = 1;
    while (rw < need && rw < kWarps) rw <<= 1;
    return rw;
}

template <int D>
size_t stats_smem(int row_warps)
{
    return (size_t)(row_warps * 32 + 2 * kTile) * Geo<D>::LD * 2 + kWarps * 32 * sizeof(float2);
}

template <int D>
size_t scores_smem(int rows_pad)
{
    return (size_t)(rows_pad + 2 * kTile) * Geo<D>::LD * 2 + (size_t)rows_pad * 12;
}

template <int D>
cudaError_t stats_impl(const QKTable& tab, const Shape& s, int chunk_tokens, float2* partial,
                       cudaStream_t st)
{
    const int rw = stats_row_warps(s.rows);
    const int chunks = (s.N + chunk_tokens - 1) / chunk_tokens;
    const int row_blocks = (s.rows + rw * 32 - 1) / (rw * 32);
    const size_t sm = stats_smem<D>(rw);
    cudaError_t e = cudaFuncSetAttribute(window_stats_kernel<D>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e != cudaSuccess) return e;
    dim3 grid(row_blocks, chunks, s.units);
    window_stats_kernel<D><<<grid, kWarps * 32, sm, st>>>(tab, s, chunk_tokens, chunks, rw, partial);
    return cudaGetLastError();
}

template <int D>
cudaError_t scores_impl(const QKTable& tab, const Shape& s, const float* lse2, float* B, float* Q,
                        float* E, cudaStream_t st)
{
    const int rows_pad = (s.rows + 15) / 16 * 16;
    const size_t sm = scores_smem<D>(rows_pad);
    cudaError_t e = cudaFuncSetAttribute(window_scores_kernel<D>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e != cudaSuccess) return e;
    const int ntiles = (s.N + kTile - 1) / kTile;
    const int tiles_per_cta = ntiles < 8 ? ntiles : 8;
    dim3 grid((ntiles + tiles_per_cta - 1) / tiles_per_cta, s.units);
    window_scores_kernel<D><<<grid, kWarps * 32, sm, st>>>(tab, s, tiles_per_cta, rows_pad, lse2,
                                                           B, Q, E);
    return cudaGetLastError();
}

}  // namespace

// largest supported G*W for a head dimension (shared-memory bound of pass 2)
int window_max_rows(int d)
{
    const size_t budget = 227 * 1024;
    const size_t ld = (size_t)(d + 8) * 2;
    const size_t fixed = 2 * kTile * ld;
    return (int)(((budget - fixed) / (ld + 12)) / 16 * 16);
}

cudaError_t launch_window_stats(const QKTable& tab, const Shape& s, int chunk_tokens,
                                float2* partial, cudaStream_t st)
{
    if (s.d == 128) return stats_impl<128>(tab, s, chunk_tokens, partial, st);
    if (s.d == 64) return stats_impl<64>(tab, s, chunk_tokens, partial, st);
    return cudaErrorInvalidValue;
}

cudaError_t launch_window_combine(const Shape& s, int chunks, const float2* partial,
                                  float* lse2, cudaStream_t st)
{
    const int threads = s.rows < 512 ? ((s.rows + 31) / 32) * 32 : 512;
    window_combine_kernel<<<s.units, threads, 0, st>>>(s, chunks, partial, lse2);
    return cudaGetLastError();
}

cudaError_t launch_window_scores(const QKTable& tab, const Shape& s, const float* lse2, float* B,
                                 float* Q, float* E, cudaStream_t st)
{
    if (s.d == 128) return scores_impl<128>(tab, s, lse2, B, Q, E, st);
    if (s.d == 64) return scores_impl<64>(tab, s, lse2, B, Q, E, st);
    return cudaErrorInvalidValue;
}

}  // namespace bacon
