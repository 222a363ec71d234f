// CUDA-core projection GEMM: the fp32 storage mode's GEMM (exact fp32 products, which the
// tensor cores do not offer) and, for bf16, a diagnostic cross-check of the tcgen05 GEMM.
// One CTA computes 128 output features x 16 tokens (x2 accumulators for SwiGLU) over the whole
// K range, then hands the tile to the shared epilogue.
#include "epilogue.cuh"

namespace dfl {
namespace {

constexpr int kTN = 128;   // features per CTA
constexpr int kTT = 16;    // tokens per CTA
constexpr int kTK = 16;    // K chunk

template <class T>
__global__ void __launch_bounds__(256) gemm_simt_kernel(const T* __restrict__ A, const T* __restrict__ A2,
                                                        const T* __restrict__ Bm, int n, int k,
                                                        int m_tok, long long a_group_rows,
                                                        long long b_group_rows, int b_shared,
                                                        int b_kgroup, int n_tiles, EpiParams ep) {
    pdl_wait();
    pdl_trigger();   // after the wait: see gemm_tc_kernel
    __shared__ float sA[2][kTN][kTK + 1];
    __shared__ float sB[kTT][kTK + 1];
    __shared__ __align__(16) float tile[2 * kTT * kTN];
    const int n_tile = blockIdx.x % n_tiles, group = blockIdx.x / n_tiles;
    const int tok0 = blockIdx.y * kTT;
    const int na = A2 ? 2 : 1;
    const int tid = threadIdx.x;
    const int f = tid & 127, tg = tid >> 7;   // feature f, tokens tg*8 .. tg*8+7
    const T* Ag = A + (size_t)group * a_group_rows * k;
    const T* A2g = A2 ? A2 + (size_t)group * a_group_rows * k : nullptr;
    const T* Bg = Bm + (size_t)(b_shared ? 0 : group) * b_group_rows * k;
    float acc[2][8];
#pragma unroll
    for (int a = 0; a < 2; ++a)
#pragma unroll
        for (int i = 0; i < 8; ++i) acc[a][i] = 0.f;
    for (int k0 = 0; k0 < k; k0 += kTK) {
        __syncthreads();
        for (int idx = tid; idx < kTN * kTK; idx += 256) {
            const int r = idx / kTK, cc = idx % kTK;
            const int row = n_tile * kTN + r, col = k0 + cc;
            const bool in = row < n && col < k;
            sA[0][r][cc] = in ? to_f(Ag[(size_t)row * k + col]) : 0.f;
            if (na == 2) sA[1][r][cc] = in ? to_f(A2g[(size_t)row * k + col]) : 0.f;
        }
        for (int idx = tid; idx < kTT * kTK; idx += 256) {
            const int r = idx / kTK, cc = idx % kTK;
            const int tok = tok0 + r, col = k0 + cc;
            float v = 0.f;
            if (tok < m_tok && col < k) {
                if (b_kgroup > 0) {   // contraction over stacked activation groups (Eq. 1)
                    const int z = col / b_kgroup;
                    v = to_f(Bm[((size_t)z * b_group_rows + tok) * b_kgroup + (col - z * b_kgroup)]);
                } else {
                    v = to_f(Bg[(size_t)tok * k + col]);
                }
            }
            sB[r][cc] = v;
        }
        __syncthreads();
        for (int a = 0; a < na; ++a)
#pragma unroll 4
            for (int cc = 0; cc < kTK; ++cc) {
                const float w = sA[a][f][cc];
#pragma unroll
                for (int i = 0; i < 8; ++i) acc[a][i] = fmaf(w, sB[tg * 8 + i][cc], acc[a][i]);
            }
    }
    for (int a = 0; a < na; ++a)
#pragma unroll
        for (int i = 0; i < 8; ++i) tile[(a * kTT + tg * 8 + i) * kTN + f] = acc[a][i];
    __syncthreads();
    if (tid < 128) apply_epilogue<T>(ep, tile, group, n_tile, tok0, tid);
}

}  // namespace

cudaError_t launch_gemm_simt(dflare_ctx* c, const GemmDesc& g, cudaStream_t s) {
    if (g.m_tok <= 0 || g.n <= 0) return cudaSuccess;
    const int n_tiles = (g.n + kTN - 1) / kTN;
    if (g.b_kgroup > 0 && (g.k % g.b_kgroup != 0 || g.groups != 1)) return cudaErrorInvalidValue;
    dim3 grid(n_tiles * g.groups, (g.m_tok + kTT - 1) / kTT);
    const long long a_gr = g.a_group_rows > 0 ? g.a_group_rows : g.n;
    if (c->cfg.dtype == DFLARE_F32)
        return launch_kernel(c->pdl, gemm_simt_kernel<float>, grid, dim3(256), 0, s,
                             (const float*)g.a, (const float*)g.a2, (const float*)g.b, g.n, g.k,
                             g.m_tok, a_gr, g.b_group_rows, g.b_shared, g.b_kgroup, n_tiles, g.ep);
    return launch_kernel(c->pdl, gemm_simt_kernel<bf16>, grid, dim3(256), 0, s, (const bf16*)g.a,
                         (const bf16*)g.a2, (const bf16*)g.b, g.n, g.k, g.m_tok, a_gr,
                         g.b_group_rows, g.b_shared, g.b_kgroup, n_tiles, g.ep);
}

}  // namespace dfl
