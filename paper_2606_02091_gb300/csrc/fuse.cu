// Adaptive layer fusion (Eq. 3, Sec. 4.1) and the bookkeeping of a context append.
//
// fusion_alpha: alpha^(i) = softmax(W^fuse_{i,:}), computed once when the weights are set
// (Sec. 4.1: the normalised weights can be cached after training).
// fuse_layers: one CTA per new position; every thread owns 8 consecutive features, reads the T
// target states of its features once with 16-byte loads (four layers in flight), forms the
// weighted sums of up to 8 draft layers in registers, then RMSNorms each sum (one block
// reduction for all layers at once). More than 8 draft layers take further passes over the same
// rows, which the previous pass left in L2.
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace dfl {
namespace {

__global__ void fusion_alpha_kernel(const float* __restrict__ w, float* __restrict__ alpha, int D,
                                    int T, int raw) {
    pdl_trigger();
    pdl_wait();
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= D) return;
    const float* row = w + (size_t)i * T;
    if (raw) {
        for (int j = 0; j < T; ++j) alpha[(size_t)i * T + j] = row[j];
        return;
    }
    float m = -INFINITY;
    for (int j = 0; j < T; ++j) m = fmaxf(m, row[j]);
    float s = 0.f;
    for (int j = 0; j < T; ++j) s += expf(row[j] - m);
    for (int j = 0; j < T; ++j) alpha[(size_t)i * T + j] = expf(row[j] - m) / s;
}

__global__ void fuse_begin_kernel(int32_t* ctx_len, int32_t* app_base, int32_t* app_cnt,
                                  const int32_t* __restrict__ n_new, int batch, int n_max,
                                  int max_ctx, uint32_t* err) {
    pdl_trigger();
    pdl_wait();
    const int b = blockIdx.x * blockDim.x + threadIdx.x;
    if (b >= batch) return;
    const int L = ctx_len[b];
    int n = n_new[b];
    if (n < 0 || n > n_max || L + n > max_ctx) {
        atomicOr(err, DFLARE_DEVERR_CAPACITY);
        n = 0;
    }
    app_base[b] = L;
    app_cnt[b] = n;
    ctx_len[b] = L + n;
}

template <class T, int DMAX>
__global__ void __launch_bounds__(512) fuse_layers_kernel(
    const T* __restrict__ H, const float* __restrict__ alpha, const T* __restrict__ gain,
    T* __restrict__ F, T* __restrict__ F_out, const int32_t* __restrict__ app_cnt, int D, int Tn,
    int batch, int n_max, int d, long long f_layer_rows, float eps) {
    pdl_trigger();
    pdl_wait();
    __shared__ float s_alpha[16 * 64];
    __shared__ float red[32][DMAX];
    const int r = blockIdx.x, b = blockIdx.y;
    for (int k = threadIdx.x; k < D * Tn; k += blockDim.x) s_alpha[k] = alpha[k];
    __syncthreads();
    if (r >= app_cnt[b]) return;
    const int e0 = threadIdx.x * 8;
    const bool act = e0 < d;
    const size_t row = (size_t)b * n_max + r;
    const size_t lstride = (size_t)batch * n_max * d;
    const T* hrow = H + row * d + (act ? e0 : 0);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;

    for (int i0 = 0; i0 < D; i0 += DMAX) {
        const int nd = min(DMAX, D - i0);
        float acc[DMAX][8];
#pragma unroll
        for (int i = 0; i < DMAX; ++i)
#pragma unroll
            for (int e = 0; e < 8; ++e) acc[i][e] = 0.f;
        if (act) {
            for (int j0 = 0; j0 < Tn; j0 += 4) {
                float h[4][8];
#pragma unroll
                for (int u = 0; u < 4; ++u)
                    if (j0 + u < Tn) load8(hrow + (size_t)(j0 + u) * lstride, h[u]);
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    if (j0 + u >= Tn) break;
#pragma unroll
                    for (int i = 0; i < DMAX; ++i) {
                        if (i < nd) {
                            const float a = s_alpha[(i0 + i) * Tn + j0 + u];
#pragma unroll
                            for (int e = 0; e < 8; ++e) acc[i][e] = fmaf(a, h[u][e], acc[i][e]);
                        }
                    }
                }
            }
        }
        // sum of squares of every draft layer's fused row, one reduction for all of them
        float ss[DMAX];
#pragma unroll
        for (int i = 0; i < DMAX; ++i) {
            float v = 0.f;
#pragma unroll
            for (int e = 0; e < 8; ++e) v = fmaf(acc[i][e], acc[i][e], v);
            ss[i] = warp_sum(v);
        }
        __syncthreads();
        if (lane == 0)
#pragma unroll
            for (int i = 0; i < DMAX; ++i) red[warp][i] = ss[i];
        __syncthreads();
#pragma unroll
        for (int i = 0; i < DMAX; ++i) {
            float s = 0.f;
            for (int w = 0; w < nw; ++w) s += red[w][i];
            ss[i] = s;
        }
        if (act) {
#pragma unroll
            for (int i = 0; i < DMAX; ++i) {
                if (i >= nd) break;
                const float inv = inv_rms(ss[i], d, eps);
                float g[8], o[8];
                load8(gain + (size_t)(i0 + i) * d + e0, g);
#pragma unroll
                for (int e = 0; e < 8; ++e) o[e] = g[e] * (acc[i][e] * inv);
                store8(F + ((size_t)(i0 + i) * f_layer_rows + row) * d + e0, o);
                if (F_out) store8(F_out + (((size_t)(i0 + i) * batch + b) * n_max + r) * d + e0, o);
            }
        }
    }
}

template <class T>
cudaError_t fuse_layers_t(dflare_ctx* c, const void* hidden, int n_max, void* fused_out,
                          cudaStream_t s) {
    const dflare_config& g = c->cfg;
    const dim3 grid(n_max, c->batch), block(((g.d / 8 + 31) / 32) * 32);
    const T* H = static_cast<const T*>(hidden);
    const T* gain = static_cast<const T*>(c->w.fuse_norm);
    T* F = static_cast<T*>(c->fused);
    T* Fo = static_cast<T*>(fused_out);
    auto kern = g.n_draft_layers <= 4 ? fuse_layers_kernel<T, 4> : fuse_layers_kernel<T, 8>;
    return launch_kernel(c->pdl, kern, grid, block, 0, s, H, (const float*)c->alpha, gain, F, Fo,
                         (const int32_t*)c->app_cnt, g.n_draft_layers, g.n_target_layers, c->batch,
                         n_max, g.d, (long long)g.max_fuse_rows, g.rms_eps);
}

}  // namespace

cudaError_t launch_fusion_alpha(dflare_ctx* c, cudaStream_t s) {
    const dflare_config& g = c->cfg;
    return launch_kernel(c->pdl, fusion_alpha_kernel, dim3(1),
                         dim3(32 * ((g.n_draft_layers + 31) / 32)), 0, s,
                         (const float*)c->w.fuse_logits, c->alpha, g.n_draft_layers,
                         g.n_target_layers, (g.flags & DFLARE_FLAG_RAW_FUSION) ? 1 : 0);
}

cudaError_t launch_fuse_begin(dflare_ctx* c, const int32_t* n_new, int n_max, cudaStream_t s) {
    return launch_kernel(c->pdl, fuse_begin_kernel, dim3(1), dim3(64), 0, s, c->ctx_len,
                         c->app_base, c->app_cnt, n_new, c->batch, n_max, c->cfg.max_ctx, c->err);
}

cudaError_t launch_fuse_layers(dflare_ctx* c, const void* hidden, int n_max, void* fused_out,
                               cudaStream_t s) {
    if (c->cfg.dtype == DFLARE_F32) return fuse_layers_t<float>(c, hidden, n_max, fused_out, s);
    return fuse_layers_t<bf16>(c, hidden, n_max, fused_out, s);
}

}  // namespace dfl
