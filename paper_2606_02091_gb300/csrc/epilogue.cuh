// Epilogues of the projection GEMMs, shared by the tcgen05 and the CUDA-core GEMM.
//
// Both GEMMs hand over a tile of fp32 accumulators for 128 consecutive output features and `nc`
// consecutive token rows, laid out [accumulator][token][feature] in shared memory. Thread t
// (0..127) writes output feature n_tile*128 + t for every token of the tile; the rotary
// embedding pairs feature j with j +- head_dim/2, which lies in the same tile because every head
// is 64 or 128 features wide and the Q, K, V regions start on multiples of 128.
#pragma once
#include "common.cuh"
#include "internal.h"

namespace dfl {

__device__ __forceinline__ float silu_f(float g) { return g / (1.0f + expf(-g)); }

template <class T>
__device__ __forceinline__ void apply_epilogue(const EpiParams& ep, const float* tile, int nc,
                                               int group, int n_tile, int tok0, int t) {
    const int n = n_tile * 128 + t;
    if (n >= ep.n) return;
    const int hd = ep.head_dim, half = hd >> 1;
    switch (ep.kind) {
        case EPI_STORE: {
            T* out = reinterpret_cast<T*>(ep.out);
            for (int c = 0; c < nc && tok0 + c < ep.m_tok; ++c)
                out[(size_t)(tok0 + c) * ep.ldo + n] = from_f<T>(tile[c * 128 + t]);
        } break;
        case EPI_F32: {
            float* out = reinterpret_cast<float*>(ep.out);
            for (int c = 0; c < nc && tok0 + c < ep.m_tok; ++c)
                out[(size_t)(tok0 + c) * ep.ldo + n] = tile[c * 128 + t];
        } break;
        case EPI_RESID: {
            for (int c = 0; c < nc && tok0 + c < ep.m_tok; ++c)
                ep.resid[(size_t)(tok0 + c) * ep.ld_resid + n] += tile[c * 128 + t];
        } break;
        case EPI_SWIGLU: {
            T* out = reinterpret_cast<T*>(ep.out);
            const float* up = tile + nc * 128;
            for (int c = 0; c < nc && tok0 + c < ep.m_tok; ++c)
                out[(size_t)(tok0 + c) * ep.ldo + n] =
                    from_f<T>(silu_f(tile[c * 128 + t]) * up[c * 128 + t]);
        } break;
        case EPI_QKV: {
            int col, ld, rot;
            T* dst;
            if (n < ep.d_q) {
                col = n; ld = ep.d_q; dst = reinterpret_cast<T*>(ep.q); rot = ep.rope;
            } else if (n < ep.d_q + ep.d_kv) {
                col = n - ep.d_q; ld = ep.d_kv; dst = reinterpret_cast<T*>(ep.kd); rot = ep.rope;
            } else {
                col = n - ep.d_q - ep.d_kv; ld = ep.d_kv; dst = reinterpret_cast<T*>(ep.vd); rot = 0;
            }
            const int j = col % hd;
            const int tp = j < half ? t + half : t - half;
            for (int c = 0; c < nc && tok0 + c < ep.m_tok; ++c) {
                const int tok = tok0 + c;
                float v = tile[c * 128 + t];
                if (rot) {
                    const int b = tok / ep.block, k = tok - b * ep.block;
                    const int pos = ep.ctx_len[b] + k;
                    const float cs = ep.rope_cos[(size_t)pos * half + (j % half)];
                    const float sn = ep.rope_sin[(size_t)pos * half + (j % half)];
                    const float y = tile[c * 128 + tp];
                    v = j < half ? v * cs - y * sn : v * cs + y * sn;
                }
                dst[(size_t)tok * ld + col] = from_f<T>(v);
            }
        } break;
        case EPI_KV_APPEND: {
            const bool is_k = n < ep.d_kv;
            const int col = is_k ? n : n - ep.d_kv;
            const int g = col / hd, j = col - g * hd;
            const int tp = j < half ? t + half : t - half;
            const int hkv = ep.d_kv / hd;
            T* cache = reinterpret_cast<T*>(is_k ? ep.kcache : ep.vcache);
            for (int c = 0; c < nc && tok0 + c < ep.m_tok; ++c) {
                const int tok = tok0 + c;
                const int b = tok / ep.n_max, r = tok - b * ep.n_max;
                if (r >= ep.app_cnt[b]) continue;
                const int pos = ep.app_base[b] + r;
                float v = tile[c * 128 + t];
                if (is_k) {
                    const float cs = ep.rope_cos[(size_t)pos * half + (j % half)];
                    const float sn = ep.rope_sin[(size_t)pos * half + (j % half)];
                    const float y = tile[c * 128 + tp];
                    v = j < half ? v * cs - y * sn : v * cs + y * sn;
                }
                const size_t row = (((size_t)group * ep.max_batch + b) * hkv + g) * ep.max_ctx + pos;
                cache[row * hd + j] = from_f<T>(v);
            }
        } break;
        default:
            break;
    }
}

}  // namespace dfl
