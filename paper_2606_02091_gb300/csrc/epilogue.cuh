// Epilogues of the projection GEMMs, shared by the tcgen05 and the CUDA-core GEMM.
//
// Both GEMMs hand over a tile of fp32 accumulators for 128 consecutive output features and 16
// consecutive token rows, laid out [accumulator][token][feature] in shared memory. Thread t
// (0..127) writes output feature n_tile*128 + t for every token of the tile; the rotary
// embedding pairs feature j with j +- head_dim/2, which lies in the same tile because every head
// is 64 or 128 features wide and the Q, K, V regions start on multiples of 128.
#pragma once
#include "common.cuh"
#include "internal.h"

namespace dfl {

constexpr int kEpiChunk = 16;   // tokens per epilogue tile

// silu(g) = g / (1 + e^-g) with the fast exponential and division intrinsics (relative error a
// few fp32 ulp, far below the bf16 rounding of the result; 1 + e^-g = inf for g < -88 gives 0)
__device__ __forceinline__ float silu_f(float g) { return __fdividef(g, 1.0f + __expf(-g)); }

// Every branch issues all of its global loads (residual values, per-token positions, rotary
// factors) before its first store, so the loads of the 16 tokens of a chunk are in flight
// together instead of each waiting behind the previous token's store.
// kAux: compile the biased, group-strided store (EPI_STORE of the fusion variants); without it
// EPI_STORE writes group 0's layout with no bias.
template <class T, bool kAux = true>
__device__ __forceinline__ void apply_epilogue(const EpiParams& ep, const float* tile, int group,
                                               int n_tile, int tok0, int t) {
    constexpr int NC = kEpiChunk;
    const int n = n_tile * 128 + t;
    if (n >= ep.n) return;
    const int hd = ep.head_dim, half = hd >> 1;
    const int nvalid = min(NC, ep.m_tok - tok0);
    if (nvalid <= 0) return;
    switch (ep.kind) {
        case EPI_STORE: {
            if constexpr (kAux) {
                T* out = reinterpret_cast<T*>(ep.out) + (size_t)group * ep.out_gstride;
                const float bv =
                    ep.bias ? to_f(reinterpret_cast<const T*>(ep.bias)[(size_t)group * ep.n + n]) : 0.f;
#pragma unroll
                for (int c = 0; c < NC; ++c)
                    if (c < nvalid)
                        out[(size_t)(tok0 + c) * ep.ldo + n] = from_f<T>(tile[c * 128 + t] + bv);
            } else {
                T* out = reinterpret_cast<T*>(ep.out);
#pragma unroll
                for (int c = 0; c < NC; ++c)
                    if (c < nvalid) out[(size_t)(tok0 + c) * ep.ldo + n] = from_f<T>(tile[c * 128 + t]);
            }
        } break;
        case EPI_F32: {
            float* out = reinterpret_cast<float*>(ep.out);
#pragma unroll
            for (int c = 0; c < NC; ++c)
                if (c < nvalid) out[(size_t)(tok0 + c) * ep.ldo + n] = tile[c * 128 + t];
        } break;
        case EPI_RESID: {
            float r[NC];
#pragma unroll
            for (int c = 0; c < NC; ++c)
                r[c] = c < nvalid ? ep.resid[(size_t)(tok0 + c) * ep.ld_resid + n] : 0.f;
#pragma unroll
            for (int c = 0; c < NC; ++c)
                if (c < nvalid) ep.resid[(size_t)(tok0 + c) * ep.ld_resid + n] = r[c] + tile[c * 128 + t];
        } break;
        case EPI_SWIGLU: {
            T* out = reinterpret_cast<T*>(ep.out);
            const float* up = tile + NC * 128;
#pragma unroll
            for (int c = 0; c < NC; ++c)
                if (c < nvalid)
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
            const int j = col % hd, jj = j % half;
            const int tp = j < half ? t + half : t - half;
            // eight tokens at a time: their positions and rotary factors are loaded together
            for (int h0 = 0; h0 < nvalid; h0 += 8) {
                float cs[8], sn[8];
                if (rot) {
                    int pos[8];
#pragma unroll
                    for (int c = 0; c < 8; ++c) {
                        const int tok = tok0 + min(h0 + c, nvalid - 1);
                        const int b = tok / ep.block;
                        pos[c] = ep.ctx_len[b] + (tok - b * ep.block);
                    }
#pragma unroll
                    for (int c = 0; c < 8; ++c) {
                        cs[c] = ep.rope_cos[(size_t)pos[c] * half + jj];
                        sn[c] = ep.rope_sin[(size_t)pos[c] * half + jj];
                    }
                }
#pragma unroll
                for (int c = 0; c < 8; ++c) {
                    if (h0 + c >= nvalid) break;
                    float v = tile[(h0 + c) * 128 + t];
                    if (rot) {
                        const float y = tile[(h0 + c) * 128 + tp];
                        v = j < half ? v * cs[c] - y * sn[c] : v * cs[c] + y * sn[c];
                    }
                    dst[(size_t)(tok0 + h0 + c) * ld + col] = from_f<T>(v);
                }
            }
        } break;
        case EPI_KV_APPEND: {
            const bool is_k = n < ep.d_kv;
            const int col = is_k ? n : n - ep.d_kv;
            const int g = col / hd, j = col - g * hd, jj = j % half;
            const int tp = j < half ? t + half : t - half;
            const int hkv = ep.d_kv / hd;
            T* cache = reinterpret_cast<T*>(is_k ? ep.kcache : ep.vcache);
            for (int h0 = 0; h0 < nvalid; h0 += 8) {
                int pos[8], ok[8], bb[8];
#pragma unroll
                for (int c = 0; c < 8; ++c) {
                    const int tok = tok0 + min(h0 + c, nvalid - 1);
                    const int b = tok / ep.n_max, r = tok - b * ep.n_max;
                    bb[c] = b;
                    ok[c] = h0 + c < nvalid && r < ep.app_cnt[b];
                    pos[c] = ep.app_base[b] + r;
                }
                float cs[8], sn[8];
                if (is_k) {
#pragma unroll
                    for (int c = 0; c < 8; ++c) {
                        const int p = ok[c] ? pos[c] : 0;
                        cs[c] = ep.rope_cos[(size_t)p * half + jj];
                        sn[c] = ep.rope_sin[(size_t)p * half + jj];
                    }
                }
#pragma unroll
                for (int c = 0; c < 8; ++c) {
                    if (!ok[c]) continue;
                    float v = tile[(h0 + c) * 128 + t];
                    if (is_k) {
                        const float y = tile[(h0 + c) * 128 + tp];
                        v = j < half ? v * cs[c] - y * sn[c] : v * cs[c] + y * sn[c];
                    }
                    const size_t row =
                        (((size_t)group * ep.max_batch + bb[c]) * hkv + g) * ep.max_ctx + pos[c];
                    cache[row * hd + j] = from_f<T>(v);
                }
            }
        } break;
        default:
            break;
    }
}

}  // namespace dfl
