// Epilogues of the projection GEMMs, shared by the tcgen05 and the CUDA-core GEMM.
//
// Both GEMMs hand over a tile of fp32 accumulators for 128 consecutive output features and 16
// consecutive token rows, laid out [accumulator][token][feature] in shared memory. Thread t
// (0..127) owns token t / 8 of the chunk and the 16 consecutive features 16 (t % 8) .. + 15 of
// the tile, so every row of output is written with 16-byte stores (two per thread for bf16, four
// for fp32) and the rotary factors of a token are read as 16-byte vectors. The rotary embedding
// pairs feature j with j +- head_dim/2, a group of 16 that lies in the same tile because every
// head is 64 or 128 features wide and the Q, K, V regions start on multiples of 128.
#pragma once
#include "common.cuh"
#include "internal.h"

namespace dfl {

constexpr int kEpiChunk = 16;   // tokens per epilogue tile

// silu(g) = g / (1 + e^-g) with the fast exponential and division intrinsics (relative error a
// few fp32 ulp, far below the bf16 rounding of the result; 1 + e^-g = inf for g < -88 gives 0)
__device__ __forceinline__ float silu_f(float g) { return __fdividef(g, 1.0f + __expf(-g)); }

__device__ __forceinline__ void ld16_smem(const float* p, float* v) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float4 q = reinterpret_cast<const float4*>(p)[i];
        v[4 * i] = q.x; v[4 * i + 1] = q.y; v[4 * i + 2] = q.z; v[4 * i + 3] = q.w;
    }
}
__device__ __forceinline__ void ld16_global(const float* p, float* v) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float4 q = __ldg(reinterpret_cast<const float4*>(p) + i);
        v[4 * i] = q.x; v[4 * i + 1] = q.y; v[4 * i + 2] = q.z; v[4 * i + 3] = q.w;
    }
}
// nv <= 16 values to dst: 16-byte stores when all 16 are valid and dst is 16-byte aligned
template <class T>
__device__ __forceinline__ void st16(T* dst, const float* v, int nv) {
    if (nv == 16 && (reinterpret_cast<uintptr_t>(dst) & 15u) == 0) {
        store8(dst, v);
        store8(dst + 8, v + 8);
    } else {
#pragma unroll
        for (int i = 0; i < 16; ++i)
            if (i < nv) dst[i] = from_f<T>(v[i]);
    }
}

// Every branch issues all of its global loads (positions, rotary factors, residual values, a
// bias) before its first store.
// kAux: compile the biased, group-strided store (EPI_STORE of the fusion variants); without it
// EPI_STORE writes group 0's layout with no bias.
template <class T, bool kAux = true>
__device__ __forceinline__ void apply_epilogue(const EpiParams& ep, const float* tile, int group,
                                               int n_tile, int tok0, int t) {
    constexpr int NC = kEpiChunk;
    const int c = t >> 3, f0 = (t & 7) * 16;
    const int tok = tok0 + c, n0 = n_tile * 128 + f0;
    if (tok >= ep.m_tok || n0 >= ep.n) return;
    const int nv = min(16, ep.n - n0);
    const float* src = tile + c * 128 + f0;
    float v[16];
    ld16_smem(src, v);
    switch (ep.kind) {
        case EPI_STORE: {
            T* out = reinterpret_cast<T*>(ep.out);
            if constexpr (kAux) {
                out += (size_t)group * ep.out_gstride;
                if (ep.bias) {
                    const T* bias = reinterpret_cast<const T*>(ep.bias) + (size_t)group * ep.n + n0;
#pragma unroll
                    for (int i = 0; i < 16; ++i)
                        if (i < nv) v[i] += to_f(bias[i]);
                }
            }
            st16(out + (size_t)tok * ep.ldo + n0, v, nv);
        } break;
        case EPI_F32:
            st16(reinterpret_cast<float*>(ep.out) + (size_t)tok * ep.ldo + n0, v, nv);
            break;
        case EPI_RESID: {
            float* dst = ep.resid + (size_t)tok * ep.ld_resid + n0;
            float r[16];
            if (nv == 16 && (reinterpret_cast<uintptr_t>(dst) & 15u) == 0) {
                ld16_global(dst, r);
            } else {
#pragma unroll
                for (int i = 0; i < 16; ++i) r[i] = i < nv ? dst[i] : 0.f;
            }
#pragma unroll
            for (int i = 0; i < 16; ++i) v[i] += r[i];
            st16(dst, v, nv);
        } break;
        case EPI_SWIGLU: {
            float up[16];
            ld16_smem(src + NC * 128, up);
#pragma unroll
            for (int i = 0; i < 16; ++i) v[i] = silu_f(v[i]) * up[i];
            st16(reinterpret_cast<T*>(ep.out) + (size_t)tok * ep.ldo + n0, v, nv);
        } break;
        case EPI_QKV: {
            // the Q, K^d and V^d regions start on multiples of 128: a group lies in one region
            const int hd = ep.head_dim, half = hd >> 1;
            int col, ld, rot;
            T* dst;
            if (n0 < ep.d_q) {
                col = n0; ld = ep.d_q; dst = reinterpret_cast<T*>(ep.q); rot = ep.rope;
            } else if (n0 < ep.d_q + ep.d_kv) {
                col = n0 - ep.d_q; ld = ep.d_kv; dst = reinterpret_cast<T*>(ep.kd); rot = ep.rope;
            } else {
                col = n0 - ep.d_q - ep.d_kv; ld = ep.d_kv; dst = reinterpret_cast<T*>(ep.vd); rot = 0;
            }
            if (rot) {
                const int j0 = col % hd, jj0 = j0 % half;
                const int b = tok / ep.block;
                const int pos = ep.ctx_len[b] + (tok - b * ep.block);
                float cs[16], sn[16], y[16];
                ld16_global(ep.rope_cos + (size_t)pos * half + jj0, cs);
                ld16_global(ep.rope_sin + (size_t)pos * half + jj0, sn);
                ld16_smem(src + (j0 < half ? half : -half), y);
#pragma unroll
                for (int i = 0; i < 16; ++i)
                    v[i] = j0 < half ? v[i] * cs[i] - y[i] * sn[i] : v[i] * cs[i] + y[i] * sn[i];
            }
            st16(dst + (size_t)tok * ld + col, v, nv);
        } break;
        case EPI_KV_APPEND: {
            const int hd = ep.head_dim, half = hd >> 1;
            const int b = tok / ep.n_max, r = tok - b * ep.n_max;
            if (r >= ep.app_cnt[b]) return;
            const int pos = ep.app_base[b] + r;
            const bool is_k = n0 < ep.d_kv;
            const int col = is_k ? n0 : n0 - ep.d_kv;
            const int g = col / hd, j0 = col - g * hd;
            if (is_k) {
                const int jj0 = j0 % half;
                float cs[16], sn[16], y[16];
                ld16_global(ep.rope_cos + (size_t)pos * half + jj0, cs);
                ld16_global(ep.rope_sin + (size_t)pos * half + jj0, sn);
                ld16_smem(src + (j0 < half ? half : -half), y);
#pragma unroll
                for (int i = 0; i < 16; ++i)
                    v[i] = j0 < half ? v[i] * cs[i] - y[i] * sn[i] : v[i] * cs[i] + y[i] * sn[i];
            }
            T* cache = reinterpret_cast<T*>(is_k ? ep.kcache : ep.vcache);
            const int hkv = ep.d_kv / hd;
            const size_t row = (((size_t)group * ep.max_batch + b) * hkv + g) * ep.max_ctx + pos;
            st16(cache + row * hd + j0, v, nv);
        } break;
        default:
            break;
    }
}

}  // namespace dfl
