// Block embedding (+ the first pre-attention RMSNorm), RMSNorm, greedy argmax, prefix
// acceptance and the synthetic target used by the benchmark loop.
#include <math.h>

#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace dfl {
namespace {

// X^0 = [E[x_t]; E[mask] x (B-1)] (Sec. 3.2: the block is the target decode token followed by
// B-1 mask positions, embedded with the target's shared table, Sec. 3.3), kept in fp32, and the
// first layer's normalised input RMSNorm(X^0) in the storage type.
// qkv32 (when given, n32 floats per block row) is cleared here, at the start of every drafted
// block, so that the first layer's Q/K^d/V^d reductions start from zero even after an aborted call.
template <class T>
__global__ void embed_kernel(const T* __restrict__ E, const int32_t* __restrict__ last_token,
                             int mask_id, int V, int B, int d, float* __restrict__ X,
                             T* __restrict__ Xn, const T* __restrict__ gain, float eps,
                             uint32_t* err, float* __restrict__ qkv32, int n32) {
    pdl_trigger();
    pdl_wait();
    __shared__ float red[32];
    const int k = blockIdx.x, b = blockIdx.y;
    if (qkv32) {
        float4* z = reinterpret_cast<float4*>(qkv32 + ((size_t)b * B + k) * n32);
        for (int i = threadIdx.x; i < n32 / 4; i += blockDim.x) z[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
    int tok = k == 0 ? last_token[b] : mask_id;
    if (tok < 0 || tok >= V) {
        if (threadIdx.x == 0) atomicOr(err, DFLARE_DEVERR_TOKEN);
        tok = 0;
    }
    const size_t row = (size_t)b * B + k;
    const int e0 = threadIdx.x * 8;
    const bool act = e0 < d;
    float v[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    float ss = 0.f;
    if (act) {
        load8(E + (size_t)tok * d + e0, v);
        store8(X + row * d + e0, v);
#pragma unroll
        for (int e = 0; e < 8; ++e) ss = fmaf(v[e], v[e], ss);
    }
    ss = block_sum(ss, red);
    if (act) {
        const float inv = inv_rms(ss, d, eps);
        float g[8], o[8];
        load8(gain + e0, g);
#pragma unroll
        for (int e = 0; e < 8; ++e) o[e] = g[e] * (v[e] * inv);
        store8(Xn + row * d + e0, o);
    }
}

// out[r] = gain * X[row(r)] / sqrt(mean(X^2) + eps). With `gather`, output row r reads the mask
// row k = r % (B-1) + 1 of sequence r / (B-1) (the LM head only needs the mask positions). With
// zero32, row r of it (n32 floats) is cleared: the fp32 sums the next Q/K^d/V^d projection adds
// into (the previous layer's attention, which read them, is complete by now).
template <class T>
__global__ void rmsnorm_kernel(const float* __restrict__ X, const T* __restrict__ gain,
                               T* __restrict__ out, int d, int B, int gather, float eps,
                               float* __restrict__ zero32, int n32) {
    pdl_trigger();
    const int e0 = threadIdx.x * 8;
    const bool act = e0 < d;
    float g[8];
    if (act) load8(gain + e0, g);   // a weight: read before the dependency wait
    pdl_wait();
    __shared__ float red[32];
    const int r = blockIdx.x;
    if (zero32) {
        float4* z = reinterpret_cast<float4*>(zero32 + (size_t)r * n32);
        for (int i = threadIdx.x; i < n32 / 4; i += blockDim.x) z[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
    const size_t in_row = gather ? (size_t)(r / (B - 1)) * B + (r % (B - 1)) + 1 : (size_t)r;
    float v[8];
    float ss = 0.f;
    if (act) {
        load8(X + in_row * d + e0, v);
#pragma unroll
        for (int e = 0; e < 8; ++e) ss = fmaf(v[e], v[e], ss);
    }
    ss = block_sum(ss, red);
    if (act) {
        const float inv = inv_rms(ss, d, eps);
        float o[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) o[e] = g[e] * (v[e] * inv);
        store8(out + (size_t)r * d + e0, o);
    }
}

// Order-preserving map of a float onto uint32 (-0 and +0 map to the same key).
__device__ __forceinline__ uint32_t ordered_key(float v) {
    uint32_t u = __float_as_uint(v);
    if (v == 0.f) u = 0u;
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Greedy argmax over the vocabulary (lowest id among equal maxima). Grid (chunks, rows): each
// CTA reduces a chunk of one row with warp shuffles and publishes (key(value), ~index) through a
// 64-bit atomicMax; the last CTA to finish turns the packed maxima into token ids and re-arms
// the slots and the counter for the next launch. NaN entries are never chosen. A row without a
// value above -inf publishes nothing; the last CTA then takes its first -inf entry (the lowest
// id among equal maxima), or id 0 when every entry is NaN.
__global__ void __launch_bounds__(256) argmax_kernel(const float* __restrict__ logits, int V,
                                                     int rows, int chunk,
                                                     unsigned long long* slot, uint32_t* cnt,
                                                     int32_t* __restrict__ tokens) {
    pdl_trigger();
    pdl_wait();
    __shared__ float sv[8];
    __shared__ int si[8];
    __shared__ int last;
    const int row = blockIdx.y;
    const int c0 = blockIdx.x * chunk, c1 = min(V, c0 + chunk);
    const float* p = logits + (size_t)row * V;
    float bv = -INFINITY;
    int bi = 0x7fffffff;
    if ((V & 3) == 0) {
        // four 16-byte loads in flight per thread (a scan with one load per iteration waits a
        // full memory round trip per 16 bytes); ids ascend within a thread, so ">" keeps the
        // lowest id of equal maxima; a load past the chunk reads as -inf, never chosen
        constexpr int U = 4;
        const int stride = blockDim.x * 4;
        for (int base = c0 + threadIdx.x * 4; base < c1; base += stride * U) {
            float4 q[U];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int i = base + u * stride;
                q[u] = i < c1 ? *reinterpret_cast<const float4*>(p + i)
                              : make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
            }
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int i = base + u * stride;
                if (q[u].x > bv) { bv = q[u].x; bi = i; }
                if (q[u].y > bv) { bv = q[u].y; bi = i + 1; }
                if (q[u].z > bv) { bv = q[u].z; bi = i + 2; }
                if (q[u].w > bv) { bv = q[u].w; bi = i + 3; }
            }
        }
    } else {
        for (int i = c0 + threadIdx.x; i < c1; i += blockDim.x) {
            const float q = p[i];
            if (q > bv) { bv = q; bi = i; }
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
        const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
        if (ov > bv || (ov == bv && oi < bi)) { bv = ov; bi = oi; }
    }
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (lane == 0) { sv[warp] = bv; si[warp] = bi; }
    __syncthreads();
    if (threadIdx.x == 0) {
        for (int w = 1; w < (int)(blockDim.x >> 5); ++w)
            if (sv[w] > bv || (sv[w] == bv && si[w] < bi)) { bv = sv[w]; bi = si[w]; }
        if (bi != 0x7fffffff) {
            const unsigned long long key =
                ((unsigned long long)ordered_key(bv) << 32) | (0xFFFFFFFFu - (uint32_t)bi);
            atomicMax(&slot[row], key);
        }
        __threadfence();
        const uint32_t prev = atomicAdd(cnt, 1u);
        last = prev == gridDim.x * gridDim.y - 1;
    }
    __syncthreads();
    if (last) {
        __threadfence();
        for (int r = threadIdx.x; r < rows; r += blockDim.x) {
            const unsigned long long key = atomicExch(&slot[r], 0ull);
            int32_t tok = (int32_t)(0xFFFFFFFFu - (uint32_t)(key & 0xFFFFFFFFull));
            if (key == 0ull) {   // no entry above -inf: a serial scan, only for such rows
                const float* pr = logits + (size_t)r * V;
                tok = 0;
                for (int i = 0; i < V; ++i)
                    if (pr[i] == -INFINITY) { tok = i; break; }
            }
            tokens[r] = tok;
        }
        if (threadIdx.x == 0) *cnt = 0;
    }
}

// Prefix acceptance (Sec. 3.2, verification): one warp per sequence; lane l compares d_{l+1}
// with g_l, the first mismatch ends the accepted prefix.
__global__ void verify_kernel(const int32_t* __restrict__ draft, const int32_t* __restrict__ target,
                              int32_t* __restrict__ accept_len, int32_t* __restrict__ next_token,
                              int batch, int B) {
    pdl_trigger();
    pdl_wait();
    const int lane = threadIdx.x & 31;
    const int b = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (b >= batch) return;
    bool mism = false;
    if (lane < B - 1) mism = draft[(size_t)b * (B - 1) + lane] != target[(size_t)b * B + lane];
    const unsigned m = __ballot_sync(0xffffffffu, mism);
    const int a = m ? __ffs(m) - 1 : B - 1;
    if (lane == 0) {
        accept_len[b] = a + 1;
        next_token[b] = target[(size_t)b * B + a];
    }
}

__global__ void synth_target_kernel(const int32_t* __restrict__ draft, const uint32_t* __restrict__ u,
                                    const int32_t* __restrict__ r, const int32_t* __restrict__ last,
                                    int n_steps, int32_t* step, uint32_t thr, int batch, int B,
                                    int32_t* __restrict__ g) {
    pdl_trigger();
    pdl_wait();
    const int s = *step % n_steps;
    for (int idx = threadIdx.x; idx < batch * B; idx += blockDim.x) {
        const int b = idx / B, k = idx % B;
        if (k == B - 1) {
            g[idx] = last[(size_t)s * batch + b];
        } else {
            const size_t o = ((size_t)s * batch + b) * (B - 1) + k;
            const int dk = draft[(size_t)b * (B - 1) + k];
            g[idx] = u[o] < thr ? dk : r[o] + (r[o] >= dk ? 1 : 0);
        }
    }
    __syncthreads();
    if (threadIdx.x == 0) *step = (s + 1) % n_steps;
}

}  // namespace

cudaError_t launch_embed(dflare_ctx* c, const int32_t* last_token, cudaStream_t s) {
    const dflare_config& g = c->cfg;
    const dim3 grid(g.block, c->batch), block(((g.d / 8 + 31) / 32) * 32);
    if (g.dtype == DFLARE_F32)
        return launch_kernel(c->pdl, embed_kernel<float>, grid, block, 0, s,
                             (const float*)c->w.embed, last_token, g.mask_token_id, g.vocab, g.block,
                             g.d, c->x, (float*)c->xn, (const float*)c->w.attn_norm, g.rms_eps,
                             c->err, (float*)nullptr, 0);
    return launch_kernel(c->pdl, embed_kernel<bf16>, grid, block, 0, s, (const bf16*)c->w.embed,
                         last_token, g.mask_token_id, g.vocab, g.block, g.d, c->x, (bf16*)c->xn,
                         (const bf16*)c->w.attn_norm, g.rms_eps, c->err, c->qkv32,
                         (g.n_q_heads + 2 * g.n_kv_heads) * g.head_dim);
}

cudaError_t launch_rmsnorm(dflare_ctx* c, const void* gain, int rows, bool gather, void* out,
                           cudaStream_t s, float* zero32) {
    const dflare_config& g = c->cfg;
    if (rows <= 0) return cudaSuccess;
    const dim3 block(((g.d / 8 + 31) / 32) * 32);
    const int n32 = (g.n_q_heads + 2 * g.n_kv_heads) * g.head_dim;
    if (g.dtype == DFLARE_F32)
        return launch_kernel(c->pdl, rmsnorm_kernel<float>, dim3(rows), block, 0, s, c->x,
                             (const float*)gain, (float*)out, g.d, g.block, gather ? 1 : 0,
                             g.rms_eps, zero32, n32);
    return launch_kernel(c->pdl, rmsnorm_kernel<bf16>, dim3(rows), block, 0, s, c->x,
                         (const bf16*)gain, (bf16*)out, g.d, g.block, gather ? 1 : 0, g.rms_eps,
                         zero32, n32);
}

cudaError_t launch_argmax(dflare_ctx* c, const float* logits, int rows, int32_t* tokens,
                          cudaStream_t s) {
    if (rows <= 0) return cudaSuccess;
    const int V = c->cfg.vocab;
    // about four CTAs per SM (measured against two: 0.5207 -> 0.5195 ms per Qwen3-4B-shaped step;
    // one: 0.5225 ms): chunks of at least 4096 ids, a multiple of 1024
    int chunks = std::max(1, (4 * c->num_sms + rows - 1) / rows);
    int chunk = (V + chunks - 1) / chunks;
    chunk = std::max(4096, ((chunk + 1023) / 1024) * 1024);
    chunks = (V + chunk - 1) / chunk;
    return launch_kernel(c->pdl, argmax_kernel, dim3(chunks, rows), dim3(256), 0, s, logits, V,
                         rows, chunk, c->amax_slot, c->amax_cnt, tokens);
}

cudaError_t launch_verify(dflare_ctx* c, const int32_t* draft, const int32_t* target,
                          int32_t* accept_len, int32_t* next_token, cudaStream_t s) {
    const int per = 4;
    return launch_kernel(c->pdl, verify_kernel, dim3((c->batch + per - 1) / per), dim3(32 * per), 0,
                         s, draft, target, accept_len, next_token, c->batch, c->cfg.block);
}

cudaError_t launch_synthetic_target(const int32_t* draft, const uint32_t* u, const int32_t* r,
                                    const int32_t* last, int n_steps, int32_t* step,
                                    uint32_t threshold, int batch, int block, int32_t* target,
                                    cudaStream_t s) {
    return launch_kernel(true, synth_target_kernel, dim3(1), dim3(256), 0, s, draft, u, r, last,
                         n_steps, step, threshold, batch, block, target);
}

}  // namespace dfl
