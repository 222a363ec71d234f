// Sampled decoding at temperature T (the temperature-1 half of Table 1).
//
// Drafting: each mask row's token is a draw from softmax(logits / T) in the Gumbel-max form,
// argmax_v (l_v / T - log(-log u_v)).
//
// Verification: the paper reports sampled decoding without its acceptance rule; this follows the
// speculative-sampling rule of the works it builds on. Draft token d_k is kept with probability
// min(1, p(d_k) / q(d_k)) (p: the target's softmax at that position, q: the draft's), i.e. when
// r_k q(d_k) < p(d_k); the first rejected position is redrawn from max(0, p - q), and when every
// draft is kept the extra token is drawn from the target's distribution after the last block row.
//
// Random numbers: Philox4x64-10 (Salmon, Moraes, Dror, Shaw, "Parallel random numbers: as easy
// as 1, 2, 3", SC'11), written here from that definition. Output word w of stream (purpose,
// step, row) is word w mod 4 of the block at counter (1 + w / 4, row, step, purpose) under key
// (seed, 0); it gives element 2w from its bits 63..41 and element 2w + 1 from its bits 31..9,
// each as (23-bit integer + 1/2) 2^-23, a value in (0, 1) that fp32 holds exactly. One block
// thus serves eight elements (the Philox rounds are the drafting kernel's main cost). The step
// is read from a device counter that the verification advances, so a captured graph of a
// draft-verify step draws fresh numbers on every replay.
#include <math.h>

#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace dfl {
namespace {

constexpr uint64_t kPhiloxM0 = 0xD2E7470EE14C6C93ull, kPhiloxM1 = 0xCA5A826395121157ull;
constexpr uint64_t kWeyl0 = 0x9E3779B97F4A7C15ull, kWeyl1 = 0xBB67AE8584CAA73Bull;
constexpr uint64_t kRngDraft = 1, kRngAccept = 2, kRngResidual = 3;
constexpr int kNone = 0x7fffffff;
constexpr int kU = 4;   // groups of four logits a thread loads at once in the vocabulary scans
constexpr int kDrawU = 2;   // groups of eight logits (one Philox block each) per thread and iteration

__device__ __forceinline__ float unit_from_bits(uint64_t x) {   // bits 63..41
    return ((float)(x >> 41) + 0.5f) * 0x1p-23f;
}
__device__ __forceinline__ float unit_from_low_bits(uint64_t x) {   // bits 31..9
    return ((float)((uint32_t)(x >> 9) & 0x7FFFFFu) + 0.5f) * 0x1p-23f;
}

// The eight uniforms of block `blk` of stream (purpose, step, row): elements 8 (blk - 1) .. + 7.
__device__ __forceinline__ void philox_uniforms(uint64_t blk, uint64_t row, uint64_t step,
                                                uint64_t purpose, uint64_t seed, float* u) {
    uint64_t c0 = blk, c1 = row, c2 = step, c3 = purpose, k0 = seed, k1 = 0;
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        if (r) {
            k0 += kWeyl0;
            k1 += kWeyl1;
        }
        const uint64_t hi0 = __umul64hi(kPhiloxM0, c0), lo0 = kPhiloxM0 * c0;
        const uint64_t hi1 = __umul64hi(kPhiloxM1, c2), lo1 = kPhiloxM1 * c2;
        c0 = hi1 ^ c1 ^ k0;
        c1 = lo1;
        c2 = hi0 ^ c3 ^ k1;
        c3 = lo0;
    }
    u[0] = unit_from_bits(c0);
    u[1] = unit_from_low_bits(c0);
    u[2] = unit_from_bits(c1);
    u[3] = unit_from_low_bits(c1);
    u[4] = unit_from_bits(c2);
    u[5] = unit_from_low_bits(c2);
    u[6] = unit_from_bits(c3);
    u[7] = unit_from_low_bits(c3);
}

__device__ __forceinline__ float gumbel(float u) { return -logf(-logf(u)); }

__device__ __forceinline__ uint32_t order_key(float v) {
    uint32_t u = __float_as_uint(v);
    if (v == 0.f) u = 0u;
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Block-wide maximum of (score, index) with the lowest index among equal scores, folded into
// slot[row] as (ordered score, ~index) by a 64-bit atomicMax. Returns true in the CTA that
// arrives last at *cnt (after a fence), which then owns every slot.
__device__ __forceinline__ bool publish_max(float bv, int bi, unsigned long long* slot_row,
                                            uint32_t* cnt, uint32_t n_ctas) {
    __shared__ float sv[8];
    __shared__ int si[8];
    __shared__ int last;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
        const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
        if (ov > bv || (ov == bv && oi < bi)) {
            bv = ov;
            bi = oi;
        }
    }
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (lane == 0) {
        sv[warp] = bv;
        si[warp] = bi;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        for (int w = 1; w < (int)(blockDim.x >> 5); ++w)
            if (sv[w] > bv || (sv[w] == bv && si[w] < bi)) {
                bv = sv[w];
                bi = si[w];
            }
        if (bi != kNone)
            atomicMax(slot_row, ((unsigned long long)order_key(bv) << 32) | (0xFFFFFFFFu - (uint32_t)bi));
        __threadfence();
        last = atomicAdd(cnt, 1u) == n_ctas - 1;
    }
    __syncthreads();
    if (last) __threadfence();
    return last;
}

__device__ __forceinline__ int32_t slot_token(unsigned long long key) {
    return (int32_t)(0xFFFFFFFFu - (uint32_t)(key & 0xFFFFFFFFull));
}

// Four consecutive logits [i, i + 4) of a row (16-byte load when the row is 16-byte aligned);
// entries at or past c1 read as NaN, which is never chosen.
__device__ __forceinline__ void load4(const float* p, int i, int c1, bool vec, float* x) {
    if (vec && i + 4 <= c1) {
        const float4 q = *reinterpret_cast<const float4*>(p + i);
        x[0] = q.x; x[1] = q.y; x[2] = q.z; x[3] = q.w;
    } else {
#pragma unroll
        for (int e = 0; e < 4; ++e) x[e] = i + e < c1 ? p[i + e] : __int_as_float(0x7fc00000);
    }
}

// ---------------------------------------------------------------------------------- drafting
// Grid (chunks, rows), chunk a multiple of 8: every thread takes groups of eight logits and the
// one Philox block that covers them.
__global__ void __launch_bounds__(256) sample_kernel(const float* __restrict__ logits, int V, int rows,
                                                     int chunk, float inv_t, uint64_t seed,
                                                     const uint64_t* __restrict__ step_dev,
                                                     unsigned long long* slot, uint32_t* cnt,
                                                     int32_t* __restrict__ tokens) {
    pdl_trigger();
    pdl_wait();
    const uint64_t step = *step_dev;
    const int row = blockIdx.y;
    const int c0 = blockIdx.x * chunk, c1 = min(V, c0 + chunk);
    const float* p = logits + (size_t)row * V;
    const bool vec = (V & 3) == 0;
    float bv = -INFINITY;
    int bi = kNone;
    // kDrawU groups of eight logits (one Philox block each) per thread and iteration, all loads
    // issued before the first block (ids ascend within a thread, so ">" keeps the lowest id of
    // equal scores)
    const int stride = blockDim.x * 8;
    for (int base = c0 + threadIdx.x * 8; base < c1; base += stride * kDrawU) {
        float x[kDrawU][8];
#pragma unroll
        for (int g = 0; g < kDrawU; ++g) {
            load4(p, base + g * stride, c1, vec, x[g]);
            load4(p, base + g * stride + 4, c1, vec, x[g] + 4);
        }
#pragma unroll
        for (int g = 0; g < kDrawU; ++g) {
            const int i = base + g * stride;
            if (i >= c1) break;
            float u[8];
            philox_uniforms(1 + (uint64_t)(i >> 3), (uint64_t)row, step, kRngDraft, seed, u);
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                const float sc = x[g][e] * inv_t + gumbel(u[e]);
                if (sc > bv) {
                    bv = sc;
                    bi = i + e;
                }
            }
        }
    }
    if (publish_max(bv, bi, &slot[row], cnt, gridDim.x * gridDim.y)) {
        for (int r = threadIdx.x; r < rows; r += blockDim.x) {
            const unsigned long long key = atomicExch(&slot[r], 0ull);
            int32_t tok = slot_token(key);
            if (key == 0ull) {   // nothing above -inf: the first -inf entry, else id 0
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

// ------------------------------------------------------------------------------ verification
// Softmax statistics (max m and sum of exp(l/T - m)) of every target row (batch x B, first) and
// every draft row (batch x (B-1)), per chunk of the vocabulary: part[row][chunk] = (m, s).
__global__ void __launch_bounds__(256) spec_stats_kernel(const float* __restrict__ target,
                                                         const float* __restrict__ draft, int V,
                                                         int n_target_rows, int chunk, float inv_t,
                                                         float2* __restrict__ part) {
    pdl_trigger();
    pdl_wait();
    const int r = blockIdx.y;
    const int c0 = blockIdx.x * chunk, c1 = min(V, c0 + chunk);
    const float* p = r < n_target_rows ? target + (size_t)r * V
                                       : draft + (size_t)(r - n_target_rows) * V;
    float m = -INFINITY, s = 0.f;
    // kU groups of four logits per thread and iteration, loaded before they are used; the
    // group's maximum updates the running maximum once, then its terms are added
    const bool vec = (V & 3) == 0;
    const int stride = blockDim.x * 4;
    for (int base = c0 + threadIdx.x * 4; base < c1; base += stride * kU) {
        float x[kU][4];
#pragma unroll
        for (int g = 0; g < kU; ++g) load4(p, base + g * stride, c1, vec, x[g]);
        float gm = -INFINITY;
#pragma unroll
        for (int g = 0; g < kU; ++g)
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                x[g][e] *= inv_t;   // NaN past the chunk: fmaxf ignores it, the test below skips it
                gm = fmaxf(gm, x[g][e]);
            }
        if (gm > m) {
            s = m > -INFINITY ? s * expf(m - gm) : 0.f;
            m = gm;
        }
        if (m > -INFINITY) {
#pragma unroll
            for (int g = 0; g < kU; ++g)
#pragma unroll
                for (int e = 0; e < 4; ++e)
                    if (x[g][e] > -INFINITY) s += expf(x[g][e] - m);
        }
    }
    __shared__ float sm[8], ss[8];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float om = __shfl_xor_sync(0xffffffffu, m, o);
        const float os = __shfl_xor_sync(0xffffffffu, s, o);
        const float M = fmaxf(m, om);
        if (M > -INFINITY) s = (m > -INFINITY ? s * expf(m - M) : 0.f) + (om > -INFINITY ? os * expf(om - M) : 0.f);
        m = M;
    }
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (lane == 0) {
        sm[warp] = m;
        ss[warp] = s;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        for (int w = 1; w < (int)(blockDim.x >> 5); ++w) {
            const float M = fmaxf(m, sm[w]);
            if (M > -INFINITY)
                s = (m > -INFINITY ? s * expf(m - M) : 0.f) + (sm[w] > -INFINITY ? ss[w] * expf(sm[w] - M) : 0.f);
            m = M;
        }
        part[(size_t)r * gridDim.x + blockIdx.x] = make_float2(m, s);
    }
}

// (max, normaliser) of one row from its chunk partials
__device__ __forceinline__ float2 row_stats(const float2* part, int row, int chunks) {
    float m = -INFINITY, s = 0.f;
#pragma unroll 8
    for (int c = 0; c < chunks; ++c) {
        const float2 q = part[(size_t)row * chunks + c];
        const float M = fmaxf(m, q.x);
        if (M > -INFINITY)
            s = (m > -INFINITY ? s * expf(m - M) : 0.f) + (q.x > -INFINITY ? q.y * expf(q.x - M) : 0.f);
        m = M;
    }
    return make_float2(m, s);
}

// One warp per sequence: lane j decides draft token d_{j+1} (target row j, draft row j, uniform
// j of the acceptance stream); a = the first rejected position (B-1 when none) goes to spec_a.
__global__ void __launch_bounds__(32) spec_accept_kernel(const float* __restrict__ target,
                                                         const float* __restrict__ draft_logits,
                                                         const int32_t* __restrict__ draft, int V,
                                                         int B, int batch, int chunks, float inv_t,
                                                         uint64_t seed, const uint64_t* __restrict__ step_dev,
                                                         const float2* __restrict__ part,
                                                         int32_t* __restrict__ spec_a, uint32_t* err) {
    pdl_trigger();
    pdl_wait();
    const int b = blockIdx.x, j = threadIdx.x;
    const uint64_t step = *step_dev;
    bool rej = false;
    if (j < B - 1) {
        const int d = draft[(size_t)b * (B - 1) + j];
        if (d < 0 || d >= V) {
            rej = true;
            atomicOr(err, DFLARE_DEVERR_TOKEN);
        } else {
            const int tr = b * B + j, dr = b * (B - 1) + j;
            const float2 st = row_stats(part, tr, chunks);
            const float2 sq = row_stats(part, batch * B + dr, chunks);
            const float p = expf(target[(size_t)tr * V + d] * inv_t - st.x) / st.y;
            const float q = expf(draft_logits[(size_t)dr * V + d] * inv_t - sq.x) / sq.y;
            float u[8];
            philox_uniforms(1 + (uint64_t)(j >> 3), (uint64_t)b, step, kRngAccept, seed, u);
            rej = !(u[j & 7] * q < p);
        }
    }
    const unsigned mask = __ballot_sync(0xffffffffu, rej);
    if (j == 0) spec_a[b] = mask ? __ffs(mask) - 1 : B - 1;
}

// Grid (chunks, batch): the replacement draw of every sequence, from max(0, p - q) at its first
// rejected position a, or from p at the last target row when every draft was kept. The last CTA
// writes accept_len = a + 1 and the token, re-arms the slots, and advances the step counter.
__global__ void __launch_bounds__(256) spec_resample_kernel(
    const float* __restrict__ target, const float* __restrict__ draft_logits, int V, int B,
    int batch, int chunk, int stat_chunks, float inv_t, uint64_t seed, uint64_t* step_dev,
    const float2* __restrict__ part, const int32_t* __restrict__ spec_a,
    unsigned long long* slot, uint32_t* cnt, int32_t* __restrict__ accept_len,
    int32_t* __restrict__ next_token) {
    pdl_trigger();
    pdl_wait();
    const uint64_t step = *step_dev;
    const int b = blockIdx.y;
    const int a = spec_a[b];
    const bool resid = a < B - 1;
    const int tr = b * B + a, dr = b * (B - 1) + a;
    const float2 st = row_stats(part, tr, stat_chunks);
    const float2 sq = resid ? row_stats(part, batch * B + dr, stat_chunks) : make_float2(0.f, 1.f);
    const float* lt = target + (size_t)tr * V;
    const float* lq = resid ? draft_logits + (size_t)dr * V : nullptr;
    const int c0 = blockIdx.x * chunk, c1 = min(V, c0 + chunk);
    const bool vec = (V & 3) == 0;
    float bv = -INFINITY;
    int bi = kNone;
    const int stride = blockDim.x * 8;
    for (int base = c0 + threadIdx.x * 8; base < c1; base += stride * kDrawU) {
        float xt[kDrawU][8], xq[kDrawU][8];
#pragma unroll
        for (int g = 0; g < kDrawU; ++g) {
            load4(lt, base + g * stride, c1, vec, xt[g]);
            load4(lt, base + g * stride + 4, c1, vec, xt[g] + 4);
            if (resid) {
                load4(lq, base + g * stride, c1, vec, xq[g]);
                load4(lq, base + g * stride + 4, c1, vec, xq[g] + 4);
            }
        }
#pragma unroll
        for (int g = 0; g < kDrawU; ++g) {
            const int i = base + g * stride;
            if (i >= c1) break;
            float u[8];
            philox_uniforms(1 + (uint64_t)(i >> 3), (uint64_t)b, step, kRngResidual, seed, u);
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                float w = expf(xt[g][e] * inv_t - st.x) / st.y;
                if (resid) w -= expf(xq[g][e] * inv_t - sq.x) / sq.y;
                if (w > 0.f) {
                    const float sc = logf(w) + gumbel(u[e]);
                    if (sc > bv) {
                        bv = sc;
                        bi = i + e;
                    }
                }
            }
        }
    }
    if (publish_max(bv, bi, &slot[b], cnt, gridDim.x * gridDim.y)) {
        for (int s = threadIdx.x; s < batch; s += blockDim.x) {
            const unsigned long long key = atomicExch(&slot[s], 0ull);
            const int as = spec_a[s];
            int32_t tok = slot_token(key);
            if (key == 0ull) {
                // max(0, p - q) vanished everywhere (or every entry was -inf): draw from p at
                // that target row instead, serially (only for such rows)
                const int r = s * B + as;
                const float2 t2 = row_stats(part, r, stat_chunks);
                const float* l = target + (size_t)r * V;
                float best = -INFINITY;
                tok = 0;
                for (int i = 0; i < V; ++i) {
                    float u[8];
                    philox_uniforms(1 + (uint64_t)(i >> 3), (uint64_t)s, step, kRngResidual, seed, u);
                    const float w = expf(l[i] * inv_t - t2.x) / t2.y;
                    if (w > 0.f) {
                        const float sc = logf(w) + gumbel(u[i & 7]);
                        if (sc > best) {
                            best = sc;
                            tok = i;
                        }
                    }
                }
            }
            accept_len[s] = as + 1;
            next_token[s] = tok;
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            *cnt = 0;
            *step_dev = step + 1;
        }
    }
}

// chunk size (a multiple of 8, at least 1024) and count for `rows` rows of V entries, about
// per_sm CTAs per SM (the scans that end in one packed atomicMax per CTA use two)
void chunking(int V, int rows, int sms, int max_chunks, int per_sm, int* chunk, int* chunks) {
    int n = std::max(1, (per_sm * sms + rows - 1) / rows);
    n = std::min(n, max_chunks);
    int c = (V + n - 1) / n;
    c = std::max(1024, ((c + 7) / 8) * 8);   // a multiple of 8: no Philox block straddles chunks
    *chunk = c;
    *chunks = (V + c - 1) / c;
}

}  // namespace

cudaError_t launch_sample(dflare_ctx* c, int rows, float inv_t, uint64_t seed, const uint64_t* step,
                          int32_t* tokens, cudaStream_t s) {
    if (rows <= 0) return cudaSuccess;
    int chunk, chunks;
    chunking(c->cfg.vocab, rows, c->num_sms, 1 << 20, 4, &chunk, &chunks);
    return launch_kernel(c->pdl, sample_kernel, dim3(chunks, rows), dim3(256), 0, s, c->logits,
                         c->cfg.vocab, rows, chunk, inv_t, seed, step, c->amax_slot, c->amax_cnt,
                         tokens);
}

cudaError_t launch_spec_stats(dflare_ctx* c, const float* target_logits, float inv_t, cudaStream_t s) {
    const int B = c->cfg.block, V = c->cfg.vocab;
    const int rows = c->batch * B + c->batch * (B - 1);
    int chunk, chunks;
    chunking(V, rows, c->num_sms, kSpecMaxChunks, 4, &chunk, &chunks);
    c->spec_chunks = chunks;
    return launch_kernel(c->pdl, spec_stats_kernel, dim3(chunks, rows), dim3(256), 0, s,
                         target_logits, (const float*)c->logits, V, c->batch * B, chunk, inv_t,
                         c->spec_part);
}

cudaError_t launch_spec_accept(dflare_ctx* c, const int32_t* draft, const float* target_logits,
                               float inv_t, uint64_t seed, const uint64_t* step, cudaStream_t s) {
    return launch_kernel(c->pdl, spec_accept_kernel, dim3(c->batch), dim3(32), 0, s, target_logits,
                         (const float*)c->logits, draft, c->cfg.vocab, c->cfg.block, c->batch,
                         c->spec_chunks, inv_t, seed, step, (const float2*)c->spec_part, c->spec_a,
                         c->err);
}

cudaError_t launch_spec_resample(dflare_ctx* c, const float* target_logits, float inv_t,
                                 uint64_t seed, uint64_t* step, int32_t* accept_len,
                                 int32_t* next_token, cudaStream_t s) {
    int chunk, chunks;
    chunking(c->cfg.vocab, c->batch, c->num_sms, 1 << 20, 2, &chunk, &chunks);
    return launch_kernel(c->pdl, spec_resample_kernel, dim3(chunks, c->batch), dim3(256), 0, s,
                         target_logits, (const float*)c->logits, c->cfg.vocab, c->cfg.block,
                         c->batch, chunk, c->spec_chunks, inv_t, seed, step,
                         (const float2*)c->spec_part, (const int32_t*)c->spec_a, c->amax_slot,
                         c->amax_cnt, accept_len, next_token);
}

}  // namespace dfl
