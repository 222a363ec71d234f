// Adaptive layer fusion (Eq. 3, Sec. 4.1) and the bookkeeping of a context append.
//
// fusion_alpha: alpha^(i) = softmax(W^fuse_{i,:}), computed once when the weights are set
// (Sec. 4.1: the normalised weights can be cached after training).
// fuse_layers: the T target rows of every new position are read once and every draft layer's
// fused, normalised row is written: a thread-block cluster per position for a handful of
// positions (one block step), one CTA per position when there are enough to fill the GPU
// (context fill).
#include <math.h>

#include <algorithm>

#include <cooperative_groups.h>

#include "common.cuh"
#include "internal.h"

namespace cg = cooperative_groups;

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

constexpr int kFuseCH = 512;       // features per CTA (64 threads x 8)
constexpr int kFuseGroups = 4;     // thread groups splitting the T target layers

// One position is handled by a cluster of ceil(d / 512) CTAs (at most 8 for d <= 4096); CTA c owns
// features [512 c, 512 c + 512). Each CTA (256 threads) stages its slice of all T target rows and
// of the D gain rows in shared memory with cp.async (one round trip). Thread group q (64 threads,
// 8 features each) forms the D weighted sums over target layers j = q, q + 4, ...; the four
// partial sums are added in group order, the CTA reduces its partial sums of squares, and the
// CTAs of the cluster exchange those partials through distributed shared memory (one gather,
// summed in rank order) before normalising.
template <class T, int DMAX>
__global__ void __launch_bounds__(256) fuse_layers_kernel(
    const T* __restrict__ H, const float* __restrict__ alpha, const T* __restrict__ gain,
    T* __restrict__ F, T* __restrict__ F_out, const int32_t* __restrict__ app_cnt, int D, int Tn,
    int batch, int n_max, int d, long long f_layer_rows, float eps) {
    pdl_trigger();
    pdl_wait();
    extern __shared__ __align__(16) uint8_t smem[];
    T* sh = reinterpret_cast<T*>(smem);          // [Tn][kFuseCH] target rows, then [D][kFuseCH] gains
    T* sg = sh + (size_t)Tn * kFuseCH;
    float* sacc = reinterpret_cast<float*>(sg + (size_t)D * kFuseCH);  // [3][DMAX][8][64]
    __shared__ float s_alpha[16 * 64];
    __shared__ float red[2][DMAX];
    __shared__ float ss_cta[DMAX];               // this CTA's partial sums of squares
    __shared__ float part[8][DMAX];              // every cluster rank's partials
    __shared__ float inv_s[DMAX];
    cg::cluster_group cluster = cg::this_cluster();
    const int C = (int)cluster.num_blocks(), cr = (int)cluster.block_rank();
    const int r = blockIdx.y, b = blockIdx.z;
    if (r >= app_cnt[b]) return;                 // the same for every CTA of the cluster
    const int tid = threadIdx.x, q = tid >> 6, t64 = tid & 63;
    const int lane = tid & 31, warp = tid >> 5;
    const int f0 = cr * kFuseCH, nf = min(kFuseCH, d - f0);
    const size_t row = (size_t)b * n_max + r;
    const size_t lstride = (size_t)batch * n_max * d;
    constexpr int EPC = 16 / sizeof(T);          // elements per 16-byte copy
    const int per_row = nf / EPC;                // <= 64 (bf16) or 128 (fp32)
    const uint32_t ssh = (uint32_t)__cvta_generic_to_shared(sh);
    // all T target rows of this slice and all D gain rows, one round trip
    for (int j = q; j < Tn + D; j += kFuseGroups) {
        const T* src = j < Tn ? H + (size_t)j * lstride + row * d + f0 : gain + (size_t)(j - Tn) * d + f0;
        for (int p = t64; p < per_row; p += 64)
            asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(
                             ssh + (uint32_t)((j * kFuseCH + p * EPC) * sizeof(T))),
                         "l"(src + p * EPC)
                         : "memory");
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
    for (int k = tid; k < D * Tn; k += blockDim.x) s_alpha[k] = alpha[k];
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    __syncthreads();
    const int e0 = t64 * 8;
    const bool act = e0 < nf;
    for (int i0 = 0; i0 < D; i0 += DMAX) {
        const int nd = min(DMAX, D - i0);
        float acc[DMAX][8];
#pragma unroll
        for (int i = 0; i < DMAX; ++i)
#pragma unroll
            for (int e = 0; e < 8; ++e) acc[i][e] = 0.f;
        if (act) {
            for (int j = q; j < Tn; j += kFuseGroups) {
                float h[8], a[DMAX];
                load8(sh + j * kFuseCH + e0, h);
#pragma unroll
                for (int i = 0; i < DMAX; ++i) a[i] = i < nd ? s_alpha[(i0 + i) * Tn + j] : 0.f;
#pragma unroll
                for (int i = 0; i < DMAX; ++i)
#pragma unroll
                    for (int e = 0; e < 8; ++e) acc[i][e] = fmaf(a[i], h[e], acc[i][e]);
            }
        }
        // groups 1..3 hand their partial sums to group 0, which adds them in group order
        if (q > 0) {
#pragma unroll
            for (int i = 0; i < DMAX; ++i)
#pragma unroll
                for (int e = 0; e < 8; ++e) sacc[(((q - 1) * DMAX + i) * 8 + e) * 64 + t64] = acc[i][e];
        }
        __syncthreads();
        if (q == 0) {
#pragma unroll
            for (int g2 = 0; g2 < kFuseGroups - 1; ++g2)
#pragma unroll
                for (int i = 0; i < DMAX; ++i)
#pragma unroll
                    for (int e = 0; e < 8; ++e) acc[i][e] += sacc[((g2 * DMAX + i) * 8 + e) * 64 + t64];
#pragma unroll
            for (int i = 0; i < DMAX; ++i) {
                float v = 0.f;
#pragma unroll
                for (int e = 0; e < 8; ++e) v = fmaf(acc[i][e], acc[i][e], v);
                v = warp_sum(v);
                if (lane == 0) red[warp][i] = v;
            }
        }
        __syncthreads();
        if (tid < DMAX) ss_cta[tid] = red[0][tid] + red[1][tid];
        cluster.sync();
        // gather every rank's partials in one round of DSMEM loads, then sum in rank order
        for (int k = tid; k < C * nd; k += blockDim.x)
            part[k / nd][k % nd] = cluster.map_shared_rank(ss_cta, k / nd)[k % nd];
        __syncthreads();
        if (tid < nd) {
            float tot = 0.f;
            for (int c = 0; c < C; ++c) tot += part[c][tid];
            inv_s[tid] = inv_rms(tot, d, eps);
        }
        __syncthreads();
        if (q == 0 && act) {
#pragma unroll
            for (int i = 0; i < DMAX; ++i) {
                if (i >= nd) break;
                float g[8], o[8];
                load8(sg + (i0 + i) * kFuseCH + e0, g);
                const float inv = inv_s[i];
#pragma unroll
                for (int e = 0; e < 8; ++e) o[e] = g[e] * (acc[i][e] * inv);
                store8(F + ((size_t)(i0 + i) * f_layer_rows + row) * d + f0 + e0, o);
                if (F_out)
                    store8(F_out + (((size_t)(i0 + i) * batch + b) * n_max + r) * d + f0 + e0, o);
            }
        }
        cluster.sync();   // peers have read ss_cta before it is reused or this CTA exits
    }
}

// Many positions (context fill): a persistent grid of one or two CTAs per SM walks the positions
// (no cluster). Warp-specialised: the last warp's first thread streams the T target rows of each
// position (d contiguous elements each) through a ring of `ns` shared-memory stages of kRB rows as
// 1-D bulk copies, the stage sequence running on across positions; the other warps (one thread
// per 8 features) consume the stages. Each stage has a "full" mbarrier (the copies landed) and an
// "empty" one that every consumer warp arrives on once it has read the stage, which is what the
// producer waits for before refilling it: no CTA barrier per stage, and up to ns - 1 stages in
// flight while one is summed. Thread t forms the D (<= DMAX) draft-layer sums of features
// [8t, 8t + 8) in registers; at the end of a position the consumer warps reduce the D sums of
// squares (warp shuffles, then the warps' partials in order) behind a named barrier. Every wait
// is bounded; a CTA that times out sets DFLARE_DEVERR_TIMEOUT and stops.
constexpr int kRB = 4;          // target rows per stage
constexpr int kMaxNS = 16;      // most stages in the ring
constexpr uint64_t kFillWaitNs = 2000000000ull;

__device__ __forceinline__ bool fill_try(uint32_t bar, uint32_t parity) {
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(bar), "r"(parity)
        : "memory");
    return done != 0;
}
// Bounded wait; the timer is read only after 64 unsuccessful polls (a %globaltimer read costs a
// few hundred ns, and most waits of the ring complete within those polls).
__device__ __forceinline__ bool fill_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag) {
    for (int i = 0; i < 64; ++i)
        if (fill_try(bar, parity)) return true;
    const uint64_t t0 = globaltimer_ns();
    for (int it = 0;; ++it) {
        if (fill_try(bar, parity)) return true;
        if ((it & 63) == 63) {
            if (*abort_flag) return false;
            if (globaltimer_ns() - t0 > kFillWaitNs) {
                *abort_flag = 1;
                return false;
            }
        }
    }
}

// Two fp32 lanes in one 64-bit register: the fill's sums use the paired FMA (fma.rn.f32x2, each
// lane rounded as a scalar fmaf), which halves the instructions of the 8 x D FMAs per row.
typedef unsigned long long f32x2;
__device__ __forceinline__ f32x2 pk2(float lo, float hi) {
    f32x2 r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}
__device__ __forceinline__ void upk2(f32x2 v, float& lo, float& hi) {
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ f32x2 fma2(f32x2 a, f32x2 b, f32x2 c) {
    f32x2 r;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
    return r;
}
// 8 consecutive elements of a staged row as four fp32 pairs
__device__ __forceinline__ void load8x2(const bf16* p, f32x2* h) {
    const uint4 u = *reinterpret_cast<const uint4*>(p);
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) h[q] = pk2(__uint_as_float(w[q] << 16), __uint_as_float(w[q] & 0xFFFF0000u));
}
__device__ __forceinline__ void load8x2(const float* p, f32x2* h) {
    const float4 a = *reinterpret_cast<const float4*>(p), b = *reinterpret_cast<const float4*>(p + 4);
    h[0] = pk2(a.x, a.y);
    h[1] = pk2(a.z, a.w);
    h[2] = pk2(b.x, b.y);
    h[3] = pk2(b.z, b.w);
}

template <class T, int DMAX>
__device__ __forceinline__ void fuse_rows_body(
    const T* __restrict__ H, const float* __restrict__ alpha, const T* __restrict__ gain,
    T* __restrict__ F, T* __restrict__ F_out, const int32_t* __restrict__ app_cnt, int D, int Tn,
    int batch, int n_max, int d, long long f_layer_rows, float eps, int ns, uint32_t* err) {
    pdl_trigger();
    extern __shared__ __align__(128) uint8_t stage_mem[];   // [ns][kRB][d]
    constexpr int DP = (DMAX + 1) & ~1;                       // DMAX rounded up to even
    __shared__ __align__(16) f32x2 s_alpha[64 * DP];          // [j][i] = (alpha_ij, alpha_ij), Tn <= 64
    __shared__ float red[16][DMAX];
    __shared__ float inv_s[DMAX];
    __shared__ __align__(8) uint64_t full_bar[kMaxNS], empty_bar[kMaxNS];
    __shared__ int abort_flag;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int n_cw = (int)(blockDim.x >> 5) - 1;   // consumer warps; the last warp produces
    const int n_ct = n_cw * 32;
    const uint32_t fb0 = (uint32_t)__cvta_generic_to_shared(&full_bar[0]);
    const uint32_t eb0 = (uint32_t)__cvta_generic_to_shared(&empty_bar[0]);
    const uint32_t sbase = (uint32_t)__cvta_generic_to_shared(stage_mem);
    if (tid == 0) {
        for (int i = 0; i < ns; ++i) {
            asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(fb0 + 8u * i) : "memory");
            asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(eb0 + 8u * i), "r"(n_cw) : "memory");
        }
        abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    pdl_wait();
    for (int k = tid; k < Tn * DP; k += blockDim.x) {
        const int j = k / DP, i = k % DP;
        const float a = i < D ? alpha[i * Tn + j] : 0.f;
        s_alpha[k] = pk2(a, a);
    }
    __syncthreads();
    volatile int* abrt = &abort_flag;
    const int n_pos = batch * n_max;
    const size_t lstride = (size_t)n_pos * d;
    const uint32_t row_bytes = (uint32_t)(d * sizeof(T));
    const int nst = (Tn + kRB - 1) / kRB;   // stages per position
    // this CTA's positions pid = blockIdx.x + k * gridDim.x that have rows to append
    auto valid = [&](int pid) { return pid % n_max < app_cnt[pid / n_max]; };
    auto next_pos = [&](int pid) {
        for (pid += gridDim.x; pid < n_pos; pid += gridDim.x)
            if (valid(pid)) return pid;
        return n_pos;
    };
    int first = (int)blockIdx.x;
    if (first < n_pos && !valid(first)) first = next_pos(first);

    if (warp == n_cw) {
        // ---------------- producer: one thread streams every stage of every position in turn
        if (lane == 0) {
            int g = 0;
            bool ok = true;
            for (int pid = first; pid < n_pos && ok; pid = next_pos(pid)) {
                for (int k = 0; k < nst; ++k, ++g) {
                    const int st = g % ns, use = g / ns;
                    if (use > 0 && !fill_wait(eb0 + 8u * st, (uint32_t)((use - 1) & 1), abrt)) {
                        ok = false;
                        break;
                    }
                    const int j0 = k * kRB, nr = min(kRB, Tn - j0);
                    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(fb0 + 8u * st),
                                 "r"((uint32_t)nr * row_bytes)
                                 : "memory");
                    for (int u = 0; u < nr; ++u)
                        asm volatile(
                            "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                                sbase + (uint32_t)(st * kRB + u) * row_bytes),
                            "l"(H + (size_t)(j0 + u) * lstride + (size_t)pid * d), "r"(row_bytes),
                            "r"(fb0 + 8u * st)
                            : "memory");
                }
            }
            // after a timeout: every issued copy lands before the CTA exits (bounded again)
            if (!ok || *abrt) {
                volatile int never = 0;
                for (int q = max(0, g - ns); q < g; ++q)
                    fill_wait(fb0 + 8u * (q % ns), (uint32_t)((q / ns) & 1), &never);
                atomicOr(err, DFLARE_DEVERR_TIMEOUT);
            }
        }
    } else {
        // ---------------- consumers: thread t owns features [8t, 8t + 8)
        const int e0 = tid * 8;
        const bool act = e0 < d;
        const T* stg = reinterpret_cast<const T*>(stage_mem);
        int g = 0;
        bool ok = true;
        for (int pid = first; pid < n_pos && ok; pid = next_pos(pid)) {
            const int b = pid / n_max, r = pid % n_max;
            f32x2 acc2[DMAX][4];
#pragma unroll
            for (int i = 0; i < DMAX; ++i)
#pragma unroll
                for (int q = 0; q < 4; ++q) acc2[i][q] = 0ull;
            for (int k = 0; k < nst; ++k, ++g) {
                const int st = g % ns;
                if (!fill_wait(fb0 + 8u * st, (uint32_t)((g / ns) & 1), abrt)) {
                    ok = false;
                    break;
                }
                if (act) {
#pragma unroll
                    for (int u = 0; u < kRB; ++u) {
                        const int j = k * kRB + u;
                        if (j >= Tn) break;
                        f32x2 h[4], a[DP];
                        load8x2(stg + (size_t)(st * kRB + u) * d + e0, h);
#pragma unroll
                        for (int i = 0; i < DP; i += 2) {
                            const uint4 a4 = *reinterpret_cast<const uint4*>(&s_alpha[j * DP + i]);
                            a[i] = ((f32x2)a4.y << 32) | a4.x;
                            a[i + 1] = ((f32x2)a4.w << 32) | a4.z;
                        }
#pragma unroll
                        for (int i = 0; i < DMAX; ++i)
#pragma unroll
                            for (int q = 0; q < 4; ++q) acc2[i][q] = fma2(a[i], h[q], acc2[i][q]);
                    }
                }
                __syncwarp();
                if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(eb0 + 8u * st) : "memory");
            }
            // the consumer warps leave the position loop together: a warp whose wait ran out sets
            // the abort flag, which every other consumer sees at the barrier below
            asm volatile("bar.sync 1, %0;" ::"r"(n_ct) : "memory");
            if (!ok || *abrt) break;
            float acc[DMAX][8];
#pragma unroll
            for (int i = 0; i < DMAX; ++i)
#pragma unroll
                for (int q = 0; q < 4; ++q) upk2(acc2[i][q], acc[i][2 * q], acc[i][2 * q + 1]);
#pragma unroll
            for (int i = 0; i < DMAX; ++i) {
                float v = 0.f;
#pragma unroll
                for (int e = 0; e < 8; ++e) v = fmaf(acc[i][e], acc[i][e], v);
                v = warp_sum(v);
                if (lane == 0) red[warp][i] = v;
            }
            asm volatile("bar.sync 1, %0;" ::"r"(n_ct) : "memory");
            if (tid < D) {
                float tot = 0.f;
                for (int w = 0; w < n_cw; ++w) tot += red[w][tid];
                inv_s[tid] = inv_rms(tot, d, eps);
            }
            asm volatile("bar.sync 1, %0;" ::"r"(n_ct) : "memory");
            if (act) {
#pragma unroll
                for (int i = 0; i < DMAX; ++i) {
                    if (i >= D) break;
                    float gg[8], o[8];
                    load8(gain + (size_t)i * d + e0, gg);
                    const float inv = inv_s[i];
#pragma unroll
                    for (int e = 0; e < 8; ++e) o[e] = gg[e] * (acc[i][e] * inv);
                    store8(F + ((size_t)i * f_layer_rows + pid) * d + e0, o);
                    if (F_out) store8(F_out + (((size_t)i * batch + b) * n_max + r) * d + e0, o);
                }
            }
        }
    }
    __syncthreads();
}

#define FUSE_ROWS_PARAMS                                                                            \
    const T *__restrict__ H, const float *__restrict__ alpha, const T *__restrict__ gain,           \
        T *__restrict__ F, T *__restrict__ F_out, const int32_t *__restrict__ app_cnt, int D,         \
        int Tn, int batch, int n_max, int d, long long f_layer_rows, float eps, int ns, uint32_t *err
#define FUSE_ROWS_ARGS H, alpha, gain, F, F_out, app_cnt, D, Tn, batch, n_max, d, f_layer_rows, eps, ns, err
// one CTA per SM (up to 512 consumer threads), or two per SM for d <= 2560 and D <= 5 (registers
// capped; eight sums of eight features do not fit without spills)
template <class T, int DMAX>
__global__ void __launch_bounds__(544, 1) fuse_rows_kernel(FUSE_ROWS_PARAMS) {
    fuse_rows_body<T, DMAX>(FUSE_ROWS_ARGS);
}
template <class T, int DMAX>
__global__ void __launch_bounds__(352, 2) fuse_rows2_kernel(FUSE_ROWS_PARAMS) {
    fuse_rows_body<T, DMAX>(FUSE_ROWS_ARGS);
}
#undef FUSE_ROWS_PARAMS
#undef FUSE_ROWS_ARGS

template <class T>
cudaError_t fuse_layers_t(dflare_ctx* c, const void* hidden, int n_max, void* fused_out,
                          cudaStream_t s) {
    const dflare_config& g = c->cfg;
    const int C = (g.d + kFuseCH - 1) / kFuseCH;
    const size_t smem = (size_t)(g.n_target_layers + g.n_draft_layers) * kFuseCH * sizeof(T) +
                        (size_t)(kFuseGroups - 1) * 8 * 8 * 64 * sizeof(float);
    const T* H = static_cast<const T*>(hidden);
    const T* gain = static_cast<const T*>(c->w.fuse_norm);
    T* F = static_cast<T*>(c->fused);
    T* Fo = static_cast<T*>(fused_out);
    // context fill: warp-specialised CTAs of d / 8 consumer threads and a producer warp, two per SM
    // when their registers allow (rings of about 100 KB), else one (about 200 KB); at most kMaxNS
    // stages of kRB rows
    const int cthreads = ((g.d / 8 + 31) / 32) * 32;
    const size_t stage_bytes = (size_t)kRB * g.d * sizeof(T);
    if ((long long)c->batch * n_max >= 2LL * c->num_sms && cthreads <= 512 && g.n_draft_layers <= 8 &&
        g.n_target_layers <= 64 && 3 * stage_bytes <= 200 * 1024) {
        const int threads = cthreads + 32;
        static PerDeviceOnce rconf;
        const cudaError_t re = rconf([] {
            for (auto k : {fuse_rows_kernel<T, 4>, fuse_rows_kernel<T, 5>, fuse_rows_kernel<T, 8>,
                           fuse_rows2_kernel<T, 4>, fuse_rows2_kernel<T, 5>, fuse_rows2_kernel<T, 8>}) {
                cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                     200 * 1024);
                if (e != cudaSuccess) return e;
            }
            return cudaSuccess;
        });
        if (re != cudaSuccess) return re;
        const int Dn = g.n_draft_layers;
        auto rk1 = Dn <= 4 ? fuse_rows_kernel<T, 4> : Dn == 5 ? fuse_rows_kernel<T, 5> : fuse_rows_kernel<T, 8>;
        auto rk2 = Dn <= 4 ? fuse_rows2_kernel<T, 4> : Dn == 5 ? fuse_rows2_kernel<T, 5> : fuse_rows2_kernel<T, 8>;
        auto rk = rk1;
        int ns = (int)std::min<size_t>(kMaxNS, (200 * 1024) / stage_bytes), per_sm = 1;
        const int ns2 = (int)std::min<size_t>(kMaxNS, (100 * 1024) / stage_bytes);
        int fit = 0;
        if (threads <= 352 && Dn <= 5 && ns2 >= 3 &&
            cudaOccupancyMaxActiveBlocksPerMultiprocessor(&fit, rk2, threads, (size_t)ns2 * stage_bytes) ==
                cudaSuccess && fit >= 2) {
            rk = rk2;
            ns = ns2;
            per_sm = 2;
        }
        const int grid = (int)std::min<long long>((long long)c->batch * n_max, (long long)per_sm * c->num_sms);
        return launch_kernel(c->pdl, rk, dim3(grid), dim3(threads), (size_t)ns * stage_bytes, s, H,
                             (const float*)c->alpha, gain, F, Fo, (const int32_t*)c->app_cnt,
                             g.n_draft_layers, g.n_target_layers, c->batch, n_max, g.d,
                             (long long)g.max_fuse_rows, g.rms_eps, ns, c->err);
    }
    auto kern = g.n_draft_layers <= 4 ? fuse_layers_kernel<T, 4> : fuse_layers_kernel<T, 8>;
    static PerDeviceOnce configured;
    const cudaError_t ce = configured([] {
        for (auto k : {fuse_layers_kernel<T, 4>, fuse_layers_kernel<T, 8>}) {
            cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 (int)((64 + 16) * kFuseCH * sizeof(T) +
                                                       (kFuseGroups - 1) * 8 * 8 * 64 * 4));
            if (e != cudaSuccess) return e;
        }
        return cudaSuccess;
    });
    if (ce != cudaSuccess) return ce;
    return launch_cluster(c->pdl, C, kern, dim3(C, n_max, c->batch), dim3(256), smem, s, H,
                          (const float*)c->alpha, gain, F, Fo, (const int32_t*)c->app_cnt,
                          g.n_draft_layers, g.n_target_layers, c->batch, n_max, g.d,
                          (long long)g.max_fuse_rows, g.rms_eps);
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
