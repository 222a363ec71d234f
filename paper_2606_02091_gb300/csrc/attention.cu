// Bidirectional block attention over [context ; block] (Sec. 3.2; keys/values per Eq. 4), as a
// split-KV ("flash-decoding") pass.
//
// For one sequence and one KV head, the queries are the B block rows of the H_q/H_kv query
// heads that share the head: B*G rows (64 for Qwen3 shapes, 128 for GPT-OSS) against L + B keys
// (context keys from the cache, then the block's own K^d / V^d). Nothing is masked: every query
// sees every key. The keys of one (sequence, head) are cut into contiguous ranges so that
// batch x H_kv x splits CTAs cover the GPU even for a single sequence.
//
// In both bf16 kernels the splits of one (sequence, head, query tile) form a thread-block
// cluster (up to 16 CTAs) and merge their partial results (O / l in fp16) through distributed
// shared memory, so the whole attention is one launch and no partial goes through HBM.
// bf16, tcgen05 (attn_tc_kernel, the default; details at its definition): 128 query rows per
// CTA as the UMMA M, 64-key K/V tiles streamed by TMA, S = Q K^T and O += P V on the fifth-
// generation tensor cores with S and O in TMEM, two softmax warpgroups on alternate tiles, one
// CTA per SM.
// bf16, mma.sync (attn_mma_kernel, DFLARE_FLAG_MMA_SYNC_ATTENTION): 64 query rows per CTA (4 warps
// x 16 rows); one thread streams 64-key K/V tiles by TMA into two 128-byte-swizzled stages;
// S = Q K^T and O += P V on mma.sync m16n8k16 with bf16 operands and fp32 accumulators, P kept in
// registers; two to four CTAs fit on an SM.
// fp32 path: a CUDA-core version of the split with partials in global memory and a second
// (combine) launch; exact fp32 products.
#include <cuda_fp16.h>
#include <math.h>

#include <algorithm>

#include <cooperative_groups.h>

#include "common.cuh"
#include "internal.h"

namespace cg = cooperative_groups;

namespace dfl {
namespace {

constexpr int kQT = 64;    // query rows per CTA
constexpr int kKT = 64;    // keys per tile

struct AttnArgs {
    const void* q;        // [batch*B][d_q]
    const void* kd;       // [batch*B][d_kv]
    const void* vd;
    const void* kc;       // this layer's cache [max_batch][H_kv][max_ctx][hd]
    const void* vc;
    const int32_t* ctx_len;
    float* part_o;        // [batch][H_kv][q_tiles][splits][64][hd]
    float* part_ml;       // [batch][H_kv][q_tiles][splits][64][2]
    uint32_t* err;        // device error word (a tile wait that timed out)
    int block_rows;       // rows of one K^d / V^d tensor-map box (min(64, max_batch * B))
    int B, G, hkv, d_q, d_kv, max_ctx, splits, q_tiles;
    float scale_log2;     // log2(e) / sqrt(hd)
    // bf16 path with the projection's fp32 sums: Q / K^d / V^d are taken from qkv32
    // ([batch*B][d_q + 2 d_kv]) with the rotary embedding at the block positions (rope != 0)
    // applied here; the CTA that holds a block tile writes its head's bf16 K^d / V^d rows to kd_w /
    // vd_w before its TMA reads them
    const float* qkv32;
    const float* rope_cos;   // [positions][hd/2]
    const float* rope_sin;
    bf16* kd_w;
    bf16* vd_w;
    int rope;
    unsigned long long* t_stamps;   // launch timing (dflare_set_timing): entry, dependency, exit
    int t_slots;
};

__device__ __forceinline__ void key_range(const AttnArgs& a, int b, int s, int& j0, int& j1, int& L) {
    L = a.ctx_len[b];
    const int total = L + a.B;
    int per = (total + a.splits - 1) / a.splits;
    per = (per + kKT - 1) / kKT * kKT;
    j0 = s * per;
    j1 = min(total, j0 + per);
}

__device__ __forceinline__ size_t part_index(const AttnArgs& a, int b, int g, int qt, int s) {
    return (((size_t)b * a.hkv + g) * a.q_tiles + qt) * a.splits + s;
}

// ------------------------------------------------------------------ bf16, mma.sync (warp-level tensor cores)

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, bool valid) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src),
                 "r"(valid ? 16 : 0)
                 : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}
__device__ __forceinline__ void mma16816(float* c, const uint32_t* a, uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, "
        "{%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
// P.V runs on bf16 operands: V as the TMA wrote it, P in [0, 1] rounded to bf16 (relative error
// at most 2^-9 per weight; the row sums l are taken from the fp32 P). Measured alternatives: P
// split into a bf16 high part and its remainder (two MMAs per step, ~2^-17) with the split merge
// in fp32 took the attention from 25.8 to 32.4 us per launch at the Qwen3-8B batch-4 shape, and
// the fp32 merge alone cost ~1 us per launch, while the hidden-state difference to the oracle
// after the first layer only went from 4.8e-3 to 3.9e-3 (the bf16 storage points amplify any
// perturbation to about an ulp within a few layers).
// 2^x with the hardware approximation (relative error about 2^-22, far below the bf16 rounding of
// P; -inf gives +0): the softmax of a tile evaluates 32 of them per thread
__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&h);
}

constexpr int kNST = 2;                   // K/V tiles in flight per CTA (two CTAs fit on an SM)
constexpr uint64_t kWaitNs = 2000000000ull;  // bound on every wait for a tile

// Tensor maps of one layer (bf16, 128-byte swizzle, boxes of 64 keys x 64 head dims):
// K and V cache [max_batch * H_kv][max_ctx][hd] and the block's K^d, V^d [H_kv][max_batch * B][hd]
// (row stride d_kv).
struct AttnMaps {
    CUtensorMap kc, vc, kd, vd;
};

__device__ __forceinline__ uint32_t smem_addr(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
// Byte offset of the 16-byte chunk c8 (head dims 8*c8 .. 8*c8+7) of key row r in a tile stored as
// [hd/64 halves][64 rows][128 bytes] with the 128-byte swizzle (chunk index XOR row % 8).
__device__ __forceinline__ uint32_t swz(int r, int c8) {
    return (uint32_t)((c8 >> 3) * 8192 + r * 128 + (((c8 & 7) ^ (r & 7)) << 4));
}
__device__ __forceinline__ bool try_wait_parity(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}
// Bounded wait. The global timer is read only once the phase has not completed within the first
// 64 polls: measured, a timer read at the start of every wait put a few hundred nanoseconds into
// each hand-off of the tcgen05 attention's pipeline.
__device__ __forceinline__ bool tile_wait(uint32_t bar, uint32_t parity) {
    for (int i = 0; i < 64; ++i)
        if (try_wait_parity(bar, parity)) return true;
    const uint64_t t0 = globaltimer_ns();
    while (true) {
        for (int i = 0; i < 64; ++i)
            if (try_wait_parity(bar, parity)) return true;
        if (globaltimer_ns() - t0 > kWaitNs) return false;
    }
}
__device__ __forceinline__ void tma_tile(uint32_t dst, const CUtensorMap* m, int x, int y, int z,
                                         uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(m)), "r"(x), "r"(y), "r"(z), "r"(bar)
        : "memory");
}

// One CTA per (key split, KV head, 64-row query tile, sequence); the `splits` CTAs of one
// (sequence, head, query tile) form a thread-block cluster. The keys are cut into tiles of 64:
// ceil(L / 64) context tiles, then one tile of the block's own B keys (K^d, V^d); the splits take
// contiguous runs of tiles whose counts differ by at most one. One thread streams the tiles with TMA into a ring of kNST swizzled stages;
// every thread waits on the stage's mbarrier, and each warp signals a stage's second mbarrier when
// it has read the tile, which is what the streaming thread waits for before refilling the stage (no
// CTA-wide barrier per tile). Each CTA runs online softmax over its keys and
// pushes its partial (O / l in fp16, running max, running sum) row by row into the shared memory
// of the CTA that merges that row (DSMEM stores); after one cluster barrier every CTA merges its
// slice of the 64 rows from its own shared memory and writes the bf16 result. No partials go
// through global memory.
template <int HD, int S>
__global__ void __launch_bounds__(128) attn_mma_kernel(const __grid_constant__ AttnMaps maps,
                                                       const AttnArgs a, bf16* __restrict__ out) {
    pdl_trigger();
    if (a.t_stamps && threadIdx.x == 0) atomicMin(a.t_stamps, (unsigned long long)globaltimer_ns());
    constexpr int LD = HD + 8;                 // padded Q row (elements)
    constexpr int PIECES = HD / 8;             // 16-byte pieces per row
    constexpr uint32_t TB = HD * 128;          // bytes of one 64-key K (or V) tile
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = smem_raw + ((1024u - (smem_addr(smem_raw) & 1023u)) & 1023u);
    bf16* Qs = reinterpret_cast<bf16*>(smem + kNST * 2 * TB);   // [kQT][LD]
    // partials pushed here by the cluster's CTAs: row lr of this CTA's slice from split p at
    // [p * RP + lr], O / l in fp16 and (running max in log2 units, running sum)
    __half* rO = reinterpret_cast<__half*>(Qs + kQT * LD);     // [kQT][HD]
    float* rML = reinterpret_cast<float*>(rO + kQT * HD);        // [kQT][2]
    uint64_t* full = reinterpret_cast<uint64_t*>(rML + 2 * kQT);   // [kNST] tile landed
    uint64_t* empty = full + kNST;                                  // [kNST] tile read by all 4 warps
    constexpr int RP = kQT / S;                                  // merged rows per CTA
    cg::cluster_group cluster = cg::this_cluster();
    const int s = (int)cluster.block_rank();
    const int g = blockIdx.y % a.hkv, qt = blockIdx.y / a.hkv, b = blockIdx.z;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int R = a.B * a.G;
    const uint32_t sbase = smem_addr(smem), fbar = smem_addr(full), ebar = smem_addr(empty);
    // rows [block_rows, 64) of the V stages are never written by the block tile's copy (its box
    // has block_rows rows): zero them once, before any copy lands in the stages
    if (a.block_rows < kKT) {
        const int zr = kKT - a.block_rows;
        for (int k = tid; k < kNST * (HD / 64) * zr * 8; k += blockDim.x) {
            const int piece = k & 7, r = a.block_rows + (k >> 3) % zr, sub = (k >> 3) / zr;
            const int st = sub / (HD / 64), h = sub % (HD / 64);
            *reinterpret_cast<uint4*>(smem + (size_t)st * 2 * TB + TB + h * 8192 + r * 128 + piece * 16) =
                make_uint4(0u, 0u, 0u, 0u);
        }
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    if (tid == 0) {
        for (int i = 0; i < kNST; ++i) {
            asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(fbar + 8u * i) : "memory");
            asm volatile("mbarrier.init.shared::cta.b64 [%0], 4;" ::"r"(ebar + 8u * i) : "memory");
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&maps.kc)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&maps.vc)) : "memory");
    }
    __syncthreads();
    // every CTA of the cluster has started before any pushes into another's shared memory (the
    // matching wait comes after the key loop)
    asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
    // The context lengths and the cached context keys/values were written before the kernel
    // that precedes this one (the Q/K^d/V^d projection, which signals its dependents only after
    // its own dependency wait), so they are complete here; Q, K^d and V^d are read after the
    // wait below.
    const int L = a.ctx_len[b];
    // the sequence's tiles: ceil(L / 64) context tiles, then the block tile; split s takes a
    // contiguous run of them (the counts differ by at most one)
    const int n_ctx_tiles = (L + kKT - 1) / kKT, T = n_ctx_tiles + 1;
    const int t0 = s * (T / S) + min(s, T % S);
    const int n_tiles = T / S + (s < T % S ? 1 : 0);
    const int n_ct = max(0, min(t0 + n_tiles, n_ctx_tiles) - t0);   // context tiles of this CTA
    // tile t -> stage t % kNST: K at [stage][0, TB), V at [stage][TB, 2 TB)
    auto issue = [&](int t) {
        const int st = t % kNST;
        const uint32_t kdst = sbase + (uint32_t)st * 2 * TB, bar = fbar + 8u * st;
        const uint32_t bytes = t < n_ct ? 2 * TB : 2u * (HD / 64) * (uint32_t)a.block_rows * 128u;
        asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
                     : "memory");
        for (int h = 0; h < HD / 64; ++h) {
            if (t < n_ct) {
                const int y = (t0 + t) * kKT, z = b * a.hkv + g;
                tma_tile(kdst + h * 8192, &maps.kc, h * 64, y, z, bar);
                tma_tile(kdst + TB + h * 8192, &maps.vc, h * 64, y, z, bar);
            } else {
                tma_tile(kdst + h * 8192, &maps.kd, h * 64, b * a.B, g, bar);
                tma_tile(kdst + TB + h * 8192, &maps.vd, h * 64, b * a.B, g, bar);
            }
        }
    };
    int issued = 0, consumed = 0;
    bool prod_ok = true;   // thread 0: every wait for an emptied stage ended in time
    // thread 0 refills the stage of tile `issued` once all four warps have read the tile that
    // used it before (tile issued - kNST)
    auto refill = [&]() {
        if (issued >= kNST)
            prod_ok = tile_wait(ebar + 8u * (issued % kNST), (uint32_t)(issued / kNST - 1) & 1u);
        if (prod_ok) issue(issued++);
    };
    // the first context tile streams in while the projection drains; the block tile waits
    if (tid == 0)
        for (; issued < min(kNST - 1, n_ct); ++issued) issue(issued);
    pdl_wait();
    if (a.t_stamps && tid == 0) atomicMin(a.t_stamps + a.t_slots, (unsigned long long)globaltimer_ns());
    if (a.qkv32 && n_tiles > n_ct) {
        // this CTA holds the block tile: its head's K^d (rotated) and V^d rows, rounded to bf16,
        // go to kd / vd for the tile's TMA load (identical values from every query tile's CTA)
        const int nb = a.B * (HD / 16), n32 = a.d_q + 2 * a.d_kv;
        for (int it = tid; it < 2 * nb; it += blockDim.x) {
            const bool is_v = it >= nb;
            const int k = (it % nb) / (HD / 16), j0 = ((it % nb) % (HD / 16)) * 8;
            const float* src = a.qkv32 + ((size_t)b * a.B + k) * n32 + a.d_q + (is_v ? a.d_kv : 0) + g * HD;
            float x1[8], x2[8], o1[8], o2[8];
            load8(src + j0, x1);
            load8(src + j0 + HD / 2, x2);
            if (!is_v && a.rope) {
                float cs[8], sn[8];
                load8(a.rope_cos + (size_t)(L + k) * (HD / 2) + j0, cs);
                load8(a.rope_sin + (size_t)(L + k) * (HD / 2) + j0, sn);
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    o1[e] = x1[e] * cs[e] - x2[e] * sn[e];
                    o2[e] = x2[e] * cs[e] + x1[e] * sn[e];
                }
            } else {
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    o1[e] = x1[e];
                    o2[e] = x2[e];
                }
            }
            bf16* dst = (is_v ? a.vd_w : a.kd_w) + ((size_t)b * a.B + k) * a.d_kv + g * HD + j0;
            store8(dst, o1);
            store8(dst + HD / 2, o2);
        }
        // the generic stores above before the tensor-memory-access reads of the block tile
        asm volatile("fence.proxy.async.global;" ::: "memory");
        __syncthreads();
    }
    if (tid == 0)
        for (; issued < min(kNST - 1, n_tiles); ++issued) issue(issued);

    float o[HD / 8][4];
#pragma unroll
    for (int i = 0; i < HD / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
    float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
    bool timed_out = false;
    if (n_tiles > 0) {
        const bf16* q = static_cast<const bf16*>(a.q);
        const uint32_t sQ = smem_addr(Qs);
        // query rows of this tile: row r -> block position r / G, head g*G + r % G
        if (a.qkv32) {
            // from the fp32 sums: the rotary embedding at position L + block position, then bf16
            const int n32 = a.d_q + 2 * a.d_kv;
            for (int idx = tid; idx < kQT * (HD / 16); idx += blockDim.x) {
                const int r = idx / (HD / 16), j0 = (idx % (HD / 16)) * 8;
                const int rr = qt * kQT + r;
                float o1[8], o2[8];
                if (rr < R) {
                    const int kpos = rr / a.G, hh = rr % a.G;
                    const float* src = a.qkv32 + ((size_t)b * a.B + kpos) * n32 + (size_t)(g * a.G + hh) * HD;
                    float x1[8], x2[8];
                    load8(src + j0, x1);
                    load8(src + j0 + HD / 2, x2);
                    if (a.rope) {
                        float cs[8], sn[8];
                        load8(a.rope_cos + (size_t)(L + kpos) * (HD / 2) + j0, cs);
                        load8(a.rope_sin + (size_t)(L + kpos) * (HD / 2) + j0, sn);
#pragma unroll
                        for (int e = 0; e < 8; ++e) {
                            o1[e] = x1[e] * cs[e] - x2[e] * sn[e];
                            o2[e] = x2[e] * cs[e] + x1[e] * sn[e];
                        }
                    } else {
#pragma unroll
                        for (int e = 0; e < 8; ++e) {
                            o1[e] = x1[e];
                            o2[e] = x2[e];
                        }
                    }
                } else {
#pragma unroll
                    for (int e = 0; e < 8; ++e) o1[e] = o2[e] = 0.f;
                }
                store8(Qs + r * LD + j0, o1);
                store8(Qs + r * LD + j0 + HD / 2, o2);
            }
        } else {
            for (int idx = tid; idx < kQT * PIECES; idx += blockDim.x) {
                const int r = idx / PIECES, pc = idx % PIECES;
                const int rr = qt * kQT + r;
                const bool ok = rr < R;
                const int kpos = ok ? rr / a.G : 0, hh = ok ? rr % a.G : 0;
                const bf16* src = q + ((size_t)b * a.B + kpos) * a.d_q + (size_t)(g * a.G + hh) * HD + pc * 8;
                cp_async16(sQ + (uint32_t)(r * LD + pc * 8) * 2, src, ok);
            }
        }
        cp_commit();
        // the query tile is complete in shared memory before the loop (the only CTA barrier on
        // this path before the loop ends; the first K/V tile is already in flight)
        cp_wait<0>();
        __syncthreads();
        uint32_t qa[HD / 16][4];
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) {
            const int row = warp * 16 + (lane & 15), col = kk * 16 + (lane >> 4) * 8;
            ldsm_x4(sQ + (uint32_t)(row * LD + col) * 2, qa[kk][0], qa[kk][1], qa[kk][2], qa[kk][3]);
        }
        for (int t = 0; t < n_tiles; ++t) {
            const int st = t % kNST;
            if (tid == 0 && prod_ok && issued < n_tiles) refill();   // tile t + kNST - 1
            const bool landed = tile_wait(fbar + 8u * st, (uint32_t)(t / kNST) & 1u);
            // each warp decides for itself (no CTA barrier inside the loop); a warp that gives
            // up stops reading tiles and arriving on the empty barriers, so thread 0's next wait
            // for an emptied stage runs out as well
            if (__any_sync(0xffffffffu, !landed || (tid == 0 && !prod_ok))) {
                timed_out = true;
                break;
            }
            ++consumed;
            // keys past the tile's valid ones get P = 0; their V rows are finite (the caches and
            // the K^d / V^d buffers are zeroed at creation and only ever hold written values),
            // so they add nothing
            const int valid = t < n_ct ? min(kKT, L - (t0 + t) * kKT) : a.B;
            const uint32_t sK = sbase + (uint32_t)st * 2 * TB, sV = sK + TB;
            // S = Q K^T for 16 rows x 64 keys
            // (k outer, keys inner: eight independent accumulators between dependent MMAs)
            float sc[8][4];
#pragma unroll
            for (int nt = 0; nt < 8; ++nt) sc[nt][0] = sc[nt][1] = sc[nt][2] = sc[nt][3] = 0.f;
#pragma unroll
            for (int kk = 0; kk < HD / 16; kk += 2) {
#pragma unroll
                for (int nt = 0; nt < 8; ++nt) {
                    const int row = nt * 8 + (lane & 7);
                    const int c8 = kk * 2 + (lane >> 3);
                    uint32_t b0, b1, b2, b3;
                    ldsm_x4(sK + swz(row, c8), b0, b1, b2, b3);
                    mma16816(sc[nt], qa[kk], b0, b1);
                    mma16816(sc[nt], qa[kk + 1], b2, b3);
                }
            }
            // mask keys past the tile's valid ones, scale into the log2 domain, online softmax
            float mx0 = m0, mx1 = m1;
#pragma unroll
            for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                    const bool ok = nt * 8 + (lane & 3) * 2 + e < valid;
                    sc[nt][e] = ok ? sc[nt][e] * a.scale_log2 : -INFINITY;
                    sc[nt][2 + e] = ok ? sc[nt][2 + e] * a.scale_log2 : -INFINITY;
                    mx0 = fmaxf(mx0, sc[nt][e]);
                    mx1 = fmaxf(mx1, sc[nt][2 + e]);
                }
            }
#pragma unroll
            for (int off = 1; off <= 2; off <<= 1) {
                mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, off));
                mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, off));
            }
            const float cr0 = ex2(m0 - mx0), cr1 = ex2(m1 - mx1);
            m0 = mx0;
            m1 = mx1;
            l0 *= cr0;
            l1 *= cr1;
#pragma unroll
            for (int i = 0; i < HD / 8; ++i) {
                o[i][0] *= cr0; o[i][1] *= cr0; o[i][2] *= cr1; o[i][3] *= cr1;
            }
#pragma unroll
            for (int nt = 0; nt < 8; ++nt) {
                sc[nt][0] = ex2(sc[nt][0] - m0);
                sc[nt][1] = ex2(sc[nt][1] - m0);
                sc[nt][2] = ex2(sc[nt][2] - m1);
                sc[nt][3] = ex2(sc[nt][3] - m1);
                l0 += sc[nt][0] + sc[nt][1];
                l1 += sc[nt][2] + sc[nt][3];
            }
            // O += P V (P from registers as the A operand; V tiles transposed by ldmatrix)
#pragma unroll
            for (int kk = 0; kk < kKT / 16; ++kk) {
                uint32_t pa[4];
                pa[0] = pack_bf16(sc[2 * kk][0], sc[2 * kk][1]);
                pa[1] = pack_bf16(sc[2 * kk][2], sc[2 * kk][3]);
                pa[2] = pack_bf16(sc[2 * kk + 1][0], sc[2 * kk + 1][1]);
                pa[3] = pack_bf16(sc[2 * kk + 1][2], sc[2 * kk + 1][3]);
#pragma unroll
                for (int nt = 0; nt < HD / 8; nt += 2) {
                    const int row = kk * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
                    const int c8 = nt + (lane >> 4);
                    uint32_t b0, b1, b2, b3;
                    ldsm_x4_t(sV + swz(row, c8), b0, b1, b2, b3);
                    mma16816(o[nt], pa, b0, b1);
                    mma16816(o[nt + 1], pa, b2, b3);
                }
            }
            __syncwarp();
            if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(ebar + 8u * st) : "memory");
        }
        cp_wait<0>();
#pragma unroll
        for (int off = 1; off <= 2; off <<= 1) {
            l0 += __shfl_xor_sync(0xffffffffu, l0, off);
            l1 += __shfl_xor_sync(0xffffffffu, l1, off);
        }
    }
    if (timed_out && lane == 0) atomicOr(a.err, DFLARE_DEVERR_TIMEOUT);
    // copies still in flight (only after a timeout) land before this shared memory is reused or
    // released; then every warp is done with the K/V stages, which the push below reuses
    if (tid == 0)
        for (int t = consumed; t < issued; ++t) tile_wait(fbar + 8u * (t % kNST), (uint32_t)(t / kNST) & 1u);
    __syncthreads();
    asm volatile("barrier.cluster.wait.aligned;" ::: "memory");
    // push the partial: query row r belongs to the merge slice of CTA r / RP, which keeps it at
    // [s * RP + r % RP]; O is normalised by l first (|O / l| <= max |V|, safe in fp16). The rows
    // are staged in this CTA's (now idle) tile memory so that the remote stores are 16 bytes wide.
    {
        __half* stg = reinterpret_cast<__half*>(smem);   // [kQT][HD]
        const int r0 = warp * 16 + (lane >> 2), r1 = r0 + 8;
        const float i0 = l0 > 0.f ? 1.0f / l0 : 0.f, i1 = l1 > 0.f ? 1.0f / l1 : 0.f;
#pragma unroll
        for (int nt = 0; nt < HD / 8; ++nt) {
            const int col = nt * 8 + (lane & 3) * 2;
            *reinterpret_cast<__half2*>(stg + r0 * HD + col) = __floats2half2_rn(o[nt][0] * i0, o[nt][1] * i0);
            *reinterpret_cast<__half2*>(stg + r1 * HD + col) = __floats2half2_rn(o[nt][2] * i1, o[nt][3] * i1);
        }
        if ((lane & 3) == 0) {
            *reinterpret_cast<float2*>(cluster.map_shared_rank(rML, r0 / RP) + 2 * (s * RP + r0 % RP)) =
                make_float2(m0, l0);
            *reinterpret_cast<float2*>(cluster.map_shared_rank(rML, r1 / RP) + 2 * (s * RP + r1 % RP)) =
                make_float2(m1, l1);
        }
        __syncthreads();
        for (int k = tid; k < kQT * PIECES; k += blockDim.x) {
            const int r = k / PIECES, pc = k % PIECES;
            *reinterpret_cast<uint4*>(cluster.map_shared_rank(rO, r / RP) + (size_t)(s * RP + r % RP) * HD + pc * 8) =
                *reinterpret_cast<const uint4*>(stg + r * HD + pc * 8);
        }
    }
    // every partial has arrived; after this barrier no CTA touches another's shared memory
    cluster.sync();
    // merge: TPR threads per row of this CTA's slice, EPT contiguous output elements per thread,
    // out = sum_p w_p (O_p / l_p) / sum_p w_p with w_p = l_p 2^(m_p - max m)
    constexpr int TPR = 128 / RP, EPT = HD / TPR;
    static_assert(EPT % 2 == 0, "merge slice must be a whole number of half2");
    const int lr = tid / TPR, lt = tid % TPR;
    const int rg = qt * kQT + s * RP + lr;
    if (rg < R) {
        float w[S];
        float M = -INFINITY;
#pragma unroll
        for (int p = 0; p < S; ++p) M = fmaxf(M, rML[2 * (p * RP + lr)]);
        float den = 0.f;
#pragma unroll
        for (int p = 0; p < S; ++p) {
            const float mp = rML[2 * (p * RP + lr)], lp = rML[2 * (p * RP + lr) + 1];
            w[p] = mp == -INFINITY ? 0.f : lp * exp2f(mp - M);
            den += w[p];
        }
        const float inv = 1.0f / den;
        const int kpos = rg / a.G, hh = rg % a.G;
        bf16* orow = out + ((size_t)b * a.B + kpos) * a.d_q + (size_t)(g * a.G + hh) * HD + lt * EPT;
#pragma unroll
        for (int q = 0; q < EPT; q += 2) {
            float v0 = 0.f, v1 = 0.f;
#pragma unroll
            for (int p = 0; p < S; ++p) {
                const float2 f = __half22float2(*reinterpret_cast<const __half2*>(rO + (size_t)(p * RP + lr) * HD + lt * EPT + q));
                v0 = fmaf(w[p], f.x, v0);
                v1 = fmaf(w[p], f.y, v1);
            }
            *reinterpret_cast<__nv_bfloat162*>(orow + q) = __floats2bfloat162_rn(v0 * inv, v1 * inv);
        }
    }
    if (a.t_stamps) {
        __syncthreads();
        if (tid == 0) atomicMax(a.t_stamps + 2 * a.t_slots, (unsigned long long)globaltimer_ns());
    }
}

// ------------------------------------------------------------------ bf16, tcgen05 (Blackwell)
//
// The same split-KV cluster attention on the fifth-generation tensor cores. One CTA per (key
// split, KV head, 128-row query tile, sequence); the 128 query rows are the UMMA M (the B x G
// rows of a KV head: 64 for the Qwen3 shapes, the rest zero; 128 for GPT-OSS, whose two 64-row
// halves then read every key tile once instead of twice). Per 64-key tile t:
//   S_t = Q K_t^T   M 128 x N 64 x K head_dim into TMEM; Q and K K-major in 128-byte-swizzled
//                   shared memory;
//   softmax         thread r of a softmax warpgroup = query row r = TMEM lane r: P_t = 2^(s - m)
//                   rounded to bf16 into a K-major swizzled shared tile, the row sum l taken from
//                   the fp32 P;
//   O += P_t V_t    M 128 x N head_dim x K 64; V read MN-major as the TMA wrote it; O stays in
//                   TMEM for the whole key range.
// Two softmax warpgroups take alternate tiles, each with its own S, P and O buffers and its own
// running (m, l), so each SM sub-partition always has a second softmax warp to switch to; their
// two partial results are combined per row at the end. Within a warpgroup the maximum m that a
// row's P and O are taken against is raised only when a tile's maximum exceeds it by more than
// 2^8; then the row's O (P V of the group's previous tile has completed by then) and its l are
// scaled by 2^(m_old - m_new) before the tile's P is written. Otherwise P <= 2^8, which bf16 and
// the fp32 accumulators carry with the same relative precision, and O / l does not depend on
// the choice of m.
// One warp streams the K/V tiles by TMA into a ring of stages. Two threads in two more warps issue
// the MMAs: one S_t as soon as tile t has landed and S_{t-2} has been read out of TMEM (so S runs
// two tiles ahead of the softmax), the other P_t V_t as soon as P_t is written. Measured: every
// M 128 MMA with N <= 128 occupies the tensor pipe for about 71 cycles, a commit-to-wait round
// trip of four MMAs takes about 740 cycles, and one thread issuing both kinds, on a sub-partition
// shared with two softmax warps, took 0.3-0.45 us per hand-off; the issuing warps sit on the
// sub-partitions that the 64-row (Qwen3-shaped) tiles leave free of softmax work.
// Every hand-off is an mbarrier with a bounded wait. The cluster may hold any number of splits
// from 1 to 16 (at one CTA per SM, the largest size whose clusters all fit at once); after the key
// loop and a cluster barrier each CTA pushes its combined partial of every query row into the
// (then idle) K/V stages of the CTA that merges that row.
constexpr int kTQ = 128;            // query rows per CTA (UMMA M)
constexpr int kTThreads = 384;      // warps 0-3, 4-7: softmax groups; 8: TMA; 9: TMEM; 10, 11: MMA
constexpr float kRescale = 8.0f;    // growth (log2) of a row maximum that triggers a rescale

constexpr int kMaxSplits = 16;     // cluster size limit (non-portable above 8)
template <int HD>
struct TcAttnLayout {
    static constexpr int NS = HD == 128 ? 4 : 10;              // 64-key K and V slots (even)
    static constexpr uint32_t TB = HD * 128;                    // one 64-key K or V tile
    static constexpr uint32_t KR = 0;                           // K ring [HD/64][NS][64 rows][128 B]
    static constexpr uint32_t VR = NS * TB;                     // V ring [NS][HD/64][64 rows][128 B]
    static constexpr uint32_t Q = NS * 2 * TB;                  // Q [HD/64][128 rows][128 B]
    static constexpr uint32_t P = Q + (uint32_t)kTQ * HD * 2;   // P [group][128 rows][64 keys] bf16
    static constexpr uint32_t BARS = P + 2u * kTQ * 128;        // mbarriers, then two words
    static constexpr int NBARS = 4 * NS + 10;
    static constexpr uint32_t BYTES = BARS + NBARS * 8 + 16;
    // head_dim 128: S of two adjacent 64-key tiles in one N 128 MMA chain (half the S MMAs; the
    // kernel is tensor-bound there); head_dim 64: S per tile (its S MMAs are cheap and the softmax
    // groups overlap better when they alternate than when they work on a pair in lockstep)
    static constexpr bool PAIR = HD == 128;
    static constexpr int W = PAIR ? 2 : 1;                      // 64-key tiles per S unit
    static_assert(NS % 2 == 0, "pairs of adjacent K slots form one N 128 operand");
    // After the key loop the (then idle) stages hold the cluster merge: the pushed partials O / l
    // in fp16 [S RP <= 128 + 15 rows][HD], their (m, l) and the merge weights [RP][S].
    static constexpr int MR = kTQ + kMaxSplits;
    static constexpr uint32_t RO = 0;
    static constexpr uint32_t RML = (uint32_t)MR * HD * 2;
    static constexpr uint32_t RW = RML + (uint32_t)MR * 8;
    static constexpr uint32_t TMEM_COLS = 512;                  // S of two tile pairs (128 each), O_A, O_B
    static_assert(RW + (uint32_t)MR * kMaxSplits * 4 <= NS * 2 * TB, "merge buffers exceed the stages");
    static_assert(1024 + BYTES <= 232448, "tcgen05 attention exceeds 227 KB of shared memory");
};
template <int HD>
size_t tc_attn_smem_bytes() { return 1024 + TcAttnLayout<HD>::BYTES; }

__device__ __forceinline__ void ta_mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void ta_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void ta_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
                 : "memory");
}
// try_wait with a suspend-time hint: the thread sleeps until the phase completes or the hint
// (ns) elapses instead of spinning, which leaves its sub-partition's issue slots to the softmax
// warps there
__device__ __forceinline__ bool try_wait_parity_sleep(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity), "r"(100000u)
        : "memory");
    return ok != 0;
}
// Bounded wait for the phase of `bar` with parity `parity`: false after kWaitNs (which sets the
// CTA's abort flag and the device error) or once another thread of the CTA has aborted. The timer
// is read only when the first (sleeping) poll has not seen the phase complete.
__device__ __noinline__ bool ta_wait_slow(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                          uint32_t* err) {
    const uint64_t t0 = globaltimer_ns();
    while (true) {
        if (try_wait_parity_sleep(bar, parity)) return true;
        if (*abort_flag) return false;
        if (globaltimer_ns() - t0 > kWaitNs) {
            *abort_flag = 1;
            atomicOr(err, DFLARE_DEVERR_TIMEOUT);
            return false;
        }
    }
}
__device__ __forceinline__ bool ta_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                        uint32_t* err) {
    if (try_wait_parity_sleep(bar, parity)) return true;
    return ta_wait_slow(bar, parity, abort_flag, err);
}
__device__ __forceinline__ void ta_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void ta_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// Shared-memory matrix descriptors (128-byte swizzle, version 1). K-major: 128-byte rows, 8-row
// groups 1024 bytes apart. MN-major (V: the head dims contiguous, the keys the contraction):
// 64-element swizzle atoms along N 8192 bytes apart, 8-key groups 1024 bytes apart.
__device__ __forceinline__ uint64_t ta_desc_k(uint32_t saddr) {
    return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
           ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}
__device__ __forceinline__ uint64_t ta_desc_mn(uint32_t saddr) {
    return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)(8192 >> 4) << 16) |
           ((uint64_t)(1024 >> 4) << 32) | ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}
__device__ __forceinline__ void ta_mma(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                       uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(idesc), "r"(accumulate)
        : "memory");
}
__device__ __forceinline__ void ta_commit(uint32_t bar) {
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
        : "memory");
}
__device__ __forceinline__ void ta_ld32(uint32_t taddr, float* v) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
        "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
          "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
          "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
          "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ void ta_st32(uint32_t taddr, const float* v) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
        "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, "
        "%17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr),
        "f"(v[0]), "f"(v[1]), "f"(v[2]), "f"(v[3]), "f"(v[4]), "f"(v[5]), "f"(v[6]), "f"(v[7]),
        "f"(v[8]), "f"(v[9]), "f"(v[10]), "f"(v[11]), "f"(v[12]), "f"(v[13]), "f"(v[14]), "f"(v[15]),
        "f"(v[16]), "f"(v[17]), "f"(v[18]), "f"(v[19]), "f"(v[20]), "f"(v[21]), "f"(v[22]), "f"(v[23]),
        "f"(v[24]), "f"(v[25]), "f"(v[26]), "f"(v[27]), "f"(v[28]), "f"(v[29]), "f"(v[30]), "f"(v[31])
        : "memory");
}
// rotate-half rotary embedding of 8 + 8 head dims (j0 .. j0+7 and j0 + hd/2 ..) at one position
__device__ __forceinline__ void rope8(const float* x1, const float* x2, const float* cs, const float* sn,
                                      float* o1, float* o2) {
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        o1[e] = x1[e] * cs[e] - x2[e] * sn[e];
        o2[e] = x2[e] * cs[e] + x1[e] * sn[e];
    }
}

template <int HD>
__global__ void __launch_bounds__(kTThreads, 1) attn_tc_kernel(const __grid_constant__ AttnMaps maps,
                                                              const AttnArgs a, bf16* __restrict__ out) {
    using LY = TcAttnLayout<HD>;
    constexpr int NS = LY::NS;
    constexpr uint32_t TB = LY::TB;
    const int S = a.splits;                     // the cluster: one CTA per split
    if (a.t_stamps && threadIdx.x == 0) atomicMin(a.t_stamps, (unsigned long long)globaltimer_ns());
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = smem_raw + ((1024u - (smem_addr(smem_raw) & 1023u)) & 1023u);
    const uint32_t sbase = smem_addr(smem);
    const uint32_t bar0 = sbase + LY::BARS;
    // kfull / vfull[NS] (the slot's K / V tile landed), kempty[NS] (the S that read it completed),
    // vempty[NS] (its P V completed); per S buffer i (S units u with u % 2 = i; a unit is a tile
    // pair at head_dim 128, a tile at 64): sfull[i] (S of the unit in TMEM), sfree[i] (read by the
    // softmax warps of the unit: 8 for a pair, 4 for a tile); per softmax group q: pready[q] (its P
    // written), odone[q] (its P V completed); one drain per MMA-issuing thread
    auto kfull_bar = [&](int st) { return bar0 + 8u * st; };
    auto kempty_bar = [&](int st) { return bar0 + 8u * (NS + st); };
    auto vfull_bar = [&](int st) { return bar0 + 8u * (2 * NS + st); };
    auto vempty_bar = [&](int st) { return bar0 + 8u * (3 * NS + st); };
    auto sfull_bar = [&](int i) { return bar0 + 8u * (4 * NS + i); };
    auto sfree_bar = [&](int i) { return bar0 + 8u * (4 * NS + 2 + i); };
    auto pready_bar = [&](int q) { return bar0 + 8u * (4 * NS + 4 + q); };
    auto odone_bar = [&](int q) { return bar0 + 8u * (4 * NS + 6 + q); };
    auto drain_bar = [&](int i) { return bar0 + 8u * (4 * NS + 8 + i); };
    uint32_t* misc = reinterpret_cast<uint32_t*>(smem + LY::BARS + LY::NBARS * 8);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(&misc[1]);
    cg::cluster_group cluster = cg::this_cluster();
    const int s = (int)cluster.block_rank();
    const int g = blockIdx.y % a.hkv, qt = blockIdx.y / a.hkv, b = blockIdx.z;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int R = a.B * a.G;
    const int rows = min(kTQ, R - qt * kTQ);    // query rows of this tile

    // rows [block_rows, 64) of the V stages are never written by the block tile's copy: zero
    // them once (P is 0 there, and 0 x garbage could be NaN)
    if (a.block_rows < kKT) {
        const int zr = kKT - a.block_rows;
        for (int k = tid; k < NS * (HD / 64) * zr * 8; k += blockDim.x) {
            const int piece = k & 7, r = a.block_rows + (k >> 3) % zr, sub = (k >> 3) / zr;
            const int st = sub / (HD / 64), h = sub % (HD / 64);
            *reinterpret_cast<uint4*>(smem + LY::VR + (size_t)st * TB + h * 8192 + r * 128 + piece * 16) =
                make_uint4(0u, 0u, 0u, 0u);
        }
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    if (tid == 0) {
        for (int i = 0; i < NS; ++i) {
            ta_mbar_init(kfull_bar(i), 1);
            ta_mbar_init(kempty_bar(i), 1);
            ta_mbar_init(vfull_bar(i), 1);
            ta_mbar_init(vempty_bar(i), 1);
        }
        for (int q = 0; q < 2; ++q) {
            ta_mbar_init(sfull_bar(q), 1);
            ta_mbar_init(sfree_bar(q), LY::PAIR ? 8 : 4);
            ta_mbar_init(pready_bar(q), 4);
            ta_mbar_init(odone_bar(q), 1);
        }
        ta_mbar_init(drain_bar(0), 1);
        ta_mbar_init(drain_bar(1), 1);
        misc[1] = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&maps.kc)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&maps.vc)) : "memory");
    }
    if (warp == 9) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_addr(&misc[0])),
                     "r"(LY::TMEM_COLS)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    ta_fence_before();
    __syncthreads();
    ta_fence_after();
    const uint32_t tmem = misc[0];
    // dependents are released only once this CTA holds its tensor memory, so a dependent CTA
    // that allocates before its own dependency wait can never hold columns this CTA waits for
    pdl_trigger();
    // The context lengths and cached keys/values were written before the kernel that precedes
    // this one (which signals its dependents only after its own dependency wait); Q, K^d and V^d
    // are read after the wait below.
    const int L = a.ctx_len[b];
    const int n_ctx_tiles = (L + kKT - 1) / kKT, T = n_ctx_tiles + 1;
    const int t0 = s * (T / S) + min(s, T % S);
    const int n_tiles = T / S + (s < T % S ? 1 : 0);
    const int n_ct = max(0, min(t0 + n_tiles, n_ctx_tiles) - t0);
    constexpr int W = LY::W;
    const int n_units = (n_tiles + W - 1) / W;   // S units: tiles W u .. W u + W - 1
    // 64-key tile t -> slot t % NS: K atom h at KR + (h NS + slot) 8192 (two adjacent slots of an
    // atom are one 128-row operand), V at VR + slot TB + h 8192
    auto issue = [&](int t, bool v) {
        const int st = t % NS;
        const uint32_t bar = v ? vfull_bar(st) : kfull_bar(st);
        ta_expect_tx(bar, t < n_ct ? TB : (HD / 64) * (uint32_t)a.block_rows * 128u);
        for (int h = 0; h < HD / 64; ++h) {
            const uint32_t dst = v ? sbase + LY::VR + (uint32_t)st * TB + h * 8192u
                                   : sbase + LY::KR + (uint32_t)(h * NS + st) * 8192u;
            if (t < n_ct)
                tma_tile(dst, v ? &maps.vc : &maps.kc, h * 64, (t0 + t) * kKT, b * a.hkv + g, bar);
            else
                tma_tile(dst, v ? &maps.vd : &maps.kd, h * 64, b * a.B, g, bar);
        }
    };
    int issued = 0;   // warps 8 (K) and 9 (V), lane 0
    // the first context tiles stream in while the projection drains; the block tile waits
    if ((warp == 8 || warp == 9) && lane == 0)
        for (; issued < min(NS, n_ct); ++issued) issue(issued, warp == 9);
    pdl_wait();
    if (a.t_stamps && tid == 0) atomicMin(a.t_stamps + a.t_slots, (unsigned long long)globaltimer_ns());
    const int n32 = a.d_q + 2 * a.d_kv;
    if (a.qkv32 && n_tiles > n_ct) {
        // this CTA holds the block tile: its head's K^d (rotated) and V^d rows, rounded to bf16,
        // go to kd / vd for the tile's TMA load (identical values from every query tile's CTA)
        const int nb = a.B * (HD / 16);
        for (int it = tid; it < 2 * nb; it += blockDim.x) {
            const bool is_v = it >= nb;
            const int k = (it % nb) / (HD / 16), j0 = ((it % nb) % (HD / 16)) * 8;
            const float* src = a.qkv32 + ((size_t)b * a.B + k) * n32 + a.d_q + (is_v ? a.d_kv : 0) + g * HD;
            float x1[8], x2[8], o1[8], o2[8];
            load8(src + j0, x1);
            load8(src + j0 + HD / 2, x2);
            if (!is_v && a.rope) {
                float cs[8], sn[8];
                load8(a.rope_cos + (size_t)(L + k) * (HD / 2) + j0, cs);
                load8(a.rope_sin + (size_t)(L + k) * (HD / 2) + j0, sn);
                rope8(x1, x2, cs, sn, o1, o2);
            } else {
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    o1[e] = x1[e];
                    o2[e] = x2[e];
                }
            }
            bf16* dst = (is_v ? a.vd_w : a.kd_w) + ((size_t)b * a.B + k) * a.d_kv + g * HD + j0;
            store8(dst, o1);
            store8(dst + HD / 2, o2);
        }
        // the generic stores above before the tensor-memory-access reads of the block tile
        asm volatile("fence.proxy.async.global;" ::: "memory");
    }
    // Q: row r of the tile is block position (qt * 128 + r) / G of query head
    // g G + (qt * 128 + r) % G, stored K-major and swizzled as [HD/64][128 rows][128 B]; rows
    // past R are zero. Four items per thread are loaded before any is converted, so that their
    // global reads are in flight together.
    if (n_tiles > 0) {
        constexpr int NQ = kTQ * (HD / 16), U = (NQ + kTThreads - 1) / kTThreads;
        const bool rot = a.qkv32 && a.rope;
        float x1[U][8], x2[U][8], cs[U][8], sn[U][8];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int idx = tid + u * kTThreads;
            const int r = idx / (HD / 16), j0 = (idx % (HD / 16)) * 8;
            const int rr = qt * kTQ + r;
            if (idx < NQ && rr < R) {
                const int kpos = rr / a.G, hh = rr % a.G;
                if (a.qkv32) {
                    const float* src = a.qkv32 + ((size_t)b * a.B + kpos) * n32 + (size_t)(g * a.G + hh) * HD;
                    load8(src + j0, x1[u]);
                    load8(src + j0 + HD / 2, x2[u]);
                    if (rot) {
                        load8(a.rope_cos + (size_t)(L + kpos) * (HD / 2) + j0, cs[u]);
                        load8(a.rope_sin + (size_t)(L + kpos) * (HD / 2) + j0, sn[u]);
                    }
                } else {
                    const bf16* src = static_cast<const bf16*>(a.q) + ((size_t)b * a.B + kpos) * a.d_q +
                                      (size_t)(g * a.G + hh) * HD;
                    load8(src + j0, x1[u]);
                    load8(src + j0 + HD / 2, x2[u]);
                }
            } else {
#pragma unroll
                for (int e = 0; e < 8; ++e) x1[u][e] = x2[u][e] = 0.f;
            }
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int idx = tid + u * kTThreads;
            if (idx >= NQ) break;
            const int r = idx / (HD / 16), j0 = (idx % (HD / 16)) * 8;
            float o1[8], o2[8];
            if (rot && qt * kTQ + r < R) {
                rope8(x1[u], x2[u], cs[u], sn[u], o1, o2);
            } else {
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    o1[e] = x1[u][e];
                    o2[e] = x2[u][e];
                }
            }
            const int c1 = j0 / 8, c2 = (j0 + HD / 2) / 8;   // 16-byte chunks of the row
            store8(reinterpret_cast<bf16*>(smem + LY::Q + (c1 >> 3) * (kTQ * 128) + r * 128 +
                                           (((c1 & 7) ^ (r & 7)) << 4)), o1);
            store8(reinterpret_cast<bf16*>(smem + LY::Q + (c2 >> 3) * (kTQ * 128) + r * 128 +
                                           (((c2 & 7) ^ (r & 7)) << 4)), o2);
        }
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    __syncthreads();

    // instruction descriptors: fp32 accumulator, bf16 A and B, M 128; S: N 64 per tile of the unit
    // (128 for a pair), both K-major; P V: N = HD, B (V) MN-major
    constexpr uint32_t kIdBase = (1u << 4) | (1u << 7) | (1u << 10) | ((128u >> 4) << 24);
    constexpr uint32_t kIdS2 = kIdBase | ((128u >> 3) << 17), kIdS1 = kIdBase | ((64u >> 3) << 17);
    constexpr uint32_t kIdO = kIdBase | (1u << 16) | (((uint32_t)HD >> 3) << 17);
    // TMEM columns: S of unit u at [128 (u % 2), + 64 W) (tile W u + h in columns 64 h + ...), O of
    // softmax group q at [256 + HD q, + HD)
    auto tS = [&](int i) { return tmem + 128u * i; };
    auto tO = [&](int q) { return tmem + 256u + (uint32_t)HD * q; };
    float m_used = -INFINITY, l = 0.f;
    bool ok = true;

    if (warp == 8 || warp == 9) {
        if (lane == 0) {
            // ---------------- TMA producers, warp 8 for K and warp 9 for V: the slot of tile t is
            // refilled once the S (K) or the P V (V) of tile t - NS has completed
            const bool v = warp == 9;
            for (; issued < n_tiles; ++issued) {
                const int st = issued % NS;
                if (issued >= NS && !(ok = ta_wait(v ? vempty_bar(st) : kempty_bar(st), (uint32_t)(issued / NS - 1) & 1u,
                                                   abort_flag, a.err)))
                    break;
                issue(issued, v);
            }
            // after an abort, the copies in flight land before the shared memory is reused
            if (!ok) {
                volatile int never = 0;
                for (int t = max(0, issued - NS); t < issued; ++t)
                    ta_wait(v ? vfull_bar(t % NS) : kfull_bar(t % NS), (uint32_t)(t / NS) & 1u, &never, a.err);
            }
        }
        __syncwarp();
    } else if (warp == 10) {
        if (lane == 0 && n_tiles > 0) {
            // ---------------- S issue (one thread): S of unit u into S buffer u % 2 once its K tiles
            // have landed and the softmax warps have read unit u - 2; descriptors advance by
            // address >> 4
            const uint64_t dQ = ta_desc_k(sbase + LY::Q);
            for (int p = 0; p < n_units && ok; ++p) {
                const int ta = W * p, i = p & 1, nsub = min(W, n_tiles - ta);
                for (int h = 0; h < nsub && ok; ++h)
                    ok = ta_wait(kfull_bar((ta + h) % NS), (uint32_t)((ta + h) / NS) & 1u, abort_flag, a.err);
                if (!ok) break;
                if (p >= 2 && !(ok = ta_wait(sfree_bar(i), (uint32_t)((p >> 1) - 1) & 1u, abort_flag, a.err))) break;
                ta_fence_after();
                const uint64_t dK = ta_desc_k(sbase + LY::KR + (uint32_t)(ta % NS) * 8192u);
                const uint32_t id = nsub == 2 ? kIdS2 : kIdS1;
#pragma unroll
                for (int kk = 0; kk < HD / 16; ++kk)
                    ta_mma(tS(i), dQ + (uint64_t)((kk >> 2) * (kTQ * 128 / 16) + (kk & 3) * 2),
                           dK + (uint64_t)((kk >> 2) * (NS * 8192 / 16) + (kk & 3) * 2), id, kk > 0 ? 1u : 0u);
                ta_commit(sfull_bar(i));
                for (int h = 0; h < nsub; ++h) ta_commit(kempty_bar((ta + h) % NS));
            }
            // every MMA this thread issued has completed before the tensor memory is released
            ta_commit(drain_bar(0));
            volatile int never = 0;
            ta_wait(drain_bar(0), 0, &never, a.err);
        }
        __syncwarp();
    } else if (warp == 11) {
        if (lane == 0 && n_tiles > 0) {
            // ---------------- P V issue (one thread): O_q += P_t V_t once the V tile has landed and
            // group q = t & 1 has written P_t; the V slot is released when this P V completes
            const uint64_t dP = ta_desc_k(sbase + LY::P);
            for (int t = 0; t < n_tiles && ok; ++t) {
                const int st = t % NS, q = t & 1;
                if (!(ok = ta_wait(vfull_bar(st), (uint32_t)(t / NS) & 1u, abort_flag, a.err))) break;
                if (!(ok = ta_wait(pready_bar(q), (uint32_t)(t >> 1) & 1u, abort_flag, a.err))) break;
                ta_fence_after();
                const uint64_t dV = ta_desc_mn(sbase + LY::VR + (uint32_t)st * TB);
                const uint64_t dPq = dP + (uint64_t)(q * (kTQ * 128 / 16));
#pragma unroll
                for (int kk = 0; kk < kKT / 16; ++kk)
                    ta_mma(tO(q), dPq + (uint64_t)(kk * 2), dV + (uint64_t)(kk * 128), kIdO,
                           (t >= 2 || kk > 0) ? 1u : 0u);
                ta_commit(odone_bar(q));
                ta_commit(vempty_bar(st));
            }
            ta_commit(drain_bar(1));
            volatile int never = 0;
            ta_wait(drain_bar(1), 0, &never, a.err);
        }
        __syncwarp();
    } else {
        // ---------------- softmax group q (warps 4q .. 4q + 3) takes tiles q, q + 2, ... (at head_dim
        // 128 the half q of every tile pair); thread = query row tid % 128 = TMEM lane. Every wait is
        // taken by the whole warp and its outcome made warp-uniform (the tcgen05 loads and stores
        // below are warp-collective).
        const int q = warp >> 2, row = tid & 127;
        const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
        const bool warp_rows = qt * kTQ + (warp & 3) * 32 < R;   // the warp holds a query row
        auto wwait = [&](uint32_t bar, uint32_t parity) {
            const bool r = ta_wait(bar, parity, abort_flag, a.err);
            return __all_sync(0xffffffffu, r) != 0;
        };
        uint8_t* const prow = smem + LY::P + (uint32_t)q * (kTQ * 128) + row * 128;
        for (int t = q; t < n_tiles && ok; t += 2) {
            const int p = t / W, i = p & 1;
            const uint32_t col = 64u * (uint32_t)(t - W * p);
            if (!(ok = wwait(sfull_bar(i), (uint32_t)(p >> 1) & 1u))) break;
            ta_fence_after();
            float sv[64];
            if (warp_rows) {
                ta_ld32(tS(i) + lane_base + col, sv);
                ta_ld32(tS(i) + lane_base + col + 32, sv + 32);
            }
            ta_fence_before();
            __syncwarp();
            if (lane == 0) ta_arrive(sfree_bar(i));
            // keys past the tile's valid count (ragged last tile, block tile) get -inf
            const int valid = t < n_ct ? min(kKT, L - (t0 + t) * kKT) : a.B;
            float mx = -INFINITY;
            if (warp_rows) {
                if (valid < kKT) {
#pragma unroll
                    for (int j = 0; j < 64; ++j) sv[j] = j < valid ? sv[j] : -INFINITY;
                }
                // row maximum of the raw scores as a tree, then in log2 units (scale > 0)
                float m8[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) m8[e] = fmaxf(sv[e], sv[8 + e]);
#pragma unroll
                for (int j = 16; j < 64; j += 8)
#pragma unroll
                    for (int e = 0; e < 8; ++e) m8[e] = fmaxf(m8[e], sv[j + e]);
                mx = fmaxf(fmaxf(fmaxf(m8[0], m8[1]), fmaxf(m8[2], m8[3])),
                           fmaxf(fmaxf(m8[4], m8[5]), fmaxf(m8[6], m8[7]))) * a.scale_log2;
            }
            // P V of the group's previous tile has completed: its O is stable and P buffer q free
            if (t >= 2 && !(ok = wwait(odone_bar(q), (uint32_t)((t >> 1) - 1) & 1u))) break;
            ta_fence_after();
            if (warp_rows) {
                const bool raise = mx > m_used + kRescale;
                if (__any_sync(0xffffffffu, raise && t >= 2)) {
                    const float alpha = raise ? ex2(m_used - mx) : 1.0f;
#pragma unroll
                    for (int c = 0; c < HD / 32; ++c) {
                        float ov[32];
                        ta_ld32(tO(q) + lane_base + c * 32, ov);
#pragma unroll
                        for (int i = 0; i < 32; ++i) ov[i] *= alpha;
                        ta_st32(tO(q) + lane_base + c * 32, ov);
                    }
                    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
                }
                if (raise) {
                    l *= ex2(m_used - mx);   // 0 on the group's first tile (m_used = -inf)
                    m_used = mx;
                }
                // P = 2^(s scale - m): one FMA and one ex2 per key; eight partial row sums
                const float neg_m = -m_used;
                float ls[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
                for (int c = 0; c < 8; ++c) {
                    float p[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        p[e] = ex2(fmaf(sv[c * 8 + e], a.scale_log2, neg_m));
                        ls[e] += p[e];
                    }
                    uint4 u;
                    u.x = pack_bf16(p[0], p[1]);
                    u.y = pack_bf16(p[2], p[3]);
                    u.z = pack_bf16(p[4], p[5]);
                    u.w = pack_bf16(p[6], p[7]);
                    *reinterpret_cast<uint4*>(prow + ((c ^ (row & 7)) << 4)) = u;
                }
                l += ((ls[0] + ls[1]) + (ls[2] + ls[3])) + ((ls[4] + ls[5]) + (ls[6] + ls[7]));
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            }
            ta_fence_before();
            __syncwarp();
            if (lane == 0) ta_arrive(pready_bar(q));
        }
        // the group's last P V has completed: O_q holds the group's whole key range
        const int last = q + ((n_tiles - 1 - q) >> 1) * 2;   // the group's last tile
        if (ok && n_tiles > q) ok = wwait(odone_bar(q), (uint32_t)(last >> 1) & 1u);
        ta_fence_after();
        // each group leaves its (m, l) per row in its own (now unused) P buffer for the push
        float2* xml = reinterpret_cast<float2*>(smem + LY::P + (uint32_t)q * (kTQ * 128));
        xml[row] = make_float2(n_tiles > q && ok ? m_used : -INFINITY, n_tiles > q && ok ? l : 0.f);
    }
    if (!ok && lane == 0) atomicOr(a.err, DFLARE_DEVERR_TIMEOUT);
    // every CTA of the cluster has finished with its stages (copies landed, MMAs drained) before
    // any partial is pushed into them
    __syncthreads();
    cluster.sync();
    // Push the partial: both groups' (m, l, O) of query row r are combined and written to CTA
    // r / RP at [s RP + r % RP]; warpgroup h (warps 4h .. 4h + 3, lane quarter = warp % 4) takes the
    // head dims [h HD/2, h HD/2 + HD/2). A group without tiles (m = -inf) contributes nothing and
    // its O is not read; the loads are guarded by warp votes, so they stay collective.
    const int RP = (rows + S - 1) / S;
    __half* rO = reinterpret_cast<__half*>(smem + LY::RO);
    float2* rML = reinterpret_cast<float2*>(smem + LY::RML);
    float* rW = reinterpret_cast<float*>(smem + LY::RW);
    if (warp < 8 && (warp & 3) * 32 < rows) {
        const int r = tid & 127, half = warp >> 2;
        const bool row_ok = r < rows;
        const float2 mlA = reinterpret_cast<const float2*>(smem + LY::P)[r];
        const float2 mlB = reinterpret_cast<const float2*>(smem + LY::P + kTQ * 128)[r];
        const bool hA = mlA.x != -INFINITY, hB = mlB.x != -INFINITY;
        const float M = fmaxf(mlA.x, mlB.x);
        const float wA = hA ? ex2(mlA.x - M) : 0.f, wB = hB ? ex2(mlB.x - M) : 0.f;
        const float lt = (hA ? mlA.y * wA : 0.f) + (hB ? mlB.y * wB : 0.f);
        const float inv = lt > 0.f ? 1.0f / lt : 0.f;
        const float cA = wA * inv, cB = wB * inv;
        const int dst_cta = row_ok ? r / RP : 0, dst_row = s * RP + (row_ok ? r % RP : 0);
        __half* dst = cluster.map_shared_rank(rO, dst_cta) + (size_t)dst_row * HD;
        const uint32_t lb = (uint32_t)((warp & 3) * 32) << 16;
        const bool anyA = __any_sync(0xffffffffu, hA), anyB = __any_sync(0xffffffffu, hB);
        if (anyA || anyB) {
#pragma unroll
            for (int c = half * (HD / 64); c < (half + 1) * (HD / 64); ++c) {
                float ov[32], ob[32];
                if (anyA) {
                    ta_ld32(tO(0) + lb + c * 32, ov);
                } else {
#pragma unroll
                    for (int i = 0; i < 32; ++i) ov[i] = 0.f;
                }
                if (anyB) ta_ld32(tO(1) + lb + c * 32, ob);
#pragma unroll
                for (int i = 0; i < 32; ++i) {
                    const float x = hA ? ov[i] * cA : 0.f;
                    ov[i] = hB ? fmaf(ob[i], cB, x) : x;
                }
                if (row_ok) {
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        uint4 u;
                        __half2* h = reinterpret_cast<__half2*>(&u);
#pragma unroll
                        for (int e = 0; e < 4; ++e) h[e] = __floats2half2_rn(ov[k * 8 + 2 * e], ov[k * 8 + 2 * e + 1]);
                        *reinterpret_cast<uint4*>(dst + c * 32 + k * 8) = u;
                    }
                }
            }
        }
        if (row_ok && half == 0)
            *cluster.map_shared_rank(rML + dst_row, dst_cta) = make_float2(hA || hB ? M : -INFINITY, lt);
    }
    // every partial has arrived; after this barrier no CTA touches another's shared memory
    ta_fence_before();
    cluster.sync();
    if (warp == 9) {
        ta_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(LY::TMEM_COLS)
                     : "memory");
    }
    // merge this CTA's rows [s RP, min(rows, s RP + RP)): the weights of the S partials of each
    // row (a partial with m = -inf weighs 0 and its O is not read), then 8 output elements per item
    const int r0 = s * RP, nr = max(0, min(rows - r0, RP));
    for (int i = tid; i < nr; i += kTThreads) {
        float M = -INFINITY;
        for (int p = 0; p < S; ++p) M = fmaxf(M, rML[p * RP + i].x);
        float den = 0.f;
        for (int p = 0; p < S; ++p) {
            const float2 ml = rML[p * RP + i];
            const float w = ml.x == -INFINITY ? 0.f : ml.y * exp2f(ml.x - M);
            rW[i * kMaxSplits + p] = w;
            den += w;
        }
        const float inv = 1.0f / den;
        for (int p = 0; p < S; ++p) rW[i * kMaxSplits + p] *= inv;
    }
    __syncthreads();
    for (int it = tid; it < nr * (HD / 8); it += kTThreads) {
        const int i = it / (HD / 8), c = it % (HD / 8);
        float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        for (int p = 0; p < S; ++p) {
            const float w = rW[i * kMaxSplits + p];
            if (w != 0.f) {
                const uint4 v = *reinterpret_cast<const uint4*>(rO + (size_t)(p * RP + i) * HD + c * 8);
                const __half2* hv = reinterpret_cast<const __half2*>(&v);
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float2 f = __half22float2(hv[e]);
                    acc[2 * e] = fmaf(w, f.x, acc[2 * e]);
                    acc[2 * e + 1] = fmaf(w, f.y, acc[2 * e + 1]);
                }
            }
        }
        const int rg = qt * kTQ + r0 + i, kpos = rg / a.G, hh = rg % a.G;
        store8(out + ((size_t)b * a.B + kpos) * a.d_q + (size_t)(g * a.G + hh) * HD + c * 8, acc);
    }
    if (a.t_stamps) {
        __syncthreads();
        if (tid == 0) atomicMax(a.t_stamps + 2 * a.t_slots, (unsigned long long)globaltimer_ns());
    }
}

// ------------------------------------------------------------------ CUDA-core path

template <class T, int HD>
__global__ void __launch_bounds__(128) attn_simt_kernel(const AttnArgs a) {
    pdl_trigger();
    pdl_wait();
    constexpr int PER = HD / 32;
    const int s = blockIdx.x, g = blockIdx.y % a.hkv, qt = blockIdx.y / a.hkv, b = blockIdx.z;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int R = a.B * a.G;
    int j_begin, j_end, L;
    key_range(a, b, s, j_begin, j_end, L);
    const size_t pidx = part_index(a, b, g, qt, s);
    float* po = a.part_o + pidx * kQT * HD;
    float* pml = a.part_ml + pidx * kQT * 2;
    const T* q = static_cast<const T*>(a.q);
    const T* kd = static_cast<const T*>(a.kd);
    const T* vd = static_cast<const T*>(a.vd);
    const T* kc = static_cast<const T*>(a.kc) + ((size_t)b * a.hkv + g) * a.max_ctx * HD;
    const T* vc = static_cast<const T*>(a.vc) + ((size_t)b * a.hkv + g) * a.max_ctx * HD;
    for (int r = warp; r < kQT; r += 4) {
        const int rr = qt * kQT + r;
        float m = -INFINITY, l = 0.f, acc[PER], qv[PER];
#pragma unroll
        for (int e = 0; e < PER; ++e) acc[e] = 0.f;
        if (rr < R && j_begin < j_end) {
            const int kpos = rr / a.G, hh = rr % a.G;
            const T* qrow = q + ((size_t)b * a.B + kpos) * a.d_q + (size_t)(g * a.G + hh) * HD;
#pragma unroll
            for (int e = 0; e < PER; ++e) qv[e] = to_f(qrow[lane + 32 * e]);
            for (int j = j_begin; j < j_end; ++j) {
                const T *kr, *vr;
                if (j < L) {
                    kr = kc + (size_t)j * HD;
                    vr = vc + (size_t)j * HD;
                } else {
                    kr = kd + ((size_t)b * a.B + (j - L)) * a.d_kv + (size_t)g * HD;
                    vr = vd + ((size_t)b * a.B + (j - L)) * a.d_kv + (size_t)g * HD;
                }
                float dot = 0.f;
#pragma unroll
                for (int e = 0; e < PER; ++e) dot = fmaf(qv[e], to_f(kr[lane + 32 * e]), dot);
                const float sc = warp_sum(dot) * a.scale_log2;
                const float mn = fmaxf(m, sc);
                const float corr = exp2f(m - mn), p = exp2f(sc - mn);
                l = l * corr + p;
#pragma unroll
                for (int e = 0; e < PER; ++e) acc[e] = fmaf(p, to_f(vr[lane + 32 * e]), acc[e] * corr);
                m = mn;
            }
        }
#pragma unroll
        for (int e = 0; e < PER; ++e) po[(size_t)r * HD + lane + 32 * e] = acc[e];
        if (lane == 0) {
            pml[2 * r] = m;
            pml[2 * r + 1] = l;
        }
    }
}

// ------------------------------------------------------------------ combine

template <class T, int HD>
__global__ void attn_combine_kernel(const AttnArgs a, T* __restrict__ out) {
    pdl_trigger();
    pdl_wait();
    const int rr = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
    const int qt = rr / kQT, r = rr % kQT;
    const int kpos = rr / a.G, hh = rr % a.G;
    float M = -INFINITY;
    for (int s = 0; s < a.splits; ++s)
        M = fmaxf(M, a.part_ml[(part_index(a, b, g, qt, s) * kQT + r) * 2]);
    float den = 0.f, num[HD / 64 > 0 ? HD / 64 : 1];
    constexpr int PER = HD / 64;
#pragma unroll
    for (int e = 0; e < PER; ++e) num[e] = 0.f;
    for (int s = 0; s < a.splits; ++s) {
        const size_t pi = part_index(a, b, g, qt, s) * kQT + r;
        const float ms = a.part_ml[pi * 2];
        if (ms == -INFINITY) continue;
        const float w = exp2f(ms - M);
        den = fmaf(w, a.part_ml[pi * 2 + 1], den);
#pragma unroll
        for (int e = 0; e < PER; ++e) num[e] = fmaf(w, a.part_o[pi * HD + threadIdx.x + 64 * e], num[e]);
    }
    T* orow = out + ((size_t)b * a.B + kpos) * a.d_q + (size_t)(g * a.G + hh) * HD;
#pragma unroll
    for (int e = 0; e < PER; ++e) orow[threadIdx.x + 64 * e] = from_f<T>(num[e] / den);
}

template <int HD>
size_t mma_smem_bytes() {   // alignment pad, K/V stages, padded Q tile, pushed partials, barriers
    return 1024 + (size_t)kNST * 2 * HD * 128 + (size_t)kQT * (HD + 8) * sizeof(bf16) +
           (size_t)kQT * HD * sizeof(__half) + (size_t)kQT * 2 * sizeof(float) + 2 * 8 * kNST;
}

template <int HD, int S>
cudaError_t launch_mma(dflare_ctx* c, const AttnMaps& maps, const AttnArgs& a, cudaStream_t s) {
    static PerDeviceOnce configured;
    cudaError_t e = configured([] {
        cudaError_t r = cudaFuncSetAttribute(attn_mma_kernel<HD, S>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)mma_smem_bytes<HD>());
        if (r == cudaSuccess && S > 8)
            r = cudaFuncSetAttribute(attn_mma_kernel<HD, S>,
                                     cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        return r;
    });
    if (e != cudaSuccess) return e;
    return launch_cluster(c->pdl, S, attn_mma_kernel<HD, S>, dim3(S, a.hkv * a.q_tiles, c->batch),
                          dim3(128), mma_smem_bytes<HD>(), s, maps, a, static_cast<bf16*>(c->attn));
}

template <int HD>
cudaError_t run_mma(dflare_ctx* c, const AttnMaps& maps, const AttnArgs& a, cudaStream_t s) {
    switch (a.splits) {
        case 1: return launch_mma<HD, 1>(c, maps, a, s);
        case 2: return launch_mma<HD, 2>(c, maps, a, s);
        case 4: return launch_mma<HD, 4>(c, maps, a, s);
        case 8: return launch_mma<HD, 8>(c, maps, a, s);
        default: return launch_mma<HD, 16>(c, maps, a, s);
    }
}

// Largest cluster the device schedules for the attention kernel (16 where non-portable clusters
// of that size fit, else 8).
template <int HD>
int max_attention_cluster() {
    static std::atomic<int> cache[64];   // per device (modulo 64): 0 = not yet queried
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        return 8;
    }
    std::atomic<int>& slot = cache[dev & 63];
    if (const int known = slot.load(std::memory_order_acquire)) return known;
    int cached = 8;
    if (cudaFuncSetAttribute(attn_mma_kernel<HD, 16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)mma_smem_bytes<HD>()) == cudaSuccess &&
        cudaFuncSetAttribute(attn_mma_kernel<HD, 16>, cudaFuncAttributeNonPortableClusterSizeAllowed,
                             1) == cudaSuccess) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(16, 1, 1);
        cfg.blockDim = dim3(128);
        cfg.dynamicSmemBytes = mma_smem_bytes<HD>();
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = 16;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        int n = 0;
        if (cudaOccupancyMaxActiveClusters(&n, attn_mma_kernel<HD, 16>, &cfg) == cudaSuccess && n > 0)
            cached = 16;
    }
    cudaGetLastError();
    slot.store(cached, std::memory_order_release);
    return cached;
}

template <int HD>
cudaError_t configure_tc() {
    static PerDeviceOnce configured;
    return configured([] {
        cudaError_t r = cudaFuncSetAttribute(attn_tc_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)tc_attn_smem_bytes<HD>());
        if (r == cudaSuccess)
            r = cudaFuncSetAttribute(attn_tc_kernel<HD>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        return r;
    });
}

template <int HD>
cudaError_t run_tc(dflare_ctx* c, const AttnMaps& maps, const AttnArgs& a, cudaStream_t s) {
    const cudaError_t e = configure_tc<HD>();
    if (e != cudaSuccess) return e;
    return launch_cluster(c->pdl, a.splits, attn_tc_kernel<HD>, dim3(a.splits, a.hkv * a.q_tiles, c->batch),
                          dim3(kTThreads), tc_attn_smem_bytes<HD>(), s, maps, a, static_cast<bf16*>(c->attn));
}

// Clusters of sp tcgen05-attention CTAs (one per SM) that the device runs at once, sp = 1 .. 16;
// queried once per device (0 where the cluster size cannot be scheduled).
template <int HD>
int tc_active_clusters(int sp) {
    static std::atomic<int> cache[64][kMaxSplits];   // per device (modulo 64): 0 = not yet queried
    int dev = 0;
    if (sp < 1 || sp > kMaxSplits || cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        return 0;
    }
    std::atomic<int>& slot = cache[dev & 63][sp - 1];
    if (const int known = slot.load(std::memory_order_acquire)) return known - 1;
    int n = 0;
    if (configure_tc<HD>() == cudaSuccess) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(sp, 1, 1);
        cfg.blockDim = dim3(kTThreads);
        cfg.dynamicSmemBytes = tc_attn_smem_bytes<HD>();
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = sp;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        if (cudaOccupancyMaxActiveClusters(&n, attn_tc_kernel<HD>, &cfg) != cudaSuccess) n = 0;
    }
    cudaGetLastError();
    slot.store(n + 1, std::memory_order_release);
    return n;
}

template <class T, int HD>
cudaError_t run_simt(dflare_ctx* c, const AttnArgs& a, cudaStream_t s) {
    cudaError_t e = launch_kernel(c->pdl, attn_simt_kernel<T, HD>,
                                  dim3(a.splits, a.hkv * a.q_tiles, c->batch), dim3(128), 0, s, a);
    if (e != cudaSuccess) return e;
    return launch_kernel(c->pdl, attn_combine_kernel<T, HD>, dim3(a.B * a.G, a.hkv, c->batch),
                         dim3(64), 0, s, a, static_cast<T*>(c->attn));
}

}  // namespace

// CUDA-core (fp32) path: enough splits for about two CTAs per SM over batch x H_kv x q_tiles,
// none shorter than 256 keys at the host's upper bound of the context length; partials go
// through global memory to a combine launch. The device derives the actual ranges from the true
// lengths, so a stale bound (e.g. a replayed graph) only costs speed.
int attention_splits(const dflare_config& g, int batch, int num_sms, int len_ub) {
    const int G = g.n_q_heads / g.n_kv_heads;
    const int q_tiles = (g.block * G + kQT - 1) / kQT;
    const int base = batch * g.n_kv_heads * q_tiles;
    // CUDA-core path: each warp walks its query rows over the split's keys one key at a time, so
    // splits of at least 64 keys, as many as give two CTAs per SM
    int sp = (2 * num_sms + base - 1) / base;
    sp = std::min(sp, (len_ub + g.block + 63) / 64);
    return std::max(1, sp);
}

// Tensor-core path: the splits of one (sequence, head, query tile) are one cluster of 1, 2, 4, 8
// or 16 CTAs, at most one per 64-key tile: the most that still run as one wave at the CTAs per SM
// the kernel fits (per_sm: two at head_dim 128, four at head_dim 64), unless that leaves a CTA
// more than 12 tiles; then as many as give about per_sm CTAs per SM in all. Measured: with a few tiles per CTA the fixed cost of a CTA (launch, first tile, partial
// push, cluster barrier, merge: ~6 us) dominates and one wave wins (Qwen3-8B-shaped batch 4,
// 32 (sequence, head) pairs at L <= 4096: 8 splits, 1.256 ms per step, against 16 splits in two
// waves, 1.327 ms); with long runs per CTA two waves of shorter CTAs overlap the next kernel
// better (GPT-OSS-shaped batch 2, L 8192: 16 splits 1.046 ms, 8 splits 1.048 ms).
int attention_cluster_splits(const dflare_config& g, int batch, int num_sms, int len_ub,
                             int max_cluster, int per_sm) {
    const int G = g.n_q_heads / g.n_kv_heads;
    const int q_tiles = (g.block * G + kQT - 1) / kQT;
    const int base = batch * g.n_kv_heads * q_tiles;
    const int tiles = (len_ub + g.block + kKT - 1) / kKT;
    const int slots = per_sm * num_sms;
    int sp = 1;
    while (sp < max_cluster && 2 * sp <= tiles && base * 2 * sp <= slots) sp *= 2;
    if ((tiles + sp - 1) / sp > 12) {
        const int want = (slots + base - 1) / base;
        while (sp < max_cluster && sp < want && 2 * sp <= tiles) sp *= 2;
    }
    return sp;
}

// CTAs of the tensor-core attention that fit on one SM (registers and shared memory; queried once
// per device): two at head_dim 128, four at head_dim 64, at most four.
template <int HD>
int attention_ctas_per_sm() {
    static std::atomic<int> cache[64];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        return 2;
    }
    std::atomic<int>& slot = cache[dev & 63];
    if (const int known = slot.load(std::memory_order_acquire)) return known;
    int n = 0;
    if (cudaFuncSetAttribute(attn_mma_kernel<HD, 16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)mma_smem_bytes<HD>()) != cudaSuccess ||
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, attn_mma_kernel<HD, 16>, 128,
                                                      mma_smem_bytes<HD>()) != cudaSuccess || n < 1)
        n = 2;
    cudaGetLastError();
    n = std::min(n, 4);
    slot.store(n, std::memory_order_release);
    return n;
}

// tcgen05 path: one CTA per SM, 128 query rows per CTA. The largest cluster size sp (1 .. 16, not
// only powers of two) for which all batch x H_kv x query-tile clusters run at once (the device's
// count of co-resident clusters of that size, queried once), with at least two 64-key tiles per
// CTA at the host's upper bound of the context length. At one CTA per SM a GB300 runs 36 clusters
// of 4, 23 of 6, 15 of 8, 8 of 12 and 7 of 16, so e.g. 16 (sequence, head) pairs take 6 splits
// (96 SMs) rather than 4, and 8 pairs take 12 rather than 8.
int attention_tc_splits(const dflare_config& g, int batch, int len_ub, int (*active)(int)) {
    const int G = g.n_q_heads / g.n_kv_heads;
    const int q_tiles = (g.block * G + kTQ - 1) / kTQ;
    const int base = batch * g.n_kv_heads * q_tiles;
    const int tiles = (len_ub + g.block + kKT - 1) / kKT;
    for (int sp = kMaxSplits; sp > 1; --sp)
        if (2 * sp <= tiles && base <= active(sp)) return sp;
    return 1;
}

static bool use_tc_attention(const dflare_config& g) {
    return g.dtype == DFLARE_BF16 && !(g.flags & DFLARE_FLAG_MMA_SYNC_ATTENTION);
}

int attention_launch_splits(const dflare_ctx* c) {
    const dflare_config& g = c->cfg;
    if (g.dtype == DFLARE_F32) return attention_splits(g, c->batch, c->num_sms, c->ctx_ub);
    if (use_tc_attention(g))
        return attention_tc_splits(g, c->batch, c->ctx_ub,
                                   g.head_dim == 64 ? tc_active_clusters<64> : tc_active_clusters<128>);
    const int maxc = g.head_dim == 64 ? max_attention_cluster<64>() : max_attention_cluster<128>();
    const int per_sm = g.head_dim == 64 ? attention_ctas_per_sm<64>() : attention_ctas_per_sm<128>();
    return attention_cluster_splits(g, c->batch, c->num_sms, c->ctx_ub, maxc, per_sm);
}

cudaError_t launch_attention(dflare_ctx* c, int layer, cudaStream_t s) {
    const dflare_config& g = c->cfg;
    AttnArgs a{};
    a.q = c->q;
    a.kd = c->kd;
    a.vd = c->vd;
    const size_t layer_elems = (size_t)g.max_batch * g.n_kv_heads * g.max_ctx * g.head_dim;
    a.kc = static_cast<const uint8_t*>(c->kcache) + layer * layer_elems * c->esz;
    a.vc = static_cast<const uint8_t*>(c->vcache) + layer * layer_elems * c->esz;
    a.ctx_len = c->ctx_len;
    a.part_o = c->attn_o;
    a.part_ml = c->attn_ml;
    a.B = g.block;
    a.G = g.n_q_heads / g.n_kv_heads;
    a.hkv = g.n_kv_heads;
    a.d_q = g.n_q_heads * g.head_dim;
    a.d_kv = g.n_kv_heads * g.head_dim;
    a.max_ctx = g.max_ctx;
    a.q_tiles = (a.B * a.G + kQT - 1) / kQT;
    a.scale_log2 = 1.4426950408889634f / sqrtf((float)g.head_dim);
    if (g.dtype == DFLARE_F32) {
        a.splits = attention_splits(g, c->batch, c->num_sms, c->ctx_ub);
        return g.head_dim == 64 ? run_simt<float, 64>(c, a, s) : run_simt<float, 128>(c, a, s);
    }
    a.err = c->err;
    if (c->qkv32 && !(g.flags & (DFLARE_FLAG_DETERMINISTIC | DFLARE_FLAG_SIMT_GEMM))) {
        a.qkv32 = c->qkv32;
        a.rope_cos = c->rope_cos;
        a.rope_sin = c->rope_sin;
        a.kd_w = static_cast<bf16*>(c->kd);
        a.vd_w = static_cast<bf16*>(c->vd);
        a.rope = (g.flags & DFLARE_FLAG_NO_BLOCK_ROPE) ? 0 : 1;
    }
    // tensor maps of every layer's K/V cache and of K^d / V^d, built once per context
    if (c->attn_maps.empty()) {
        std::vector<CUtensorMap> m((size_t)2 * g.n_draft_layers + 2);
        const uint64_t hd = (uint64_t)g.head_dim;
        const uint32_t box[3] = {64u, (uint32_t)kKT, 1u};
        const uint32_t bbox[3] = {64u, (uint32_t)std::min(kKT, g.max_batch * g.block), 1u};
        for (int i = 0; i < g.n_draft_layers; ++i)
            for (int kv = 0; kv < 2; ++kv) {
                const uint8_t* base = static_cast<const uint8_t*>(kv ? c->vcache : c->kcache) + i * layer_elems * c->esz;
                const uint64_t dims[3] = {hd, (uint64_t)g.max_ctx, (uint64_t)g.max_batch * g.n_kv_heads};
                const uint64_t strides[2] = {hd * 2, (uint64_t)g.max_ctx * hd * 2};
                if (!encode_tma_bf16(&m[2 * i + kv], base, 3, dims, strides, box)) return cudaErrorInvalidValue;
            }
        for (int kv = 0; kv < 2; ++kv) {
            const uint64_t dims[3] = {hd, (uint64_t)g.max_batch * g.block, (uint64_t)g.n_kv_heads};
            const uint64_t strides[2] = {(uint64_t)a.d_kv * 2, hd * 2};
            if (!encode_tma_bf16(&m[2 * g.n_draft_layers + kv], kv ? c->vd : c->kd, 3, dims, strides, bbox))
                return cudaErrorInvalidValue;
        }
        c->attn_maps.swap(m);
    }
    AttnMaps maps;
    maps.kc = c->attn_maps[2 * layer];
    maps.vc = c->attn_maps[2 * layer + 1];
    maps.kd = c->attn_maps[2 * g.n_draft_layers];
    maps.vd = c->attn_maps[2 * g.n_draft_layers + 1];
    a.block_rows = std::min(kKT, g.max_batch * g.block);
    a.splits = attention_launch_splits(c);
    if (c->t_stamps && c->t_next < c->t_slots) {
        a.t_stamps = c->t_stamps + c->t_next++;
        a.t_slots = c->t_slots;
    }
    if (use_tc_attention(g)) {
        a.q_tiles = (a.B * a.G + kTQ - 1) / kTQ;
        return g.head_dim == 64 ? run_tc<64>(c, maps, a, s) : run_tc<128>(c, maps, a, s);
    }
    return g.head_dim == 64 ? run_mma<64>(c, maps, a, s) : run_mma<128>(c, maps, a, s);
}

}  // namespace dfl
