// Bidirectional block attention over [context ; block] (Sec. 3.2; keys/values per Eq. 4), as a
// split-KV ("flash-decoding") pass.
//
// For one sequence and one KV head, the queries are the B block rows of the H_q/H_kv query
// heads that share the head: B*G rows (64 for Qwen3 shapes, 128 for GPT-OSS) against L + B keys
// (context keys from the cache, then the block's own K^d / V^d). Nothing is masked: every query
// sees every key. The keys of one (sequence, head) are cut into contiguous ranges so that
// batch x H_kv x splits CTAs cover the GPU even for a single sequence.
//
// bf16 path: 64 query rows per CTA (4 warps x 16 rows); one thread streams 64-key K/V tiles by
// TMA into two 128-byte-swizzled stages; S = Q K^T and O += P V on mma.sync m16n8k16 with bf16
// operands and fp32 accumulators, P kept in registers; two CTAs fit on an SM. The splits of one
// (sequence, head, query tile) form a thread-block cluster (up to 16 CTAs) and merge their
// partial results (O / l in fp16) through distributed shared memory, so the whole attention is
// one launch and no partial goes through HBM.
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

// ------------------------------------------------------------------ bf16, tensor cores

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
__device__ __forceinline__ bool tile_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok = 0;
    const uint64_t t0 = globaltimer_ns();
    while (true) {
        asm volatile(
            "{\n\t.reg .pred p;\n\t"
            "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
            "selp.u32 %0, 1, 0, p;\n\t}"
            : "=r"(ok)
            : "r"(bar), "r"(parity)
            : "memory");
        if (ok) return true;
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

int attention_launch_splits(const dflare_ctx* c) {
    const dflare_config& g = c->cfg;
    if (g.dtype == DFLARE_F32) return attention_splits(g, c->batch, c->num_sms, c->ctx_ub);
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
    const int maxc = g.head_dim == 64 ? max_attention_cluster<64>() : max_attention_cluster<128>();
    const int per_sm = g.head_dim == 64 ? attention_ctas_per_sm<64>() : attention_ctas_per_sm<128>();
    a.splits = attention_cluster_splits(g, c->batch, c->num_sms, c->ctx_ub, maxc, per_sm);
    if (c->t_stamps && c->t_next < c->t_slots) {
        a.t_stamps = c->t_stamps + c->t_next++;
        a.t_slots = c->t_slots;
    }
    return g.head_dim == 64 ? run_mma<64>(c, maps, a, s) : run_mma<128>(c, maps, a, s);
}

}  // namespace dfl
