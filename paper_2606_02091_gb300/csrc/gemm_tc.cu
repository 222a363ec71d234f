// Weight-streaming projection GEMM on the sm_103a tensor cores (tcgen05 + TMEM + TMA).
//
// Every projection of the draft path (context K/V of Eq. 4, Q/K^d/V^d, attention output, SwiGLU
// gate/up and down, LM head) multiplies a few activation rows (batch * B tokens, at most a few
// hundred) by a large weight matrix, so each weight byte is used only m_tok times: the kernel is
// bound by HBM bandwidth while m_tok is below ~280. The layout is therefore "swap AB": the
// 128-row UMMA M dimension runs over weight rows (output features) and the small token count is
// the UMMA N dimension (16..256), so one instruction covers a 128 x bn x 16 piece.
//
// Work unit = (group, 128-feature tile, token tile, K split); for an LM head over 128+ token rows,
// a pair of adjacent 128-feature tiles (two accumulators over one activation tile); a context
// fill's units run only over the token tiles that hold appended rows. A
// persistent grid of one CTA per SM walks the units. Per CTA (192 threads):
//   warp 4    TMA producer: per stage, kbs consecutive 128x64 bf16 weight tiles (+ the up tiles
//             for SwiGLU) and the matching bn x 64 activation tiles, 128-byte swizzled; weights
//             carry an L2 evict-first hint (each byte is read once per step). Weights do not
//             depend on the previous kernel: the first ring of stages gets its weight tiles
//             before griddepcontrol.wait, the activation tiles after it.
//   warp 5    allocates TMEM, issues tcgen05.mma (one thread), commits stages back to the
//             producer and finished accumulators to the epilogue; two accumulator buffers let
//             the next unit's MMAs overlap the current unit's epilogue.
//   warps 0-3 epilogue: tcgen05.ld of the accumulator (thread t = TMEM lane t = feature t),
//             split-K reduction through a global workspace (the last CTA of a tile sums the
//             partials in split order, so results are deterministic), then the fused epilogue.
//             Residual rows are loaded before the accumulator is waited for.
// Every wait on an mbarrier is bounded (2 s); on a timeout the CTA sets DFLARE_DEVERR_TIMEOUT,
// stops issuing work, drains what it issued and frees its TMEM.
#include <cudaTypedefs.h>

#include <algorithm>
#include <cstring>
#include <mutex>

#include "epilogue.cuh"

namespace dfl {
namespace {

constexpr int kThreads = 192;
constexpr int kBM = 128;
constexpr int kBK = 64;
constexpr int kChunk = 16;
constexpr int kMaxStages = 8;
constexpr uint64_t kTimeoutNs = 2000000000ull;
constexpr int kSmemLimit = 227 * 1024;
constexpr uint32_t kABytes = kBM * kBK * 2;   // one 128 x 64 bf16 weight tile
constexpr int kMaxTokList = 1024;             // token tiles a compacted launch can list

struct TcArgs {
    CUtensorMap map_a, map_a2, map_b;   // weights, up weights (SwiGLU), activations
    int n_units, n_tiles, tok_tiles, splits, kb_per_split, k_blocks;
    int bn, n_a, stages, n_bufs, tmem_cols;
    int pair;                  // 1: a unit is two adjacent 128-row tiles of one weight matrix
                               // (the second accumulator takes rows 128..255 of the pair)
    int compact;               // EPI_KV_APPEND: skip the token tiles that hold no appended row
    int kbs;                   // 64-wide k-blocks per pipeline stage
    uint32_t b_bytes;          // bytes of one activation sub-tile (bn x 64 bf16)
    int evict_first;           // stream the weights with an L2 evict-first policy
    uint32_t idesc;
    uint32_t stage_bytes;
    float* ws;
    uint32_t* tile_cnt;
    uint32_t* err;
    EpiParams ep;
    // activation addressing of the kAux instance only
    int b_kg;                  // > 0: activation group z holds contraction indices [z b_kg, (z+1) b_kg)
    int b_gsel;                // 1: activation group = weight group; 0: one activation group for all
    int resid_red;             // EPI_RESID: each split adds its partial to resid with L2 reductions
    int resid_vec;             // ... as 16-byte reductions of token-major rows (aligned residual)
    unsigned long long* t_stamps;   // launch timing: entry, dependency met, exit (nullptr: off)
    int t_slots;
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
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
// Bounded wait: false when the CTA aborted or this wait timed out.
__device__ __noinline__ bool bar_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                      uint32_t* err) {
    for (int i = 0; i < 128; ++i)
        if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = globaltimer_ns();
    while (true) {
        for (int i = 0; i < 128; ++i)
            if (mbar_try_wait(bar, parity)) return true;
        if (*abort_flag) return false;
        if (globaltimer_ns() - t0 > kTimeoutNs) {
            *abort_flag = 1;
            atomicOr(err, DFLARE_DEVERR_TIMEOUT);
            return false;
        }
    }
}
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* map, int x, int y,
                                            int z, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(bar)
        : "memory");
}
__device__ __forceinline__ void tma_load_3d_hint(uint32_t dst, const CUtensorMap* map, int x, int y,
                                                 int z, uint32_t bar, uint64_t policy) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        ".L2::cache_hint [%0], [%1, {%2, %3, %4}], [%5], %6;" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(bar), "l"(policy)
        : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// Shared-memory matrix descriptor: K-major operand, rows of 128 bytes, 128-byte swizzle,
// 8-row core-matrix groups 1024 bytes apart (SBO), descriptor version 1.
__device__ __forceinline__ uint64_t smem_desc(uint32_t saddr) {
    return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
           ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}
__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                          uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(idesc), "r"(accumulate)
        : "memory");
}
__device__ __forceinline__ void umma_commit(uint32_t bar) {
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
        : "memory");
}
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float* v) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
          "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ void epi_bar() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

__device__ __forceinline__ uint32_t atom_add_acq_rel(uint32_t* p, uint32_t v) {
    uint32_t old;
    asm volatile("atom.add.acq_rel.gpu.global.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
    return old;
}

// The kernel's loop constants, copied out of the parameter block into registers (the block is
// addressed for the tensor maps, so every asm with a memory clobber would otherwise reload them).
struct Geom {
    int n_units, n_tiles, tok_tiles, splits, kb_per_split, k_blocks, n_a, kbs, bn, n_bufs, pair;
    uint32_t b_bytes, stage_bytes, idesc;
    const int* tok_list;       // token tiles in unit order (compacted launches), else nullptr
};
struct Unit {
    int group, n_tile, tok_tile, split, tile_id, kb0, kb1;
};
__device__ __forceinline__ Unit decode_unit(const Geom& a, int u) {
    Unit x;
    x.split = u % a.splits;
    x.tile_id = u / a.splits;
    int t = x.tile_id;
    x.tok_tile = t % a.tok_tiles;
    if (a.tok_list) x.tok_tile = a.tok_list[x.tok_tile];
    t /= a.tok_tiles;
    x.n_tile = t % a.n_tiles;
    x.group = t / a.n_tiles;
    x.kb0 = x.split * a.kb_per_split;
    x.kb1 = min(a.k_blocks, x.kb0 + a.kb_per_split);
    return x;
}

// EPI_RESID with the residual values already in registers: resid[tok][n] += acc.
__device__ __forceinline__ void load_resid(const EpiParams& ep, int n_tile, int tok0, int t, float* r) {
    const int n = n_tile * 128 + t;
    const int nvalid = min(kChunk, ep.m_tok - tok0);
#pragma unroll
    for (int c = 0; c < kChunk; ++c)
        r[c] = (n < ep.n && c < nvalid) ? ep.resid[(size_t)(tok0 + c) * ep.ld_resid + n] : 0.f;
}
__device__ __forceinline__ void resid_epilogue(const EpiParams& ep, const float* tile, int n_tile,
                                               int tok0, int t, const float* r) {
    const int n = n_tile * 128 + t;
    if (n >= ep.n) return;
    const int nvalid = min(kChunk, ep.m_tok - tok0);
#pragma unroll
    for (int c = 0; c < kChunk; ++c)
        if (c < nvalid) ep.resid[(size_t)(tok0 + c) * ep.ld_resid + n] = r[c] + tile[c * 128 + t];
}

// kAux = false: the projections of the draft step (every activation group belongs to its weight
// group; the epilogues without bias). kAux = true adds the activation addressing of the fusion
// variants (a shared activation group, a contraction across stacked groups) and the biased store;
// it is a separate instance so that the draft step's code is not touched by it.
template <bool kAux>
__global__ void __launch_bounds__(kThreads, 1) gemm_tc_kernel(const __grid_constant__ TcArgs args) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t pad = (1024u - (raw & 1023u)) & 1023u;
    uint8_t* smem = smem_raw + pad;
    const uint32_t sbase = raw + pad;
    Geom G;
    G.n_units = args.n_units;
    G.n_tiles = args.n_tiles;
    G.tok_tiles = args.tok_tiles;
    G.splits = args.splits;
    G.kb_per_split = args.kb_per_split;
    G.k_blocks = args.k_blocks;
    G.n_a = args.n_a;
    G.kbs = args.kbs;
    G.bn = args.bn;
    G.n_bufs = args.n_bufs;
    G.pair = args.pair;
    G.tok_list = nullptr;
    G.b_bytes = args.b_bytes;
    G.stage_bytes = args.stage_bytes;
    G.idesc = args.idesc;
    uint32_t* const err = args.err;
    const int S = args.stages;
    float* epi = reinterpret_cast<float*>(smem + (size_t)S * G.stage_bytes);
    uint64_t* bars = reinterpret_cast<uint64_t*>(epi + G.n_a * kChunk * 128);
    uint32_t* misc = reinterpret_cast<uint32_t*>(bars + 2 * S + 5);
    const uint32_t bar0 = smem_u32(bars);
    auto full_bar = [&](int s) { return bar0 + 8u * s; };
    auto empty_bar = [&](int s) { return bar0 + 8u * (S + s); };
    auto tfull_bar = [&](int b) { return bar0 + 8u * (2 * S + b); };
    auto tempty_bar = [&](int b) { return bar0 + 8u * (2 * S + 2 + b); };
    const uint32_t drain_bar = bar0 + 8u * (2 * S + 4);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    unsigned long long* const tst = args.t_stamps;
    if (tst && threadIdx.x == 0) atomicMin(tst, (unsigned long long)globaltimer_ns());
    if (warp == 4 && lane == 0) {
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&args.map_a)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&args.map_b)) : "memory");
        if (G.n_a == 2)
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&args.map_a2)) : "memory");
    }
    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(full_bar(s), 1);
            mbar_init(empty_bar(s), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(tfull_bar(b), 1);
            mbar_init(tempty_bar(b), 128);
        }
        mbar_init(drain_bar, 1);
        misc[1] = 0;
        misc[2] = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    // Compacted launch (a context fill of sequences with different lengths, token row
    // b * n_max + r): after the dependency wait, warp 0 lists the token tiles that hold at least
    // one appended row (r < app_cnt[b]); units then run over the listed tiles only.
    int* const tok_list = reinterpret_cast<int*>(misc + 4);
    if (args.compact) {
        pdl_wait();
        if (tst && threadIdx.x == 0) atomicMin(tst + args.t_slots, (unsigned long long)globaltimer_ns());
        if (warp == 0) {
            const int nm = args.ep.n_max;
            int cnt = 0;
            for (int base = 0; base < args.tok_tiles; base += 32) {
                const int tt = base + lane;
                bool v = false;
                if (tt < args.tok_tiles) {
                    const int r0 = tt * G.bn, r1 = min(args.ep.m_tok, r0 + G.bn);
                    for (int b = r0 / nm; b <= (r1 - 1) / nm && !v; ++b)
                        v = args.ep.app_cnt[b] > max(0, r0 - b * nm);
                }
                const unsigned m = __ballot_sync(0xffffffffu, v);
                if (v) tok_list[cnt + __popc(m & ((1u << lane) - 1u))] = tt;
                cnt += __popc(m);
            }
            if (lane == 0) misc[3] = (uint32_t)cnt;
        }
    }
    if (warp == 5) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_u32(&misc[0])),
                     "r"(args.tmem_cols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = misc[0];
    volatile int* abort_flag = reinterpret_cast<volatile int*>(&misc[1]);
    if (args.compact) {
        G.n_units = args.n_units / args.tok_tiles * (int)misc[3];
        G.tok_tiles = (int)misc[3];
        G.tok_list = tok_list;
    }
    const int acc_cols = G.n_a * G.bn;

    if (warp == 4) {
        if (lane == 0) {
            // ---------------- TMA producer
            const CUtensorMap* mA = &args.map_a;
            const CUtensorMap* mA2 = &args.map_a2;
            const CUtensorMap* mB = &args.map_b;
            int stage = 0;
            uint32_t phase = 0, issued = 0, issued_phase = 0;
            bool ok = true;
            uint64_t policy = 0;
            const bool evict_first = args.evict_first != 0;
            if (evict_first)
                asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(policy));
            const uint32_t b_base = kABytes * G.n_a * G.kbs;
            const uint32_t tx = kABytes * G.n_a + G.b_bytes;
            // first weight row of a unit in both maps (a pair's second map starts 128 rows in)
            const int row_step = kBM << G.pair;
            // Weights do not depend on the previous kernel: the first ring of stages gets its
            // weight tiles before griddepcontrol.wait, the activation tiles after it.
            int pend_kx[kMaxStages], pend_nk[kMaxStages], pend_tok[kMaxStages], pend_grp[kMaxStages];
            uint32_t pend_st[kMaxStages];
            int npend = 0;
            bool waited = args.compact != 0;   // a compacted launch waited before the unit list
            auto load_b = [&](uint32_t st, int kx0, int nk, int tok_tile, int group, uint32_t bar) {
                if constexpr (kAux) {
                    for (int j = 0; j < nk; ++j) {
                        int bx = kx0 + j * kBK, bz = group * args.b_gsel;
                        if (args.b_kg > 0) {   // contraction over stacked activation groups (Eq. 1)
                            bz = bx / args.b_kg;
                            bx -= bz * args.b_kg;
                        }
                        tma_load_3d(st + b_base + j * G.b_bytes, mB, bx, tok_tile * G.bn, bz, bar);
                    }
                } else {
                    for (int j = 0; j < nk; ++j)
                        tma_load_3d(st + b_base + j * G.b_bytes, mB, kx0 + j * kBK, tok_tile * G.bn, group, bar);
                }
            };
            for (int u = blockIdx.x; u < G.n_units && ok; u += gridDim.x) {
                const Unit x = decode_unit(G, u);
                for (int kb = x.kb0; kb < x.kb1; kb += G.kbs) {
                    const int nk = min(G.kbs, x.kb1 - kb);
                    if (!bar_wait(empty_bar(stage), phase ^ 1u, abort_flag, err)) {
                        ok = false;
                        break;
                    }
                    const uint32_t st = sbase + (uint32_t)stage * G.stage_bytes;
                    mbar_expect_tx(full_bar(stage), (uint32_t)nk * tx);
                    for (int j = 0; j < nk; ++j) {
                        const int kx = (kb + j) * kBK;
                        if (evict_first) {
                            tma_load_3d_hint(st + j * kABytes, mA, kx, x.n_tile * row_step, x.group,
                                             full_bar(stage), policy);
                            if (G.n_a == 2)
                                tma_load_3d_hint(st + (G.kbs + j) * kABytes, mA2, kx, x.n_tile * row_step,
                                                 x.group, full_bar(stage), policy);
                        } else {
                            tma_load_3d(st + j * kABytes, mA, kx, x.n_tile * row_step, x.group, full_bar(stage));
                            if (G.n_a == 2)
                                tma_load_3d(st + (G.kbs + j) * kABytes, mA2, kx, x.n_tile * row_step, x.group,
                                            full_bar(stage));
                        }
                    }
                    if (waited) {
                        load_b(st, kb * kBK, nk, x.tok_tile, x.group, full_bar(stage));
                    } else {
                        pend_kx[npend] = kb * kBK;
                        pend_nk[npend] = nk;
                        pend_tok[npend] = x.tok_tile;
                        pend_grp[npend] = x.group;
                        pend_st[npend] = (uint32_t)stage;
                        if (++npend == S) {
                            pdl_wait();
                            if (tst) atomicMin(tst + args.t_slots, (unsigned long long)globaltimer_ns());
                            waited = true;
                            for (int i = 0; i < npend; ++i)
                                load_b(sbase + pend_st[i] * G.stage_bytes, pend_kx[i], pend_nk[i],
                                       pend_tok[i], pend_grp[i], full_bar(pend_st[i]));
                        }
                    }
                    issued |= 1u << stage;
                    issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
                    if (++stage == S) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
            if (!waited) {
                pdl_wait();
                if (tst) atomicMin(tst + args.t_slots, (unsigned long long)globaltimer_ns());
                for (int i = 0; i < npend; ++i)
                    load_b(sbase + pend_st[i] * G.stage_bytes, pend_kx[i], pend_nk[i], pend_tok[i],
                           pend_grp[i], full_bar(pend_st[i]));
            }
            // make sure no copy is still landing in shared memory when the CTA exits
            for (int s = 0; s < S; ++s)
                if (issued & (1u << s)) {
                    volatile int never = 0;
                    bar_wait(full_bar(s), (issued_phase >> s) & 1u, ok ? &never : abort_flag, err);
                }
        }
    } else if (warp == 5) {
        if (lane == 0) {
            // ---------------- MMA issuer
            int stage = 0, acc = 0;
            uint32_t phase = 0, acc_phase = 0;
            bool ok = true;
            const uint32_t b_base = kABytes * G.n_a * G.kbs;
            for (int u = blockIdx.x; u < G.n_units && ok; u += gridDim.x) {
                const Unit x = decode_unit(G, u);
                if (!bar_wait(tempty_bar(acc), acc_phase ^ 1u, abort_flag, err)) break;
                tc_fence_after();
                const uint32_t d0 = tmem + (uint32_t)(acc * acc_cols);
                for (int kb = x.kb0; kb < x.kb1; kb += G.kbs) {
                    const int nk = min(G.kbs, x.kb1 - kb);
                    if (!bar_wait(full_bar(stage), phase, abort_flag, err)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t st = sbase + (uint32_t)stage * G.stage_bytes;
                    for (int j = 0; j < nk; ++j) {
                        const uint64_t da = smem_desc(st + j * kABytes);
                        const uint64_t da2 = smem_desc(st + (G.kbs + j) * kABytes);
                        const uint64_t db = smem_desc(st + b_base + j * G.b_bytes);
#pragma unroll
                        for (int k = 0; k < kBK / 16; ++k) {
                            const uint32_t accum = (kb > x.kb0 || j > 0 || k > 0) ? 1u : 0u;
                            umma_bf16(d0, da + 2 * k, db + 2 * k, G.idesc, accum);
                            if (G.n_a == 2) umma_bf16(d0 + G.bn, da2 + 2 * k, db + 2 * k, G.idesc, accum);
                        }
                    }
                    umma_commit(empty_bar(stage));
                    if (++stage == S) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
                if (!ok) break;
                umma_commit(tfull_bar(acc));
                if (G.n_bufs == 2) {
                    acc ^= 1;
                    if (acc == 0) acc_phase ^= 1u;
                } else {
                    acc_phase ^= 1u;
                }
            }
            // all issued MMAs complete before TMEM is released
            umma_commit(drain_bar);
            volatile int never = 0;
            bar_wait(drain_bar, 0, &never, err);
        }
    } else {
        // ---------------- epilogue warps 0-3 (thread t <-> TMEM lane t <-> feature t of a tile)
        pdl_wait();
        // dependents may start once every CTA has passed its own dependency wait: everything the
        // kernels before this one wrote is then complete (the attention that follows the Q/K^d/V^d
        // projection reads the context cache before its own wait)
        if (threadIdx.x == 0) pdl_trigger();
        const int t = threadIdx.x;
        int acc = 0;
        uint32_t acc_phase = 0;
        const int bn = G.bn, na = G.n_a;
        float* const ws = args.ws;
        uint32_t* const tile_cnt = args.tile_cnt;
        const bool resid = args.ep.kind == EPI_RESID && bn == kChunk;
        const bool resid_red = args.ep.kind == EPI_RESID && args.resid_red && !args.resid_vec;
        const bool red32 = args.ep.kind == EPI_RED32 || (args.ep.kind == EPI_RESID && args.resid_red && args.resid_vec);
        float* const red_out = args.ep.kind == EPI_RED32 ? reinterpret_cast<float*>(args.ep.out) : args.ep.resid;
        const int red_ld = args.ep.kind == EPI_RED32 ? args.ep.ldo : args.ep.ld_resid;
        for (int u = blockIdx.x; u < G.n_units; u += gridDim.x) {
            const Unit x = decode_unit(G, u);
            if (resid_red) {
                // resid += acc with fp32 reductions in L2: every split adds its own partial sum,
                // with no workspace, no tile counter and no read of the residual (the order of
                // the additions, and so the last bit of the sum, can vary between runs)
                if (!bar_wait(tfull_bar(acc), acc_phase, abort_flag, err)) break;
                tc_fence_after();
                const uint32_t taddr = tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)(acc * acc_cols);
                const int n = x.n_tile * 128 + t;
                for (int c0 = 0; c0 < bn; c0 += kChunk) {
                    float v[kChunk];
                    tmem_ld16(taddr + (uint32_t)c0, v);
                    if (c0 + kChunk >= bn) {
                        tc_fence_before();
                        mbar_arrive(tempty_bar(acc));
                    }
                    const int tok0 = x.tok_tile * bn + c0;
                    const int nvalid = min(kChunk, args.ep.m_tok - tok0);
                    if (n < args.ep.n) {
                        float* dst = args.ep.resid + (size_t)tok0 * args.ep.ld_resid + n;
#pragma unroll
                        for (int c = 0; c < kChunk; ++c)
                            if (c < nvalid)
                                asm volatile("red.global.add.f32 [%0], %1;" ::"l"(dst + (size_t)c * args.ep.ld_resid),
                                             "f"(v[c])
                                             : "memory");
                    }
                }
                if (G.n_bufs == 2) {
                    acc ^= 1;
                    if (acc == 0) acc_phase ^= 1u;
                } else {
                    acc_phase ^= 1u;
                }
                continue;
            }
            if (red32) {
                // out += acc with fp32 L2 reductions (EPI_RED32, and the residual projections when
                // the residual rows are 16-byte aligned): each 16-token chunk is turned token-major
                // in shared memory, then every thread adds 16 consecutive features of one token
                // with four 16-byte reductions (no workspace, no tile counter, no read back; the
                // order of the additions, and so the last bit of a sum, can vary between runs)
                if (!bar_wait(tfull_bar(acc), acc_phase, abort_flag, err)) break;
                tc_fence_after();
                const uint32_t taddr = tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)(acc * acc_cols);
                const int cc = t >> 3, f0 = (t & 7) * 16;
                const int n0 = x.n_tile * 128 + f0;
                float* const out32 = red_out;
                for (int c0 = 0; c0 < bn; c0 += kChunk) {
                    float v[kChunk];
                    tmem_ld16(taddr + (uint32_t)c0, v);
                    if (c0 + kChunk >= bn) {
                        tc_fence_before();
                        mbar_arrive(tempty_bar(acc));
                    }
#pragma unroll
                    for (int c = 0; c < kChunk; ++c) epi[c * 128 + t] = v[c];
                    epi_bar();
                    const int tok = x.tok_tile * bn + c0 + cc;
                    if (tok < args.ep.m_tok && n0 < args.ep.n) {
                        float* dst = out32 + (size_t)tok * red_ld + n0;
                        const float* srow = epi + cc * 128 + f0;
#pragma unroll
                        for (int q4 = 0; q4 < 4; ++q4) {
                            const float4 w4 = *reinterpret_cast<const float4*>(srow + 4 * q4);
                            asm volatile("red.global.add.v4.f32 [%0], {%1, %2, %3, %4};" ::"l"(dst + 4 * q4),
                                         "f"(w4.x), "f"(w4.y), "f"(w4.z), "f"(w4.w)
                                         : "memory");
                        }
                    }
                    epi_bar();
                }
                if (G.n_bufs == 2) {
                    acc ^= 1;
                    if (acc == 0) acc_phase ^= 1u;
                } else {
                    acc_phase ^= 1u;
                }
                continue;
            }
            // the residual rows do not depend on the accumulator: load them before waiting
            float rr[kChunk];
            if (resid) load_resid(args.ep, x.n_tile, x.tok_tile * bn, t, rr);
            if (!bar_wait(tfull_bar(acc), acc_phase, abort_flag, err)) break;
            tc_fence_after();
            const uint32_t taddr = tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)(acc * acc_cols);
            bool final_tile = true;
            if (G.splits > 1) {
                // partial layout per (tile, split): [accumulator][16-token chunk][feature][16]
                float* dst = ws + (size_t)(x.tile_id * G.splits + x.split) * na * bn * 128;
                for (int a = 0; a < na; ++a)
                    for (int c0 = 0; c0 < bn; c0 += kChunk) {
                        float v[kChunk];
                        tmem_ld16(taddr + (uint32_t)(a * bn + c0), v);
                        float4* d4 = reinterpret_cast<float4*>(
                            dst + ((size_t)(a * (bn / kChunk) + c0 / kChunk) * 128 + t) * kChunk);
#pragma unroll
                        for (int k = 0; k < kChunk / 4; ++k)
                            d4[k] = make_float4(v[4 * k], v[4 * k + 1], v[4 * k + 2], v[4 * k + 3]);
                    }
                tc_fence_before();
                mbar_arrive(tempty_bar(acc));
                // the CTA barrier orders every thread's partial before thread 0's release; its
                // acquire (when last) orders the other partials before the reads below
                epi_bar();
                if (t == 0) {
                    const uint32_t prev = atom_add_acq_rel(&tile_cnt[x.tile_id], 1u);
                    misc[2] = (prev == (uint32_t)(G.splits - 1)) ? 1u : 0u;
                    if (prev == (uint32_t)(G.splits - 1)) tile_cnt[x.tile_id] = 0;
                }
                epi_bar();
                final_tile = misc[2] != 0;
            }
            if (final_tile) {
                for (int c0 = 0; c0 < bn; c0 += kChunk) {
                    for (int a = 0; a < na; ++a) {
                        float v[kChunk];
                        if (G.splits == 1) {
                            tmem_ld16(taddr + (uint32_t)(a * bn + c0), v);
                        } else {
                            // sum the splits in split order (deterministic); four 16-byte loads
                            // per split, several splits in flight
                            float4 acc4[kChunk / 4];
#pragma unroll
                            for (int k = 0; k < kChunk / 4; ++k) acc4[k] = make_float4(0.f, 0.f, 0.f, 0.f);
                            const size_t off = ((size_t)(a * (bn / kChunk) + c0 / kChunk) * 128 + t) * kChunk;
#pragma unroll 4
                            for (int s = 0; s < G.splits; ++s) {
                                const float4* src = reinterpret_cast<const float4*>(
                                    ws + (size_t)(x.tile_id * G.splits + s) * na * bn * 128 + off);
#pragma unroll
                                for (int k = 0; k < kChunk / 4; ++k) {
                                    const float4 w4 = __ldcg(src + k);
                                    acc4[k].x += w4.x;
                                    acc4[k].y += w4.y;
                                    acc4[k].z += w4.z;
                                    acc4[k].w += w4.w;
                                }
                            }
#pragma unroll
                            for (int k = 0; k < kChunk / 4; ++k) {
                                v[4 * k] = acc4[k].x;
                                v[4 * k + 1] = acc4[k].y;
                                v[4 * k + 2] = acc4[k].z;
                                v[4 * k + 3] = acc4[k].w;
                            }
                        }
#pragma unroll
                        for (int c = 0; c < kChunk; ++c) epi[(a * kChunk + c) * 128 + t] = v[c];
                    }
                    epi_bar();
                    if (resid)
                        resid_epilogue(args.ep, epi, x.n_tile, x.tok_tile * bn + c0, t, rr);
                    else if (G.pair)   // two 128-feature tiles, one per accumulator
                        for (int a = 0; a < 2; ++a)
                            apply_epilogue<bf16, kAux>(args.ep, epi + a * kChunk * 128, x.group,
                                                       2 * x.n_tile + a, x.tok_tile * bn + c0, t);
                    else
                        apply_epilogue<bf16, kAux>(args.ep, epi, x.group, x.n_tile, x.tok_tile * bn + c0, t);
                    epi_bar();
                }
            }
            if (G.splits == 1) {
                tc_fence_before();
                mbar_arrive(tempty_bar(acc));
            }
            if (G.n_bufs == 2) {
                acc ^= 1;
                if (acc == 0) acc_phase ^= 1u;
            } else {
                acc_phase ^= 1u;
            }
        }
    }
    __syncthreads();
    if (tst && threadIdx.x == 0) atomicMax(tst + 2 * args.t_slots, (unsigned long long)globaltimer_ns());
    if (warp == 5) {
        __syncwarp();
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                     "r"(args.tmem_cols)
                     : "memory");
    }
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

// bf16 tensor [groups][rows][k] (row stride k, group stride group_rows rows) -> 3-D tensor map
// with a box of 64 (k) x box_rows x 1, 128-byte swizzle, zero fill outside the tensor.
bool make_map(CUtensorMap* m, const void* base, int k, int rows, int groups, long long group_rows,
              int box_rows) {
    auto enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[3] = {(cuuint64_t)k, (cuuint64_t)rows, (cuuint64_t)groups};
    cuuint64_t strides[2] = {(cuuint64_t)k * 2, (cuuint64_t)group_rows * k * 2};
    cuuint32_t box[3] = {(cuuint32_t)kBK, (cuuint32_t)box_rows, 1};
    cuuint32_t es[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box,
               es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

bool encode_tma_bf16(CUtensorMap* m, const void* base, int rank, const uint64_t* dims,
                     const uint64_t* strides_bytes, const uint32_t* box) {
    auto enc = encode_fn();
    if (!enc || rank < 1 || rank > 5) return false;
    cuuint64_t d[5], st[4];
    cuuint32_t bx[5], es[5];
    for (int i = 0; i < rank; ++i) {
        d[i] = dims[i];
        bx[i] = box[i];
        es[i] = 1;
        if (i + 1 < rank) st[i] = strides_bytes[i];
    }
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, (cuuint32_t)rank, const_cast<void*>(base), d, st, bx,
               es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

cudaError_t launch_gemm_tc(dflare_ctx* c, const GemmDesc& g, cudaStream_t s, std::string* why) {
    if (g.m_tok <= 0 || g.n <= 0) return cudaSuccess;
    TcArgs a;
    memset(&a, 0, sizeof(a));
    a.bn = g.m_tok <= 256 ? ((g.m_tok + 15) / 16) * 16 : 256;
    // With token tiles of 128 or more rows the GEMM is bound by the tensor pipeline, not by HBM:
    // two adjacent 128-row weight tiles can then share one activation tile (two accumulators, as
    // the SwiGLU gate and up tiles do), a third fewer shared-memory bytes per FLOP. At 256 token
    // rows the pair fills all 512 TMEM columns, so a unit's epilogue no longer overlaps the next
    // unit's MMAs: pairs pay only for the cheap fp32-logit epilogue (the LM head), and only when
    // their wave count times ~1.8 single-tile units beats the single tiles' wave count.
    // Measured: batch-16 step 1.965 -> 1.947 ms (the LM head); the context fill's K/V projection
    // with its rotary epilogue lost (Qwen3-4B shape 822 -> 640 TFLOP/s).
    {
        const long long u1 = (long long)g.groups * ((g.n + kBM - 1) / kBM) * ((g.m_tok + a.bn - 1) / a.bn);
        const long long u2 = (long long)g.groups * ((g.n + 2 * kBM - 1) / (2 * kBM)) * ((g.m_tok + a.bn - 1) / a.bn);
        const long long w1 = (u1 + c->num_sms - 1) / c->num_sms, w2 = (u2 + c->num_sms - 1) / c->num_sms;
        a.pair = (!g.a2 && a.bn >= 128 && g.n > kBM && g.force_splits <= 0 &&
                  g.ep.kind == EPI_F32 && 9 * w2 < 5 * w1) ? 1 : 0;
    }
    a.n_a = (g.a2 || a.pair) ? 2 : 1;
    a.tok_tiles = (g.m_tok + a.bn - 1) / a.bn;
    a.n_tiles = (g.n + (kBM << a.pair) - 1) / (kBM << a.pair);
    a.k_blocks = (g.k + kBK - 1) / kBK;
    const int tiles = g.groups * a.n_tiles * a.tok_tiles;
    const int sms = c->num_sms;
    // split-K choice: the most splits that still run as one wave (tiles * splits <= SMs), within
    // the workspace and counter capacity. Measured: a second wave of split units is slower than
    // fewer, longer units even when it shortens every unit (d 4096 gate/up: 3 splits over 288
    // units 97 us, 1 split over 96 units 42 us), so no split count that spills into a second
    // wave is taken.
    int best = 1;
    for (int sp = 2; sp <= 16 && sp <= a.k_blocks / 2 && tiles * sp <= sms; ++sp) {
        const int kbp = (a.k_blocks + sp - 1) / sp;
        const int spn = (a.k_blocks + kbp - 1) / kbp;
        const size_t need = (size_t)tiles * spn * a.n_a * a.bn * 128;
        if (need > c->ws_floats || tiles > c->tile_cnt_n) break;
        best = spn;
    }
    // Shared-memory budget: up to 227 KB (one CTA per SM; measured faster than two smaller CTAs
    // per SM, with or without programmatic dependent launch). Stage size: four 64-wide k-blocks
    // (512 contiguous bytes of every weight row; 128-byte rows per request leave DRAM bandwidth
    // unused), fewer when two stages do not fit.
    const int epi_bytes = a.n_a * kChunk * 128 * 4;
    // a context fill over several token tiles lists the tiles that hold appended rows (the
    // sequences of one call can have very different lengths: rows past app_cnt are padding)
    a.compact = (g.ep.kind == EPI_KV_APPEND && a.tok_tiles > 1 && a.tok_tiles <= kMaxTokList) ? 1 : 0;
    const int misc_bytes = 16 + (a.compact ? 4 * kMaxTokList : 0);
    const int fixed = 1024 + epi_bytes + 8 * (2 * kMaxStages + 5) + misc_bytes;
    const int budget = g.max_smem > 0 ? std::min(g.max_smem, kSmemLimit) : kSmemLimit;
    if (g.kbs > 0) {
        a.kbs = g.kbs;
    } else {
        a.kbs = 4;
        while (a.kbs > 1 && 2 * a.kbs * (kBM * kBK * 2 * a.n_a + a.bn * kBK * 2) > budget - fixed)
            a.kbs >>= 1;
    }
    if (g.force_splits > 0) best = std::min(g.force_splits, a.k_blocks);
    a.kb_per_split = (a.k_blocks + best - 1) / best;
    // (split ranges are not rounded to whole stages: the producer issues a partial last stage,
    // and balanced ranges beat 512-byte-aligned ones, e.g. Q/K^d/V^d 14/14/12 k-blocks rather
    // than 16/16/8: 0.5265 -> 0.5221 ms per Qwen3-4B-shaped step)
    a.splits = (a.k_blocks + a.kb_per_split - 1) / a.kb_per_split;
    if (a.splits > 1 && ((size_t)tiles * a.splits * a.n_a * a.bn * 128 > c->ws_floats || tiles > c->tile_cnt_n)) {
        if (why) *why = "tcgen05 GEMM: split-K workspace too small";
        return cudaErrorInvalidValue;
    }
    a.n_units = tiles * a.splits;
    a.b_bytes = (uint32_t)a.bn * kBK * 2;
    a.stage_bytes = (uint32_t)a.kbs * (kABytes * a.n_a + a.b_bytes);
    a.evict_first = g.evict_first >= 0 ? 1 : 0;
    a.stages = std::min(kMaxStages, (budget - fixed) / (int)a.stage_bytes);
    if (a.stages < 2) {
        if (why) *why = "tcgen05 GEMM: tile does not fit in shared memory";
        return cudaErrorInvalidValue;
    }
    const int smem = 1024 + a.stages * (int)a.stage_bytes + epi_bytes + 8 * (2 * a.stages + 5) + misc_bytes;
    a.n_bufs = (2 * a.n_a * a.bn <= 512) ? 2 : 1;
    int cols = 32;
    while (cols < a.n_bufs * a.n_a * a.bn) cols <<= 1;
    a.tmem_cols = cols;
    // kind::f16 instruction descriptor: fp32 accumulate, bf16 A and B, both K-major,
    // N = bn (bits 17-22, N >> 3), M = 128 (bits 24-28, M >> 4)
    a.idesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(a.bn >> 3) << 17) |
              ((uint32_t)(kBM >> 4) << 24);
    a.ws = c->ws;
    a.tile_cnt = c->tile_cnt;
    a.err = c->err;
    a.ep = g.ep;
    // weights: groups of n rows, a_group_rows apart; activations: one group per weight group, one
    // group shared by all (b_shared), or k / b_kgroup groups that the contraction runs across
    const long long a_gr = g.a_group_rows > 0 ? g.a_group_rows : g.n;
    a.b_kg = g.b_kgroup;
    a.resid_red = (c->cfg.flags & DFLARE_FLAG_DETERMINISTIC) ? 0 : 1;
    a.resid_vec = g.ep.kind == EPI_RESID && g.ep.n % 16 == 0 && g.ep.ld_resid % 4 == 0 &&
                  (reinterpret_cast<uintptr_t>(g.ep.resid) & 15u) == 0;
    a.b_gsel = g.b_shared ? 0 : 1;
    const int b_k = g.b_kgroup > 0 ? g.b_kgroup : g.k;
    const int b_groups = g.b_kgroup > 0 ? g.k / g.b_kgroup : (g.b_shared ? 1 : g.groups);
    const long long b_gr = g.b_group_rows > 0 ? g.b_group_rows : g.m_tok;
    if (g.b_kgroup > 0 && (g.b_kgroup % kBK != 0 || g.k % g.b_kgroup != 0 || g.groups != 1)) {
        if (why) *why = "tcgen05 GEMM: b_kgroup must be a multiple of 64 that divides k, with one group";
        return cudaErrorInvalidValue;
    }
    // a pair's second tile: the same matrix from row 128 on (rows past its end read as zeros)
    const void* a2 = g.a2 ? g.a2 : a.pair ? static_cast<const void*>(static_cast<const bf16*>(g.a) + (size_t)kBM * g.k)
                                          : g.a;
    if (!make_map(&a.map_a, g.a, g.k, g.n, g.groups, a_gr, kBM) ||
        !make_map(&a.map_a2, a2, g.k, a.pair ? g.n - kBM : g.n, g.groups, a_gr, kBM) ||
        !make_map(&a.map_b, g.b, b_k, g.m_tok, b_groups, b_gr, a.bn)) {
        if (why) *why = "cuTensorMapEncodeTiled failed (alignment or driver entry point)";
        return cudaErrorInvalidValue;
    }
    const bool aux = g.b_kgroup > 0 || g.b_shared || g.ep.bias || g.ep.out_gstride;
    static PerDeviceOnce configured[2];
    const cudaError_t ce = configured[aux]([aux] {
        return cudaFuncSetAttribute(aux ? gemm_tc_kernel<true> : gemm_tc_kernel<false>,
                                    cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemLimit);
    });
    if (ce != cudaSuccess) return ce;
    const int grid = std::min(a.n_units, sms);
    if (c->t_stamps && c->t_next < c->t_slots) {
        a.t_stamps = c->t_stamps + c->t_next++;
        a.t_slots = c->t_slots;
    }
    return launch_kernel(c->pdl, aux ? gemm_tc_kernel<true> : gemm_tc_kernel<false>, dim3(grid),
                         dim3(kThreads), smem, s, a);
}

}  // namespace dfl
