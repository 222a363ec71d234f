// The C ABI of libdflare (include/dflare.h): argument checks, device memory of a context, and the
// launch sequence of the three calls of the draft path.
#include <math.h>
#include <string.h>

#include <algorithm>
#include <cmath>
#include <map>
#include <mutex>
#include <string>
#include <vector>

#include "internal.h"

using namespace dfl;

namespace dfl {
int attention_splits(const dflare_config& g, int batch, int num_sms, int len_ub);
}

namespace {

thread_local std::string g_create_error;

dflare_status fail(dflare_ctx* c, dflare_status st, const std::string& m) {
    if (c)
        c->msg = m;
    else
        g_create_error = m;
    return st;
}

#define CUDA_TRY(expr)                                                                     \
    do {                                                                                   \
        cudaError_t e_ = (expr);                                                           \
        if (e_ != cudaSuccess)                                                             \
            return fail(c, DFLARE_ECUDA, std::string(#expr) + ": " + cudaGetErrorString(e_)); \
    } while (0)

bool check_config(const dflare_config* g, std::string* why) {
    auto bad = [&](const char* m) {
        *why = std::string("invalid config: ") + m;
        return false;
    };
    if (!g) return bad("null");
    if (g->d < 64 || g->d % 64 != 0 || g->d > 4096) return bad("d must be a multiple of 64 in [64, 4096]");
    if (g->n_draft_layers < 1 || g->n_draft_layers > 16) return bad("n_draft_layers must be in [1, 16]");
    if (g->n_target_layers < 1 || g->n_target_layers > 64) return bad("n_target_layers must be in [1, 64]");
    if (g->head_dim != 64 && g->head_dim != 128) return bad("head_dim must be 64 or 128");
    if (g->n_kv_heads < 1 || g->n_q_heads < 1 || g->n_q_heads % g->n_kv_heads != 0)
        return bad("n_q_heads must be a positive multiple of n_kv_heads");
    if ((g->n_q_heads * g->head_dim) % 128 != 0 || (g->n_kv_heads * g->head_dim) % 128 != 0)
        return bad("n_q_heads*head_dim and n_kv_heads*head_dim must be multiples of 128");
    if (g->ffn < 64 || g->ffn % 64 != 0) return bad("ffn must be a positive multiple of 64");
    if (g->vocab < 2) return bad("vocab must be >= 2");
    if (g->mask_token_id < 0 || g->mask_token_id >= g->vocab) return bad("mask_token_id outside [0, vocab)");
    if (g->block < 1 || g->block > 32) return bad("block must be in [1, 32]");
    if (g->max_batch < 1 || g->max_batch > 64) return bad("max_batch must be in [1, 64]");
    if (g->max_ctx < 1 || g->max_ctx > (1 << 22)) return bad("max_ctx must be in [1, 2^22]");
    if (g->max_fuse_rows < 1 || g->max_fuse_rows > (1 << 20)) return bad("max_fuse_rows must be in [1, 2^20]");
    if (!(g->rms_eps >= 0.f) || !isfinite(g->rms_eps)) return bad("rms_eps must be finite and >= 0");
    if (!(g->rope_theta > 0.f) || !isfinite(g->rope_theta)) return bad("rope_theta must be finite and > 0");
    if (g->dtype != DFLARE_BF16 && g->dtype != DFLARE_F32) return bad("dtype must be DFLARE_BF16 or DFLARE_F32");
    if (g->flags & ~(DFLARE_FLAG_NO_BLOCK_ROPE | DFLARE_FLAG_RAW_FUSION | DFLARE_FLAG_SIMT_GEMM |
                     DFLARE_FLAG_SERIAL_LAUNCH | DFLARE_FLAG_SHARED_KV | DFLARE_FLAG_FUSION_FC |
                     DFLARE_FLAG_DFLASH_FC | DFLARE_FLAG_DETERMINISTIC | DFLARE_FLAG_MMA_SYNC_ATTENTION))
        return bad("unknown flag bits");
    if ((g->flags & DFLARE_FLAG_DFLASH_FC) &&
        (g->flags & (DFLARE_FLAG_RAW_FUSION | DFLARE_FLAG_FUSION_FC)))
        return bad("DFLARE_FLAG_DFLASH_FC replaces the layer-wise fusion: no RAW_FUSION or FUSION_FC");
    return true;
}

template <class P>
cudaError_t dalloc(P** p, size_t bytes, std::vector<void*>& owned) {
    void* q = nullptr;
    cudaError_t e = cudaMalloc(&q, bytes < 256 ? 256 : bytes);
    if (e == cudaSuccess) {
        owned.push_back(q);
        *p = static_cast<P*>(q);
    }
    return e;
}

// Device allocations of each context, freed by dflare_destroy.
std::mutex g_own_mu;
std::map<const dflare_ctx*, std::vector<void*>> g_owned;

void free_all(dflare_ctx* c) {
    std::vector<void*> v;
    {
        std::lock_guard<std::mutex> lk(g_own_mu);
        auto it = g_owned.find(c);
        if (it != g_owned.end()) {
            v.swap(it->second);
            g_owned.erase(it);
        }
    }
    for (void* p : v) cudaFree(p);
}

bool use_tc(const dflare_ctx* c) {
    return c->cfg.dtype == DFLARE_BF16 && !(c->cfg.flags & DFLARE_FLAG_SIMT_GEMM);
}

dflare_status gemm(dflare_ctx* c, const GemmDesc& g, cudaStream_t s) {
    cudaError_t e;
    std::string why;
    if (use_tc(c))
        e = launch_gemm_tc(c, g, s, &why);
    else
        e = launch_gemm_simt(c, g, s);
    if (e != cudaSuccess)
        return fail(c, DFLARE_ECUDA, "GEMM launch: " + (why.empty() ? std::string(cudaGetErrorString(e)) : why));
    return DFLARE_OK;
}

EpiParams epi_base(const dflare_ctx* c) {
    EpiParams ep;
    memset(&ep, 0, sizeof(ep));
    const dflare_config& g = c->cfg;
    ep.d_q = g.n_q_heads * g.head_dim;
    ep.d_kv = g.n_kv_heads * g.head_dim;
    ep.head_dim = g.head_dim;
    ep.block = g.block;
    ep.max_ctx = g.max_ctx;
    ep.max_batch = g.max_batch;
    ep.rope_cos = c->rope_cos;
    ep.rope_sin = c->rope_sin;
    return ep;
}

// Calls the user's trace hook around one launch (see dflare_set_trace).
struct Trace {
    dflare_ctx* c;
    const char* name;
    cudaStream_t s;
    Trace(dflare_ctx* c_, const char* n, cudaStream_t s_) : c(c_), name(n), s(s_) {
        if (c->trace_fn) c->trace_fn(c->trace_user, name, 0, s);
    }
    ~Trace() {
        if (c->trace_fn) c->trace_fn(c->trace_user, name, 1, s);
    }
};

dflare_status traced_gemm(dflare_ctx* c, const char* name, const GemmDesc& g, cudaStream_t s) {
    Trace t(c, name, s);
    return gemm(c, g, s);
}

const uint8_t* at(const void* base, size_t elems, size_t esz) {
    return static_cast<const uint8_t*>(base) + elems * esz;
}

// Repeated calls with the same operands run as one CUDA graph: the first call of a new operand
// set runs its launches directly, the second is captured (thread-local capture on the caller's
// stream) and launched, later ones replay the graph. The kernels' parameters depend only on the
// operands in the key and on state that is fixed for the context (the weights: set_weights drops
// the graphs); everything that varies from step to step (context lengths, accepted counts, step
// counters) is read by the kernels from device memory. Calls made while the stream is being
// captured, with a trace hook or GEMM timing set, or on the legacy default stream run directly.
void drop_slot(GraphSlot& sl) {
    if (sl.exec) cudaGraphExecDestroy(sl.exec);
    sl = GraphSlot{};
}
void drop_graph(CallGraph& cg) {
    for (GraphSlot& sl : cg.slot) drop_slot(sl);
}
template <class F>
dflare_status graphed(dflare_ctx* c, CallGraph& cg, const uint64_t* key, int nk, cudaStream_t s, F&& body) {
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (!s || c->trace_fn || c->t_stamps || nk > GraphSlot::kKeyLen || cudaStreamIsCapturing(s, &cs) != cudaSuccess ||
        cs != cudaStreamCaptureStatusNone) {
        cudaGetLastError();
        return body();
    }
    const size_t kb = (size_t)nk * sizeof(uint64_t);
    GraphSlot* sl = nullptr;
    for (GraphSlot& x : cg.slot)
        if (x.seen && memcmp(x.key, key, kb) == 0) sl = &x;
    if (!sl) {   // a new operand set: run it directly and remember it (evicting the oldest)
        sl = &cg.slot[0];
        for (GraphSlot& x : cg.slot)
            if (x.used < sl->used) sl = &x;
        drop_slot(*sl);
        memcpy(sl->key, key, kb);
        sl->seen = true;
        sl->used = ++cg.clock;
        return body();
    }
    sl->used = ++cg.clock;
    if (sl->exec) {
        if (cudaGraphLaunch(sl->exec, s) == cudaSuccess) return DFLARE_OK;
        cudaGetLastError();
        drop_slot(*sl);
        return body();
    }
    // the second call with these operands: capture it
    if (cudaStreamBeginCapture(s, cudaStreamCaptureModeThreadLocal) != cudaSuccess) {
        cudaGetLastError();
        return body();
    }
    const dflare_status st = body();
    cudaGraph_t graph = nullptr;
    const cudaError_t e = cudaStreamEndCapture(s, &graph);
    if (st != DFLARE_OK || e != cudaSuccess || !graph) {
        if (graph) cudaGraphDestroy(graph);
        cudaGetLastError();
        drop_slot(*sl);
        return st != DFLARE_OK ? st : body();   // nothing ran while capturing: run it now
    }
    cudaGraphExec_t exec = nullptr;
    const cudaError_t ei = cudaGraphInstantiate(&exec, graph, 0);
    cudaGraphDestroy(graph);
    if (ei != cudaSuccess || cudaGraphLaunch(exec, s) != cudaSuccess) {
        if (exec) cudaGraphExecDestroy(exec);
        cudaGetLastError();
        drop_slot(*sl);
        return body();
    }
    sl->exec = exec;
    return DFLARE_OK;
}

dflare_status fuse_context_launches(dflare_ctx* c, const void* hidden, const int32_t* n_new,
                                    int n_max, void* fused_out, cudaStream_t s) {
    const dflare_config& g = c->cfg;
    const int m_tok = c->batch * n_max;
    const size_t d_q = (size_t)g.n_q_heads * g.head_dim, d_kv = (size_t)g.n_kv_heads * g.head_dim;
    {
        Trace t(c, "fuse_begin", s);
        CUDA_TRY(launch_fuse_begin(c, n_new, n_max, s));
    }
    // ctx_src: what the context K/V projection reads, [groups][ctx_rows][d]
    const void* ctx_src = c->fused;
    long long ctx_rows = g.max_fuse_rows;
    int ctx_shared = 0;
    if (g.flags & DFLARE_FLAG_DFLASH_FC) {
        // Eq. 1: c_t = W_fc [h^(1); ...; h^(T)] + b_fc as one GEMM whose contraction runs over
        // the T stacked target layers of target_hidden; one c for every draft layer
        GemmDesc fc{};
        fc.a = c->w.dflash_fc_w;
        fc.b = hidden;
        fc.groups = 1;
        fc.n = g.d;
        fc.k = g.n_target_layers * g.d;
        fc.m_tok = m_tok;
        fc.b_group_rows = m_tok;
        fc.b_kgroup = g.d;
        fc.ep = epi_base(c);
        fc.ep.kind = EPI_STORE;
        fc.ep.m_tok = m_tok;
        fc.ep.n = g.d;
        fc.ep.out = fused_out ? fused_out : c->fused;
        fc.ep.ldo = g.d;
        fc.ep.bias = c->w.dflash_fc_b;
        dflare_status st = traced_gemm(c, "gemm_dflash_fc", fc, s);
        if (st != DFLARE_OK) return st;
        ctx_src = fc.ep.out;
        ctx_rows = m_tok;
        ctx_shared = 1;
    } else {
        const bool fc_after = g.flags & DFLARE_FLAG_FUSION_FC;
        {
            Trace t(c, "fuse_layers", s);
            CUDA_TRY(launch_fuse_layers(c, hidden, n_max, fc_after ? nullptr : fused_out, s));
        }
        if (fc_after) {
            // "+FC": F'^(i) = F^(i) W_fc^(i)T + b_fc^(i), one d x d GEMM per draft layer
            GemmDesc fc{};
            fc.a = c->w.fusion_fc_w;
            fc.b = c->fused;
            fc.groups = g.n_draft_layers;
            fc.n = g.d;
            fc.k = g.d;
            fc.m_tok = m_tok;
            fc.b_group_rows = g.max_fuse_rows;
            fc.ep = epi_base(c);
            fc.ep.kind = EPI_STORE;
            fc.ep.m_tok = m_tok;
            fc.ep.n = g.d;
            fc.ep.out = fused_out ? fused_out : c->fused_fc;
            fc.ep.ldo = g.d;
            fc.ep.out_gstride = (fused_out ? (long long)m_tok : g.max_fuse_rows) * g.d;
            fc.ep.bias = c->w.fusion_fc_b;
            dflare_status st = traced_gemm(c, "gemm_fusion_fc", fc, s);
            if (st != DFLARE_OK) return st;
            ctx_src = fc.ep.out;
            ctx_rows = fused_out ? (long long)m_tok : g.max_fuse_rows;
        }
    }
    GemmDesc gd{};
    if (g.flags & (DFLARE_FLAG_SHARED_KV | DFLARE_FLAG_DFLASH_FC)) {
        // W_K^d / W_V^d: rows [d_q, d_q + 2 d_kv) of each layer's w_qkv
        gd.a = at(c->w.w_qkv, d_q * g.d, c->esz);
        gd.a_group_rows = (long long)(d_q + 2 * d_kv);
    } else {
        gd.a = c->w.w_kv_ctx;
    }
    gd.b = ctx_src;
    gd.b_shared = ctx_shared;
    gd.groups = g.n_draft_layers;
    gd.n = (int)(2 * d_kv);
    gd.k = g.d;
    gd.m_tok = m_tok;
    gd.b_group_rows = ctx_rows;
    gd.ep = epi_base(c);
    gd.ep.kind = EPI_KV_APPEND;
    gd.ep.m_tok = gd.m_tok;
    gd.ep.n = gd.n;
    gd.ep.kcache = c->kcache;
    gd.ep.vcache = c->vcache;
    gd.ep.app_base = c->app_base;
    gd.ep.app_cnt = c->app_cnt;
    gd.ep.n_max = n_max;
    return traced_gemm(c, "gemm_kv_ctx", gd, s);
}

}  // namespace

namespace dfl {
void noalloc_set_error(const std::string& message) { g_create_error = message; }
}  // namespace dfl

extern "C" {

dflare_status dflare_create(const dflare_config* cfg, dflare_ctx** out) {
    dflare_ctx* c = nullptr;
    std::string why;
    if (!out) return fail(nullptr, DFLARE_EINVAL, "out is NULL");
    *out = nullptr;
    if (!check_config(cfg, &why)) return fail(nullptr, DFLARE_EINVAL, why);
    c = new dflare_ctx();
    c->cfg = *cfg;
    c->esz = cfg->dtype == DFLARE_BF16 ? 2 : 4;
    c->pdl = !(cfg->flags & DFLARE_FLAG_SERIAL_LAUNCH);
    std::vector<void*> owned;
    auto bail = [&](dflare_status st, const std::string& m) {
        for (void* p : owned) cudaFree(p);
        delete c;
        return fail(nullptr, st, m);
    };
    cudaError_t e = cudaGetDevice(&c->device);
    if (e != cudaSuccess) return bail(DFLARE_ECUDA, std::string("cudaGetDevice: ") + cudaGetErrorString(e));
    e = cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, c->device);
    if (e != cudaSuccess) return bail(DFLARE_ECUDA, std::string("cudaDeviceGetAttribute: ") + cudaGetErrorString(e));
    const dflare_config& g = c->cfg;
    const size_t esz = c->esz;
    const size_t d = g.d, D = g.n_draft_layers, B = g.block, V = g.vocab, F = g.ffn;
    const size_t d_q = (size_t)g.n_q_heads * g.head_dim, d_kv = (size_t)g.n_kv_heads * g.head_dim;
    const size_t rows = (size_t)g.max_batch * B, mrows = (size_t)g.max_batch * (B > 1 ? B - 1 : 1);
    const size_t kv = D * g.max_batch * d_kv * (size_t)g.max_ctx;
    // split-KV partial buffers sized for the largest batch x splits product
    const int G = g.n_q_heads / g.n_kv_heads;
    const int q_tiles = (g.block * G + 63) / 64;
    size_t part_rows = 1;   // split-KV partials in global memory: the fp32 path only
    for (int b = 1; b <= g.max_batch && g.dtype == DFLARE_F32; ++b) {
        const size_t r = (size_t)b * g.n_kv_heads * q_tiles * attention_splits(g, b, c->num_sms, g.max_ctx) * 64;
        if (r > part_rows) part_rows = r;
    }
    c->ws_floats = (size_t)8 << 20;
    c->tile_cnt_n = 8192;
#define ALLOC(ptr, bytes)                                                                    \
    do {                                                                                     \
        e = dalloc(&(ptr), (bytes), owned);                                                  \
        if (e != cudaSuccess)                                                                \
            return bail(DFLARE_ENOMEM, std::string("cudaMalloc(" #ptr ", ") +               \
                                           std::to_string((size_t)(bytes)) + "): " +           \
                                           cudaGetErrorString(e));                           \
    } while (0)
    ALLOC(c->kcache, kv * esz);
    ALLOC(c->vcache, kv * esz);
    ALLOC(c->ctx_len, g.max_batch * sizeof(int32_t));
    ALLOC(c->app_base, g.max_batch * sizeof(int32_t));
    ALLOC(c->app_cnt, g.max_batch * sizeof(int32_t));
    ALLOC(c->alpha, D * g.n_target_layers * sizeof(float));
    ALLOC(c->fused, D * (size_t)g.max_fuse_rows * d * esz);
    if (g.flags & DFLARE_FLAG_FUSION_FC) ALLOC(c->fused_fc, D * (size_t)g.max_fuse_rows * d * esz);
    ALLOC(c->x, rows * d * sizeof(float));
    ALLOC(c->xn, rows * d * esz);
    ALLOC(c->q, rows * d_q * esz);
    ALLOC(c->kd, rows * d_kv * esz);
    ALLOC(c->vd, rows * d_kv * esz);
    if (g.dtype == DFLARE_BF16) ALLOC(c->qkv32, rows * (d_q + 2 * d_kv) * sizeof(float));
    ALLOC(c->attn, rows * d_q * esz);
    ALLOC(c->act, rows * F * esz);
    ALLOC(c->xh, mrows * d * esz);
    ALLOC(c->logits, mrows * V * sizeof(float));
    ALLOC(c->attn_o, part_rows * g.head_dim * sizeof(float));
    ALLOC(c->attn_ml, part_rows * 2 * sizeof(float));
    ALLOC(c->ws, c->ws_floats * sizeof(float));
    ALLOC(c->tile_cnt, (size_t)c->tile_cnt_n * sizeof(uint32_t));
    ALLOC(c->amax_slot, rows * sizeof(unsigned long long));
    ALLOC(c->tgt_tok, rows * sizeof(int32_t));
    ALLOC(c->spec_part, (size_t)g.max_batch * (2 * B - 1) * kSpecMaxChunks * sizeof(float2));
    ALLOC(c->spec_a, g.max_batch * sizeof(int32_t));
    ALLOC(c->amax_cnt, sizeof(uint32_t));
    const size_t half = g.head_dim / 2, npos = (size_t)g.max_ctx + B;
    ALLOC(c->rope_cos, npos * half * sizeof(float));
    ALLOC(c->rope_sin, npos * half * sizeof(float));
    ALLOC(c->err, sizeof(uint32_t));
#undef ALLOC
    // zero what must start at zero (counters, lengths, error word, stale-row buffers)
    struct Z { void* p; size_t n; } zs[] = {
        {c->ctx_len, g.max_batch * sizeof(int32_t)}, {c->app_base, g.max_batch * sizeof(int32_t)},
        {c->app_cnt, g.max_batch * sizeof(int32_t)}, {c->tile_cnt, (size_t)c->tile_cnt_n * 4},
        {c->amax_slot, rows * 8}, {c->amax_cnt, 4}, {c->err, 4},
        {c->fused, D * (size_t)g.max_fuse_rows * d * esz}, {c->x, rows * d * 4},
        // every row the attention reads past the valid keys holds a written value or zero
        {c->kcache, kv * esz}, {c->vcache, kv * esz}, {c->kd, rows * d_kv * esz},
        {c->vd, rows * d_kv * esz}, {c->qkv32, c->qkv32 ? rows * (d_q + 2 * d_kv) * 4 : 0}};
    for (auto& z : zs) {
        if (!z.p || !z.n) continue;
        e = cudaMemset(z.p, 0, z.n);
        if (e != cudaSuccess) return bail(DFLARE_ECUDA, std::string("cudaMemset: ") + cudaGetErrorString(e));
    }
    // rotary table: cos/sin of pos * theta^(-2j/hd), evaluated in double, stored as float
    {
        std::vector<float> cs(npos * half), sn(npos * half);
        for (size_t j = 0; j < half; ++j) {
            const double inv = pow((double)g.rope_theta, -2.0 * (double)j / (double)g.head_dim);
            for (size_t p = 0; p < npos; ++p) {
                const double ang = (double)p * inv;
                cs[p * half + j] = (float)cos(ang);
                sn[p * half + j] = (float)sin(ang);
            }
        }
        e = cudaMemcpy(c->rope_cos, cs.data(), cs.size() * 4, cudaMemcpyHostToDevice);
        if (e == cudaSuccess) e = cudaMemcpy(c->rope_sin, sn.data(), sn.size() * 4, cudaMemcpyHostToDevice);
        if (e != cudaSuccess) return bail(DFLARE_ECUDA, std::string("rotary table upload: ") + cudaGetErrorString(e));
    }
    {
        std::lock_guard<std::mutex> lk(g_own_mu);
        g_owned[c] = owned;
    }
    c->batch = g.max_batch;
    *out = c;
    return DFLARE_OK;
}

dflare_status dflare_destroy(dflare_ctx* c) {
    if (!c) return DFLARE_OK;
    DeviceGuard dg(c->device);
    cudaDeviceSynchronize();
    drop_graph(c->draft_graph);
    drop_graph(c->fuse_graph);
    free_all(c);
    delete c;
    return DFLARE_OK;
}

dflare_status dflare_set_weights(dflare_ctx* c, const dflare_weights* w, void* stream) {
    if (!c) return fail(nullptr, DFLARE_EINVAL, "ctx is NULL");
    DeviceGuard dg(c->device);
    if (!w) return fail(c, DFLARE_EINVAL, "weights is NULL");
    const unsigned fl = c->cfg.flags;
    const bool dflash = fl & DFLARE_FLAG_DFLASH_FC;
    // (pointer, name, read under the context's flags)
    struct Need { const void* p; const char* name; bool used; } need[] = {
        {w->fuse_logits, "fuse_logits", !dflash},
        {w->fuse_norm, "fuse_norm", !dflash},
        {w->w_kv_ctx, "w_kv_ctx", !dflash && !(fl & DFLARE_FLAG_SHARED_KV)},
        {w->attn_norm, "attn_norm", true}, {w->w_qkv, "w_qkv", true}, {w->w_o, "w_o", true},
        {w->mlp_norm, "mlp_norm", true}, {w->w_gate, "w_gate", true}, {w->w_up, "w_up", true},
        {w->w_down, "w_down", true}, {w->final_norm, "final_norm", true}, {w->embed, "embed", true},
        {w->lm_head, "lm_head", true},
        {w->fusion_fc_w, "fusion_fc_w", (fl & DFLARE_FLAG_FUSION_FC) != 0},
        {w->fusion_fc_b, "fusion_fc_b", (fl & DFLARE_FLAG_FUSION_FC) != 0},
        {w->dflash_fc_w, "dflash_fc_w", dflash}, {w->dflash_fc_b, "dflash_fc_b", dflash}};
    for (const Need& n : need) {
        if (!n.used) continue;
        if (!n.p) return fail(c, DFLARE_EINVAL, std::string("weight ") + n.name + " is NULL");
        if (reinterpret_cast<uintptr_t>(n.p) % 16 != 0)
            return fail(c, DFLARE_EINVAL, std::string("weight ") + n.name + " is not 16-byte aligned");
    }
    c->w = *w;
    drop_graph(c->draft_graph);   // captured launches hold the previous weights' tensor maps
    drop_graph(c->fuse_graph);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (!dflash) CUDA_TRY(launch_fusion_alpha(c, s));
    c->weights_set = true;
    return DFLARE_OK;
}

dflare_status dflare_reset(dflare_ctx* c, int batch, void* stream) {
    if (!c) return fail(nullptr, DFLARE_EINVAL, "ctx is NULL");
    DeviceGuard dg(c->device);
    if (batch < 1 || batch > c->cfg.max_batch)
        return fail(c, DFLARE_ECAPACITY, "batch outside [1, max_batch]");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    c->batch = batch;
    c->ctx_ub = 0;
    CUDA_TRY(cudaMemsetAsync(c->ctx_len, 0, c->cfg.max_batch * sizeof(int32_t), s));
    return DFLARE_OK;
}

dflare_status dflare_fuse_context(dflare_ctx* c, const void* hidden, const int32_t* n_new,
                                  int n_max, void* fused_out, void* stream) {
    if (!c) return fail(nullptr, DFLARE_EINVAL, "ctx is NULL");
    DeviceGuard dg(c->device);
    if (!c->weights_set) return fail(c, DFLARE_ESTATE, "dflare_set_weights has not been called");
    if (!hidden || !n_new) return fail(c, DFLARE_EINVAL, "target_hidden or n_new is NULL");
    if (n_max < 1) return fail(c, DFLARE_EINVAL, "n_max must be >= 1");
    if ((long long)c->batch * n_max > c->cfg.max_fuse_rows)
        return fail(c, DFLARE_ECAPACITY, "batch * n_max exceeds max_fuse_rows");
    if (n_max > c->cfg.max_ctx) return fail(c, DFLARE_ECAPACITY, "n_max exceeds max_ctx");
    if (reinterpret_cast<uintptr_t>(hidden) % 16 || reinterpret_cast<uintptr_t>(fused_out) % 16)
        return fail(c, DFLARE_EINVAL, "target_hidden and fused_out must be 16-byte aligned");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const uint64_t key[] = {(uint64_t)c->batch, (uint64_t)(uintptr_t)hidden, (uint64_t)(uintptr_t)n_new,
                            (uint64_t)n_max, (uint64_t)(uintptr_t)fused_out};
    const dflare_status st = graphed(c, c->fuse_graph, key, 5, s, [&] {
        return fuse_context_launches(c, hidden, n_new, n_max, fused_out, s);
    });
    if (st == DFLARE_OK) c->ctx_ub = std::min(c->cfg.max_ctx, c->ctx_ub + n_max);
    return st;
}

}  // extern "C"

namespace {

// Sampling parameters of dflare_draft_block_sampled (null: greedy).
struct Sampling {
    float inv_t;
    uint64_t seed;
    const uint64_t* step;
};

dflare_status draft_block_impl(dflare_ctx* c, const int32_t* last_token, int32_t* draft_tokens,
                               float* logits_out, float* hidden_out, void* stream,
                               const Sampling* smp) {
    if (!c) return fail(nullptr, DFLARE_EINVAL, "ctx is NULL");
    if (!c->weights_set) return fail(c, DFLARE_ESTATE, "dflare_set_weights has not been called");
    // with B = 1 the block has no mask rows: nothing is drafted and draft_tokens may be NULL
    if (!last_token || (!draft_tokens && c->cfg.block > 1))
        return fail(c, DFLARE_EINVAL, "last_token or draft_tokens is NULL");
    const dflare_config& g = c->cfg;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const size_t esz = c->esz, d = g.d, B = g.block, F = g.ffn;
    const size_t d_q = (size_t)g.n_q_heads * g.head_dim, d_kv = (size_t)g.n_kv_heads * g.head_dim;
    const int rows = c->batch * g.block;
    const size_t hid_stride = (size_t)c->batch * B * d;
    {
        Trace t(c, "embed", s);
        CUDA_TRY(launch_embed(c, last_token, s));
    }
    if (hidden_out)
        CUDA_TRY(cudaMemcpyAsync(hidden_out, c->x, hid_stride * 4, cudaMemcpyDeviceToDevice, s));
    // bf16 tensor-core path: the Q/K^d/V^d splits add their fp32 partials into qkv32 with L2
    // reductions and the attention applies the rotary embedding and rounds as it loads them (no
    // split-K workspace, tile counter or last-CTA epilogue on the critical path); qkv32 is cleared
    // by the embedding (first layer) and by each pre-attention RMSNorm. The deterministic mode
    // keeps the fixed-order reduction.
    const bool red32 = c->qkv32 && !(g.flags & (DFLARE_FLAG_DETERMINISTIC | DFLARE_FLAG_SIMT_GEMM));
    for (int i = 0; i < g.n_draft_layers; ++i) {
        if (i > 0) {
            Trace t(c, "rmsnorm", s);
            CUDA_TRY(launch_rmsnorm(c, at(c->w.attn_norm, i * d, esz), rows, false, c->xn, s,
                                    red32 ? c->qkv32 : nullptr));
        }
        // Q = X~ W_Q, K^d = X~ W_K^d, V^d = X~ W_V^d with the rotary embedding (Eq. 4)
        GemmDesc q{};
        q.a = at(c->w.w_qkv, i * (d_q + 2 * d_kv) * d, esz);
        q.b = c->xn;
        q.groups = 1;
        q.n = (int)(d_q + 2 * d_kv);
        q.k = g.d;
        q.m_tok = rows;
        q.b_group_rows = rows;
        q.ep = epi_base(c);
        q.ep.kind = EPI_QKV;
        q.ep.m_tok = rows;
        q.ep.n = q.n;
        q.ep.q = c->q;
        q.ep.kd = c->kd;
        q.ep.vd = c->vd;
        q.ep.ctx_len = c->ctx_len;
        q.ep.rope = (g.flags & DFLARE_FLAG_NO_BLOCK_ROPE) ? 0 : 1;
        if (red32) {
            q.ep.kind = EPI_RED32;
            q.ep.out = c->qkv32;
            q.ep.ldo = q.n;
        }
        dflare_status st = traced_gemm(c, "gemm_qkv", q, s);
        if (st != DFLARE_OK) return st;
        // bidirectional attention over [context ; block] (Sec. 3.2)
        {
            Trace t(c, "attention", s);
            CUDA_TRY(launch_attention(c, i, s));
        }
        // X += O W_O
        GemmDesc o{};
        o.a = at(c->w.w_o, i * d * d_q, esz);
        o.b = c->attn;
        o.groups = 1;
        o.n = g.d;
        o.k = (int)d_q;
        o.m_tok = rows;
        o.b_group_rows = rows;
        o.ep = epi_base(c);
        o.ep.kind = EPI_RESID;
        o.ep.m_tok = rows;
        o.ep.n = g.d;
        o.ep.resid = c->x;
        o.ep.ld_resid = g.d;
        if ((st = traced_gemm(c, "gemm_o", o, s)) != DFLARE_OK) return st;
        // SwiGLU MLP: X += W_down (silu(X~ W_gate) * (X~ W_up))
        {
            Trace t(c, "rmsnorm", s);
            CUDA_TRY(launch_rmsnorm(c, at(c->w.mlp_norm, i * d, esz), rows, false, c->xn, s));
        }
        GemmDesc gu{};
        gu.a = at(c->w.w_gate, i * F * d, esz);
        gu.a2 = at(c->w.w_up, i * F * d, esz);
        gu.b = c->xn;
        gu.groups = 1;
        gu.n = g.ffn;
        gu.k = g.d;
        gu.m_tok = rows;
        gu.b_group_rows = rows;
        gu.ep = epi_base(c);
        gu.ep.kind = EPI_SWIGLU;
        gu.ep.m_tok = rows;
        gu.ep.n = g.ffn;
        gu.ep.out = c->act;
        gu.ep.ldo = g.ffn;
        if ((st = traced_gemm(c, "gemm_gate_up", gu, s)) != DFLARE_OK) return st;
        GemmDesc dn{};
        dn.a = at(c->w.w_down, i * d * F, esz);
        dn.b = c->act;
        dn.groups = 1;
        dn.n = g.d;
        dn.k = g.ffn;
        dn.m_tok = rows;
        dn.b_group_rows = rows;
        dn.ep = epi_base(c);
        dn.ep.kind = EPI_RESID;
        dn.ep.m_tok = rows;
        dn.ep.n = g.d;
        dn.ep.resid = c->x;
        dn.ep.ld_resid = g.d;
        if ((st = traced_gemm(c, "gemm_down", dn, s)) != DFLARE_OK) return st;
        if (hidden_out)
            CUDA_TRY(cudaMemcpyAsync(hidden_out + (size_t)(i + 1) * hid_stride, c->x, hid_stride * 4,
                                     cudaMemcpyDeviceToDevice, s));
    }
    if (g.block < 2) return DFLARE_OK;
    // final RMSNorm of the mask rows, LM head, greedy argmax (Sec. 3.2)
    const int mrows = c->batch * (g.block - 1);
    {
        Trace t(c, "rmsnorm", s);
        CUDA_TRY(launch_rmsnorm(c, c->w.final_norm, mrows, true, c->xh, s));
    }
    GemmDesc h{};
    h.a = c->w.lm_head;
    h.b = c->xh;
    h.groups = 1;
    h.n = g.vocab;
    h.k = g.d;
    h.m_tok = mrows;
    h.b_group_rows = mrows;
    h.ep = epi_base(c);
    h.ep.kind = EPI_F32;
    h.ep.m_tok = mrows;
    h.ep.n = g.vocab;
    h.ep.out = c->logits;
    h.ep.ldo = g.vocab;
    dflare_status st = traced_gemm(c, "gemm_lm_head", h, s);
    if (st != DFLARE_OK) return st;
    if (smp) {
        Trace t(c, "sample", s);
        CUDA_TRY(launch_sample(c, mrows, smp->inv_t, smp->seed, smp->step, draft_tokens, s));
    } else {
        Trace t(c, "argmax", s);
        CUDA_TRY(launch_argmax(c, c->logits, mrows, draft_tokens, s));
    }
    if (logits_out)
        CUDA_TRY(cudaMemcpyAsync(logits_out, c->logits, (size_t)mrows * g.vocab * 4,
                                 cudaMemcpyDeviceToDevice, s));
    return DFLARE_OK;
}

bool bad_temperature(float t) { return !(t > 0.f) || !std::isfinite(t) || !std::isfinite(1.0f / t); }

}  // namespace

extern "C" {

dflare_status dflare_draft_block(dflare_ctx* c, const int32_t* last_token, int32_t* draft_tokens,
                                 float* logits_out, float* hidden_out, void* stream) {
    if (!c) return fail(nullptr, DFLARE_EINVAL, "ctx is NULL");
    DeviceGuard dg(c->device);
    const uint64_t key[] = {(uint64_t)c->batch, (uint64_t)(uintptr_t)last_token,
                            (uint64_t)(uintptr_t)draft_tokens, (uint64_t)(uintptr_t)logits_out,
                            (uint64_t)(uintptr_t)hidden_out, (uint64_t)attention_launch_splits(c), 0, 0, 0, 0};
    return graphed(c, c->draft_graph, key, 10, static_cast<cudaStream_t>(stream), [&] {
        return draft_block_impl(c, last_token, draft_tokens, logits_out, hidden_out, stream, nullptr);
    });
}

dflare_status dflare_draft_block_sampled(dflare_ctx* c, const int32_t* last_token, float temperature,
                                         uint64_t seed, const uint64_t* step, int32_t* draft_tokens,
                                         float* logits_out, float* hidden_out, void* stream) {
    if (!c) return fail(nullptr, DFLARE_EINVAL, "ctx is NULL");
    DeviceGuard dg(c->device);
    if (bad_temperature(temperature)) return fail(c, DFLARE_EINVAL, "temperature must be finite and > 0");
    if (!step) return fail(c, DFLARE_EINVAL, "step is NULL");
    const Sampling smp{1.0f / temperature, seed, step};
    uint32_t tbits;
    memcpy(&tbits, &smp.inv_t, 4);
    const uint64_t key[] = {(uint64_t)c->batch, (uint64_t)(uintptr_t)last_token,
                            (uint64_t)(uintptr_t)draft_tokens, (uint64_t)(uintptr_t)logits_out,
                            (uint64_t)(uintptr_t)hidden_out, (uint64_t)attention_launch_splits(c),
                            1, seed, (uint64_t)tbits, (uint64_t)(uintptr_t)step};
    return graphed(c, c->draft_graph, key, 10, static_cast<cudaStream_t>(stream), [&] {
        return draft_block_impl(c, last_token, draft_tokens, logits_out, hidden_out, stream, &smp);
    });
}

dflare_status dflare_verify_accept(dflare_ctx* c, const int32_t* draft, const int32_t* target,
                                   int32_t* accept_len, int32_t* next_token, void* stream) {
    if (!c) return fail(nullptr, DFLARE_EINVAL, "ctx is NULL");
    DeviceGuard dg(c->device);
    if (!target || !accept_len || !next_token || (!draft && c->cfg.block > 1))
        return fail(c, DFLARE_EINVAL, "a verification buffer is NULL");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    Trace t(c, "verify", s);
    CUDA_TRY(launch_verify(c, draft, target, accept_len, next_token, s));
    return DFLARE_OK;
}

dflare_status dflare_verify_logits(dflare_ctx* c, const int32_t* draft, const float* target_logits,
                                   int32_t* accept_len, int32_t* next_token, void* stream) {
    if (!c) return fail(nullptr, DFLARE_EINVAL, "ctx is NULL");
    DeviceGuard dg(c->device);
    if (!target_logits || !accept_len || !next_token || (!draft && c->cfg.block > 1))
        return fail(c, DFLARE_EINVAL, "a verification buffer is NULL");
    if (reinterpret_cast<uintptr_t>(target_logits) % 16)
        return fail(c, DFLARE_EINVAL, "target_logits must be 16-byte aligned");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    {
        Trace t(c, "argmax_target", s);
        CUDA_TRY(launch_argmax(c, target_logits, c->batch * c->cfg.block, c->tgt_tok, s));
    }
    Trace t(c, "verify", s);
    CUDA_TRY(launch_verify(c, draft, c->tgt_tok, accept_len, next_token, s));
    return DFLARE_OK;
}

dflare_status dflare_verify_sampled(dflare_ctx* c, const int32_t* draft, const float* target_logits,
                                    float temperature, uint64_t seed, uint64_t* step,
                                    int32_t* accept_len, int32_t* next_token, void* stream) {
    if (!c) return fail(nullptr, DFLARE_EINVAL, "ctx is NULL");
    DeviceGuard dg(c->device);
    if (!target_logits || !accept_len || !next_token || !step || (!draft && c->cfg.block > 1))
        return fail(c, DFLARE_EINVAL, "a verification buffer is NULL");
    if (bad_temperature(temperature)) return fail(c, DFLARE_EINVAL, "temperature must be finite and > 0");
    if (reinterpret_cast<uintptr_t>(target_logits) % 16)
        return fail(c, DFLARE_EINVAL, "target_logits must be 16-byte aligned");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const float inv_t = 1.0f / temperature;
    {
        Trace t(c, "spec_stats", s);
        CUDA_TRY(launch_spec_stats(c, target_logits, inv_t, s));
    }
    {
        Trace t(c, "spec_accept", s);
        CUDA_TRY(launch_spec_accept(c, draft, target_logits, inv_t, seed, step, s));
    }
    Trace t(c, "spec_resample", s);
    CUDA_TRY(launch_spec_resample(c, target_logits, inv_t, seed, step, accept_len, next_token, s));
    return DFLARE_OK;
}

dflare_status dflare_read_kv(dflare_ctx* c, int layer, int seq, int pos0, int n, void* k_out,
                             void* v_out, void* stream) {
    if (!c) return fail(nullptr, DFLARE_EINVAL, "ctx is NULL");
    DeviceGuard dg(c->device);
    const dflare_config& g = c->cfg;
    if (layer < 0 || layer >= g.n_draft_layers || seq < 0 || seq >= g.max_batch || pos0 < 0 || n < 0 ||
        (long long)pos0 + n > g.max_ctx)
        return fail(c, DFLARE_EINVAL, "layer, seq or position range out of bounds");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const size_t hd = g.head_dim, esz = c->esz;
    for (int h = 0; h < g.n_kv_heads; ++h) {
        const size_t row0 = (((size_t)layer * g.max_batch + seq) * g.n_kv_heads + h) * g.max_ctx + pos0;
        if (k_out)
            CUDA_TRY(cudaMemcpy2DAsync(static_cast<uint8_t*>(k_out) + h * hd * esz, g.n_kv_heads * hd * esz,
                                       static_cast<uint8_t*>(c->kcache) + row0 * hd * esz, hd * esz,
                                       hd * esz, n, cudaMemcpyDeviceToDevice, s));
        if (v_out)
            CUDA_TRY(cudaMemcpy2DAsync(static_cast<uint8_t*>(v_out) + h * hd * esz, g.n_kv_heads * hd * esz,
                                       static_cast<uint8_t*>(c->vcache) + row0 * hd * esz, hd * esz,
                                       hd * esz, n, cudaMemcpyDeviceToDevice, s));
    }
    return DFLARE_OK;
}

dflare_status dflare_ctx_lens(dflare_ctx* c, int32_t* host, void* stream) {
    if (!c) return fail(nullptr, DFLARE_EINVAL, "ctx is NULL");
    DeviceGuard dg(c->device);
    if (!host) return fail(c, DFLARE_EINVAL, "ctx_len_host is NULL");
    CUDA_TRY(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)));
    CUDA_TRY(cudaMemcpy(host, c->ctx_len, c->batch * sizeof(int32_t), cudaMemcpyDeviceToHost));
    return DFLARE_OK;
}

dflare_status dflare_device_error(dflare_ctx* c, uint32_t* bits, void* stream) {
    if (!c) return fail(nullptr, DFLARE_EINVAL, "ctx is NULL");
    DeviceGuard dg(c->device);
    if (!bits) return fail(c, DFLARE_EINVAL, "bits_host is NULL");
    CUDA_TRY(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)));
    CUDA_TRY(cudaMemcpy(bits, c->err, sizeof(uint32_t), cudaMemcpyDeviceToHost));
    CUDA_TRY(cudaMemset(c->err, 0, sizeof(uint32_t)));
    return *bits ? DFLARE_EDEVICE : DFLARE_OK;
}

dflare_status dflare_set_trace(dflare_ctx* c, dflare_trace_fn fn, void* user) {
    if (!c) return fail(nullptr, DFLARE_EINVAL, "ctx is NULL");
    c->trace_fn = fn;
    c->trace_user = user;
    return DFLARE_OK;
}

dflare_status dflare_set_timing(dflare_ctx* c, unsigned long long* stamps, int slots) {
    if (!c) return fail(nullptr, DFLARE_EINVAL, "ctx is NULL");
    if (slots < 0) return fail(c, DFLARE_EINVAL, "slots < 0");
    c->t_stamps = slots > 0 ? stamps : nullptr;
    c->t_slots = c->t_stamps ? slots : 0;
    c->t_next = 0;
    return DFLARE_OK;
}

const char* dflare_last_error(const dflare_ctx* c) {
    return c ? c->msg.c_str() : g_create_error.c_str();
}

dflare_status dflare_synthetic_target(const int32_t* draft, const uint32_t* u, const int32_t* r,
                                      const int32_t* last, int n_steps, int32_t* step,
                                      uint32_t threshold, int batch, int block, int32_t* target,
                                      void* stream) {
    dflare_ctx* c = nullptr;
    // with B = 1 there are no drafts: draft_tokens, u and r are empty and may be NULL
    if (!last || !step || !target || ((!draft || !u || !r) && block > 1))
        return fail(nullptr, DFLARE_EINVAL, "a synthetic-target buffer is NULL");
    if (n_steps < 1 || batch < 1 || block < 1 || block > 32)
        return fail(nullptr, DFLARE_EINVAL, "n_steps, batch or block out of range");
    CUDA_TRY(launch_synthetic_target(draft, u, r, last, n_steps, step, threshold, batch, block,
                                     target, static_cast<cudaStream_t>(stream)));
    return DFLARE_OK;
}

}  // extern "C"
