// Host-side internals of libdflare: the context object and the kernel launchers.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>
#include <string>
#include <vector>

#include "dflare.h"

namespace dfl {

constexpr int kSpecMaxChunks = 64;   // vocabulary chunks per row of the sampled verification

// Epilogue kinds of the projection GEMMs (applied to a 128-feature x token tile in fp32).
enum EpiKind : int {
    EPI_STORE = 0,      // out[g][tok][n] = acc (+ bias[g][n])    (storage type)
    EPI_F32 = 1,        // out[tok][n] = acc                      (fp32: logits)
    EPI_RESID = 2,      // resid[tok][n] += acc                   (fp32 residual stream)
    EPI_QKV = 3,        // Q / K^d / V^d with rotary embedding on Q and K^d at the block positions
    EPI_KV_APPEND = 4,  // context K^t (rotated) / V^t appended to the layer's cache
    EPI_SWIGLU = 5,     // out[tok][n] = silu(gate) * up          (two accumulators)
    EPI_RED32 = 6       // out[tok][n] += acc with fp32 L2 reductions (every split adds its part)
};

struct EpiParams {
    int kind;
    int m_tok;             // valid token rows per group
    int n;                 // valid output features per group
    void* out;             // EPI_STORE / EPI_F32 / EPI_SWIGLU
    int ldo;
    float* resid;          // EPI_RESID
    int ld_resid;
    void* q;               // EPI_QKV outputs: [tok][d_q], [tok][d_kv], [tok][d_kv]
    void* kd;
    void* vd;
    int d_q, d_kv;
    const int32_t* ctx_len;  // EPI_QKV: block row k of sequence b sits at ctx_len[b] + k
    int block;
    void* kcache;          // EPI_KV_APPEND: [D][max_batch][H_kv][max_ctx][hd]
    void* vcache;
    const int32_t* app_base;  // first new position of each sequence
    const int32_t* app_cnt;   // rows appended per sequence
    int n_max;             // token row tok = b * n_max + r
    int max_ctx;
    int max_batch;
    int head_dim;
    const float* rope_cos;   // [positions][hd/2]
    const float* rope_sin;
    int rope;              // apply the rotary embedding (EPI_QKV)
    long long out_gstride; // EPI_STORE: elements between the groups' outputs
    const void* bias;      // EPI_STORE: optional [groups][n] storage-type bias added to acc
};

// One projection GEMM: out = epilogue(B x A^T) per group, where A holds `groups` stacked weight
// matrices [N][K] (row-major, out x in) and B holds the activations, m_tok valid rows per group
// with `b_group_rows` rows between groups.
struct GemmDesc {
    const void* a;
    const void* a2;        // second weight matrix for EPI_SWIGLU (up), else nullptr
    const void* b;
    int groups;
    int n, k, m_tok;
    long long b_group_rows;
    long long a_group_rows = 0;  // rows between weight groups (0 = n)
    int b_shared = 0;      // 1: every group reads the same activations (group 0 of b)
    int b_kgroup = 0;      // > 0 (groups == 1): b holds k / b_kgroup stacked [m_tok][b_kgroup]
                           // blocks, b_group_rows rows apart, and contraction index kk reads
                           // block kk / b_kgroup at column kk % b_kgroup
    EpiParams ep;
    int kbs = 0;           // tcgen05 GEMM: 64-wide k-blocks per pipeline stage (0 = default)
    int max_smem = 0;      // tcgen05 GEMM: shared-memory budget per CTA in bytes (0 = default)
    int evict_first = 0;   // tcgen05 GEMM: weights with an L2 evict-first policy (0 = yes, -1 = no)
    int force_splits = 0;  // tcgen05 GEMM: K splits (0 = chosen from the wave count)
};

}  // namespace dfl

// Calls of the library replayed as CUDA graphs (see graphed() in dflare_api.cu): a few operand
// sets per call type, least recently used first out (a caller that double-buffers its inputs
// alternates between two).
// Makes the context's device current for the duration of an API call and restores the caller's
// device afterwards (a process may drive contexts on several GPUs from one thread).
struct DeviceGuard {
    int prev = -1;
    explicit DeviceGuard(int dev) {
        int cur = -1;
        if (cudaGetDevice(&cur) == cudaSuccess && cur != dev && cudaSetDevice(dev) == cudaSuccess) prev = cur;
    }
    ~DeviceGuard() {
        if (prev >= 0) cudaSetDevice(prev);
    }
    DeviceGuard(const DeviceGuard&) = delete;
    DeviceGuard& operator=(const DeviceGuard&) = delete;
};

// cudaFuncSetAttribute acts on the current device only: a launcher runs its configuration once per
// device (devices are told apart modulo 64).
struct PerDeviceOnce {
    std::atomic<uint64_t> mask{0};
    template <class F>
    cudaError_t operator()(F&& configure) {
        int dev = 0;
        cudaError_t e = cudaGetDevice(&dev);
        if (e != cudaSuccess) return e;
        const uint64_t bit = 1ull << (dev & 63);
        if (mask.load(std::memory_order_acquire) & bit) return cudaSuccess;
        e = configure();
        if (e == cudaSuccess) mask.fetch_or(bit, std::memory_order_acq_rel);
        return e;
    }
};

struct GraphSlot {
    static constexpr int kKeyLen = 10;
    uint64_t key[kKeyLen] = {};
    bool seen = false;
    cudaGraphExec_t exec = nullptr;
    uint64_t used = 0;
};
struct CallGraph {
    static constexpr int kSlots = 4;
    GraphSlot slot[kSlots];
    uint64_t clock = 0;
};

struct dflare_ctx {
    dflare_config cfg;
    int device = 0;
    int num_sms = 0;
    int batch = 0;
    int ctx_ub = 0;            // host-side upper bound of every sequence's context length
    bool pdl = true;           // programmatic dependent launch between the library's kernels
    bool weights_set = false;
    dflare_weights w{};
    size_t esz = 2;            // bytes per storage element

    void* kcache = nullptr;    // [D][max_batch][H_kv][max_ctx][hd]
    void* vcache = nullptr;
    int32_t* ctx_len = nullptr;    // [max_batch]
    int32_t* app_base = nullptr;   // [max_batch]
    int32_t* app_cnt = nullptr;    // [max_batch]
    float* alpha = nullptr;        // [D][T]
    void* fused = nullptr;         // [D][max_fuse_rows][d]
    void* fused_fc = nullptr;      // [D][max_fuse_rows][d], DFLARE_FLAG_FUSION_FC only
    float* x = nullptr;            // [max_batch*B][d] residual stream
    void* xn = nullptr;            // [max_batch*B][d] normalised activations
    void* q = nullptr;             // [max_batch*B][d_q]
    void* kd = nullptr;            // [max_batch*B][d_kv]
    void* vd = nullptr;
    float* qkv32 = nullptr;        // [max_batch*B][d_q + 2 d_kv] fp32 sums of the Q/K^d/V^d splits (bf16 path)
    void* attn = nullptr;          // [max_batch*B][d_q]
    void* act = nullptr;           // [max_batch*B][F]
    void* xh = nullptr;            // [max_batch*(B-1)][d]
    float* logits = nullptr;       // [max_batch*(B-1)][V]
    float* attn_o = nullptr;       // split-KV partial outputs
    float* attn_ml = nullptr;      // split-KV partial (max, sum)
    int attn_splits = 1;
    // tensor maps of the bf16 attention: per layer K and V cache, then K^d and V^d (built on first use)
    std::vector<CUtensorMap> attn_maps;
    float* ws = nullptr;           // split-K workspace
    size_t ws_floats = 0;
    uint32_t* tile_cnt = nullptr;  // split-K arrival counters
    int tile_cnt_n = 0;
    unsigned long long* amax_slot = nullptr;  // packed (value, index) per logits row [max_batch*B]
    int32_t* tgt_tok = nullptr;    // [max_batch*B] target argmax of dflare_verify_logits
    float2* spec_part = nullptr;   // [max_batch*(2B-1)][kSpecMaxChunks] softmax partials (m, s)
    int spec_chunks = 1;           // vocabulary chunks of the current sampled verification
    int32_t* spec_a = nullptr;     // [max_batch] first rejected draft position
    uint32_t* amax_cnt = nullptr;
    float* rope_cos = nullptr;     // [max_ctx + B][hd/2]
    float* rope_sin = nullptr;
    uint32_t* err = nullptr;       // device error word
    CallGraph draft_graph, fuse_graph;   // graphs of repeated dflare_draft_block / _fuse_context calls
    dflare_trace_fn trace_fn = nullptr;
    void* trace_user = nullptr;
    unsigned long long* t_stamps = nullptr;   // GEMM and attention launch timing (dflare_set_timing)
    int t_slots = 0;
    int t_next = 0;
    std::string msg;
};

namespace dfl {

// Launch with cudaLaunchKernelEx; `pdl` adds programmatic stream serialisation, so the kernel may
// start while its predecessor drains (every kernel of the library calls griddepcontrol.wait
// before it touches memory a predecessor writes or reads).
template <typename... KArgs, typename... Args>
inline cudaError_t launch_kernel(bool pdl, void (*kernel)(KArgs...), dim3 grid, dim3 block,
                                 size_t smem, cudaStream_t s, Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// As launch_kernel, with thread-block clusters of `cluster_x` CTAs along x.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_cluster(bool pdl, int cluster_x, void (*kernel)(KArgs...), dim3 grid,
                                  dim3 block, size_t smem, cudaStream_t s, Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = cluster_x;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 2 : 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// Sets the message dflare_last_error(NULL) returns (for entry points without a context).
void noalloc_set_error(const std::string& message);

// launchers (each returns the first CUDA error it meets)
cudaError_t launch_gemm_tc(dflare_ctx* c, const GemmDesc& g, cudaStream_t s, std::string* why);
// the split count the next attention launch takes (the only launch parameter that depends on the
// host-side context-length bound)
int attention_launch_splits(const dflare_ctx* c);
// bf16 tensor map with a 128-byte swizzle and zero fill outside the tensor (dims innermost first;
// strides_bytes for dims 1..rank-1); false when the driver rejects it.
bool encode_tma_bf16(CUtensorMap* m, const void* base, int rank, const uint64_t* dims,
                     const uint64_t* strides_bytes, const uint32_t* box);
cudaError_t launch_gemm_simt(dflare_ctx* c, const GemmDesc& g, cudaStream_t s);
cudaError_t launch_fusion_alpha(dflare_ctx* c, cudaStream_t s);
cudaError_t launch_fuse_begin(dflare_ctx* c, const int32_t* n_new, int n_max, cudaStream_t s);
cudaError_t launch_fuse_layers(dflare_ctx* c, const void* hidden, int n_max, void* fused_out,
                               cudaStream_t s);
cudaError_t launch_embed(dflare_ctx* c, const int32_t* last_token, cudaStream_t s);
// zero32 (optional): the fp32 Q/K^d/V^d sums of the next projection, rows x (d_q + 2 d_kv), cleared
cudaError_t launch_rmsnorm(dflare_ctx* c, const void* gain, int rows, bool gather_mask_rows,
                           void* out, cudaStream_t s, float* zero32 = nullptr);
cudaError_t launch_attention(dflare_ctx* c, int layer, cudaStream_t s);
cudaError_t launch_argmax(dflare_ctx* c, const float* logits, int rows, int32_t* tokens,
                          cudaStream_t s);
cudaError_t launch_sample(dflare_ctx* c, int rows, float inv_t, uint64_t seed, const uint64_t* step,
                          int32_t* tokens, cudaStream_t s);
cudaError_t launch_spec_stats(dflare_ctx* c, const float* target_logits, float inv_t, cudaStream_t s);
cudaError_t launch_spec_accept(dflare_ctx* c, const int32_t* draft, const float* target_logits,
                               float inv_t, uint64_t seed, const uint64_t* step, cudaStream_t s);
cudaError_t launch_spec_resample(dflare_ctx* c, const float* target_logits, float inv_t,
                                 uint64_t seed, uint64_t* step, int32_t* accept_len,
                                 int32_t* next_token, cudaStream_t s);
cudaError_t launch_verify(dflare_ctx* c, const int32_t* draft, const int32_t* target,
                          int32_t* accept_len, int32_t* next_token, cudaStream_t s);
cudaError_t launch_synthetic_target(const int32_t* draft, const uint32_t* u, const int32_t* r,
                                    const int32_t* last, int n_steps, int32_t* step,
                                    uint32_t threshold, int batch, int block, int32_t* target,
                                    cudaStream_t s);

}  // namespace dfl
