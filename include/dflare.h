/*
 * dflare.h -- C ABI of a GB300 (sm_103a) library for the per-step draft path of DFlare,
 * block-diffusion speculative decoding with layer-wise target fusion (arxiv 2606.02091).
 *
 * One block step of the path is three calls, in this order:
 *   dflare_fuse_context   Eq. 3 (Sec. 4.1) layer-wise fusion of the target's hidden states at the
 *                         newly committed positions, then Eq. 4 (Sec. 4.2) projection of each
 *                         draft layer's fused context to keys/values, appended to that layer's
 *                         context KV cache.
 *   dflare_draft_block    Sec. 3.2 drafting phase: one forward pass over the block
 *                         [x_t ; B-1 mask positions] with bidirectional attention over
 *                         [context ; block] (keys/values per Eq. 4), RMSNorm, SwiGLU MLP, LM head
 *                         and greedy argmax at the B-1 mask positions.
 *   dflare_verify_accept  Sec. 3.2 verification phase: the acceptance length is the longest
 *                         prefix of drafts matching the target's own argmax, plus one, and the
 *                         target's extra token becomes the next x_t.
 *
 * Conventions shared by every call:
 * - Pointers named *_dev are device pointers, *_host host pointers. Device buffers passed in are
 *   borrowed: the caller owns them and keeps them valid until the stream has executed the call.
 * - `stream` is a cudaStream_t passed as void* (NULL = the legacy default stream). Every call is
 *   stream-ordered and asynchronous unless it says otherwise; none allocates memory except
 *   dflare_create (and the CUDA graphs below).
 * - dflare_fuse_context, dflare_draft_block and dflare_draft_block_sampled replay repeated calls
 *   as CUDA graphs: the second call with the same operands (context batch, buffer pointers,
 *   sampling parameters) on a non-legacy stream that is not being captured is captured and
 *   launched, later ones are replayed (host cost of a few microseconds). Results are those of the
 *   direct launches. dflare_set_weights discards the graphs.
 * - Errors: argument checks happen on the host before anything is enqueued and return a status
 *   at once. Errors found by kernels (a token id out of range, a context that would overflow)
 *   set bits of a device error word read by dflare_device_error. Asynchronous CUDA errors are
 *   reported as DFLARE_ECUDA by the next call that checks the stream. dflare_last_error returns
 *   a message for the last failing call on a context.
 * - Storage types: bf16 (default) or fp32 (dflare_config.dtype). "T" below is that type. Integer
 *   arrays are int32, row-major.
 * - One context serves one stream at a time; calls on one context must not overlap.
 * - Devices: a context lives on the device that was current at dflare_create. Every call on it
 *   makes that device current while it runs and restores the caller's device before returning,
 *   so one thread may drive contexts on several GPUs; `stream` must belong to that device.
 */
#ifndef DFLARE_H
#define DFLARE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    DFLARE_OK = 0,
    DFLARE_EINVAL = 1,      /* bad argument: null pointer, size out of range, bad config field */
    DFLARE_ECAPACITY = 2,   /* a size exceeds what the context was created for */
    DFLARE_ECUDA = 3,       /* a CUDA runtime or driver call failed */
    DFLARE_ESTATE = 4,      /* call out of order, e.g. drafting before dflare_set_weights */
    DFLARE_ENOMEM = 5,      /* device allocation failed (dflare_create only) */
    DFLARE_EDEVICE = 6      /* dflare_device_error found a kernel-reported error */
} dflare_status;

typedef enum { DFLARE_BF16 = 0, DFLARE_F32 = 1 } dflare_dtype;

/* dflare_config.flags */
#define DFLARE_FLAG_NO_BLOCK_ROPE 0x1u  /* no rotary embedding on the block's queries and keys
                                           (context keys keep theirs); used to test that the
                                           block is permutation-equivariant over mask rows */
#define DFLARE_FLAG_RAW_FUSION    0x2u  /* alpha = W^fuse without the softmax: the "-Softmax"
                                           ablation of Sec. 6.3 (Table 2) */
#define DFLARE_FLAG_SIMT_GEMM     0x4u  /* bf16 only: run the projections, MLP and LM head on the
                                           CUDA-core GEMM instead of the tcgen05 tensor-core
                                           GEMM (a diagnostic cross-check; fp32 always uses it) */
#define DFLARE_FLAG_SERIAL_LAUNCH 0x8u  /* launch every kernel fully serialised on its stream
                                           instead of with programmatic dependent launch (which
                                           lets a kernel's prologue and weight prefetch overlap the
                                           previous kernel's tail); for measurements */
#define DFLARE_FLAG_SHARED_KV     0x10u /* the "-KVProj" ablation of Sec. 6.3 (Table 2): context
                                           keys/values use the layer's own W_K^d / W_V^d (rows
                                           [d_q, d_q + 2 d_kv) of w_qkv) instead of W^t of Eq. 4;
                                           w_kv_ctx is not read and may be NULL */
#define DFLARE_FLAG_FUSION_FC     0x20u /* the "+FC" ablation of Sec. 6.3 (Table 2): one more
                                           fully-connected layer per draft layer after the fusion,
                                           F'^(i) = F^(i) W_fc^(i)T + b_fc^(i) (weights fusion_fc_w,
                                           fusion_fc_b), which then feeds Eq. 4 in place of F^(i) */
#define DFLARE_FLAG_DFLASH_FC     0x40u /* the DFlash baseline of Sec. 2.2-2.3: one context feature
                                           c_t = W_fc [h_t^(1); ...; h_t^(T)] + b_fc (Eq. 1) for
                                           every draft layer, projected by the layer's own W_K /
                                           W_V as in Eq. 2 (weights dflash_fc_w, dflash_fc_b);
                                           fuse_logits, fuse_norm and w_kv_ctx are not read and
                                           may be NULL. Cannot be combined with RAW_FUSION or
                                           FUSION_FC (DFLARE_EINVAL) */

#define DFLARE_FLAG_DETERMINISTIC 0x80u /* bitwise-reproducible runs: the split-K partial sums of
                                           the residual projections (W_O, W_down) are reduced in
                                           a fixed order by the last CTA of each tile. Without it
                                           every split adds its partial to the fp32 residual
                                           stream with L2 reductions, which is faster but leaves
                                           the order of those additions, and so the last bit of
                                           the residual, free to vary between runs (the
                                           verification decides every emitted token either way) */
#define DFLARE_FLAG_MMA_SYNC_ATTENTION 0x100u /* bf16 only: run the attention on the mma.sync
                                           (warp-level) tensor-core kernel, 64 query rows per CTA
                                           with P in registers, instead of the tcgen05 kernel
                                           (a cross-check and a measurement baseline) */

/* Device error word bits (dflare_device_error) */
#define DFLARE_DEVERR_TOKEN     0x1u    /* a token id outside [0, vocab) was read (clamped to 0) */
#define DFLARE_DEVERR_CAPACITY  0x2u    /* ctx_len + n_new > max_ctx, or n_new outside [0, n_max]:
                                           that sequence appended nothing */
#define DFLARE_DEVERR_TIMEOUT   0x4u    /* a pipeline wait inside a GEMM gave up (results invalid) */

typedef struct {
    int d;                /* hidden size; multiple of 64 */
    int n_draft_layers;   /* D, 1..16 */
    int n_target_layers;  /* T, 1..64: target layers fused by Eq. 3 */
    int n_q_heads;        /* query heads; a multiple of n_kv_heads */
    int n_kv_heads;       /* key/value heads */
    int head_dim;         /* 64 or 128; n_q_heads*head_dim and n_kv_heads*head_dim multiples of 128 */
    int ffn;              /* SwiGLU width; multiple of 64 */
    int vocab;            /* V >= 2 */
    int block;            /* B, 1..32: x_t plus B-1 mask positions */
    int max_batch;        /* sequences per call, 1..64 */
    int max_ctx;          /* context capacity per sequence (positions) */
    int max_fuse_rows;    /* largest batch * n_max of one dflare_fuse_context call */
    int mask_token_id;    /* token id of the mask positions, in [0, vocab) */
    float rms_eps;        /* epsilon of every RMSNorm */
    float rope_theta;     /* rotary base */
    int dtype;            /* dflare_dtype */
    unsigned flags;       /* DFLARE_FLAG_* */
} dflare_config;

/*
 * Draft weights (device pointers, borrowed until dflare_destroy or the next dflare_set_weights).
 * Linear maps are row-major [out_features][in_features]; per-layer tensors are stacked over the
 * D draft layers. Sizes use d_q = n_q_heads*head_dim, d_kv = n_kv_heads*head_dim, F = ffn.
 * Every pointer must be 16-byte aligned.
 */
typedef struct {
    const float* fuse_logits;  /* [D][T] fp32: W^fuse of Eq. 3 (alpha = softmax of each row) */
    const void* fuse_norm;     /* [D][d] T: gain of the RMSNorm in Eq. 3, per draft layer */
    const void* w_kv_ctx;      /* [D][2*d_kv][d] T: rows [0,d_kv) W_K^t, rows [d_kv,2d_kv) W_V^t (Eq. 4) */
    const void* attn_norm;     /* [D][d] T: pre-attention RMSNorm gain */
    const void* w_qkv;         /* [D][d_q+2*d_kv][d] T: rows W_Q, then W_K^d, then W_V^d (Eq. 4) */
    const void* w_o;           /* [D][d][d_q] T: attention output projection */
    const void* mlp_norm;      /* [D][d] T: pre-MLP RMSNorm gain */
    const void* w_gate;        /* [D][F][d] T */
    const void* w_up;          /* [D][F][d] T */
    const void* w_down;        /* [D][d][F] T */
    const void* final_norm;    /* [d] T: RMSNorm before the LM head */
    const void* embed;         /* [V][d] T: token embedding shared with the target (Sec. 3.3) */
    const void* lm_head;       /* [V][d] T: LM head shared with the target (Sec. 3.3) */
    /* read only under the flag named; NULL otherwise */
    const void* fusion_fc_w;   /* [D][d][d] T: DFLARE_FLAG_FUSION_FC, per-layer FC after Eq. 3 */
    const void* fusion_fc_b;   /* [D][d] T: DFLARE_FLAG_FUSION_FC, its bias */
    const void* dflash_fc_w;   /* [d][T*d] T: DFLARE_FLAG_DFLASH_FC, W_fc of Eq. 1 (column j*d+e
                                  multiplies element e of target layer j's state) */
    const void* dflash_fc_b;   /* [d] T: DFLARE_FLAG_DFLASH_FC, b_fc of Eq. 1 */
} dflare_weights;

typedef struct dflare_ctx dflare_ctx;

/* Validate `cfg` (host only: returns DFLARE_EINVAL without touching the GPU when a field is out
 * of range), then allocate the context on the current device: the per-layer context KV caches
 * (2 * D * max_batch * max_ctx * d_kv elements of T), activation buffers sized for max_batch and
 * max_fuse_rows, and a rotary table. On success *out owns all of it until dflare_destroy. */
dflare_status dflare_create(const dflare_config* cfg, dflare_ctx** out);

/* Free everything dflare_create allocated (synchronises the device first). NULL is a no-op. */
dflare_status dflare_destroy(dflare_ctx* ctx);

/* Borrow the draft weights and precompute alpha^(i) = softmax(W^fuse_{i,:}) once (Eq. 3; Sec. 4.1
 * notes the weights can be cached after training). Enqueued on `stream`. */
dflare_status dflare_set_weights(dflare_ctx* ctx, const dflare_weights* w, void* stream);

/* Start `batch` (1..max_batch) empty sequences: every context length becomes 0. */
dflare_status dflare_reset(dflare_ctx* ctx, int batch, void* stream);

/*
 * Fuse and append newly committed context positions (Eq. 3, Eq. 4; Sec. 3.2 "target context
 * tokens" injected into every draft layer's KV cache).
 *   target_hidden_dev  [T][batch][n_max][d] T: hidden states h^(j) of the T fused target layers
 *                      at the new positions of each sequence, layer-major as a target emits them;
 *                      rows r >= n_new[b] are ignored.
 *   n_new_dev          [batch] int32: positions to append per sequence, each in [0, n_max]
 *                      (typically the previous step's accept_len, or the prompt length first).
 *   n_max              row stride of target_hidden; batch * n_max <= max_fuse_rows.
 *   fused_out_dev      optional [D][batch][n_max][d] T: the context representation each layer
 *                      projects: f^(i) of Eq. 3 (with DFLARE_FLAG_FUSION_FC: the FC's output
 *                      F'^(i)); with DFLARE_FLAG_DFLASH_FC only slot 0 is written, with c_t of
 *                      Eq. 1, which every layer shares. Rows r >= n_new[b] are unspecified.
 * Sequence b's new rows get positions ctx_len[b] .. ctx_len[b]+n_new[b]-1; keys are rotated at
 * those positions and cached; ctx_len[b] grows by n_new[b]. A sequence that would exceed max_ctx
 * appends nothing and sets DFLARE_DEVERR_CAPACITY.
 */
dflare_status dflare_fuse_context(dflare_ctx* ctx, const void* target_hidden_dev,
                                  const int32_t* n_new_dev, int n_max, void* fused_out_dev,
                                  void* stream);

/*
 * Draft one block per sequence (Sec. 3.2, drafting phase, with Eq. 4's keys/values).
 *   last_token_dev    [batch] int32: the target decode token x_t of each sequence, at position
 *                     ctx_len[b]; the B-1 mask positions follow at ctx_len[b]+1 ..
 *   draft_tokens_dev  [batch][B-1] int32 out: greedy argmax at each mask position (ties -> lowest id);
 *                     may be NULL when B = 1 (no mask positions, nothing is drafted).
 *   logits_out_dev    optional [batch][B-1][V] fp32 out: the LM-head logits at the mask positions.
 *   hidden_out_dev    optional [D+1][batch][B][d] fp32 out: the block rows after the embedding and
 *                     after every draft layer (the residual stream, kept in fp32).
 * Needs dflare_set_weights; every sequence needs ctx_len >= 0 (an empty context is allowed).
 */
dflare_status dflare_draft_block(dflare_ctx* ctx, const int32_t* last_token_dev,
                                 int32_t* draft_tokens_dev, float* logits_out_dev,
                                 float* hidden_out_dev, void* stream);

/*
 * Prefix acceptance (Sec. 3.2, verification phase).
 *   draft_tokens_dev   [batch][B-1] int32: d_1 .. d_{B-1}.
 *   target_argmax_dev  [batch][B] int32: g_0 .. g_{B-1}, the target's argmax after block rows
 *                      0 .. B-1 (g_{k-1} checks d_k).
 *   accept_len_dev     [batch] int32 out: tau = a + 1 in [1, B], a = longest prefix with
 *                      d_k == g_{k-1} for all k <= a.
 *   next_token_dev     [batch] int32 out: g_a, the target's extra token (the next x_t).
 * The caller then fuses the tau committed positions' target states with dflare_fuse_context
 * (n_new = accept_len).
 */
dflare_status dflare_verify_accept(dflare_ctx* ctx, const int32_t* draft_tokens_dev,
                                   const int32_t* target_argmax_dev, int32_t* accept_len_dev,
                                   int32_t* next_token_dev, void* stream);

/*
 * Prefix acceptance from the target's logits (Sec. 3.2, verification phase, with the target's
 * greedy predictions taken here): g_k = argmax_v target_logits[b][k][v] (lowest id among equal
 * maxima; NaN entries are never chosen, a row of NaN gives id 0), then exactly
 * dflare_verify_accept on g.
 *   draft_tokens_dev     [batch][B-1] int32: d_1 .. d_{B-1}.
 *   target_logits_dev    [batch][B][V] fp32, 16-byte aligned: the target's logits after block
 *                        rows 0 .. B-1 (row k predicts position t+k+1).
 *   accept_len_dev, next_token_dev  as in dflare_verify_accept.
 * Uses the context's own scratch, so calls on one context must be stream-ordered.
 */
dflare_status dflare_verify_logits(dflare_ctx* ctx, const int32_t* draft_tokens_dev,
                                   const float* target_logits_dev, int32_t* accept_len_dev,
                                   int32_t* next_token_dev, void* stream);

/*
 * Sampled decoding at temperature T (Table 1's temperature-1 rows). The paper does not state its
 * acceptance rule for sampling; these calls use the speculative-sampling rule of the works it
 * builds on. Random numbers are Philox4x64-10 streams (Salmon et al., SC'11): element v of
 * stream (purpose, step, row) comes from word x = word (v/2) mod 4 of the block at counter
 * (1 + v/8, row, step, purpose), key (seed, 0): ((x >> 41) + 1/2) * 2^-23 for even v,
 * (((x >> 9) & 0x7FFFFF) + 1/2) * 2^-23 for odd v. Purposes: 1 draft draws (row =
 * b*(B-1) + k-1, v = token id), 2 acceptance draws (row = b, v = k-1), 3 replacement draws
 * (row = b, v = token id). `step_dev` is a uint64 device counter read by both calls;
 * dflare_verify_sampled adds 1 to it when it finishes, so a captured draft-verify graph draws
 * fresh numbers on every replay.
 *
 * dflare_draft_block_sampled: dflare_draft_block with d_k drawn from softmax(logits_k / T)
 * (Gumbel-max: argmax_v l_v / T - log(-log u_v), lowest id among equal scores) instead of the
 * argmax. temperature must be finite and > 0 (DFLARE_EINVAL otherwise).
 */
dflare_status dflare_draft_block_sampled(dflare_ctx* ctx, const int32_t* last_token_dev,
                                         float temperature, uint64_t seed,
                                         const uint64_t* step_dev, int32_t* draft_tokens_dev,
                                         float* logits_out_dev, float* hidden_out_dev,
                                         void* stream);

/*
 * dflare_verify_sampled: speculative-sampling verification of the block the last
 * dflare_draft_block[_sampled] on this context drafted (its logits are kept in the context).
 * With p_k = softmax(target_logits[b][k-1] / T) and q_k = softmax(draft logits of d_k / T),
 * d_k is kept when r_k * q_k(d_k) < p_k(d_k) (r_k the acceptance draw); a = the number of kept
 * drafts before the first rejection; accept_len = a + 1. next_token is drawn from
 * max(0, p_{a+1} - q_{a+1}) when a < B-1 (from p_{a+1} if that vanishes everywhere), else from
 * softmax(target_logits[b][B-1] / T).
 *   draft_tokens_dev   [batch][B-1] int32 (an id outside [0, V) is rejected and sets
 *                      DFLARE_DEVERR_TOKEN).
 *   target_logits_dev  [batch][B][V] fp32, 16-byte aligned.
 *   step_dev           the counter described above (incremented on the device).
 */
dflare_status dflare_verify_sampled(dflare_ctx* ctx, const int32_t* draft_tokens_dev,
                                    const float* target_logits_dev, float temperature,
                                    uint64_t seed, uint64_t* step_dev, int32_t* accept_len_dev,
                                    int32_t* next_token_dev, void* stream);

/* Copy n cached context rows [pos0, pos0+n) of draft layer `layer`, sequence `seq`, into
 * k_out_dev / v_out_dev, each [n][n_kv_heads][head_dim] T (keys already rotated). Either output
 * may be NULL. Rows past the current context hold stale data. */
dflare_status dflare_read_kv(dflare_ctx* ctx, int layer, int seq, int pos0, int n,
                             void* k_out_dev, void* v_out_dev, void* stream);

/* Synchronous: wait for `stream`, then copy the `batch` current context lengths to ctx_len_host. */
dflare_status dflare_ctx_lens(dflare_ctx* ctx, int32_t* ctx_len_host, void* stream);

/* Synchronous: wait for `stream`, copy the device error word (DFLARE_DEVERR_* bits) to
 * *bits_host and clear it. Returns DFLARE_EDEVICE when a bit was set, else DFLARE_OK. */
dflare_status dflare_device_error(dflare_ctx* ctx, uint32_t* bits_host, void* stream);

/* Optional tracing. When set, fn(user, name, phase, stream) is called on the host right before
 * (phase 0) and right after (phase 1) the library enqueues each of its kernel launches on
 * `stream` (name: "fuse_begin", "fuse_layers", "gemm_fusion_fc", "gemm_dflash_fc",
 * "gemm_kv_ctx", "embed", "rmsnorm", "gemm_qkv",
 * "attention", "gemm_o", "gemm_gate_up", "gemm_down", "gemm_lm_head", "argmax", "sample",
 * "argmax_target", "verify", "spec_stats", "spec_accept", "spec_resample").
 * A caller can record CUDA events there, also while the stream is being captured into a graph.
 * fn = NULL turns tracing off. */
typedef void (*dflare_trace_fn)(void* user, const char* name, int phase, void* stream);
dflare_status dflare_set_trace(dflare_ctx* ctx, dflare_trace_fn fn, void* user);

/* Optional device-side timing of the projection GEMM launches (the tcgen05 kernel behind every
 * "gemm_*" trace name) and of the bf16 attention launches ("attention"). stamps_dev: caller-owned device array of 3 * slots uint64, laid out as
 * [0, slots) first-CTA entry times, [slots, 2 slots) times at which the first CTA's dependency
 * on the previous kernel was met, [2 slots, 3 slots) last-CTA exit times, all in %globaltimer
 * nanoseconds. After this call, timed launch number k (GEMM and attention launches in issue
 * order, counted from this call, k < slots) folds its CTAs' times into slot k with atomicMin (entry, dependency) and atomicMax
 * (exit); later launches are not timed. The caller sets the first two ranges to all-ones and the
 * third to zero before the launches it reads, and may capture the launches into a CUDA graph
 * (the slot numbers are fixed at capture). Adds two global atomics per CTA while enabled.
 * stamps_dev = NULL (or slots = 0) turns timing off. Calls made with timing on launch directly
 * (they are not replayed from the library's own graphs). */
dflare_status dflare_set_timing(dflare_ctx* ctx, unsigned long long* stamps_dev, int slots);

/* Message of the last failing call on ctx (or of the last failing dflare_create when ctx is
 * NULL). Never NULL; valid until the next call on the same context. */
const char* dflare_last_error(const dflare_ctx* ctx);

/*
 * Not part of the method: a stand-in for the target model's verification argmax, used by the
 * benchmark loop and tests so a whole step stays on the device. For each sequence b and
 * k = 1..B-1, with step s = *step_dev % n_steps:
 *   g[b][k-1] = d[b][k-1]                       if u[s][b][k-1] < threshold (uint32 compare)
 *             = r[s][b][k-1] + (r >= d[b][k-1]) otherwise (a uniform token other than d_k),
 *   g[b][B-1] = last[s][b];
 * then *step_dev += 1. Tables: u [n_steps][batch][B-1] uint32, r [n_steps][batch][B-1] int32 in
 * [0, V-1), last [n_steps][batch] int32. threshold = floor(p * 2^32) for match probability p.
 * With B = 1 the draft, u and r tables are empty and may be NULL.
 */
dflare_status dflare_synthetic_target(const int32_t* draft_tokens_dev, const uint32_t* u_dev,
                                      const int32_t* r_dev, const int32_t* last_dev, int n_steps,
                                      int32_t* step_dev, uint32_t threshold, int batch, int block,
                                      int32_t* target_argmax_dev, void* stream);

/* Largest number of rows dflare_argmax_noalloc accepts. */
#define DFLARE_NOALLOC_MAX_ROWS 4096

/*
 * Greedy argmax over rows of fp32 logits that allocates nothing (the paper has no counterpart:
 * this is a library utility, with the same tie rule as the drafted tokens -- the lowest token id
 * among equal maxima).
 *   logits_dev  [rows][vocab] fp32 (caller-owned, device)
 *   tokens_dev  [rows] int32 out (caller-owned, device)
 * It is for callers that cannot allocate device memory: serving loops that fix their memory
 * budget at start-up and forbid allocation afterwards, code that must avoid the implicit
 * device synchronisation of cudaMalloc/cudaFree, or allocator-free embeddings. The call uses a
 * fixed scratch array compiled into the library (one 8-byte slot per row plus a counter,
 * DFLARE_NOALLOC_MAX_ROWS rows, held by every GPU that loads the library until the process
 * exits); it calls no cudaMalloc, cudaFree or allocating library routine.
 * - rows > DFLARE_NOALLOC_MAX_ROWS returns DFLARE_ECAPACITY (message in dflare_last_error(NULL)).
 * - A call made outside stream capture looks up the scratch array's device address (and the
 *   SM count) with the calling thread's current device; a call made while `stream` is being
 *   captured uses the values of the last call outside capture on that device. So make the first
 *   call on a device before capturing a stream into a CUDA graph (a first call inside a capture
 *   returns DFLARE_ECUDA), and after cudaDeviceReset make one call outside capture before
 *   capturing again: the reset invalidates the address held for capture.
 * - Every call on a device shares the same scratch array, which keeps the last call's contents;
 *   each call clears the part it uses on `stream` before its kernel. Calls that overlap on the
 *   GPU (on different streams, or from several host threads) race on the scratch and give wrong
 *   tokens: serialise them.
 */
dflare_status dflare_argmax_noalloc(const float* logits_dev, int rows, int vocab,
                                    int32_t* tokens_dev, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* DFLARE_H */
