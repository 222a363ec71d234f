// dflare_argmax_noalloc: greedy argmax over caller-provided fp32 logit rows that allocates
// nothing. Its scratch (one packed (value, index) slot per row and an arrival counter) is a
// file-scope __device__ array, so the call never asks the CUDA runtime or any library for
// memory. Callers that cannot allocate (a serving loop with a fixed memory budget that forbids
// allocation after start-up, code that must not trigger the implicit device synchronisation
// cudaMalloc/cudaFree can cause, an allocator-free embedding) can use it on their own logits,
// e.g. a target model's verification logits.
#include <math.h>

#include <mutex>
#include <string>

#include "common.cuh"
#include "internal.h"

// Scratch shared by every call on a device (DFLARE_NOALLOC_MAX_ROWS 8-byte slots and one counter,
// padded to 256 bytes); each call clears the part it uses before its kernel runs.
static __device__ __align__(256) unsigned long long g_noalloc_slot[DFLARE_NOALLOC_MAX_ROWS];
static __device__ __align__(256) unsigned int g_noalloc_count[64];

namespace dfl {
namespace {

struct Scratch {
    unsigned long long* slot = nullptr;
    unsigned int* count = nullptr;
};

// Device addresses of the two arrays, looked up once per device with that device current
// (in host code the symbols only name host-side stand-ins).
std::mutex g_mu;
Scratch g_scratch[64];

cudaError_t scratch_for_current_device(Scratch* out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_scratch[dev].slot) {
        Scratch s;
        e = cudaGetSymbolAddress(reinterpret_cast<void**>(&s.slot), g_noalloc_slot);
        if (e != cudaSuccess) return e;
        e = cudaGetSymbolAddress(reinterpret_cast<void**>(&s.count), g_noalloc_count);
        if (e != cudaSuccess) return e;
        g_scratch[dev] = s;
    }
    *out = g_scratch[dev];
    return cudaSuccess;
}

__device__ __forceinline__ uint32_t order_key(float v) {
    uint32_t u = __float_as_uint(v);
    if (v == 0.f) u = 0u;
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Grid (chunks, rows): each CTA reduces one vocabulary chunk of one row (lowest index among
// equal maxima) and folds (ordered value, ~index) into the row's slot with a 64-bit atomicMax;
// the last CTA to arrive writes the token ids. NaN entries are never chosen; a row with no value
// above -inf gets its first -inf entry (id 0 when every entry is NaN).
__global__ void __launch_bounds__(256) argmax_noalloc_kernel(const float* __restrict__ logits,
                                                             int V, int rows, int chunk,
                                                             unsigned long long* slot,
                                                             unsigned int* count,
                                                             int32_t* __restrict__ tokens) {
    __shared__ float sv[8];
    __shared__ int si[8];
    __shared__ int last;
    const int row = blockIdx.y;
    const int c0 = blockIdx.x * chunk, c1 = min(V, c0 + chunk);
    const float* p = logits + (size_t)row * V;
    float bv = -INFINITY;
    int bi = 0x7fffffff;
    for (int i = c0 + threadIdx.x; i < c1; i += blockDim.x) {
        const float q = p[i];
        if (q > bv) { bv = q; bi = i; }
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
        if (bi != 0x7fffffff)
            atomicMax(&slot[row], ((unsigned long long)order_key(bv) << 32) | (0xFFFFFFFFu - (uint32_t)bi));
        __threadfence();
        last = atomicAdd(count, 1u) == gridDim.x * gridDim.y - 1;
    }
    __syncthreads();
    if (last) {
        __threadfence();
        for (int r = threadIdx.x; r < rows; r += blockDim.x) {
            const unsigned long long key = atomicAdd(&slot[r], 0ull);
            int32_t tok = (int32_t)(0xFFFFFFFFu - (uint32_t)(key & 0xFFFFFFFFull));
            if (key == 0ull) {   // no entry above -inf: a serial scan, only for such rows
                const float* pr = logits + (size_t)r * V;
                tok = 0;
                for (int i = 0; i < V; ++i)
                    if (pr[i] == -INFINITY) { tok = i; break; }
            }
            tokens[r] = tok;
        }
    }
}

}  // namespace
}  // namespace dfl

extern "C" dflare_status dflare_argmax_noalloc(const float* logits_dev, int rows, int vocab,
                                               int32_t* tokens_dev, void* stream) {
    if (!logits_dev || !tokens_dev) {
        dfl::noalloc_set_error("dflare_argmax_noalloc: logits or tokens is NULL");
        return DFLARE_EINVAL;
    }
    if (rows < 1 || vocab < 1) {
        dfl::noalloc_set_error("dflare_argmax_noalloc: rows and vocab must be >= 1");
        return DFLARE_EINVAL;
    }
    if (rows > DFLARE_NOALLOC_MAX_ROWS) {
        dfl::noalloc_set_error("dflare_argmax_noalloc: rows exceeds DFLARE_NOALLOC_MAX_ROWS (" +
                               std::to_string(DFLARE_NOALLOC_MAX_ROWS) + ")");
        return DFLARE_ECAPACITY;
    }
    dfl::Scratch sc;
    cudaError_t e = dfl::scratch_for_current_device(&sc);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(sc.slot, 0, (size_t)rows * sizeof(unsigned long long), s);
    if (e == cudaSuccess) e = cudaMemsetAsync(sc.count, 0, sizeof(unsigned int), s);
    if (e == cudaSuccess) {
        int chunks = (vocab + 8191) / 8192;
        if (chunks < 1) chunks = 1;
        const int chunk = (vocab + chunks - 1) / chunks;
        dfl::argmax_noalloc_kernel<<<dim3(chunks, rows), 256, 0, s>>>(logits_dev, vocab, rows, chunk,
                                                                       sc.slot, sc.count, tokens_dev);
        e = cudaGetLastError();
    }
    if (e != cudaSuccess) {
        dfl::noalloc_set_error(std::string("dflare_argmax_noalloc: ") + cudaGetErrorString(e));
        return DFLARE_ECUDA;
    }
    return DFLARE_OK;
}
