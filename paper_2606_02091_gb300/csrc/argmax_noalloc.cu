// dflare_argmax_noalloc: greedy argmax over caller-provided fp32 logit rows that allocates
// nothing. Its scratch (one packed (value, index) slot per row and an arrival counter) is a
// file-scope __device__ array, so the call never asks the CUDA runtime or any library for
// memory. Callers that cannot allocate (a serving loop with a fixed memory budget that forbids
// allocation after start-up, code that must not trigger the implicit device synchronisation
// cudaMalloc/cudaFree can cause, an allocator-free embedding) can use it on their own logits,
// e.g. a target model's verification logits.
#include <math.h>

#include <algorithm>
#include <cstdint>
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
    int num_sms = 0;
};

// Device addresses of the two arrays (in host code the symbols only name host-side stand-ins)
// and the SM count, per device. A call made outside stream capture looks them up again with the
// device current (cheap), so a context rebuilt after cudaDeviceReset gets the new addresses; a
// call made during capture uses the values of the last call outside capture on that device.
std::mutex g_mu;
Scratch g_scratch[64];

cudaError_t scratch_for_current_device(cudaStream_t stream, Scratch* out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    e = cudaStreamIsCapturing(stream, &cs);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lk(g_mu);
    if (cs == cudaStreamCaptureStatusNone) {
        Scratch s;
        e = cudaGetSymbolAddress(reinterpret_cast<void**>(&s.slot), g_noalloc_slot);
        if (e != cudaSuccess) return e;
        e = cudaGetSymbolAddress(reinterpret_cast<void**>(&s.count), g_noalloc_count);
        if (e != cudaSuccess) return e;
        e = cudaDeviceGetAttribute(&s.num_sms, cudaDevAttrMultiProcessorCount, dev);
        if (e != cudaSuccess) return e;
        g_scratch[dev] = s;
    } else if (!g_scratch[dev].slot) {
        return cudaErrorStreamCaptureUnsupported;   // first call on this device inside a capture
    }
    *out = g_scratch[dev];
    return cudaSuccess;
}

__device__ __forceinline__ uint32_t order_key(float v) {
    uint32_t u = __float_as_uint(v);
    if (v == 0.f) u = 0u;
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__device__ __forceinline__ void take(float q, int i, float& bv, int& bi) {
    if (q > bv) { bv = q; bi = i; }   // NaN never compares greater; equal values keep the lower id
}

// Grid (chunks, rows): each CTA reduces one vocabulary chunk of one row (lowest index among
// equal maxima) and folds (ordered value, ~index) into the row's slot with a 64-bit atomicMax;
// the last CTA to arrive writes the token ids. With vec4 (rows 16-byte aligned, chunk a multiple
// of 4) every thread keeps four 16-byte loads in flight. NaN entries are never chosen; a row
// with no value above -inf gets its first -inf entry (id 0 when every entry is NaN).
__global__ void __launch_bounds__(256) argmax_noalloc_kernel(const float* __restrict__ logits,
                                                             int V, int rows, int chunk, int vec4,
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
    if (vec4) {
        const float4* p4 = reinterpret_cast<const float4*>(p);
        const int q0 = c0 >> 2, q1 = c1 >> 2;   // whole float4 groups; V % 4 == 0 here
        for (int q = q0 + threadIdx.x; q < q1; q += 4 * blockDim.x) {
            float4 f[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int qq = q + j * blockDim.x;
                f[j] = qq < q1 ? __ldg(p4 + qq) : make_float4(NAN, NAN, NAN, NAN);
            }
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int i = 4 * (q + j * blockDim.x);
                take(f[j].x, i, bv, bi);
                take(f[j].y, i + 1, bv, bi);
                take(f[j].z, i + 2, bv, bi);
                take(f[j].w, i + 3, bv, bi);
            }
        }
    } else {
        for (int i = c0 + threadIdx.x; i < c1; i += blockDim.x) take(p[i], i, bv, bi);
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
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = dfl::scratch_for_current_device(s, &sc);
    if (e == cudaSuccess) e = cudaMemsetAsync(sc.slot, 0, (size_t)rows * sizeof(unsigned long long), s);
    if (e == cudaSuccess) e = cudaMemsetAsync(sc.count, 0, sizeof(unsigned int), s);
    if (e == cudaSuccess) {
        // about four CTAs of 256 threads per SM over all rows, at least 1024 logits per CTA
        const int target = 4 * (sc.num_sms > 0 ? sc.num_sms : 1);
        int chunks = (target + rows - 1) / rows;
        chunks = std::max(1, std::min(chunks, (vocab + 1023) / 1024));
        const bool vec4 = vocab % 4 == 0 && (reinterpret_cast<uintptr_t>(logits_dev) & 15u) == 0;
        int chunk = (vocab + chunks - 1) / chunks;
        if (vec4) chunk = (chunk + 3) & ~3;
        chunks = (vocab + chunk - 1) / chunk;
        dfl::argmax_noalloc_kernel<<<dim3(chunks, rows), 256, 0, s>>>(logits_dev, vocab, rows, chunk,
                                                                       vec4 ? 1 : 0, sc.slot, sc.count,
                                                                       tokens_dev);
        e = cudaGetLastError();
    }
    if (e != cudaSuccess) {
        dfl::noalloc_set_error(std::string("dflare_argmax_noalloc: ") + cudaGetErrorString(e));
        return DFLARE_ECUDA;
    }
    return DFLARE_OK;
}
