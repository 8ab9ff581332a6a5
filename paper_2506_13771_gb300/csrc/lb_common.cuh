// lb_common.cuh -- device-side types and primitives shared by the LittleBit
// kernels (sm_103a).  Internal to liblittlebit.so.
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "littlebit.h"

namespace lb {

constexpr int kMaxRank = 1024;
constexpr unsigned long long kWaitLimitNs = 1000000000ull;  // 1 s per grid-wide wait

// Workspace header (first 256 bytes of every workspace).
//   word 0    : sticky error word (an lb_status once a kernel failed); cleared
//               only by littlebit_poll_error
//   word 1    : grid-barrier arrival counter
//   word 2    : count of CTAs that finished a stack launch
//   word 3    : launch epoch of the single-token kernel (selects which of its
//               two exchange-word buffers a launch uses)
//   words 4-5 : 64-bit fingerprint of the linears a stack workspace was
//               prepared for (littlebit_stack_prepare)
constexpr size_t kWsHeader = 256;
constexpr int kErrWord = 0;
constexpr int kCounterWord = 1;
constexpr int kDoneWord = 2;
constexpr int kEpochWord = 3;  // launches of the single-token kernel on this workspace
constexpr int kPlanWord = 4;

#ifndef LB_S1_WORDS
#define LB_S1_WORDS 1
#endif
// Stage 1 of the single-token kernels (k_decode, k_decode_multi) runs on the
// first s1_ctas(W, N) CTAs of the grid, at least kS1Words of the W input
// words each, the others holding none; an exchange element takes one
// contribution per stage-1 CTA.  (Concentrating stage 1 on fewer CTAs cuts
// the exchange's atomics but lengthens those CTAs' share of the ±1 sums:
// 2 words per CTA measured slower than 1 on the 4096 x 11008 r512 shape.)
constexpr int kS1Words = LB_S1_WORDS;
__host__ __device__ inline int s1_ctas(int W, int N) {
    const int n = (W + kS1Words - 1) / kS1Words;
    return n < 1 ? 1 : (n > N ? N : n);
}
// Input words [w0, w0 + nw) of CTA c.
__host__ __device__ inline void s1_slice(int W, int N, int c, int &w0, int &nw) {
    const int n = s1_ctas(W, N);
    if (c >= n) {
        w0 = 0;
        nw = 0;
        return;
    }
    w0 = (int)((long long)c * W / n);
    nw = (int)((long long)(c + 1) * W / n) - w0;
}

// Device copy of one linear (paths 0..n_paths-1).
struct LinDesc {
    int d_in, d_out, n_paths, r[2];
    const uint32_t *v[2];
    const uint32_t *u[2];
    const uint16_t *g[2];
    const uint16_t *l[2];
    const uint16_t *h[2];
};

__host__ inline LinDesc make_desc(const lb_linear &L) {
    LinDesc d{};
    d.d_in = L.d_in;
    d.d_out = L.d_out;
    d.n_paths = L.n_paths;
    for (int p = 0; p < L.n_paths; ++p) {
        d.r[p] = L.path[p].r;
        d.v[p] = L.path[p].v_bits;
        d.u[p] = L.path[p].u_bits;
        d.g[p] = L.path[p].g;
        d.l[p] = L.path[p].l;
        d.h[p] = L.path[p].h;
    }
    return d;
}

// ---------------------------------------------------------------- numbers

__device__ __forceinline__ float half_bits_to_float(uint16_t b) {
    return __half2float(__ushort_as_half(b));
}

__device__ __forceinline__ float bf16_bits_to_float(uint16_t b) {
    return __uint_as_float(static_cast<uint32_t>(b) << 16);
}

// fp32 -> bf16 bits, round to nearest even (finite inputs).
__device__ __forceinline__ uint16_t float_to_bf16_bits(float f) {
    return __bfloat16_as_ushort(__float2bfloat16_rn(f));
}

// x with its sign flipped when bit k of word is set (the +-1 product of Eq. 2).
__device__ __forceinline__ float apply_sign(float x, uint32_t word, int k) {
    return __uint_as_float(__float_as_uint(x) ^ ((word >> k) << 31));
}

// ---------------------------------------------------------------- memory ordering

__device__ __forceinline__ unsigned ld_acquire_gpu(const unsigned *p) {
    unsigned v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ unsigned ld_relaxed_gpu(const unsigned *p) {
    unsigned v;
    asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ void red_release_gpu_add(unsigned *p, unsigned v) {
    asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ void red_add_f32(float *p, float v) {
    asm volatile("red.global.add.f32 [%0], %1;" ::"l"(p), "f"(v) : "memory");
}

__device__ __forceinline__ unsigned long long globaltimer_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Grid-wide barrier over a monotonic arrival counter: every CTA adds one
// arrival per barrier; barrier number b (0-based) completes when the counter
// reaches n_ctas * (b + 1).  Writes made by the CTA before the call (including
// red.add reductions) are visible to every CTA after it.  The wait is bounded:
// after kWaitLimitNs, or once another CTA has recorded an error, the CTA
// records LB_ERR_TIMEOUT (first writer wins) and the call returns false; the
// caller must then return from the kernel.
__device__ __forceinline__ bool grid_barrier(unsigned *ws_words, unsigned target) {
    __shared__ int s_ok;
    __syncthreads();
    if (threadIdx.x == 0) {
        unsigned *counter = ws_words + kCounterWord;
        unsigned *err = ws_words + kErrWord;
        __threadfence();
        red_release_gpu_add(counter, 1u);
        int ok = 1;
        unsigned long long t0 = globaltimer_ns();
        while (ld_acquire_gpu(counter) < target) {
            if (ld_relaxed_gpu(err) != 0u) {
                ok = 0;
                break;
            }
            if (globaltimer_ns() - t0 > kWaitLimitNs) {
                atomicCAS(err, 0u, static_cast<unsigned>(LB_ERR_TIMEOUT));
                ok = 0;
                break;
            }
        }
        s_ok = ok;
    }
    __syncthreads();
    return s_ok != 0;
}

// Sum of v over the block, returned to every thread (blockDim.x <= 1024).
__device__ __forceinline__ float block_sum(float v) {
    __shared__ float s_part[32];
    __shared__ float s_total;
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) s_part[warp] = v;
    __syncthreads();
    if (warp == 0) {
        const int nw = (blockDim.x + 31) >> 5;
        float s = lane < nw ? s_part[lane] : 0.f;
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        if (lane == 0) s_total = s;
    }
    __syncthreads();
    const float total = s_total;
    __syncthreads();
    return total;
}

}  // namespace lb
