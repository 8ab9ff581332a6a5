// lb_pack.cu -- Eq. 2 sign packing on the device: +-1 int8 -> uint32 words,
// 32 signs per word along the reduction dimension, bit = 1 <=> -1, LSB first.
#include "lb_common.cuh"
#include "lb_kernels.h"

namespace lb {

namespace {

// One thread per output word.
//   U layout: word (o, w) holds signs[o][32w + k], k = 0..31.
//   V layout: word (w, j) holds signs[32w + k][j], k = 0..31.
__global__ void k_pack(const int8_t *__restrict__ signs, int64_t rows, int64_t cols, int layout,
                       uint32_t *__restrict__ out, int32_t *bad) {
    const int64_t n_words = layout == LB_PACK_U ? rows * ((cols + 31) / 32)
                                                : ((rows + 31) / 32) * cols;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < n_words;
         idx += stride) {
        int64_t base, step, n_valid;
        if (layout == LB_PACK_U) {
            const int64_t nw = (cols + 31) / 32;
            const int64_t o = idx / nw, w = idx - o * nw;
            base = o * cols + 32 * w;
            step = 1;
            n_valid = min((int64_t)32, cols - 32 * w);
        } else {
            const int64_t w = idx / cols, j = idx - w * cols;
            base = 32 * w * cols + j;
            step = cols;
            n_valid = min((int64_t)32, rows - 32 * w);
        }
        uint32_t word = 0;
        bool invalid = false;
        for (int k = 0; k < n_valid; ++k) {
            const int8_t v = signs[base + k * step];
            word |= (uint32_t)(v == -1) << k;
            invalid |= (v != 1 && v != -1);
        }
        out[idx] = word;
        if (invalid && bad) atomicExch(bad, 1);
    }
}

}  // namespace

cudaError_t launch_pack(const int8_t *signs, int64_t rows, int64_t cols, int layout,
                        uint32_t *out, int32_t *bad, cudaStream_t s) {
    const int64_t n_words = layout == LB_PACK_U ? rows * ((cols + 31) / 32)
                                                : ((rows + 31) / 32) * cols;
    int64_t blocks = (n_words + 255) / 256;
    if (blocks > 65535) blocks = 65535;
    k_pack<<<(unsigned)blocks, 256, 0, s>>>(signs, rows, cols, layout, out, bad);
    return cudaGetLastError();
}

}  // namespace lb
