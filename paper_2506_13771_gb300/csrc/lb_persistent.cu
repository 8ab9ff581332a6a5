// lb_persistent.cu -- bounded-wait diagnostic: a one-CTA kernel whose grid
// barrier can never complete (littlebit_selftest_wait_timeout).  It checks,
// without faulting or hanging the GPU, that a wait which runs out records
// LB_ERR_TIMEOUT in the workspace and that later launches on that workspace
// return early until the error is polled.
#include "lb_common.cuh"
#include "lb_kernels.h"

namespace lb {

namespace {

// One CTA waits at a grid barrier that needs two arrivals: only its own comes,
// so the bounded wait must run out and record LB_ERR_TIMEOUT.
__global__ void k_wait_timeout(unsigned *ws_words) {
    if (ld_relaxed_gpu(ws_words + kErrWord) != 0u) return;
    if (!grid_barrier(ws_words, 2u)) return;
}

}  // namespace

cudaError_t launch_wait_timeout(unsigned *ws_words, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(ws_words + kCounterWord, 0, sizeof(unsigned), s);
    if (e != cudaSuccess) return e;
    k_wait_timeout<<<1, 32, 0, s>>>(ws_words);
    return cudaGetLastError();
}

}  // namespace lb
