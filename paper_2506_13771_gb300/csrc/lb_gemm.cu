// lb_gemm.cu -- C[M][N] (+)= A[M][K] B[N][K]^T on the 5th-generation tensor
// cores with TF32 operands and fp32 accumulation (tcgen05.mma kind::tf32,
// accumulators in TMEM), for the QAT products of lb_qat.cu.
//
// A and B are fp32, row-major with K contiguous (K-major), their rows
// 16-byte aligned; both stream by TMA in 32-element (128-byte, 128-byte
// swizzled) K-stages.  One CTA computes 128 x BN output tiles (BN = 64, 128
// or 256 by N), persistently: CTAs walk the tiles t = blockIdx.x + k
// gridDim.x and keep two TMEM accumulators, so the epilogue of one tile
// overlaps the K loop of the next.  Warp 0 issues the copies into a ring of
// as many stages as fit 192 KB, warp 1 issues four MMAs (K = 8 each) per
// stage from one thread and hands the stage back with tcgen05.commit, warps
// 2..9 read the accumulator out (warp w: TMEM lanes 32 (w % 4) .., one half
// of the columns) and store it through a shared-memory transpose so every
// store instruction writes whole row segments.  A long K over few tiles is
// split into S slices whose fp32 partials go to a workspace and are added in
// slice order by a second kernel (deterministic).  Every wait is bounded
// (about one second); on a timeout the CTA records LB_ERR_TIMEOUT in the
// error word, the other roles stop, the CTA lets its copies and MMAs land,
// frees its TMEM and returns.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <mutex>

#include "lb_common.cuh"
#include "lb_kernels.h"

namespace lb {

namespace {

constexpr int GM = 128;         // tile rows (MMA M)
constexpr int GK = 32;          // K per stage: 32 fp32 = one 128-byte swizzle row
constexpr int kGThreads = 320;  // warp 0 copies, warp 1 MMAs, warps 2..9 epilogue
constexpr int kGMaxStages = 8;
constexpr int kGRing = 192 * 1024;
constexpr int kGPitch = 33;     // staging rows padded to 33 floats (no bank conflicts)
constexpr int kGStage = 32 * kGPitch * 4;
constexpr int kGSmem = kGRing + 8 * kGStage + 1024;
static_assert(kGSmem <= 232448, "shared memory");

extern __shared__ __align__(1024) unsigned char g_gsmem[];

struct GemmParams {
    int M, N, K;
    float *C;
    long long ldc;
    int accumulate;  // C += A B^T (else C = A B^T); with split > 1 the reduction applies it
    int bn, tiles_n, split, n_tiles;
    float *part;     // split > 1: [split][M][N] partials
    unsigned *err;
    // optional second output C2[m][n] = C[m][n] * scale2[n] at ldc2 (not with accumulate)
    float *C2;
    const float *scale2;
    long long ldc2;
};

struct GemmBars {
    uint64_t full[kGMaxStages], empty[kGMaxStages], acc_full[2], acc_empty[2];
};

__device__ __forceinline__ uint32_t gs(const void *p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void gmb_init(uint64_t *b, unsigned n) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(gs(b)), "r"(n) : "memory");
}
__device__ __forceinline__ void gmb_expect_tx(uint64_t *b, unsigned bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(gs(b)),
                 "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ bool gmb_test(uint64_t *b, unsigned parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(gs(b)), "r"(parity)
        : "memory");
    return ok != 0;
}
__device__ __forceinline__ bool gmb_try(uint64_t *b, unsigned parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(gs(b)), "r"(parity)
        : "memory");
    return ok != 0;
}
// Bounded waits: spinning test_wait for the single-thread roles, try_wait
// for the epilogue warps; both give up early once another role failed.
__device__ bool gmb_spin(uint64_t *b, unsigned parity, volatile int *fail) {
    if (gmb_test(b, parity)) return true;
    const unsigned long long t0 = globaltimer_ns();
    while (!gmb_test(b, parity)) {
        if (*fail || globaltimer_ns() - t0 > kWaitLimitNs) return false;
    }
    return true;
}
__device__ bool gmb_wait(uint64_t *b, unsigned parity, volatile int *fail) {
    if (gmb_try(b, parity)) return true;
    const unsigned long long t0 = globaltimer_ns();
    while (!gmb_try(b, parity)) {
        if ((fail && *fail) || globaltimer_ns() - t0 > kWaitLimitNs) return false;
    }
    return true;
}
__device__ __forceinline__ void gtma_2d(void *dst, const CUtensorMap *map, int x, int y,
                                        uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];" ::"r"(gs(dst)),
        "l"(map), "r"(x), "r"(y), "r"(gs(bar))
        : "memory");
}
// K-major, 128-byte swizzle, 8-row groups 1024 bytes apart, version 1.
__device__ __forceinline__ uint64_t gdesc(uint32_t saddr) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFF) >> 4);
    d |= (uint64_t)1 << 16;
    d |= (uint64_t)(1024 >> 4) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
}
// Instruction descriptor, kind::tf32: D f32 (bits 4-5 = 1), A and B tf32
// (bits 7-9 and 10-12 = 2), both K-major, N >> 3 at bit 17, M >> 4 at bit 24.
__host__ __device__ constexpr uint32_t gidesc(int M, int N) {
    return (1u << 4) | (2u << 7) | (2u << 10) | ((uint32_t)(N >> 3) << 17) |
           ((uint32_t)(M >> 4) << 24);
}
__device__ __forceinline__ void mma_tf32(uint32_t d, uint64_t a, uint64_t b, uint32_t idesc,
                                         uint32_t acc) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n\t}" ::"r"(d),
        "l"(a), "l"(b), "r"(idesc), "r"(acc)
        : "memory");
}
__device__ __forceinline__ void gcommit(uint64_t *bar) {
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
            gs(bar))
        : "memory");
}
__device__ __forceinline__ void gfence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void gfence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void gtmem_ld32(uint32_t taddr, float (&v)[32]) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
        "%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n\t"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
          "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
          "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
          "=r"(r[31])
        : "r"(taddr)
        : "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

__global__ void __launch_bounds__(kGThreads, 1)
    k_gemm_tf32(const __grid_constant__ CUtensorMap amap, const __grid_constant__ CUtensorMap bmap,
                const __grid_constant__ GemmParams P) {
    __shared__ GemmBars B;
    __shared__ uint32_t s_tmem;
    __shared__ int s_fail;
    unsigned char *smem = reinterpret_cast<unsigned char *>(
        (reinterpret_cast<uintptr_t>(g_gsmem) + 1023) & ~(uintptr_t)1023);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    volatile int *fail = &s_fail;
    if (ld_relaxed_gpu(P.err) != 0u) return;
    const int bn = P.bn;
    const int SB = (GM + bn) * GK * 4;  // one stage: A then B
    const int nst = min(kGMaxStages, kGRing / SB);
    const int KT = (P.K + GK - 1) / GK;
    const uint32_t idesc = gidesc(GM, bn);
    if (threadIdx.x == 0) {
        for (int s = 0; s < kGMaxStages; ++s) {
            gmb_init(B.full + s, 1);
            gmb_init(B.empty + s, 1);
        }
        for (int b = 0; b < 2; ++b) {
            gmb_init(B.acc_full + b, 1);
            gmb_init(B.acc_empty + b, 8);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        s_fail = 0;
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         gs(&s_tmem)),
                     "r"(2 * bn < 32 ? 32 : 2 * bn)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    gfence_before();
    __syncthreads();
    gfence_after();
    const uint32_t tmem = s_tmem;
    auto give_up = [&]() {
        *fail = 1;
        atomicCAS(P.err, 0u, static_cast<unsigned>(LB_ERR_TIMEOUT));
    };
    // tile t -> row origin m0, column origin n0, K slice z: stages [kb, kb + kc)
    auto tile = [&](int t, int &m0, int &n0, int &z, int &kb, int &kc) {
        const int nt = t % P.tiles_n, rest = t / P.tiles_n;
        z = rest % P.split;
        m0 = (rest / P.split) * GM;
        n0 = nt * bn;
        kb = (int)((long long)z * KT / P.split);
        kc = (int)((long long)(z + 1) * KT / P.split) - kb;
    };
    auto advance = [&](int &s, unsigned &ph) {
        if (++s == nst) {
            s = 0;
            ph ^= 1u;
        }
    };
    int loads = 0, mmas = 0;

    if (warp == 0) {
        if (lane == 0) {
            bool ok = true;
            int s = 0;
            unsigned ph = 0;
            for (int t = blockIdx.x; t < P.n_tiles && ok; t += gridDim.x) {
                int m0, n0, z, kb, kc;
                tile(t, m0, n0, z, kb, kc);
                for (int i = 0; i < kc; ++i) {
                    if (loads >= nst && !gmb_spin(B.empty + s, ph ^ 1u, fail)) {
                        give_up();
                        ok = false;
                        break;
                    }
                    gmb_expect_tx(B.full + s, (unsigned)SB);
                    gtma_2d(smem + s * SB, &amap, (kb + i) * GK, m0, B.full + s);
                    gtma_2d(smem + s * SB + GM * GK * 4, &bmap, (kb + i) * GK, n0, B.full + s);
                    ++loads;
                    advance(s, ph);
                }
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            bool ok = true;
            int ti = 0, s = 0;
            unsigned ph = 0;
            for (int t = blockIdx.x; t < P.n_tiles && ok; t += gridDim.x, ++ti) {
                int m0, n0, z, kb, kc;
                tile(t, m0, n0, z, kb, kc);
                const int b = ti & 1;
                if (ti >= 2 && !gmb_spin(B.acc_empty + b, (unsigned)(((ti >> 1) - 1) & 1), fail)) {
                    give_up();
                    break;
                }
                gfence_after();
                const uint32_t d = tmem + (uint32_t)(b * bn);
                for (int i = 0; i < kc; ++i) {
                    if (!gmb_spin(B.full + s, ph, fail)) {
                        give_up();
                        ok = false;
                        break;
                    }
                    gfence_after();
                    const uint32_t a0 = gs(smem + s * SB), b0 = a0 + GM * GK * 4;
#pragma unroll
                    for (int k = 0; k < GK / 8; ++k)
                        mma_tf32(d, gdesc(a0 + 32 * k), gdesc(b0 + 32 * k), idesc,
                                 (i > 0 || k > 0) ? 1u : 0u);
                    gcommit(B.empty + s);
                    ++mmas;
                    advance(s, ph);
                }
                if (ok) gcommit(B.acc_full + b);
            }
        }
        __syncwarp();
    } else {
        // epilogue: warp w reads TMEM lanes 32 (w % 4) .. +31 (tile rows) and
        // one half of the tile's 32-column chunks
        const int wq = warp & 3, half = (warp - 2) >> 2;
        const int nchunk = bn / 32;
        const int c0 = 32 * (half * nchunk / 2), c1 = 32 * ((half + 1) * nchunk / 2);
        const uint32_t lane_base = tmem + ((uint32_t)(32 * wq) << 16);
        float *stg = reinterpret_cast<float *>(smem + kGRing + (warp - 2) * kGStage);
        int ti = 0;
        for (int t = blockIdx.x; t < P.n_tiles; t += gridDim.x, ++ti) {
            int m0, n0, z, kb, kc;
            tile(t, m0, n0, z, kb, kc);
            const int b = ti & 1;
            const bool got = gmb_wait(B.acc_full + b, (unsigned)((ti >> 1) & 1), fail);
            if (!__all_sync(0xffffffffu, got)) {
                if (lane == 0) give_up();
                break;
            }
            gfence_after();
            float *dst = P.split > 1 ? P.part + (size_t)z * P.M * P.N : P.C;
            const long long ld = P.split > 1 ? P.N : P.ldc;
            const bool acc = P.split == 1 && P.accumulate;
            const bool two = P.split == 1 && P.C2 != nullptr;
            for (int cb = c0; cb < c1; cb += 32) {
                float v[32];
                gtmem_ld32(lane_base + (uint32_t)(b * bn + cb), v);
                // lane = tile row: through shared memory so that each store
                // instruction writes 32 consecutive columns of one row
#pragma unroll
                for (int j = 0; j < 32; ++j) stg[lane * kGPitch + j] = v[j];
                __syncwarp();
                const int col = n0 + cb + lane;
                if (acc) {
                    // every old value in flight before the first store
                    float old[32];
#pragma unroll
                    for (int rr = 0; rr < 32; ++rr) {
                        const int row = m0 + 32 * wq + rr;
                        old[rr] = row < P.M && col < P.N ? dst[(size_t)row * ld + col] : 0.f;
                    }
#pragma unroll
                    for (int rr = 0; rr < 32; ++rr) {
                        const int row = m0 + 32 * wq + rr;
                        if (row < P.M && col < P.N)
                            dst[(size_t)row * ld + col] = old[rr] + stg[rr * kGPitch + lane];
                    }
                } else {
                    const float s2 = two && col < P.N ? P.scale2[col] : 0.f;
#pragma unroll 8
                    for (int rr = 0; rr < 32; ++rr) {
                        const int row = m0 + 32 * wq + rr;
                        if (row < P.M && col < P.N) {
                            const float x = stg[rr * kGPitch + lane];
                            dst[(size_t)row * ld + col] = x;
                            if (two) P.C2[(size_t)row * P.ldc2 + col] = x * s2;
                        }
                    }
                }
                __syncwarp();
            }
            gfence_before();
            __syncwarp();
            if (lane == 0)
                asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(gs(B.acc_empty + b))
                             : "memory");
        }
    }
    if (__syncthreads_or(*fail)) {
        // let every issued copy and MMA land before the CTA goes away
        if (threadIdx.x == 0)
            for (int i = loads - nst; i < loads; ++i)
                if (i >= 0) gmb_wait(B.full + i % nst, (unsigned)((i / nst) & 1), nullptr);
        if (threadIdx.x == 32)
            for (int i = mmas - nst; i < mmas; ++i)
                if (i >= 0) gmb_wait(B.empty + i % nst, (unsigned)((i / nst) & 1), nullptr);
    }
    gfence_before();
    __syncthreads();
    if (warp == 1)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                     "r"(2 * bn < 32 ? 32 : 2 * bn)
                     : "memory");
}

// C (+)= sum over the split slices, in slice order.
__global__ void k_gemm_reduce(const __grid_constant__ GemmParams P) {
    const long long n = (long long)P.M * P.N;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n;
         i += (long long)gridDim.x * blockDim.x) {
        float s = 0.f;
        for (int z = 0; z < P.split; ++z) s += P.part[(size_t)z * n + i];
        const int row = (int)(i / P.N), col = (int)(i - (long long)row * P.N);
        float *c = P.C + (size_t)row * P.ldc + col;
        *c = P.accumulate ? *c + s : s;
        if (P.C2) P.C2[(size_t)row * P.ldc2 + col] = s * P.scale2[col];
    }
}

PFN_cuTensorMapEncodeTiled_v12000 g_genc = nullptr;
std::once_flag g_genc_once;

bool genc() {
    std::call_once(g_genc_once, [] {
        void *fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            g_genc = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    });
    return g_genc != nullptr;
}

// 2-D map over an fp32 [rows][ld] operand with K = k valid columns, box 32 x
// box_rows, 128-byte swizzle; reads beyond k or rows return zero.
bool gmap(CUtensorMap *m, const GemmOperand &A, int box_rows) {
    const cuuint64_t dims[2] = {(cuuint64_t)A.k, (cuuint64_t)A.rows};
    const cuuint64_t strides[1] = {(cuuint64_t)A.ld * 4};
    const cuuint32_t box[2] = {(cuuint32_t)GK, (cuuint32_t)box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return g_genc(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float *>(A.p), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int gemm_bn(int N) { return N <= 64 ? 64 : N <= 128 ? 128 : 256; }

// K slices: when the output tiles cannot fill the SMs and K is long, split K
// so that tiles x slices is about the SM count (at least 8 stages a slice).
int gemm_split(int M, int N, int K, int sms) {
    const int bn = gemm_bn(N);
    const int tiles = ((M + GM - 1) / GM) * ((N + bn - 1) / bn);
    const int KT = (K + GK - 1) / GK;
    int s = sms / std::max(1, tiles);
    s = std::min(s, KT / 8);
    s = std::min(s, 16);
    return std::max(1, s);
}

int gemm_sms() {
    static int sms[64];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
    if (sms[dev] == 0) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
            n <= 0)
            return 0;
        sms[dev] = n;
    }
    return sms[dev];
}

cudaError_t gemm_setup() {
    static std::mutex mu;
    static bool done[64];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(mu);
    if (dev >= 0 && dev < 64 && done[dev]) return cudaSuccess;
    e = cudaFuncSetAttribute(k_gemm_tf32, cudaFuncAttributeMaxDynamicSharedMemorySize, kGSmem);
    if (e == cudaSuccess && dev >= 0 && dev < 64) done[dev] = true;
    return e;
}

}  // namespace

bool gemm_operand_ok(const GemmOperand &A) {
    return A.p && A.rows >= 1 && A.k >= 1 && A.ld >= A.k && A.ld % 4 == 0 &&
           (reinterpret_cast<uintptr_t>(A.p) & 15u) == 0;
}

size_t gemm_part_floats(int M, int N, int K) {
    const int sms = 152;  // a bound: the split never exceeds what the SM count allows
    const int s = gemm_split(M, N, K, std::max(sms, gemm_sms()));
    return s > 1 ? (size_t)s * M * N : 0;
}

cudaError_t gemm_tf32(const GemmOperand &A, const GemmOperand &B, float *C, long long ldc,
                      bool accumulate, float *part, size_t part_floats, unsigned *err,
                      cudaStream_t s, float *C2, const float *scale2, long long ldc2) {
    if (!gemm_operand_ok(A) || !gemm_operand_ok(B) || A.k != B.k || !C || ldc < B.rows)
        return cudaErrorInvalidValue;
    if (C2 && (accumulate || !scale2 || ldc2 < B.rows)) return cudaErrorInvalidValue;
    if (!genc()) return cudaErrorNotSupported;
    const int sms = gemm_sms();
    if (sms <= 0) return cudaErrorInvalidDevice;
    cudaError_t e = gemm_setup();
    if (e != cudaSuccess) return e;
    GemmParams P{};
    P.M = A.rows;
    P.N = B.rows;
    P.K = A.k;
    P.C = C;
    P.ldc = ldc;
    P.accumulate = accumulate ? 1 : 0;
    P.bn = gemm_bn(P.N);
    P.tiles_n = (P.N + P.bn - 1) / P.bn;
    P.split = gemm_split(P.M, P.N, P.K, sms);
    if (P.split > 1 && (!part || part_floats < (size_t)P.split * P.M * P.N)) P.split = 1;
    P.n_tiles = ((P.M + GM - 1) / GM) * P.tiles_n * P.split;
    P.part = part;
    P.err = err;
    P.C2 = C2;
    P.scale2 = scale2;
    P.ldc2 = ldc2;
    CUtensorMap am, bm;
    if (!gmap(&am, A, GM) || !gmap(&bm, B, P.bn)) return cudaErrorInvalidValue;
    const int grid = std::min(P.n_tiles, sms);
    k_gemm_tf32<<<grid, kGThreads, kGSmem, s>>>(am, bm, P);
    e = cudaGetLastError();
    if (e != cudaSuccess || P.split == 1) return e;
    const long long n = (long long)P.M * P.N;
    k_gemm_reduce<<<(int)std::min<long long>((n + 255) / 256, (long long)sms * 8), 256, 0, s>>>(P);
    return cudaGetLastError();
}

}  // namespace lb
