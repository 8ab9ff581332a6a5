// lb_prefill.cu -- many-token LittleBit forward on the 5th-generation tensor
// cores (tcgen05, fp16 operands, fp32 accumulators in TMEM).
//
// Prop. 1 (LittleBit, arXiv 2506.13771) as two dense contractions:
//   stage 1   z = fp16( l . (X diag(g) V_sign) )     [T x N1],  N1 = sum_p r_p
//   stage 2   Y = z [diag(h_p) U_p,sign]_p^T          [T x d_out]  (Eq. 6 sum
//             over the paths is the K dimension of this GEMM)
// Below four token tiles the sign factors never exist in memory as numbers:
// each CTA unpacks the +-1 bits of its K-slice into shared memory as +-g
// (stage 1) or +-h (stage 2) fp16 values, in the tensor cores' 128-byte-
// swizzled K-major layout.  The bits come from shared memory too: stage 1
// bulk-copies each K-stage's two V word rows (and its 64 g values) on the
// stage's mbarrier beside the TMA of X; stage 2 bulk-copies the tile's U rows
// and h once per CTA.  X arrives by TMA (bf16) and is converted to fp16 in
// shared memory (exact for |x| < 65504).  From four token tiles on, every
// tile would repeat the unpacking, so the operands are expanded to +-g / +-h
// fp16 matrices in the workspace once per call and both GEMMs stream them by
// TMA.  That path is ONE cooperative launch (k_fused, one CTA per SM): the
// expansion, stage 1 over all its tiles, the reduction of its K slices and
// stage 2 run as phases separated by grid barriers, and each tile phase is
// persistent, with two TMEM accumulators so the epilogue of one tile overlaps
// the K loop of the next.  z goes to the workspace as fp16 and comes back by
// TMA.  For long runs whose N1 is a multiple of 512 the expanded path runs
// instead on SM pairs (k_pair, tcgen05 cta_group::2, three launches chained
// by programmatic dependent launch; see the 2-SM section below).  Stage 2 of
// both forms writes y by TMA tensor stores from a swizzled staging tile per
// epilogue warp.
//
// One CTA computes a 128 x BN tile (BN <= 256 fp32 TMEM columns) with
// specialised warps: warp 0 issues the TMA / bulk copies of each 64-element
// K-stage into a 4-deep shared-memory ring, warps 2..9 unpack and convert a
// stage as soon as it lands (only without the pre-pass), and warp 1 issues
// its MMAs (tcgen05.mma, one thread) as soon as the stage is ready;
// tcgen05.commit hands the stage back to the copy warp.  Per stage, full /
// ready / empty mbarriers order the three roles, so no CTA-wide barrier sits
// in the K loop; the two single-thread roles poll with test_wait, which
// notices a completed phase sooner than a suspended try_wait.  Every wait is
// bounded (about one second); on a timeout the CTA records LB_ERR_TIMEOUT, the
// other roles stop, the CTA waits for its own copies and MMAs in flight,
// frees its TMEM and returns.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <mutex>

#include "lb_common.cuh"
#include "lb_kernels.h"

namespace lb {

namespace {

constexpr int BM = 128;       // tokens per tile (MMA M)
constexpr int BN = 256;       // columns per tile (MMA N)
constexpr int BK = 64;        // K per stage: 64 fp16 = one 128-byte swizzle row
constexpr int STAGES = 4;
// Warp roles: 0 issues the TMA / bulk copies, 1 issues the MMAs, 2..9 unpack
// and convert each K-stage and then read the accumulator out.
constexpr int kThreads = 320;
constexpr int kWork = 256;     // threads of the unpacking / epilogue warps
constexpr int kWorkWarps = kWork / 32;
constexpr int A_BYTES = BM * BK * 2;   // 16 KB
constexpr int B_BYTES = BN * BK * 2;   // 32 KB
// stage 1: per stage, the two V word rows of the stage's 64 inputs for the
// tile's columns (2 x BN words) and the 64 g values of each path
constexpr int SRC_BYTES = 2 * BN * 4 + 2 * 64 * 2;
constexpr int MAX_R = 512;  // ranks up to this take the tensor-core path
// stage 2: once per CTA, the tile's U rows (BN x R words per path) and h
constexpr int SLAB_U_BYTES = BN * (MAX_R / 32) * 4;
constexpr int SLAB_BYTES = 2 * SLAB_U_BYTES + 2 * BN * 2;
// Layout: the A|B stage ring (1024-byte aligned stages, as the 128-byte
// swizzle requires), then stage 1's ring of sign words or stage 2's slab.
constexpr int RING_BYTES = STAGES * (A_BYTES + B_BYTES);
template <bool STAGE1>
__host__ __device__ constexpr int smem_bytes() {
    return RING_BYTES + (STAGE1 ? STAGES * SRC_BYTES : SLAB_BYTES) + 1024;
}
static_assert(smem_bytes<true>() <= 232448 && smem_bytes<false>() <= 232448, "shared memory");
// The persistent form: the A|B ring, then (stage 2) one output staging tile
// per epilogue warp: 32 rows x 128 bytes (64 bf16 or 32 fp32 columns) in the
// 128-byte-swizzled layout of the y tensor map, which a TMA store writes out.
constexpr int kMaxStages = 8;
constexpr int kStageBytes = 32 * 128;
constexpr int kTilesSmem = RING_BYTES + kWorkWarps * kStageBytes + 1024;
static_assert(kTilesSmem <= 232448, "shared memory");

extern __shared__ __align__(1024) unsigned char p_smem[];

// ---------------------------------------------------------------- PTX helpers

__device__ __forceinline__ uint32_t su32(const void *p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mb_init(uint64_t *b, unsigned n) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(su32(b)), "r"(n) : "memory");
}
__device__ __forceinline__ void mb_expect_tx(uint64_t *b, unsigned bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(su32(b)),
                 "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ bool mb_try(uint64_t *b, unsigned parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(su32(b)), "r"(parity)
        : "memory");
    return ok != 0;
}

// Bounded wait (every calling thread); false after the limit.
__device__ bool mb_wait(uint64_t *b, unsigned parity) {
    if (mb_try(b, parity)) return true;
    const unsigned long long t0 = globaltimer_ns();
    while (!mb_try(b, parity))
        if (globaltimer_ns() - t0 > kWaitLimitNs) return false;
    return true;
}

// The same, giving up early once another role of the CTA has failed.
__device__ bool mb_wait_role(uint64_t *b, unsigned parity, volatile int *fail) {
    if (mb_try(b, parity)) return true;
    const unsigned long long t0 = globaltimer_ns();
    while (!mb_try(b, parity)) {
        if (*fail) return false;
        if (globaltimer_ns() - t0 > kWaitLimitNs) return false;
    }
    return true;
}

__device__ __forceinline__ bool mb_test(uint64_t *b, unsigned parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(su32(b)), "r"(parity)
        : "memory");
    return ok != 0;
}

// mb_wait_role for the single-thread roles on the pipeline's critical path
// (copy issuer, MMA issuer): a test_wait spin, which sees a completed phase
// sooner than a suspended try_wait wakes up.
__device__ bool mb_spin_role(uint64_t *b, unsigned parity, volatile int *fail) {
    if (mb_test(b, parity)) return true;
    const unsigned long long t0 = globaltimer_ns();
    while (!mb_test(b, parity)) {
        if (*fail) return false;
        if (globaltimer_ns() - t0 > kWaitLimitNs) return false;
    }
    return true;
}

__device__ __forceinline__ void tma_load_2d(void *dst, const CUtensorMap *map, int x, int y,
                                            uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];" ::"r"(su32(dst)),
        "l"(map), "r"(x), "r"(y), "r"(su32(bar))
        : "memory");
}

// Fire-and-forget prefetch of one TMA box into L2.
__device__ __forceinline__ void tma_prefetch_2d(const CUtensorMap *map, int x, int y) {
    asm volatile("cp.async.bulk.prefetch.tensor.2d.L2.global.tile [%0, {%1, %2}];" ::"l"(map),
                 "r"(x), "r"(y)
                 : "memory");
}

__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Shared-memory matrix descriptor: K-major, 128-byte swizzle, 8-row groups
// 1024 bytes apart (stride byte offset), descriptor version 1.
__device__ __forceinline__ uint64_t smem_desc(uint32_t saddr) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFF) >> 4);      // start address
    d |= (uint64_t)1 << 16;                        // leading byte offset (unused when swizzled)
    d |= (uint64_t)(1024 >> 4) << 32;              // stride byte offset
    d |= (uint64_t)1 << 46;                        // version
    d |= (uint64_t)2 << 61;                        // 128-byte swizzle
    return d;
}

// Instruction descriptor, kind::f16: D f32, A f16, B f16, both K-major, M x N.
__host__ __device__ constexpr uint32_t instr_desc(int M, int N) {
    return (1u << 4) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ void mma_f16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                        uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// The same with A (M rows x 16 K, two fp16 per 32-bit column, row m in lane
// m) read from TMEM at a_taddr.
__device__ __forceinline__ void mma_f16_ta(uint32_t tmem_d, uint32_t a_taddr, uint64_t bdesc,
                                           uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(tmem_d),
        "r"(a_taddr), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

__device__ __forceinline__ void mma_commit(uint64_t *bar) {
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
            su32(bar))
        : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// 32 consecutive fp32 columns of this thread's TMEM lane.  The load and its
// wait are one asm statement: tcgen05.ld fills the registers asynchronously,
// so no instruction may read (or copy) them before tcgen05.wait::ld.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
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

// 32 consecutive 32-bit columns of this thread's TMEM lane from r; the store
// and its wait are one asm statement.
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,"
        "%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};\n\t"
        "tcgen05.wait::st.sync.aligned;" ::"r"(taddr),
        "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
        "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]),
        "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]),
        "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]),
        "r"(r[29]), "r"(r[30]), "r"(r[31])
        : "memory");
}

// Byte offset of the 16-byte chunk c (0..7) of row n in a K-major tile with
// 128-byte rows, 128-byte swizzle (chunk index XOR row mod 8).
__device__ __forceinline__ int sw128(int n, int c) {
    return (n >> 3) * 1024 + (n & 7) * 128 + ((c ^ (n & 7)) << 4);
}

// 8 fp16 values: scale[k] with its sign flipped where bit k of bits is set.
__device__ __forceinline__ uint4 signed8(uint32_t bits, uint4 mag) {
    // bit 2i -> bit 15 of word i, bit 2i+1 -> bit 31 of word i
    uint4 r;
    r.x = mag.x ^ (((bits << 15) & 0x8000u) | ((bits << 30) & 0x80000000u));
    r.y = mag.y ^ (((bits << 13) & 0x8000u) | ((bits << 28) & 0x80000000u));
    r.z = mag.z ^ (((bits << 11) & 0x8000u) | ((bits << 26) & 0x80000000u));
    r.w = mag.w ^ (((bits << 9) & 0x8000u) | ((bits << 24) & 0x80000000u));
    return r;
}

struct PrefillParams {
    LinDesc L;
    int T, N1, d_out;
    int bn1;           // stage-1 tile width: N1 if N1 <= 256, else 256
    int bn2;           // k_prefill's stage-2 tile width: 256, 128 or 64 (enough tiles for the SMs)
    int off1;          // column offset of path 1 in the N1 concatenation (= r_0)
    uint16_t *z;       // stage 1 output / stage 2 input, fp16 [T][N1]
    float *z32;        // stage 1 output in fp32 instead of z (latent entry point), or null
    float *zpart;      // split stage 1: fp32 partial sums [split][T][N1] (before l)
    int split;         // stage-1 K slices (gridDim.z of stage 1)
    int pair;          // stage 1 in 128 x 512 column-pair tiles (k_fused)
    int expanded;      // B operands pre-expanded to fp16 (bv, bu): the k_fused path
    uint16_t *bv;      // [N1][d_in]: +-g_p[k] at (column n of path p, input k)
    uint16_t *bu;      // [d_out][N1]: +-h_p[o] at (output o, column n of path p)
    void *y;           // stage 2 output [T][d_out]
    int y_fp32;
    unsigned *ws_words;
};

// Fill B stage with the +-scale values of K-chunk kc for columns [n0, n0+bn),
// from sign words and scales already in shared memory (src: stage 1's
// per-stage words and g; slab: stage 2's U rows and h).
template <bool STAGE1>
__device__ __forceinline__ void unpack_b(const PrefillParams &P, unsigned char *Bs,
                                         const unsigned char *src, const unsigned char *slab,
                                         int kc, int n0, int bn, int tid) {
    const uint32_t *words = reinterpret_cast<const uint32_t *>(src);
    const uint16_t *gs = reinterpret_cast<const uint16_t *>(src + 2 * BN * 4);
    // each item = four 16-byte chunks (32 K values, one sign word) of one B
    // row: half hf of row n
    for (int item = tid; item < bn * 2; item += kWork) {
        const int n = item >> 1, hf = item & 1;
        uint32_t word = 0u;
        bool live = false;
        uint4 mag[4];
        if (STAGE1) {
            const int col = n0 + n;
            live = col < P.N1;
            if (live) {
                const int p = col >= P.off1 ? 1 : 0;
                // inputs 64kc + 32hf .. +31: word row hf
                word = words[hf * BN + n];
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    mag[q] = *reinterpret_cast<const uint4 *>(gs + p * 64 + 8 * (4 * hf + q));
            }
        } else {
            const int o = n0 + n;
            live = o < P.d_out;
            if (live) {
                const int k0 = 64 * kc;
                const int p = k0 >= P.off1 ? 1 : 0, j0 = k0 - (p ? P.off1 : 0);
                const int R = ((p ? P.L.r[1] : P.L.r[0]) + 31) >> 5;
                const uint32_t *U = reinterpret_cast<const uint32_t *>(slab + p * SLAB_U_BYTES);
                const uint16_t *h =
                    reinterpret_cast<const uint16_t *>(slab + 2 * SLAB_U_BYTES) + p * BN;
                word = U[n * R + (j0 >> 5) + hf];
                const uint32_t hb = h[n];
                const uint32_t hh = hb | (hb << 16);
#pragma unroll
                for (int q = 0; q < 4; ++q) mag[q] = make_uint4(hh, hh, hh, hh);
            }
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const uint4 v =
                live ? signed8((word >> (8 * q)) & 0xffu, mag[q]) : make_uint4(0, 0, 0, 0);
            *reinterpret_cast<uint4 *>(Bs + sw128(n, 4 * hf + q)) = v;
        }
    }
}

__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, unsigned bytes,
                                         uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
            "r"(su32(dst)),
        "l"(src), "r"(bytes), "r"(su32(bar))
        : "memory");
}

__device__ __forceinline__ void mb_expect_only(uint64_t *b, unsigned bytes) {
    asm volatile("mbarrier.expect_tx.relaxed.cta.shared::cta.b64 [%0], %1;" ::"r"(su32(b)),
                 "r"(bytes)
                 : "memory");
}

// In-place bf16 -> fp16 of the A stage (layout-preserving, elementwise),
// NT threads.
template <int NT = kWork>
__device__ __forceinline__ void convert_a(unsigned char *As, int tid) {
    for (int i = tid; i < A_BYTES / 16; i += NT) {
        uint4 *p = reinterpret_cast<uint4 *>(As) + i;
        uint4 u = *p;
        uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const float lo = __uint_as_float(w[k] << 16), hi = __uint_as_float(w[k] & 0xffff0000u);
            const __half2 h = __floats2half2_rn(lo, hi);
            w[k] = *reinterpret_cast<const uint32_t *>(&h);
        }
        *p = make_uint4(w[0], w[1], w[2], w[3]);
    }
}

// One 32-column chunk of a finished accumulator row: columns c0 .. c0 + 31 of
// output row `row` (stage 1: z, or the fp32 partial sums of K slice zslice
// when nsplit > 1; stage 2: y).
template <bool STAGE1>
__device__ __forceinline__ void store_chunk(const PrefillParams &P, const float (&v)[32], int row,
                                            int c0, int zslice, int nsplit) {
    if (STAGE1 && nsplit > 1) {
        // fp32 partial sums of this K slice; the reduction applies l
        if (c0 < P.N1) {
            float4 *dst = reinterpret_cast<float4 *>(
                P.zpart + ((size_t)zslice * P.T + row) * P.N1 + c0);
#pragma unroll
            for (int q = 0; q < 8; ++q)
                dst[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
        }
    } else if (STAGE1 && P.z32) {
        // z = l . t as fp32
        if (c0 < P.N1) {
            const int p = c0 >= P.off1 ? 1 : 0;  // 32 | off1
            const int j0 = c0 - (p ? P.off1 : 0);
            const uint16_t *lp = (p ? P.L.l[1] : P.L.l[0]) + j0;
            float4 *dst = reinterpret_cast<float4 *>(P.z32 + (size_t)row * P.N1 + c0);
#pragma unroll
            for (int q = 0; q < 8; ++q)
                dst[q] = make_float4(v[4 * q] * half_bits_to_float(__ldg(lp + 4 * q)),
                                     v[4 * q + 1] * half_bits_to_float(__ldg(lp + 4 * q + 1)),
                                     v[4 * q + 2] * half_bits_to_float(__ldg(lp + 4 * q + 2)),
                                     v[4 * q + 3] * half_bits_to_float(__ldg(lp + 4 * q + 3)));
        }
    } else if (STAGE1) {
        // z = l . t as fp16
        uint32_t packed[16];
#pragma unroll
        for (int i = 0; i < 32; i += 2) {
            float a = 0.f, b = 0.f;
            const int c = c0 + i;
            if (c < P.N1) {
                const int p = c >= P.off1 ? 1 : 0;
                const int j = c - (p ? P.off1 : 0);
                const uint16_t *lp = p ? P.L.l[1] : P.L.l[0];
                a = v[i] * half_bits_to_float(__ldg(lp + j));
                b = v[i + 1] * half_bits_to_float(__ldg(lp + j + 1));
            }
            const __half2 h = __floats2half2_rn(a, b);
            packed[i >> 1] = *reinterpret_cast<const uint32_t *>(&h);
        }
        if (c0 < P.N1) {
            uint4 *dst = reinterpret_cast<uint4 *>(P.z + (size_t)row * P.N1 + c0);
#pragma unroll
            for (int q = 0; q < 4; ++q)
                dst[q] = make_uint4(packed[4 * q], packed[4 * q + 1], packed[4 * q + 2],
                                    packed[4 * q + 3]);
        }
    } else {
        if (P.y_fp32) {
            float *dst = static_cast<float *>(P.y) + (size_t)row * P.d_out + c0;
            if (c0 + 32 <= P.d_out && (P.d_out & 3) == 0) {
#pragma unroll
                for (int q = 0; q < 8; ++q)
                    reinterpret_cast<float4 *>(dst)[q] =
                        make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
            } else {
#pragma unroll
                for (int i = 0; i < 32; ++i)
                    if (c0 + i < P.d_out) dst[i] = v[i];
            }
        } else {
            uint16_t *dst = static_cast<uint16_t *>(P.y) + (size_t)row * P.d_out + c0;
            if (c0 + 32 <= P.d_out && (P.d_out & 7) == 0) {
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    uint32_t w[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        w[e] = (uint32_t)float_to_bf16_bits(v[8 * q + 2 * e]) |
                               ((uint32_t)float_to_bf16_bits(v[8 * q + 2 * e + 1]) << 16);
                    reinterpret_cast<uint4 *>(dst)[q] = make_uint4(w[0], w[1], w[2], w[3]);
                }
            } else {
#pragma unroll
                for (int i = 0; i < 32; ++i)
                    if (c0 + i < P.d_out) dst[i] = float_to_bf16_bits(v[i]);
            }
        }
    }
}

template <bool STAGE1>
__global__ void __launch_bounds__(kThreads, 1)
    k_prefill(const __grid_constant__ CUtensorMap amap, const __grid_constant__ PrefillParams P) {
    __shared__ __align__(8) uint64_t full[STAGES], ready[STAGES], empty[STAGES];
    __shared__ __align__(8) uint64_t slab_bar, acc_bar;
    __shared__ uint32_t s_tmem;
    __shared__ int s_fail;
    unsigned char *smem = reinterpret_cast<unsigned char *>(
        (reinterpret_cast<uintptr_t>(p_smem) + 1023) & ~(uintptr_t)1023);
    constexpr int SB = A_BYTES + B_BYTES;
    unsigned char *slab = smem + RING_BYTES;
    const int bn = STAGE1 ? P.bn1 : P.bn2;
    const int m0 = blockIdx.x * BM, n0 = blockIdx.y * (STAGE1 ? BN : bn);
    const int K = STAGE1 ? P.L.d_in : P.N1;
    // stage 1 may be split along K: slice z of split takes chunks [kbeg, kbeg + KC)
    const int KT = K / BK, nsplit = STAGE1 ? P.split : 1;
    const int kbeg = (int)((long long)blockIdx.z * KT / nsplit);
    const int KC = (int)((long long)(blockIdx.z + 1) * KT / nsplit) - kbeg;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    volatile int *fail = &s_fail;
    if (ld_relaxed_gpu(P.ws_words + kErrWord) != 0u) return;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mb_init(full + s, 1);
            mb_init(ready + s, kWorkWarps);
            mb_init(empty + s, 1);
        }
        mb_init(&slab_bar, 1);
        mb_init(&acc_bar, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        s_fail = 0;
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         su32(&s_tmem)),
                     "r"(BN)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = s_tmem;
    const uint32_t idesc = instr_desc(BM, bn);

    auto A_of = [&](int s) { return smem + s * SB; };
    auto B_of = [&](int s) { return smem + s * SB + A_BYTES; };
    auto S_of = [&](int s) { return smem + RING_BYTES + s * SRC_BYTES; };
    auto give_up = [&]() {
        *fail = 1;
        atomicCAS(P.ws_words + kErrWord, 0u, static_cast<unsigned>(LB_ERR_TIMEOUT));
    };
    int loads_issued = 0, mmas_issued = 0;  // K-chunks loaded / multiplied
    // The x / z tile of the CTA's K-chunk i (chunk kbeg + i of the layer) by
    // TMA; in stage 1 also the chunk's two V word rows for the tile's columns
    // and the chunk's g values, by bulk copy.
    auto issue_load = [&](int i) {
        const int s = i % STAGES, kc = kbeg + i;
        uint64_t *b = full + s;
        if (STAGE1) {
            unsigned char *src = S_of(s);
            for (int p = 0; p < P.L.n_paths; ++p) {
                const int c0 = p ? P.off1 : 0, c1 = p ? P.N1 : P.off1;
                const int lo = max(n0, c0), hi = min(n0 + bn, c1);
                if (lo >= hi) continue;
                const int r = p ? P.L.r[1] : P.L.r[0];
                const uint32_t *V = p ? P.L.v[1] : P.L.v[0];
                for (int wr = 0; wr < 2; ++wr) {
                    const unsigned bytes = (unsigned)(hi - lo) * 4;
                    mb_expect_only(b, bytes);
                    bulk_g2s(src + wr * BN * 4 + (lo - n0) * 4,
                             V + (size_t)(2 * kc + wr) * r + (lo - c0), bytes, b);
                }
                mb_expect_only(b, 128);
                bulk_g2s(src + 2 * BN * 4 + p * 128, (p ? P.L.g[1] : P.L.g[0]) + 64 * kc, 128, b);
            }
        }
        mb_expect_tx(b, A_BYTES);
        tma_load_2d(A_of(s), &amap, kc * BK, m0, b);
    };

    if (warp == 0) {
        // ---------------- producer: copies for chunk i once the MMAs of
        //                  chunk i - STAGES have released its stage
        if (lane == 0) {
            if (!STAGE1) {
                // the tile's U rows and h of every path, once
                const int nrows = min(bn, P.d_out - n0);
                for (int p = 0; p < P.L.n_paths; ++p) {
                    const int R = ((p ? P.L.r[1] : P.L.r[0]) + 31) >> 5;
                    mb_expect_only(&slab_bar, (unsigned)(nrows * R * 4 + nrows * 2));
                    bulk_g2s(slab + p * SLAB_U_BYTES, (p ? P.L.u[1] : P.L.u[0]) + (size_t)n0 * R,
                             (unsigned)(nrows * R * 4), &slab_bar);
                    bulk_g2s(slab + 2 * SLAB_U_BYTES + p * BN * 2,
                             (p ? P.L.h[1] : P.L.h[0]) + n0, (unsigned)(nrows * 2), &slab_bar);
                }
                asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(su32(&slab_bar))
                             : "memory");
            }
            for (int i = 0; i < KC; ++i) {
                const int s = i % STAGES;
                if (i >= STAGES &&
                    !mb_spin_role(empty + s, (unsigned)((i / STAGES - 1) & 1), fail)) {
                    give_up();
                    break;
                }
                issue_load(i);
                ++loads_issued;
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        // ---------------- MMA issuer
        if (lane == 0) {
            for (int i = 0; i < KC; ++i) {
                const int s = i % STAGES;
                if (!mb_spin_role(ready + s, (unsigned)((i / STAGES) & 1), fail)) {
                    give_up();
                    break;
                }
                tc_fence_after();
                const uint32_t a0 = su32(A_of(s)), b0 = su32(B_of(s));
#pragma unroll
                for (int k = 0; k < BK / 16; ++k)
                    mma_f16(tmem, smem_desc(a0 + 32 * k), smem_desc(b0 + 32 * k), idesc,
                            (i > 0 || k > 0) ? 1u : 0u);
                mma_commit(empty + s);
                ++mmas_issued;
            }
            if (mmas_issued == KC) mma_commit(&acc_bar);
        }
        __syncwarp();
    } else {
        // ---------------- unpacking warps: +-scale B and fp16 A of each stage
        const int tid = threadIdx.x - 64;
        bool ok = STAGE1 || mb_wait_role(&slab_bar, 0, fail);
        if (!ok) give_up();
        for (int i = 0; i < KC && ok; ++i) {
            const int s = i % STAGES;
            if (!mb_wait_role(full + s, (unsigned)((i / STAGES) & 1), fail)) {
                give_up();
                break;
            }
            unpack_b<STAGE1>(P, B_of(s), S_of(s), slab, kbeg + i, n0, bn, tid);
            if (STAGE1) convert_a(A_of(s), tid);
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0)
                asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(su32(ready + s))
                             : "memory");
        }
    }
    // the accumulator is complete when the last commit lands
    bool ok = true;
    if (warp >= 2 && KC > 0 && !mb_wait_role(&acc_bar, 0, fail)) {
        if (lane == 0) give_up();
        ok = false;
    }
    ok = __syncthreads_and(ok && !*fail) != 0;
    if (!ok) {
        // let every issued copy and MMA land before the CTA goes away: for
        // each stage wait (bounded) for the phase of its last issued use
        if (threadIdx.x == 0) {
            for (int i = loads_issued - STAGES; i < loads_issued; ++i)
                if (i >= 0) mb_wait(full + i % STAGES, (unsigned)((i / STAGES) & 1));
            if (!STAGE1) mb_wait(&slab_bar, 0);
        }
        if (threadIdx.x == 32)
            for (int i = mmas_issued - STAGES; i < mmas_issued; ++i)
                if (i >= 0) mb_wait(empty + i % STAGES, (unsigned)((i / STAGES) & 1));
        __syncthreads();
    } else if (warp >= 2) {
        tc_fence_after();
        // epilogue: warp w reads TMEM lanes 32(w%4) .. +31 (tile rows) and
        // one half of the tile's 32-column chunks
        const int wq = warp & 3, half = (warp - 2) >> 2, nchunk = bn / 32;
        const int row = m0 + 32 * wq + lane;
        const uint32_t lane_base = tmem + ((uint32_t)(32 * wq) << 16);
        const int cb0 = 32 * (half * nchunk / 2), cb1 = 32 * ((half + 1) * nchunk / 2);
        for (int cb = cb0; cb < cb1; cb += 32) {
            float v[32];
            tmem_ld32(lane_base + cb, v);
            if (row >= P.T) continue;
            store_chunk<STAGE1>(P, v, row, n0 + cb, blockIdx.z, nsplit);
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                     "r"(BN)
                     : "memory");
}

// TMA store of a shared-memory tile (this CTA's) into the tensor map at
// (x, y); out-of-range rows and columns are not written.
__device__ __forceinline__ void tma_store_2d(const CUtensorMap *map, int x, int y, const void *src) {
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];" ::"l"(
                     map),
                 "r"(x), "r"(y), "r"(su32(src))
                 : "memory");
}
__device__ __forceinline__ void bulk_commit() {
    asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}
// until this thread's bulk stores have read their shared-memory sources
__device__ __forceinline__ void bulk_wait_read0() {
    asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
// until this thread's bulk stores are complete
__device__ __forceinline__ void bulk_wait0() {
    asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}

// Stage 2 output of one warp: its 32 accumulator rows (thread = row) and
// columns [c0, c1) of the tile at TMEM address taddr, written through the
// warp's 4 KB staging tile by TMA stores of 32 rows x 128 bytes (64 bf16 or
// 32 fp32 columns) at (col0 + c, row0).  The staging tile is 128-byte
// swizzled (16-byte chunk q of row n at n * 128 + ((q ^ n % 8) << 4)), so
// each warp-wide 16-byte store hits every bank four times, the minimum.
// Lane 0 issues the stores and waits for the previous one to have read the
// tile before the warp refills it; it must call bulk_wait0() before the CTA
// ends.
__device__ __forceinline__ void store_y_tma(const CUtensorMap *ymap, int y_fp32, uint32_t taddr,
                                            int c0, int c1, int row0, int col0,
                                            unsigned char *stg, int lane) {
    const int G = y_fp32 ? 32 : 64;
    for (int c = c0; c < c1; c += G) {
        float v[32], w[32];
        tmem_ld32(taddr + (uint32_t)c, v);
        if (!y_fp32) tmem_ld32(taddr + (uint32_t)(c + 32), w);
        if (lane == 0) bulk_wait_read0();
        __syncwarp();
        unsigned char *rowp = stg + (lane >> 3) * 1024 + (lane & 7) * 128;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            uint4 u;
            if (y_fp32) {
                u = make_uint4(__float_as_uint(v[4 * q]), __float_as_uint(v[4 * q + 1]),
                               __float_as_uint(v[4 * q + 2]), __float_as_uint(v[4 * q + 3]));
            } else {
                const float *f = q < 4 ? v + 8 * q : w + 8 * (q - 4);
                u = make_uint4((uint32_t)float_to_bf16_bits(f[0]) |
                                   ((uint32_t)float_to_bf16_bits(f[1]) << 16),
                               (uint32_t)float_to_bf16_bits(f[2]) |
                                   ((uint32_t)float_to_bf16_bits(f[3]) << 16),
                               (uint32_t)float_to_bf16_bits(f[4]) |
                                   ((uint32_t)float_to_bf16_bits(f[5]) << 16),
                               (uint32_t)float_to_bf16_bits(f[6]) |
                                   ((uint32_t)float_to_bf16_bits(f[7]) << 16));
            }
            *reinterpret_cast<uint4 *>(rowp + ((q ^ (lane & 7)) << 4)) = u;
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
            tma_store_2d(ymap, col0 + c, row0, stg);
            bulk_commit();
        }
    }
}

// The item loops below run inside k_fused at ten warps per SM, so each
// thread gathers the inputs of kBatch items (independent loads in flight)
// before it computes and stores them, and walks its items of a [rows][cols]
// index space by stepping (row, col) instead of dividing a flat index.
constexpr int kBatch = 8;

struct ItemWalk {
    int row, col, drow, dcol, cols;
    __device__ ItemWalk(long long i0, long long di, int cols_)
        : row((int)(i0 / cols_)), col((int)(i0 % cols_)), drow((int)(di / cols_)),
          dcol((int)(di % cols_)), cols(cols_) {}
    __device__ __forceinline__ void step() {
        row += drow;
        col += dcol;
        if (col >= cols) {
            col -= cols;
            ++row;
        }
    }
};

// z = l . (sum over the K slices of the partial t), as fp16 (or fp32 into z32),
// four columns per item; items i0, i0 + di, ... of [T][N1 / 4].  MANY: the
// stand-alone reduction of k_prefill's up to 32 slices, which batches the
// loads of several slices of one item; else (k_fused's few slices) the loads
// of several items of one slice.
template <bool MANY = false>
__device__ __forceinline__ void reduce_z_items(const PrefillParams &P, long long i0, long long di) {
    constexpr int kB = kBatch / 2;
    ItemWalk w(i0, di, P.N1 / 4);
    const size_t slice = (size_t)P.T * P.N1;
    while (w.row < P.T) {
        int row[kB], c[kB];
        float4 a[kB];
#pragma unroll
        for (int k = 0; k < kB; ++k) {
            row[k] = w.row;
            c[k] = 4 * w.col;
            a[k] = make_float4(0.f, 0.f, 0.f, 0.f);
            w.step();
        }
        if (MANY) {
            // up to kZ slices' loads in flight at a time; the sums run in slice
            // order (with up to 32 slices and few tokens the slices, not the
            // items, are what a thread has many of)
            constexpr int kZ = 8;
            for (int z0 = 0; z0 < P.split; z0 += kZ) {
#pragma unroll
                for (int k = 0; k < kB; ++k) {
                    if (row[k] >= P.T) continue;
                    const float *src = P.zpart + z0 * slice + (size_t)row[k] * P.N1 + c[k];
                    float4 b[kZ];
#pragma unroll
                    for (int q = 0; q < kZ; ++q)
                        if (z0 + q < P.split)
                            b[q] = *reinterpret_cast<const float4 *>(src + q * slice);
#pragma unroll
                    for (int q = 0; q < kZ; ++q)
                        if (z0 + q < P.split) {
                            a[k].x += b[q].x;
                            a[k].y += b[q].y;
                            a[k].z += b[q].z;
                            a[k].w += b[q].w;
                        }
                }
            }
        } else {
            for (int z = 0; z < P.split; ++z) {
#pragma unroll
                for (int k = 0; k < kB; ++k) {
                    if (row[k] < P.T) {
                        const float4 b = *reinterpret_cast<const float4 *>(
                            P.zpart + z * slice + (size_t)row[k] * P.N1 + c[k]);
                        a[k].x += b.x;
                        a[k].y += b.y;
                        a[k].z += b.z;
                        a[k].w += b.w;
                    }
                }
            }
        }
#pragma unroll
        for (int k = 0; k < kB; ++k) {
            if (row[k] >= P.T) continue;
            const int p = c[k] >= P.off1 ? 1 : 0, j = c[k] - (p ? P.off1 : 0);  // 4 | off1
            const uint2 lb = __ldg(reinterpret_cast<const uint2 *>((p ? P.L.l[1] : P.L.l[0]) + j));
            const float l0 = half_bits_to_float(lb.x & 0xffffu), l1 = half_bits_to_float(lb.x >> 16);
            const float l2 = half_bits_to_float(lb.y & 0xffffu), l3 = half_bits_to_float(lb.y >> 16);
            const size_t e = (size_t)row[k] * P.N1 + c[k];
            if (P.z32) {
                *reinterpret_cast<float4 *>(P.z32 + e) =
                    make_float4(a[k].x * l0, a[k].y * l1, a[k].z * l2, a[k].w * l3);
                continue;
            }
            const __half2 h0 = __floats2half2_rn(a[k].x * l0, a[k].y * l1);
            const __half2 h1 = __floats2half2_rn(a[k].z * l2, a[k].w * l3);
            *reinterpret_cast<uint2 *>(P.z + e) =
                make_uint2(*reinterpret_cast<const uint32_t *>(&h0),
                           *reinterpret_cast<const uint32_t *>(&h1));
        }
    }
}

// bv[n][k] = +-g_p[k]: input k of column n (column j of path p) of V_sign,
// eight inputs (one 16-byte chunk) per item; items of [N1][d_in / 8].
__device__ __forceinline__ void expand_v_items(const PrefillParams &P, long long i0, long long di) {
    ItemWalk w(i0, di, P.L.d_in / 8);
    while (w.row < P.N1) {
        int n[kBatch], k0[kBatch];
        uint32_t word[kBatch];
        uint4 mag[kBatch];
#pragma unroll
        for (int k = 0; k < kBatch; ++k) {
            n[k] = w.row;
            k0[k] = 8 * w.col;
            w.step();
            word[k] = 0u;
            mag[k] = make_uint4(0u, 0u, 0u, 0u);
            if (n[k] < P.N1) {
                const int p = n[k] >= P.off1 ? 1 : 0, j = n[k] - (p ? P.off1 : 0);
                const int r = p ? P.L.r[1] : P.L.r[0];
                word[k] = __ldg((p ? P.L.v[1] : P.L.v[0]) + (size_t)(k0[k] >> 5) * r + j);
                mag[k] = __ldg(reinterpret_cast<const uint4 *>((p ? P.L.g[1] : P.L.g[0]) + k0[k]));
            }
        }
#pragma unroll
        for (int k = 0; k < kBatch; ++k)
            if (n[k] < P.N1)
                *reinterpret_cast<uint4 *>(P.bv + (size_t)n[k] * P.L.d_in + k0[k]) =
                    signed8((word[k] >> (k0[k] & 31)) & 0xffu, mag[k]);
    }
}

// bu[o][n] = +-h_p[o]: column n (column j of path p) of row o of U_sign,
// eight columns per item; items of [d_out][N1 / 8].
__device__ __forceinline__ void expand_u_items(const PrefillParams &P, long long i0, long long di) {
    ItemWalk w(i0, di, P.N1 / 8);
    while (w.row < P.d_out) {
        int o[kBatch], n0[kBatch];
        uint32_t word[kBatch], hb[kBatch];
#pragma unroll
        for (int k = 0; k < kBatch; ++k) {
            o[k] = w.row;
            n0[k] = 8 * w.col;
            w.step();
            word[k] = hb[k] = 0u;
            if (o[k] < P.d_out) {
                const int p = n0[k] >= P.off1 ? 1 : 0, j0 = n0[k] - (p ? P.off1 : 0);
                const int R = ((p ? P.L.r[1] : P.L.r[0]) + 31) >> 5;
                word[k] = __ldg((p ? P.L.u[1] : P.L.u[0]) + (size_t)o[k] * R + (j0 >> 5));
                hb[k] = __ldg((p ? P.L.h[1] : P.L.h[0]) + o[k]);
            }
        }
#pragma unroll
        for (int k = 0; k < kBatch; ++k) {
            if (o[k] >= P.d_out) continue;
            const int p = n0[k] >= P.off1 ? 1 : 0, j0 = n0[k] - (p ? P.off1 : 0);
            const uint32_t hh = hb[k] | (hb[k] << 16);
            *reinterpret_cast<uint4 *>(P.bu + (size_t)o[k] * P.N1 + n0[k]) =
                signed8((word[k] >> (j0 & 31)) & 0xffu, make_uint4(hh, hh, hh, hh));
        }
    }
}

// mbarriers of one persistent tile phase.  Each phase of the fused kernel has
// its own set, so that no late arrival of one phase lands on the other's.
struct PhaseBars {
    uint64_t full[kMaxStages], ready[kMaxStages], empty[kMaxStages], acc_full[2], acc_empty[2];
};

__device__ __forceinline__ void fence_proxy_async_global() {
    asm volatile("fence.proxy.async.global;" ::: "memory");
}

// One persistent tile phase over pre-expanded B operands (A and B both
// stream by TMA; in stage 1 four warps convert each bf16 x stage to fp16, in
// place or, where the accumulators leave room, into a TMEM ring that the
// MMAs read A from): the CTAs walk the tiles t = blockIdx.x, blockIdx.x + gridDim.x, ...
// (column tile fastest, then K slice, then token tile) and keep two fp32
// accumulators in TMEM (2 x BN columns), so the epilogue warps read out tile
// t while the MMA warp already accumulates tile t + gridDim.x and the copy
// warp keeps streaming K-stages across tile boundaries.  acc_full[b] is
// committed by the MMA warp when accumulator b holds a finished tile;
// acc_empty[b] collects one arrival per epilogue warp once it has read b.
// Every thread of the CTA calls this; false once a wait of this CTA ran out
// (every copy and MMA it issued has landed by then).
template <bool STAGE1>
__device__ bool run_tiles(const CUtensorMap *amap, const CUtensorMap *bmap,
                          const CUtensorMap *ymap, const PrefillParams &P, int tiles_n,
                          int nsplit, int n_tiles, PhaseBars &B, uint32_t tmem,
                          unsigned char *smem, volatile int *fail,
                          bool expand_u_meanwhile = false) {
    // stage 1 streams x as bf16: warps 2..5 convert each A stage to fp16 (in
    // place or into TMEM, below) and warps 6..9 run the epilogue; stage 2
    // uses all eight for it
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int bn = STAGE1 ? P.bn1 : BN;
    const int KT = (STAGE1 ? P.L.d_in : P.N1) / BK;
    // the ring holds as many stages as fit: narrower B tiles, deeper ring
    // (bn 64 / 128 / 192 / 256 -> 8 / 6 / 4 / 4 stages of 24 / 32 / 40 / 48 KB)
    const int SB = A_BYTES + bn * BK * 2;
    const int nst = min(kMaxStages, RING_BYTES / SB);
    const uint32_t idesc = instr_desc(BM, bn);
    // Stage 1 with tiles at most 128 wide, or with at most one tile per CTA
    // (which then uses accumulator 0 only): the accumulators take TMEM
    // columns [0, 256) and the conversion warps put each stage's fp16 A into
    // a TMEM ring at columns 256 + 32 s (at most eight stages of 32 columns),
    // from which the MMAs read it: no fp16 A in shared memory (per K-stage 64
    // instead of 96 KB of shared-memory traffic at bn = 128, 96 instead of
    // 128 KB at bn = 256).
    const bool a_tm = STAGE1 && (bn <= 128 || n_tiles <= (int)gridDim.x);
    const int acc_stride = a_tm ? 128 : BN;
    constexpr int kATmCol = 2 * 128;
    auto give_up = [&]() {
        *fail = 1;
        atomicCAS(P.ws_words + kErrWord, 0u, static_cast<unsigned>(LB_ERR_TIMEOUT));
    };
    // tile t -> token tile origin m0, column origin n0, K chunks [kbeg, kbeg + kc)
    auto tile = [&](int t, int &m0, int &n0, int &z, int &kbeg, int &kc) {
        const int nt = t % tiles_n, rest = t / tiles_n;
        z = rest % nsplit;
        m0 = (rest / nsplit) * BM;
        n0 = nt * bn;
        kbeg = (int)((long long)z * KT / nsplit);
        kc = (int)((long long)(z + 1) * KT / nsplit) - kbeg;
    };
    int loads_issued = 0, mmas_issued = 0;  // K-stages over all of this CTA's tiles
    // ring cursor: stage s and the parity ph of its current use
    auto advance = [&](int &s, unsigned &ph) {
        if (++s == nst) {
            s = 0;
            ph ^= 1u;
        }
    };

    if (warp == 0) {
        // ---------------- copy warp
        if (lane == 0) {
            // the operands may have been written by other CTAs of this launch
            // (generic proxy) before the grid barrier that led here
            fence_proxy_async_global();
            bool ok = true;
            int s = 0;
            unsigned ph = 0;
            for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x) {
                int m0, n0, z, kbeg, kc;
                tile(t, m0, n0, z, kbeg, kc);
                for (int i = 0; i < kc; ++i) {
                    // a stage's previous use must have been multiplied
                    if (loads_issued >= nst && !mb_spin_role(B.empty + s, ph ^ 1u, fail)) {
                        give_up();
                        ok = false;
                        break;
                    }
                    uint64_t *b = B.full + s;
                    mb_expect_tx(b, (unsigned)SB);
                    tma_load_2d(smem + s * SB, amap, (kbeg + i) * BK, m0, b);
                    tma_load_2d(smem + s * SB + A_BYTES, bmap, (kbeg + i) * BK, n0, b);
                    ++loads_issued;
                    advance(s, ph);
                }
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        // ---------------- MMA warp
        if (lane == 0) {
            bool ok = true;
            int ti = 0, s = 0;
            unsigned ph = 0;
            for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x, ++ti) {
                int m0, n0, z, kbeg, kc;
                tile(t, m0, n0, z, kbeg, kc);
                const int b = ti & 1;
                if (ti >= 2 &&
                    !mb_spin_role(B.acc_empty + b, (unsigned)(((ti >> 1) - 1) & 1), fail)) {
                    give_up();
                    break;
                }
                tc_fence_after();
                const uint32_t d = tmem + (uint32_t)(b * acc_stride);
                for (int i = 0; i < kc; ++i) {
                    // stage 1: the stage is ready once its A half is fp16
                    if (!mb_spin_role(STAGE1 ? B.ready + s : B.full + s, ph, fail)) {
                        give_up();
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t a0 = su32(smem + s * SB), b0 = su32(smem + s * SB + A_BYTES);
                    if (a_tm) {
                        const uint32_t at = tmem + (uint32_t)(kATmCol + 32 * s);
#pragma unroll
                        for (int k = 0; k < BK / 16; ++k)
                            mma_f16_ta(d, at + 8 * k, smem_desc(b0 + 32 * k), idesc,
                                       (i > 0 || k > 0) ? 1u : 0u);
                    } else {
#pragma unroll
                        for (int k = 0; k < BK / 16; ++k)
                            mma_f16(d, smem_desc(a0 + 32 * k), smem_desc(b0 + 32 * k), idesc,
                                    (i > 0 || k > 0) ? 1u : 0u);
                    }
                    mma_commit(B.empty + s);
                    ++mmas_issued;
                    advance(s, ph);
                }
                if (ok) mma_commit(B.acc_full + b);
            }
        }
        __syncwarp();
    } else if (STAGE1 && warp < 6) {
        // ---------------- conversion warps: bf16 -> fp16 of each A stage
        const int tid = threadIdx.x - 64;
        int s = 0;
        unsigned ph = 0;
        bool ok = true;
        for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x) {
            int m0, n0, z, kbeg, kc;
            tile(t, m0, n0, z, kbeg, kc);
            for (int i = 0; i < kc; ++i, advance(s, ph)) {
                const bool got = mb_wait_role(B.full + s, ph, fail);
                if (!__all_sync(0xffffffffu, got)) {
                    if (lane == 0) give_up();
                    ok = false;
                    break;
                }
                if (a_tm) {
                    // this lane's row n = 32 (w % 4) + lane of the 128-byte-
                    // swizzled bf16 stage into its TMEM lane as fp16
                    const int n = 32 * (warp & 3) + lane;
                    const unsigned char *rowp = smem + s * SB + (n >> 3) * 1024 + (n & 7) * 128;
                    uint32_t r[32];
#pragma unroll
                    for (int c = 0; c < 8; ++c) {
                        const uint4 u =
                            *reinterpret_cast<const uint4 *>(rowp + ((c ^ (n & 7)) << 4));
                        const uint32_t w4[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const __half2 h = __floats2half2_rn(
                                __uint_as_float(w4[e] << 16), __uint_as_float(w4[e] & 0xffff0000u));
                            r[4 * c + e] = *reinterpret_cast<const uint32_t *>(&h);
                        }
                    }
                    tmem_st32(tmem + ((uint32_t)(32 * (warp & 3)) << 16) +
                                  (uint32_t)(kATmCol + 32 * s),
                              r);
                    tc_fence_before();
                } else {
                    convert_a<128>(smem + s * SB, tid);
                    fence_proxy_async_smem();
                }
                __syncwarp();
                if (lane == 0)
                    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(su32(B.ready + s))
                                 : "memory");
            }
        }
    } else {
        // ---------------- epilogue warps: warp w reads TMEM lanes 32(w%4) ..
        //                  +31 (tile rows) and its share of the tile's columns
        //                  (all of them in stage 1, one half in stage 2)
        const int wq = warp & 3, nchunk = bn / 32;
        const int half = STAGE1 ? 0 : (warp - 2) >> 2, halves = STAGE1 ? 1 : 2;
        const uint32_t lane_base = tmem + ((uint32_t)(32 * wq) << 16);
        const int cb0 = 32 * (half * nchunk / halves), cb1 = 32 * ((half + 1) * nchunk / halves);
        // stage 1 of a forward: the epilogue warps of all CTAs expand stage
        // 2's +-h operand while the first tiles accumulate
        if (STAGE1 && expand_u_meanwhile)
            expand_u_items(P, blockIdx.x * 128LL + (threadIdx.x - 192), gridDim.x * 128LL);
        int ti = 0;
        for (int t = blockIdx.x; t < n_tiles; t += gridDim.x, ++ti) {
            int m0, n0, z, kbeg, kc;
            tile(t, m0, n0, z, kbeg, kc);
            const int b = ti & 1;
            // the vote reconverges the warp (each lane leaves the wait on its
            // own) before the warp-collective tcgen05.ld, and makes the
            // outcome uniform
            const bool got = mb_wait_role(B.acc_full + b, (unsigned)((ti >> 1) & 1), fail);
            if (!__all_sync(0xffffffffu, got)) {
                if (lane == 0) give_up();
                break;
            }
            tc_fence_after();
            const int row = m0 + 32 * wq + lane;
            if (STAGE1) {
                for (int cb = cb0; cb < cb1; cb += 32) {
                    float v[32];
                    tmem_ld32(lane_base + (uint32_t)(b * acc_stride + cb), v);
                    if (row < P.T) store_chunk<STAGE1>(P, v, row, n0 + cb, z, nsplit);
                }
            } else {
                store_y_tma(ymap, P.y_fp32, lane_base + (uint32_t)(b * BN), cb0, cb1, m0 + 32 * wq,
                            n0, smem + RING_BYTES + (warp - 2) * kStageBytes, lane);
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0)
                asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(su32(B.acc_empty + b))
                             : "memory");
        }
        if (!STAGE1 && lane == 0) bulk_wait0();  // this warp's output stores
        __syncwarp();
    }
    if (__syncthreads_or(*fail)) {
        // let every issued copy and MMA land before the CTA goes away
        if (threadIdx.x == 0)
            for (int i = loads_issued - nst; i < loads_issued; ++i)
                if (i >= 0) mb_wait(B.full + i % nst, (unsigned)((i / nst) & 1));
        if (threadIdx.x == 32)
            for (int i = mmas_issued - nst; i < mmas_issued; ++i)
                if (i >= 0) mb_wait(B.empty + i % nst, (unsigned)((i / nst) & 1));
        __syncthreads();
        return false;
    }
    return true;
}

// The split stage 1 of the non-persistent path (k_prefill) reduces its K
// slices in a launch of its own.
__global__ void k_reduce_z(const __grid_constant__ PrefillParams P) {
    reduce_z_items<true>(P, blockIdx.x * (long long)blockDim.x + threadIdx.x,
                         (long long)gridDim.x * blockDim.x);
}

// Column-pair form of stage 1 for long token runs (N1 a multiple of 512):
// one CTA computes a 128 x 512 tile as two 256-wide MMAs that share each
// converted A stage, which halves the shared-memory traffic of A and of the
// bf16 -> fp16 conversion per flop.  The two accumulators fill all of TMEM,
// so a tile's epilogue does not overlap the next tile's K loop (stage 1's K
// loop is long: d_in).  K-stages are 32 wide (64-byte rows, 64-byte
// swizzle): 8 KB of A and 2 x 16 KB of B, five in the ring.
constexpr int BK2 = 32;
constexpr int A2_BYTES = BM * BK2 * 2;
constexpr int B2_HALF = BN * BK2 * 2;
constexpr int SB2 = A2_BYTES + 2 * B2_HALF;
constexpr int NST2 = 5;
static_assert(NST2 * SB2 + 1024 <= kTilesSmem && NST2 <= kMaxStages, "pair ring");

// Shared-memory matrix descriptor: K-major, 64-byte swizzle, 8-row groups
// 512 bytes apart, descriptor version 1.
__device__ __forceinline__ uint64_t smem_desc_sw64(uint32_t saddr) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFF) >> 4);  // start address
    d |= (uint64_t)1 << 16;                    // leading byte offset (unused when swizzled)
    d |= (uint64_t)(512 >> 4) << 32;           // stride byte offset
    d |= (uint64_t)1 << 46;                    // version
    d |= (uint64_t)4 << 61;                    // 64-byte swizzle
    return d;
}

__device__ bool run_tiles_pair(const CUtensorMap *amap, const CUtensorMap *bmap,
                               const PrefillParams &P, int n_pairs, int n_tiles, PhaseBars &B,
                               uint32_t tmem, unsigned char *smem, volatile int *fail,
                               bool expand_u_meanwhile) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int KT = P.L.d_in / BK2;
    const uint32_t idesc = instr_desc(BM, BN);
    auto give_up = [&]() {
        *fail = 1;
        atomicCAS(P.ws_words + kErrWord, 0u, static_cast<unsigned>(LB_ERR_TIMEOUT));
    };
    // tile t -> token tile origin m0, column origin n0 (512 columns)
    auto tile = [&](int t, int &m0, int &n0) {
        m0 = (t / n_pairs) * BM;
        n0 = (t % n_pairs) * 2 * BN;
    };
    int loads_issued = 0, mmas_issued = 0;
    auto advance = [&](int &s, unsigned &ph) {
        if (++s == NST2) {
            s = 0;
            ph ^= 1u;
        }
    };

    if (warp == 0) {
        // ---------------- copy warp
        if (lane == 0) {
            fence_proxy_async_global();
            bool ok = true;
            int s = 0;
            unsigned ph = 0;
            for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x) {
                int m0, n0;
                tile(t, m0, n0);
                for (int i = 0; i < KT; ++i) {
                    if (loads_issued >= NST2 && !mb_spin_role(B.empty + s, ph ^ 1u, fail)) {
                        give_up();
                        ok = false;
                        break;
                    }
                    uint64_t *b = B.full + s;
                    unsigned char *st = smem + s * SB2;
                    mb_expect_tx(b, (unsigned)SB2);
                    tma_load_2d(st, amap, i * BK2, m0, b);
                    tma_load_2d(st + A2_BYTES, bmap, i * BK2, n0, b);
                    tma_load_2d(st + A2_BYTES + B2_HALF, bmap, i * BK2, n0 + BN, b);
                    ++loads_issued;
                    advance(s, ph);
                }
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        // ---------------- MMA warp: both halves of the tile per K-step
        if (lane == 0) {
            bool ok = true;
            int ti = 0, s = 0;
            unsigned ph = 0;
            for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x, ++ti) {
                if (ti >= 1 &&
                    !mb_spin_role(B.acc_empty, (unsigned)((ti - 1) & 1), fail)) {
                    give_up();
                    break;
                }
                tc_fence_after();
                for (int i = 0; i < KT; ++i) {
                    if (!mb_spin_role(B.ready + s, ph, fail)) {
                        give_up();
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t a0 = su32(smem + s * SB2), b0 = a0 + A2_BYTES;
#pragma unroll
                    for (int k = 0; k < BK2 / 16; ++k) {
                        const uint64_t ad = smem_desc_sw64(a0 + 32 * k);
                        const uint32_t acc = (i > 0 || k > 0) ? 1u : 0u;
                        mma_f16(tmem, ad, smem_desc_sw64(b0 + 32 * k), idesc, acc);
                        mma_f16(tmem + BN, ad, smem_desc_sw64(b0 + B2_HALF + 32 * k), idesc, acc);
                    }
                    mma_commit(B.empty + s);
                    ++mmas_issued;
                    advance(s, ph);
                }
                if (ok) mma_commit(B.acc_full);
            }
        }
        __syncwarp();
    } else if (warp < 6) {
        // ---------------- conversion warps: bf16 -> fp16 of each A stage
        const int tid = threadIdx.x - 64;
        int s = 0;
        unsigned ph = 0;
        bool ok = true;
        for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x) {
            for (int i = 0; i < KT; ++i, advance(s, ph)) {
                const bool got = mb_wait_role(B.full + s, ph, fail);
                if (!__all_sync(0xffffffffu, got)) {
                    if (lane == 0) give_up();
                    ok = false;
                    break;
                }
                uint4 *a = reinterpret_cast<uint4 *>(smem + s * SB2);
                for (int q = tid; q < A2_BYTES / 16; q += 128) {
                    uint4 u = a[q];
                    uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float lo = __uint_as_float(w[e] << 16),
                                    hi = __uint_as_float(w[e] & 0xffff0000u);
                        const __half2 h = __floats2half2_rn(lo, hi);
                        w[e] = *reinterpret_cast<const uint32_t *>(&h);
                    }
                    a[q] = make_uint4(w[0], w[1], w[2], w[3]);
                }
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0)
                    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(su32(B.ready + s))
                                 : "memory");
            }
        }
    } else {
        // ---------------- epilogue warps: TMEM lanes 32(w%4) .. +31, all 512 columns
        const int wq = warp & 3;
        const uint32_t lane_base = tmem + ((uint32_t)(32 * wq) << 16);
        if (expand_u_meanwhile)
            expand_u_items(P, blockIdx.x * 128LL + (threadIdx.x - 192), gridDim.x * 128LL);
        int ti = 0;
        for (int t = blockIdx.x; t < n_tiles; t += gridDim.x, ++ti) {
            int m0, n0;
            tile(t, m0, n0);
            const bool got = mb_wait_role(B.acc_full, (unsigned)(ti & 1), fail);
            if (!__all_sync(0xffffffffu, got)) {
                if (lane == 0) give_up();
                break;
            }
            tc_fence_after();
            const int row = m0 + 32 * wq + lane;
            for (int cb = 0; cb < 2 * BN; cb += 32) {
                float v[32];
                tmem_ld32(lane_base + (uint32_t)cb, v);
                if (row < P.T) store_chunk<true>(P, v, row, n0 + cb, 0, 1);
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0)
                asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(su32(B.acc_empty))
                             : "memory");
        }
    }
    if (__syncthreads_or(*fail)) {
        if (threadIdx.x == 0)
            for (int i = loads_issued - NST2; i < loads_issued; ++i)
                if (i >= 0) mb_wait(B.full + i % NST2, (unsigned)((i / NST2) & 1));
        if (threadIdx.x == 32)
            for (int i = mmas_issued - NST2; i < mmas_issued; ++i)
                if (i >= 0) mb_wait(B.empty + i % NST2, (unsigned)((i / NST2) & 1));
        __syncthreads();
        return false;
    }
    return true;
}


// ------------------------------------------------ 2-SM tiles (cta_group::2)
//
// For long token runs the expanded path can also run on SM pairs: a cluster
// of two CTAs computes a 256-token tile with tcgen05.mma.cta_group::2
// (M = 256, N = 256).  Each CTA holds 128 rows of A and 128 of the 256 B
// rows of each MMA in its own shared memory; the MMA, issued by one thread
// of the even CTA (the leader), reads both CTAs' halves and leaves rows
// 128 c .. 128 c + 127 of D in the TMEM of CTA c.  Per SM, the B operand's
// shared-memory traffic (its TMA write and the MMA's read) halves against
// the 1-SM tile of the same work.
//   stage 1: 256 x 512 tiles (two N = 256 MMAs over each converted A stage,
//            all 512 TMEM columns), 64-wide K-stages of 48 KB, four deep;
//   stage 2: 256 x 256 tiles, two accumulators, 32 KB stages, six deep.
// Every CTA's copy warp loads its own halves.  In stage 1 they complete on
// its own `full` barrier, its conversion warps then arrive on the leader's
// `ready` barrier, and the leader's MMA thread waits for that; in stage 2
// both CTAs' copies complete on the leader's `full` barrier (the 2-SM form
// of the TMA copy) and the MMA thread waits for it.  The leader's
// tcgen05.commit arrives on the `empty` (or `acc_full`) barrier of both CTAs
// at once (multicast).  The epilogue warps of both CTAs read their own TMEM
// and arrive on the leader's `acc_empty`.  These kernels are cluster
// launches of their own (expansion, stage 1, stage 2: three launches), not
// cooperative, as they need no grid barrier.
constexpr int kPairRows = 128;                  // rows of A and of each B half per CTA
constexpr int PM = 2 * kPairRows;               // tokens per pair tile (MMA M)
constexpr int PA_BYTES = kPairRows * BK * 2;    // 16 KB
constexpr int PB_BYTES = kPairRows * BK * 2;    // 16 KB
constexpr int PSB1 = PA_BYTES + 2 * PB_BYTES;   // stage 1: A, two B halves
constexpr int PSB2 = PA_BYTES + PB_BYTES;       // stage 2: A, one B half
constexpr int PNST1 = RING_BYTES / PSB1;        // 4
constexpr int PNST2 = RING_BYTES / PSB2;        // 6
static_assert(PNST1 >= 2 && PNST2 <= kMaxStages, "pair rings");

__device__ __forceinline__ unsigned pair_rank() {
    unsigned r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
__device__ __forceinline__ unsigned pair_ctas() {
    unsigned n;
    asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(n));
    return n;
}
// shared::cluster address of a barrier of this CTA in the CTA of rank `rank`
__device__ __forceinline__ uint32_t bar_in(const uint64_t *b, unsigned rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(su32(b)), "r"(rank));
    return r;
}
// Arrive on a barrier of the other CTA (or this one) of the pair.  Default
// semantics (release at CTA scope): a release at cluster scope serialised
// the arriving thread (about 1 us per arrival) and halved the pipeline's
// rate.  What it orders is either TMA-written data, complete before the
// arriving thread saw its own barrier, or the conversion warps' stores,
// published to the tensor cores' async proxy by fence.proxy.async before
// the arrival.
__device__ __forceinline__ void mb_arrive_remote(uint32_t cluster_addr) {
    asm volatile("mbarrier.arrive.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}
// A wait with its own limit (the teardown's short waits).
__device__ bool mb_wait_ns(uint64_t *b, unsigned parity, unsigned long long limit) {
    if (mb_try(b, parity)) return true;
    const unsigned long long t0 = globaltimer_ns();
    while (!mb_try(b, parity))
        if (globaltimer_ns() - t0 > limit) return false;
    return true;
}
// TMA load into this CTA's shared memory that completes on a barrier of
// the pair's leader (a shared::cluster address): the 2-SM form of the copy.
__device__ __forceinline__ void tma_load_2d_lead(void *dst, const CUtensorMap *map, int x, int y,
                                                 uint32_t lead_bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];" ::"r"(su32(dst)),
        "l"(map), "r"(x), "r"(y), "r"(lead_bar)
        : "memory");
}
__device__ __forceinline__ void pair_sync() {
    asm volatile("barrier.cluster.arrive.release;\n\tbarrier.cluster.wait.acquire;" ::: "memory");
}
__device__ __forceinline__ void mma_f16_pair(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                             uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
// arrive once on barrier b of both CTAs of the pair when the MMAs issued so
// far have completed
__device__ __forceinline__ void mma_commit_pair(uint64_t *bar) {
    asm volatile(
        "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
        " [%0], %1;" ::"r"(su32(bar)),
        "h"((uint16_t)3)
        : "memory");
}

// One 2-SM tile phase; launched with clusters of two CTAs, grid even.
// amap: x (stage 1, bf16) or z (stage 2), boxes of 64 x 128; bmap: the
// expanded B operand (bv or bu), boxes of 64 x 128.  Stage 1's epilogue
// warps expand the +-h operand of stage 2 first when expand_u is set.
template <bool STAGE1>
__global__ void __launch_bounds__(kThreads, 1)
    k_pair(const __grid_constant__ CUtensorMap amap, const __grid_constant__ CUtensorMap bmap,
           const __grid_constant__ CUtensorMap ymap, const __grid_constant__ PrefillParams P,
           int tiles_n, int n_tiles, int expand_u) {
    __shared__ PhaseBars B;
    __shared__ uint32_t s_tmem;
    __shared__ int s_fail;
    unsigned char *smem = reinterpret_cast<unsigned char *>(
        (reinterpret_cast<uintptr_t>(p_smem) + 1023) & ~(uintptr_t)1023);
    // A launch that formed no pairs (a profiler may replay it without
    // clusters) must not touch another CTA or issue a 2-SM instruction.
    if (pair_ctas() != 2) {
        if (threadIdx.x == 0)
            atomicCAS(P.ws_words + kErrWord, 0u, static_cast<unsigned>(LB_ERR_UNSUPPORTED));
        return;
    }
    constexpr int SB = STAGE1 ? PSB1 : PSB2, NST = STAGE1 ? PNST1 : PNST2;
    constexpr int kEpiWarps = STAGE1 ? 4 : kWorkWarps;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const unsigned rank = pair_rank();
    const bool leader = rank == 0;
    const int pair = blockIdx.x >> 1, n_pairs = gridDim.x >> 1;
    const int KT = (STAGE1 ? P.L.d_in : P.N1) / BK;
    volatile int *fail = &s_fail;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kMaxStages; ++s) {
            mb_init(B.full + s, 1);
            mb_init(B.ready + s, 2 * 4);  // stage 1: the conversion warps of both CTAs
            mb_init(B.empty + s, 1);
        }
        for (int b = 0; b < 2; ++b) {
            mb_init(B.acc_full + b, 1);
            mb_init(B.acc_empty + b, 2 * kEpiWarps);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        s_fail = 0;
    }
    if (warp == 1) {
        // one warp of each CTA of the pair, together
        asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         su32(&s_tmem)),
                     "r"(2 * BN)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    pair_sync();  // both CTAs' barriers exist before any arrival from the other
    tc_fence_after();
    const uint32_t tmem = s_tmem;
    // Launched as a programmatic dependent of the previous kernel: the set-up
    // above overlapped its tail; its results (the expanded operands, z) are
    // read only after it has completed.  The next launch may start its own
    // set-up on the SMs this one leaves free.
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

    auto give_up = [&]() {
        *fail = 1;
        atomicCAS(P.ws_words + kErrWord, 0u, static_cast<unsigned>(LB_ERR_TIMEOUT));
    };
    // tile t -> token origin m0 of the pair tile, column origin n0
    auto tile = [&](int t, int &m0, int &n0) {
        m0 = (t / tiles_n) * PM;
        n0 = (t % tiles_n) * (STAGE1 ? 2 * BN : BN);
    };
    auto advance = [&](int &s, unsigned &ph) {
        if (++s == NST) {
            s = 0;
            ph ^= 1u;
        }
    };
    int loads_issued = 0, mmas_issued = 0;

    if (warp == 0) {
        // ---------------- copy warp: this CTA's rows of A and of each B half
        if (lane == 0) {
            const uint32_t lead_full = bar_in(B.full, 0);
            bool ok = true;
            int s = 0;
            unsigned ph = 0;
            for (int t = pair; t < n_tiles && ok; t += n_pairs) {
                int m0, n0;
                tile(t, m0, n0);
                const int ra = m0 + kPairRows * (int)rank, rb = n0 + kPairRows * (int)rank;
                for (int i = 0; i < KT; ++i) {
                    if (loads_issued >= NST && !mb_spin_role(B.empty + s, ph ^ 1u, fail)) {
                        give_up();
                        ok = false;
                        break;
                    }
                    uint64_t *b = B.full + s;
                    unsigned char *st = smem + s * SB;
                    if (STAGE1) {
                        // own barrier: the conversion warps wait for it
                        mb_expect_tx(b, (unsigned)SB);
                        tma_load_2d(st, &amap, i * BK, ra, b);
                        tma_load_2d(st + PA_BYTES, &bmap, i * BK, rb, b);
                        tma_load_2d(st + PA_BYTES + PB_BYTES, &bmap, i * BK, rb + BN, b);
                    } else {
                        // both CTAs' halves complete on the leader's barrier
                        if (leader) mb_expect_tx(b, 2u * SB);
                        const uint32_t lb = lead_full + 8u * (uint32_t)s;
                        tma_load_2d_lead(st, &amap, i * BK, ra, lb);
                        tma_load_2d_lead(st + PA_BYTES, &bmap, i * BK, rb, lb);
                    }
                    ++loads_issued;
                    advance(s, ph);
                }
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        if (leader && lane == 0) {
            // ---------------- MMA thread (leader only)
            const uint32_t idesc = instr_desc(PM, BN);
            bool ok = true;
            int ti = 0, s = 0;
            unsigned ph = 0;
            for (int t = pair; t < n_tiles && ok; t += n_pairs, ++ti) {
                const int b = STAGE1 ? 0 : (ti & 1), uses = STAGE1 ? ti : (ti >> 1);
                if (uses >= 1 &&
                    !mb_spin_role(B.acc_empty + b, (unsigned)((uses - 1) & 1), fail)) {
                    give_up();
                    break;
                }
                tc_fence_after();
                const uint32_t d = tmem + (uint32_t)(b * BN);
                // the MMAs of one K-stage into the accumulator
                auto issue = [&](int i) {
                    const uint32_t a0 = su32(smem + s * SB), b0 = a0 + PA_BYTES;
#pragma unroll
                    for (int k = 0; k < BK / 16; ++k) {
                        const uint64_t ad = smem_desc(a0 + 32 * k);
                        const uint32_t acc = (i > 0 || k > 0) ? 1u : 0u;
                        mma_f16_pair(d, ad, smem_desc(b0 + 32 * k), idesc, acc);
                        if (STAGE1)
                            mma_f16_pair(d + BN, ad, smem_desc(b0 + PB_BYTES + 32 * k), idesc,
                                         acc);
                    }
                    mma_commit_pair(B.empty + s);
                    ++mmas_issued;
                    advance(s, ph);
                };
                // Stage 2 waits for two stages at once and issues them back to
                // back: each wait of this thread costs the tensor pipe a gap
                // whether or not the stage has landed (4096 x 4096 r512,
                // T = 8192: 112.3 -> 109.5 us; groups of 4: 114.3).  Stage 1
                // waits on its conversion warps, and grouping there delays
                // the MMAs (groups of 2: 119.5 us); so does grouping the 1-SM
                // kernel's stage 2 (133.8 -> 137.9 us).
                constexpr int G = STAGE1 ? 1 : 2;
                if (G > 1 && KT % G == 0) {
                    for (int i = 0; i < KT; i += G) {
                        int s2 = s;
                        unsigned ph2 = ph;
                        bool got = true;
#pragma unroll
                        for (int j = 0; j < G; ++j) {
                            got = got && mb_spin_role(STAGE1 ? B.ready + s2 : B.full + s2, ph2,
                                                      fail);
                            advance(s2, ph2);
                        }
                        if (!got) {
                            give_up();
                            ok = false;
                            break;
                        }
                        tc_fence_after();
#pragma unroll
                        for (int j = 0; j < G; ++j) issue(i + j);
                    }
                } else {
                    for (int i = 0; i < KT; ++i) {
                        if (!mb_spin_role(STAGE1 ? B.ready + s : B.full + s, ph, fail)) {
                            give_up();
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        issue(i);
                    }
                }
                if (ok) mma_commit_pair(B.acc_full + b);
            }
        }
        __syncwarp();
    } else if (STAGE1 && warp < 6) {
        // ---------------- conversion warps: bf16 -> fp16 of this CTA's A rows
        const int tid = threadIdx.x - 64;
        const uint32_t rdy = bar_in(B.ready, 0);
        int s = 0;
        unsigned ph = 0;
        bool ok = true;
        for (int t = pair; t < n_tiles && ok; t += n_pairs) {
            for (int i = 0; i < KT; ++i, advance(s, ph)) {
                const bool got = mb_wait_role(B.full + s, ph, fail);
                if (!__all_sync(0xffffffffu, got)) {
                    if (lane == 0) give_up();
                    ok = false;
                    break;
                }
                convert_a<128>(smem + s * SB, tid);
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) mb_arrive_remote(rdy + 8u * (uint32_t)s);
            }
        }
    } else {
        // ---------------- epilogue warps: TMEM lanes 32(w%4) .. +31 of this
        //                  CTA (tile rows 128 rank + ...), stage 1 all 512
        //                  columns, stage 2 one half of 256
        const int wq = warp & 3;
        const int half = STAGE1 ? 0 : (warp - 2) >> 2;
        const int cb0 = STAGE1 ? 0 : half * (BN / 2), cb1 = STAGE1 ? 2 * BN : cb0 + BN / 2;
        const uint32_t lane_base = tmem + ((uint32_t)(32 * wq) << 16);
        const uint32_t aempty = bar_in(B.acc_empty, 0);
        if (STAGE1 && expand_u)
            expand_u_items(P, blockIdx.x * 128LL + (threadIdx.x - 192), gridDim.x * 128LL);
        int ti = 0;
        for (int t = pair; t < n_tiles; t += n_pairs, ++ti) {
            int m0, n0;
            tile(t, m0, n0);
            const int b = STAGE1 ? 0 : (ti & 1), uses = STAGE1 ? ti : (ti >> 1);
            const bool got = mb_wait_role(B.acc_full + b, (unsigned)(uses & 1), fail);
            if (!__all_sync(0xffffffffu, got)) {
                if (lane == 0) give_up();
                break;
            }
            tc_fence_after();
            const int row0 = m0 + kPairRows * (int)rank + 32 * wq;
            if (STAGE1) {
                for (int cb = cb0; cb < cb1; cb += 32) {
                    float v[32];
                    tmem_ld32(lane_base + (uint32_t)(b * BN + cb), v);
                    if (row0 + lane < P.T) store_chunk<true>(P, v, row0 + lane, n0 + cb, 0, 1);
                }
            } else {
                store_y_tma(&ymap, P.y_fp32, lane_base + (uint32_t)(b * BN), cb0, cb1, row0, n0,
                            smem + RING_BYTES + (warp - 2) * kStageBytes, lane);
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mb_arrive_remote(aempty + 8u * (uint32_t)b);
        }
        if (!STAGE1 && lane == 0) bulk_wait0();  // this warp's output stores
        __syncwarp();
    }

    // Teardown.  After a failure, let this CTA's copies (and, in the leader,
    // its MMAs) land.  Every CTA then waits for the arrivals of the MMAs
    // that read its last stages (they come from the leader's commits; on a
    // failure some never come, hence the short limit), so that nothing
    // lands in a CTA that has left; both CTAs meet before the TMEM is freed.
    if (__syncthreads_or(*fail)) {
        if (threadIdx.x == 0) {
            if (STAGE1 || leader) {
                for (int i = loads_issued - NST; i < loads_issued; ++i)
                    if (i >= 0) mb_wait(B.full + i % NST, (unsigned)((i / NST) & 1));
            } else {
                // stage 2's odd CTA: its copies complete on the leader's
                // barriers, which it cannot wait on; a copy lands within
                // microseconds of its issue
                const unsigned long long t0 = globaltimer_ns();
                while (globaltimer_ns() - t0 < 100000ull) __nanosleep(1000);
            }
        }
        if (threadIdx.x == 32)
            for (int i = mmas_issued - NST; i < mmas_issued; ++i)
                if (i >= 0) mb_wait(B.empty + i % NST, (unsigned)((i / NST) & 1));
    }
    if (threadIdx.x == 0)
        for (int i = loads_issued - NST; i < loads_issued; ++i)
            if (i >= 0) mb_wait_ns(B.empty + i % NST, (unsigned)((i / NST) & 1), 200000ull);
    tc_fence_before();
    pair_sync();
    tc_fence_after();
    if (warp == 1)
        asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                     "r"(2 * BN)
                     : "memory");
}

// The +-g V_sign (and +-h U_sign) expansion of the 2-SM path, a plain launch
// of kExpandPerSm CTAs per SM (its loads are latency-bound: more warps in
// flight).
constexpr int kExpandPerSm = 2;
__global__ void __launch_bounds__(kThreads, kExpandPerSm) k_expand(const __grid_constant__ PrefillParams P,
                                                     int flags) {
    const long long gi = blockIdx.x * (long long)blockDim.x + threadIdx.x;
    const long long gn = (long long)gridDim.x * blockDim.x;
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    if (flags & 1) expand_v_items(P, gi, gn);
    if (flags & 2) expand_u_items(P, gi, gn);
}

// What one launch of k_fused does, in this order: expand V and / or U, stage
// 1 (and the reduction of its K slices), stage 2.
enum : int { kDoExpandV = 1, kDoExpandU = 2, kDoStage1 = 4, kDoStage2 = 8 };
struct FusedPlan {
    int flags;
    int tiles_n1, split, n_tiles1;  // stage 1: column tiles, K slices, work units
    int tiles_n2, n_tiles2;         // stage 2: column tiles, tiles
};

// The many-token forward (or either half of it) in ONE cooperative launch of
// one CTA per SM: the +-g / +-h operand expansion, stage 1 over all its
// tiles, the reduction of its K slices, and stage 2, separated by grid
// barriers.  Writes that a later phase reads by TMA are published with a
// proxy fence before the barrier.  The last CTA out resets the barrier
// counter, so the next launch on the workspace starts from zero; a launch
// that fails leaves the sticky error word set, and littlebit_poll_error
// clears both.
__global__ void __launch_bounds__(kThreads, 1)
    k_fused(const __grid_constant__ CUtensorMap xmap, const __grid_constant__ CUtensorMap bvmap,
            const __grid_constant__ CUtensorMap zmap, const __grid_constant__ CUtensorMap bumap,
            const __grid_constant__ CUtensorMap ymap, const __grid_constant__ PrefillParams P,
            const __grid_constant__ FusedPlan F) {
    __shared__ PhaseBars bars[2];
    __shared__ uint32_t s_tmem;
    __shared__ int s_fail;
    unsigned char *smem = reinterpret_cast<unsigned char *>(
        (reinterpret_cast<uintptr_t>(p_smem) + 1023) & ~(uintptr_t)1023);
    const int warp = threadIdx.x >> 5;
    volatile int *fail = &s_fail;
    if (ld_relaxed_gpu(P.ws_words + kErrWord) != 0u) return;
    const unsigned n_ctas = gridDim.x;

    if (threadIdx.x == 0) {
        for (int ph = 0; ph < 2; ++ph) {
            PhaseBars &B = bars[ph];
            for (int s = 0; s < kMaxStages; ++s) {
                mb_init(B.full + s, 1);
                mb_init(B.ready + s, 4);
                mb_init(B.empty + s, 1);
            }
            for (int b = 0; b < 2; ++b) {
                mb_init(B.acc_full + b, 1);
                mb_init(B.acc_empty + b, ph == 0 ? 4 : kWorkWarps);
            }
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        s_fail = 0;
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         su32(&s_tmem)),
                     "r"(2 * BN)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = s_tmem;
    const long long gi = blockIdx.x * (long long)blockDim.x + threadIdx.x;
    const long long gn = (long long)gridDim.x * blockDim.x;
    unsigned nbar = 0;  // grid barriers passed
    bool ok = true;

    // U is expanded up front only without a stage 1 to hide it in
    const bool u_in_stage1 = (F.flags & kDoStage1) && (F.flags & kDoExpandU);
    if (F.flags & (kDoExpandV | kDoExpandU)) {
        if (threadIdx.x == 32) {
            // while the operands expand: the A stages of this CTA's first tile
            // (x or z, inputs of the call) into L2
            const bool s1 = F.flags & kDoStage1;
            const int t = blockIdx.x, tiles_n = s1 ? F.tiles_n1 : F.tiles_n2;
            const int kstep = (s1 && P.pair) ? BK2 : BK;
            const int nsplit = s1 ? F.split : 1, KT = (s1 ? P.L.d_in : P.N1) / kstep;
            if (t < (s1 ? F.n_tiles1 : F.n_tiles2)) {
                const int rest = t / tiles_n, z = rest % nsplit, m0 = (rest / nsplit) * BM;
                const int kbeg = (int)((long long)z * KT / nsplit);
                const int kc = (int)((long long)(z + 1) * KT / nsplit) - kbeg;
                for (int i = 0; i < kc && i < 16; ++i)
                    tma_prefetch_2d(s1 ? &xmap : &zmap, (kbeg + i) * kstep, m0);
            }
        }
        if (F.flags & kDoExpandV) expand_v_items(P, gi, gn);
        if ((F.flags & kDoExpandU) && !u_in_stage1) expand_u_items(P, gi, gn);
        fence_proxy_async_global();
        ok = grid_barrier(P.ws_words, n_ctas * ++nbar);
    }
    if (ok && (F.flags & kDoStage1)) {
        ok = P.pair ? run_tiles_pair(&xmap, &bvmap, P, F.tiles_n1, F.n_tiles1, bars[0], tmem,
                                     smem, fail, u_in_stage1)
                    : run_tiles<true>(&xmap, &bvmap, nullptr, P, F.tiles_n1, F.split, F.n_tiles1, bars[0],
                                      tmem, smem, fail, u_in_stage1);
        if (ok && F.split > 1) {
            ok = grid_barrier(P.ws_words, n_ctas * ++nbar);
            if (ok) reduce_z_items(P, gi, gn);
        }
        if (ok && (F.flags & kDoStage2)) {
            fence_proxy_async_global();
            ok = grid_barrier(P.ws_words, n_ctas * ++nbar);
        }
    }
    if (ok && (F.flags & kDoStage2))
        ok = run_tiles<false>(&zmap, &bumap, &ymap, P, F.tiles_n2, 1, F.n_tiles2, bars[1], tmem, smem,
                              fail);
    if (ok && threadIdx.x == 0) {
        // every CTA counted here has passed its last barrier
        __threadfence();
        if (atomicAdd(P.ws_words + kDoneWord, 1u) == n_ctas - 1) {
            atomicExch(P.ws_words + kCounterWord, 0u);
            atomicExch(P.ws_words + kDoneWord, 0u);
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                     "r"(2 * BN)
                     : "memory");
}

// ---------------------------------------------------------------- host side

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;

bool encoder() {
    std::call_once(g_encode_once, [] {
        void *fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    });
    return g_encode != nullptr;
}

// 2-D map over a row-major [rows][cols] 16-bit matrix, box BK x BM with the
// 128-byte swizzle (or, narrow, BK2 x BM with the 64-byte swizzle of the
// column-pair stage 1), out-of-range rows read as zero.
bool make_map(CUtensorMap *m, const void *base, CUtensorMapDataType dt, int64_t rows,
              int64_t cols, int box_rows = BM, bool narrow = false) {
    const cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    const cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
    const cuuint32_t box[2] = {(cuuint32_t)(narrow ? BK2 : BK), (cuuint32_t)box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return g_encode(m, dt, 2, const_cast<void *>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE,
                    narrow ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The output map of stage 2's TMA stores: [T][d_out] bf16 or fp32, boxes of
// 32 rows x 128 bytes (64 or 32 columns), 128-byte swizzle.
bool make_ymap(CUtensorMap *m, void *y, int y_fp32, int64_t T, int64_t d_out) {
    const int es = y_fp32 ? 4 : 2;
    const cuuint64_t dims[2] = {(cuuint64_t)d_out, (cuuint64_t)T};
    const cuuint64_t strides[1] = {(cuuint64_t)d_out * es};
    const cuuint32_t box[2] = {(cuuint32_t)(128 / es), 32};
    const cuuint32_t estr[2] = {1, 1};
    return g_encode(m, y_fp32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16,
                    2, y, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                    CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

// The kernels' shared-memory opt-in, once per device (a host call that
// would otherwise sit between the launches of every forward).
static cudaError_t set_smem_attributes() {
    static std::mutex mu;
    static bool done[64];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(mu);
    if (dev >= 0 && dev < 64 && done[dev]) return cudaSuccess;
    e = cudaFuncSetAttribute(k_prefill<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             smem_bytes<true>());
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(k_fused, cudaFuncAttributeMaxDynamicSharedMemorySize, kTilesSmem);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(k_prefill<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 smem_bytes<false>());
    if (e == cudaSuccess && dev >= 0 && dev < 64) done[dev] = true;
    return e;
}

// SM count of the current device (cached per device); 0 when it cannot be
// read, which the cooperative launch turns into an error (its grid must be
// exactly one CTA per SM, never a guess).
static int device_sms() {
    static int sms[64];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
    if (sms[dev] == 0) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
            return 0;
        sms[dev] = n;
    }
    return sms[dev];
}

bool prefill_supported(const lb_linear &L, int64_t T) {
    if (T < 1 || T > (1LL << 30)) return false;
    if (L.d_in % BK != 0 || L.d_out % 8 != 0) return false;
    for (int p = 0; p < L.n_paths; ++p)
        if (L.path[p].r % BK != 0 || L.path[p].r > MAX_R) return false;
    return encoder();
}

namespace {
size_t n1_of(const lb_linear &L) {
    size_t n1 = 0;
    for (int p = 0; p < L.n_paths; ++p) n1 += (size_t)L.path[p].r;
    return n1;
}
// Stage-1 K slices: enough CTAs to fill about 148 SMs, at least two K-chunks
// per slice, at most 32 slices (a function of the shapes only, so the
// workspace size does not depend on the device).
bool expanded_of(const lb_linear &, int64_t T);
bool pair_of(const lb_linear &L, int64_t T);
int split_of(const lb_linear &L, int64_t T) {
    if (pair_of(L, T)) return 1;
    const int64_t n1 = (int64_t)n1_of(L), bn1 = n1 <= BN ? n1 : BN;
    const int64_t tiles = ((T + BM - 1) / BM) * ((n1 + bn1 - 1) / bn1);
    const int64_t kc = L.d_in / BK;
    int64_t s = 148 / tiles;
    s = std::min<int64_t>(s, kc / 2);
    s = std::min<int64_t>(s, 32);
    return s < 2 ? 1 : (int)s;
}
size_t z16_bytes(const lb_linear &L, int64_t T) {
    return ((size_t)T * n1_of(L) * 2 + 255) & ~(size_t)255;
}
size_t zpart_bytes(const lb_linear &L, int64_t T) {
    const int S = split_of(L, T);
    return S > 1 ? ((size_t)S * T * n1_of(L) * 4 + 255) & ~(size_t)255 : 0;
}
// From four token tiles on, every tile would unpack the same sign bits: the
// B operands are expanded to fp16 once per call instead (workspace).
bool expanded_of(const lb_linear &, int64_t T) { return (T + BM - 1) / BM >= 4; }
// Stage 1 in 128 x 512 column-pair tiles once there are enough of them to
// fill most SMs without splitting K.
bool pair_of(const lb_linear &L, int64_t T) {
    const int64_t n1 = (int64_t)n1_of(L);
    return expanded_of(L, T) && n1 % (2 * BN) == 0 && ((T + BM - 1) / BM) * (n1 / (2 * BN)) >= 96;
}
size_t bv_bytes(const lb_linear &L) { return ((size_t)n1_of(L) * L.d_in * 2 + 255) & ~(size_t)255; }
size_t bu_bytes(const lb_linear &L) { return ((size_t)L.d_out * n1_of(L) * 2 + 255) & ~(size_t)255; }
}  // namespace

size_t prefill_ws_bytes(const lb_linear &L, int64_t T) {
    return z16_bytes(L, T) + zpart_bytes(L, T) +
           (expanded_of(L, T) ? bv_bytes(L) + bu_bytes(L) : 0);
}

namespace {
PrefillParams params_of(const lb_linear &L, int64_t T, unsigned *ws_words, void *ws) {
    PrefillParams P{};
    P.L = make_desc(L);
    P.T = (int)T;
    P.N1 = (int)n1_of(L);
    P.off1 = L.path[0].r;
    P.bn1 = P.N1 <= BN ? P.N1 : BN;
    // k_prefill's stage 2 (fewer than four token tiles): the narrowest of
    // 256 / 128 / 64 columns whose tiles still fit one wave of 148 CTAs (one
    // per SM: the CTA unpacks its U rows for every K-stage, so with few
    // tokens the rows per CTA set the time, and a second wave doubles it)
    {
        const int64_t tm = (T + BM - 1) / BM;
        P.bn2 = BN;
        while (P.bn2 > 64 && tm * ((L.d_out + P.bn2 / 2 - 1) / (P.bn2 / 2)) <= 148) P.bn2 /= 2;
    }
    P.d_out = L.d_out;
    char *wsb = static_cast<char *>(ws);
    P.z = reinterpret_cast<uint16_t *>(wsb);
    P.split = split_of(L, T);
    P.pair = pair_of(L, T) ? 1 : 0;
    P.zpart = reinterpret_cast<float *>(wsb + z16_bytes(L, T));
    P.expanded = expanded_of(L, T) ? 1 : 0;
    P.bv = reinterpret_cast<uint16_t *>(wsb + z16_bytes(L, T) + zpart_bytes(L, T));
    P.bu = reinterpret_cast<uint16_t *>(wsb + z16_bytes(L, T) + zpart_bytes(L, T) + bv_bytes(L));
    P.ws_words = ws_words;
    return P;
}
}  // namespace

namespace {
// One cooperative launch of k_fused, one CTA per SM (the grid barriers need
// every CTA resident).  Maps of phases the plan skips are never read.
cudaError_t launch_fused(const CUtensorMap &xmap, const CUtensorMap &bvmap,
                         const CUtensorMap &zmap, const CUtensorMap &bumap,
                         const CUtensorMap &ymap, const PrefillParams &P, const FusedPlan &F,
                         cudaStream_t s) {
    void *args[] = {const_cast<CUtensorMap *>(&xmap), const_cast<CUtensorMap *>(&bvmap),
                    const_cast<CUtensorMap *>(&zmap), const_cast<CUtensorMap *>(&bumap),
                    const_cast<CUtensorMap *>(&ymap), const_cast<PrefillParams *>(&P),
                    const_cast<FusedPlan *>(&F)};
    const int sms = device_sms();
    if (sms <= 0) return cudaErrorInvalidDevice;
    return cudaLaunchCooperativeKernel((const void *)k_fused, dim3(sms), dim3(kThreads), args,
                                       kTilesSmem, s);
}

// Stage-1 and stage-2 tilings of the persistent phases.
void plan_stage1(const PrefillParams &P, FusedPlan &F) {
    const int tm = (P.T + BM - 1) / BM;
    const int tn = P.pair ? P.N1 / (2 * BN) : (P.N1 + P.bn1 - 1) / P.bn1;
    F.tiles_n1 = tn;
    F.split = P.split;
    F.n_tiles1 = tm * tn * P.split;
}
void plan_stage2(const PrefillParams &P, FusedPlan &F) {
    const int tm = (P.T + BM - 1) / BM, tn = (P.d_out + BN - 1) / BN;
    F.tiles_n2 = tn;
    F.n_tiles2 = tm * tn;
}
}  // namespace

namespace {
// The 2-SM path is the default for the column-pair shapes; LB_PREFILL_2SM=0
// selects the 1-SM form (k_fused) instead, for comparison.
bool two_sm_enabled() {
    const char *e = getenv("LB_PREFILL_2SM");
    return !(e && e[0] == '0');
}

cudaError_t launch_pair_kernel(bool stage1, const CUtensorMap &amap, const CUtensorMap &bmap,
                               const CUtensorMap &ymap, const PrefillParams &P, int tiles_n,
                               int n_tiles, int expand_u, int grid, cudaStream_t s) {
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = kTilesSmem;
    cfg.stream = s;
    cudaLaunchAttribute at[2];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = 2;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    at[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = at;
    cfg.numAttrs = 2;
    return stage1 ? cudaLaunchKernelEx(&cfg, k_pair<true>, amap, bmap, ymap, P, tiles_n, n_tiles,
                                       expand_u)
                  : cudaLaunchKernelEx(&cfg, k_pair<false>, amap, bmap, ymap, P, tiles_n, n_tiles,
                                       expand_u);
}

// The expanded path on SM pairs, in stream order: the +-g V_sign expansion
// (and +-h U_sign when stage 1 does not run), stage 1 in 256 x 512 tiles
// (its epilogue warps expand +-h U_sign meanwhile when stage 2 follows),
// stage 2 in 256 x 256 tiles.  x is read by stage 1, P.z is stage 1's output
// and stage 2's input.
cudaError_t launch_pair(const lb_linear &L, const uint16_t *x, int64_t T, const PrefillParams &P,
                        bool stage1, bool stage2, cudaStream_t s) {
    CUtensorMap xmap{}, bvmap{}, zmap{}, bumap{}, ymap{};
    if (stage1 &&
        (!make_map(&xmap, x, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, T, L.d_in, kPairRows) ||
         !make_map(&bvmap, P.bv, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, P.N1, L.d_in, kPairRows)))
        return cudaErrorInvalidValue;
    if (stage2 &&
        (!make_map(&zmap, P.z, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, T, P.N1, kPairRows) ||
         !make_map(&bumap, P.bu, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, L.d_out, P.N1, kPairRows) ||
         !make_ymap(&ymap, P.y, P.y_fp32, T, L.d_out)))
        return cudaErrorInvalidValue;
    static std::once_flag once;
    static cudaError_t attr = cudaSuccess;
    std::call_once(once, [] {
        attr = cudaFuncSetAttribute(k_pair<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    kTilesSmem);
        if (attr == cudaSuccess)
            attr = cudaFuncSetAttribute(k_pair<false>,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize, kTilesSmem);
    });
    if (attr != cudaSuccess) return attr;
    const int sms = device_sms() & ~1;
    if (sms <= 0) return cudaErrorInvalidDevice;
    k_expand<<<kExpandPerSm * sms, kThreads, 0, s>>>(P, (stage1 ? 1 : 0) | (stage1 ? 0 : 2));
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const int tm = (int)((T + PM - 1) / PM);
    if (stage1) {
        const int tn1 = P.N1 / (2 * BN), n1 = tm * tn1;
        e = launch_pair_kernel(true, xmap, bvmap, ymap, P, tn1, n1, stage2 ? 1 : 0,
                               std::min(sms, 2 * n1), s);
        if (e != cudaSuccess) return e;
    }
    if (stage2) {
        const int tn2 = (P.d_out + BN - 1) / BN, n2 = tm * tn2;
        e = launch_pair_kernel(false, zmap, bumap, ymap, P, tn2, n2, 0, std::min(sms, 2 * n2), s);
    }
    return e;
}
}  // namespace

cudaError_t launch_prefill_latent(const lb_linear &L, const uint16_t *x, int64_t T, uint16_t *z16,
                                  float *z32, unsigned *ws_words, void *ws, cudaStream_t s) {
    if (!encoder()) return cudaErrorNotSupported;
    PrefillParams P = params_of(L, T, ws_words, ws);
    P.z = z16;
    P.z32 = z32;
    CUtensorMap xmap, bvmap{}, none{};
    if (!make_map(&xmap, x, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, T, L.d_in, BM, P.pair))
        return cudaErrorInvalidValue;
    if (P.expanded &&
        !make_map(&bvmap, P.bv, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, P.N1, L.d_in, P.bn1, P.pair))
        return cudaErrorInvalidValue;
    if (P.expanded && P.pair && two_sm_enabled()) return launch_pair(L, x, T, P, true, false, s);
    cudaError_t e = set_smem_attributes();
    if (e != cudaSuccess) return e;
    if (P.expanded) {
        FusedPlan F{};
        F.flags = kDoExpandV | kDoStage1;
        plan_stage1(P, F);
        return launch_fused(xmap, bvmap, none, none, none, P, F, s);
    }
    const int tm = (int)((T + BM - 1) / BM), tn = (P.N1 + P.bn1 - 1) / P.bn1;
    const dim3 g1((unsigned)tm, (unsigned)tn, (unsigned)P.split);
    k_prefill<true><<<g1, kThreads, smem_bytes<true>(), s>>>(xmap, P);
    e = cudaGetLastError();
    if (e != cudaSuccess || P.split <= 1) return e;
    const long long groups = (long long)T * (P.N1 / 4);
    const int blocks = (int)std::min<long long>((groups + 255) / 256, 148 * 8);
    k_reduce_z<<<blocks, 256, 0, s>>>(P);
    return cudaGetLastError();
}

cudaError_t launch_prefill_expand(const lb_linear &L, const uint16_t *z16, int64_t T, void *y,
                                  int y_fp32, unsigned *ws_words, void *ws, cudaStream_t s) {
    if (!encoder()) return cudaErrorNotSupported;
    PrefillParams P = params_of(L, T, ws_words, ws);
    P.z = const_cast<uint16_t *>(z16);
    P.y = y;
    P.y_fp32 = y_fp32;
    CUtensorMap zmap, bumap{}, ymap{}, none{};
    if (!make_map(&zmap, z16, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, T, P.N1)) return cudaErrorInvalidValue;
    if (P.expanded && !make_ymap(&ymap, y, y_fp32, T, L.d_out)) return cudaErrorInvalidValue;
    if (P.expanded && !make_map(&bumap, P.bu, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, L.d_out, P.N1, BN))
        return cudaErrorInvalidValue;
    if (P.expanded && P.pair && two_sm_enabled())
        return launch_pair(L, nullptr, T, P, false, true, s);
    cudaError_t e = set_smem_attributes();
    if (e != cudaSuccess) return e;
    if (P.expanded) {
        FusedPlan F{};
        F.flags = kDoExpandU | kDoStage2;
        plan_stage2(P, F);
        return launch_fused(none, none, zmap, bumap, ymap, P, F, s);
    }
    const int tm = (int)((T + BM - 1) / BM), tn = (L.d_out + P.bn2 - 1) / P.bn2;
    const dim3 g2((unsigned)tm, (unsigned)tn);
    k_prefill<false><<<g2, kThreads, smem_bytes<false>(), s>>>(zmap, P);
    return cudaGetLastError();
}


cudaError_t launch_prefill(const lb_linear &L, const uint16_t *x, int64_t T, void *y, int y_fp32,
                           unsigned *ws_words, void *ws, cudaStream_t s) {
    uint16_t *z16 = static_cast<uint16_t *>(ws);  // the workspace starts with z
    if (!encoder()) return cudaErrorNotSupported;
    PrefillParams P = params_of(L, T, ws_words, ws);
    if (!P.expanded) {
        cudaError_t e = launch_prefill_latent(L, x, T, z16, nullptr, ws_words, ws, s);
        if (e != cudaSuccess) return e;
        return launch_prefill_expand(L, z16, T, y, y_fp32, ws_words, ws, s);
    }
    // both stages in one launch
    P.z = z16;
    P.y = y;
    P.y_fp32 = y_fp32;
    if (P.pair && two_sm_enabled()) return launch_pair(L, x, T, P, true, true, s);
    CUtensorMap xmap, bvmap, zmap, bumap, ymap;
    if (!make_map(&xmap, x, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, T, L.d_in, BM, P.pair) ||
        !make_map(&bvmap, P.bv, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, P.N1, L.d_in, P.bn1, P.pair) ||
        !make_map(&zmap, z16, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, T, P.N1) ||
        !make_map(&bumap, P.bu, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, L.d_out, P.N1, BN) ||
        !make_ymap(&ymap, y, y_fp32, T, L.d_out))
        return cudaErrorInvalidValue;
    cudaError_t e = set_smem_attributes();
    if (e != cudaSuccess) return e;
    FusedPlan F{};
    F.flags = kDoExpandV | kDoExpandU | kDoStage1 | kDoStage2;
    plan_stage1(P, F);
    plan_stage2(P, F);
    return launch_fused(xmap, bvmap, zmap, bumap, ymap, P, F, s);
}

}  // namespace lb
