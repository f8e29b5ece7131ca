// Dense weight gradient G = dY X^T on the 5th-generation tensor cores
// (tcgen05, kind::tf32, float32 accumulation in tensor memory).
//
// G is M x K with G[i, j] = sum_c dY[i, c] X[j, c]; both operands keep the
// reduction index c contiguous, i.e. both are "K-major" in GEMM terms
// (GEMM M = rows of dY, GEMM N = rows of X, GEMM K = the batch columns).
//
// One CTA computes a 128 x 256 tile of G:
//  * warp 0, one lane: TMA producer. Each stage holds a 128 x 32 slice of dY
//    and a 256 x 32 slice of X (32 floats = 128 bytes per row, 128-byte
//    swizzle), 48 KB per stage, 4 stages, tracked by full/empty mbarriers.
//  * warp 1, one lane: allocates 256 TMEM columns and issues
//    tcgen05.mma (M=128, N=256, K=8) four times per stage, then
//    tcgen05.commit to release the stage and finally to signal the epilogue.
//  * warps 2-5: epilogue. Each warp reads its 32 TMEM lanes (= 32 rows of the
//    tile) with tcgen05.ld 32x32b, 32 columns at a time, and stores them.
// Operands are fed as float32; the tensor core uses their TF32 part. Rows
// and reduction columns beyond the matrix are zero-filled by TMA.
//
// Every mbarrier wait is bounded: a wait that runs out sets CSRT_DEV_TIMEOUT
// in the workspace status word and the CTA drains what it issued, frees its
// tensor memory and exits instead of hanging.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "common.cuh"

namespace csrt {

constexpr int kTcBM = 128;
constexpr int kTcBN = 256;
constexpr int kTcBK = 32;                       // floats per row per stage (128 bytes)
constexpr int kTcStages = 4;
constexpr int kTcABytes = kTcBM * kTcBK * 4;    // 16 KB
constexpr int kTcBBytes = kTcBN * kTcBK * 4;    // 32 KB
constexpr int kTcStageBytes = kTcABytes + kTcBBytes;
constexpr int kTcSmemBytes = kTcStages * kTcStageBytes + 1024 /*align*/ + 256 /*barriers*/;
constexpr int kTcThreads = 192;
constexpr unsigned kTcWaitLimit = 1u << 22;     // polls before a wait gives up

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t *bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
                 : "memory");
}

// Bounded wait for the phase with the given parity to complete.
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity) {
    const uint32_t addr = smem_u32(bar);
    for (unsigned i = 0; i < kTcWaitLimit; ++i) {
        uint32_t done;
        asm volatile(
            "{\n .reg .pred p;\n mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n"
            " selp.u32 %0, 1, 0, p;\n}\n"
            : "=r"(done)
            : "r"(addr), "r"(parity)
            : "memory");
        if (done) return true;
        if (i > 64) __nanosleep(32);
    }
    return false;
}

__device__ __forceinline__ void tma_load_2d(void *dst, const CUtensorMap *map, int x, int y, uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
        ::"r"(smem_u32(dst)), "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
        : "memory");
}

// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle, 8-row
// groups 1024 bytes apart (SBO), descriptor version 1.
__device__ __forceinline__ uint64_t smem_desc_sw128(const void *p) {
    const uint64_t addr = smem_u32(p);
    uint64_t d = 0;
    d |= (addr & 0x3FFFFull) >> 4;          // start address
    d |= (uint64_t)1 << 16;                 // leading byte offset (unused for swizzled K-major)
    d |= (uint64_t)(1024 >> 4) << 32;       // stride byte offset
    d |= (uint64_t)1 << 46;                 // version
    d |= (uint64_t)2 << 61;                 // 128-byte swizzle
    return d;
}

// Instruction descriptor, kind::tf32: D = F32, A = B = TF32, both K-major.
constexpr uint32_t kTcIdesc = (1u << 4) | (2u << 7) | (2u << 10) | ((uint32_t)(kTcBN >> 3) << 17) |
                              ((uint32_t)(kTcBM >> 4) << 24);

__device__ __forceinline__ void mma_tf32(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t accumulate) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n}\n"
        ::"r"(tmem_d), "l"(adesc), "l"(bdesc), "r"(kTcIdesc), "r"(accumulate)
        : "memory");
}

__device__ __forceinline__ void mma_commit(uint64_t *bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
                 : "memory");
}

__device__ __forceinline__ void tmem_ld_32cols(uint32_t taddr, uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

struct TcArgs {
    float *g;
    int32_t m, k, n;
    WsHeader *hdr;
};

__global__ void __launch_bounds__(kTcThreads, 1)
    gemm_tf32_tc_kernel(const __grid_constant__ CUtensorMap map_a, const __grid_constant__ CUtensorMap map_b,
                        TcArgs a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sa = smem;
    uint8_t *sb = smem + kTcStages * kTcABytes;
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + kTcStages * kTcStageBytes);
    uint64_t *empty = full + kTcStages;
    uint64_t *acc_full = empty + kTcStages;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(acc_full + 1);
    __shared__ int s_failed;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m0 = blockIdx.y * kTcBM;     // rows of G (rows of dY)
    const int n0 = blockIdx.x * kTcBN;     // columns of G (rows of X)
    const int num_kb = (a.n + kTcBK - 1) / kTcBK;

    if (threadIdx.x == 0) {
        s_failed = 0;
        for (int s = 0; s < kTcStages; ++s) {
            mbar_init(full + s, 1);
            mbar_init(empty + s, 1);
        }
        mbar_init(acc_full, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&map_a)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&map_b)) : "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                     "r"(kTcBN)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        if (lane == 0) {
            // producer: stage kb % S, waiting for the MMA of kb - S to release it
            int issued = 0;
            for (int kb = 0; kb < num_kb; ++kb) {
                const int s = kb % kTcStages;
                if (kb >= kTcStages && !mbar_wait(empty + s, ((kb / kTcStages) & 1) ^ 1)) {
                    s_failed = 1;
                    break;
                }
                mbar_expect_tx(full + s, kTcStageBytes);
                tma_load_2d(sa + s * kTcABytes, &map_a, kb * kTcBK, m0, full + s);
                tma_load_2d(sb + s * kTcBBytes, &map_b, kb * kTcBK, n0, full + s);
                issued = kb + 1;
            }
            // drain: every issued load must land before the CTA may exit
            for (int kb = imax(0, issued - kTcStages); kb < issued; ++kb)
                if (!mbar_wait(full + kb % kTcStages, (kb / kTcStages) & 1)) s_failed = 1;
        }
    } else if (warp == 1) {
        if (lane == 0) {
            bool ok = true;
            for (int kb = 0; kb < num_kb; ++kb) {
                const int s = kb % kTcStages;
                if (!mbar_wait(full + s, (kb / kTcStages) & 1)) {
                    ok = false;
                    break;
                }
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
#pragma unroll
                for (int k = 0; k < kTcBK / 8; ++k) {
                    const uint64_t ad = smem_desc_sw128(sa + s * kTcABytes + k * 32);
                    const uint64_t bd = smem_desc_sw128(sb + s * kTcBBytes + k * 32);
                    mma_tf32(tmem, ad, bd, (kb > 0 || k > 0) ? 1u : 0u);
                }
                mma_commit(empty + s);
            }
            if (!ok) s_failed = 1;
            mma_commit(acc_full);   // also fires when no MMA was issued
        }
    } else {
        // epilogue warps 2..5: TMEM lanes 32*(warp % 4) .. +31
        const bool ok = __all_sync(0xffffffffu, mbar_wait(acc_full, 0));
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const int quarter = warp & 3;
        const int row = m0 + quarter * 32 + lane;
        if (!ok && lane == 0) s_failed = 1;
        if (ok) {
            const bool vec = (a.k % 4) == 0;
            for (int c = 0; c < kTcBN; c += 32) {
                uint32_t r[32];
                tmem_ld_32cols(tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)c, r);
                if (row < a.m) {
                    float *dst = a.g + (int64_t)row * a.k + n0 + c;
                    const int left = a.k - (n0 + c);
                    if (vec && left >= 32) {
#pragma unroll
                        for (int j = 0; j < 32; j += 4)
                            *reinterpret_cast<float4 *>(dst + j) =
                                make_float4(__uint_as_float(r[j]), __uint_as_float(r[j + 1]),
                                            __uint_as_float(r[j + 2]), __uint_as_float(r[j + 3]));
                    } else {
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            if (j < left) dst[j] = __uint_as_float(r[j]);
                    }
                }
            }
        }
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (threadIdx.x == 0 && s_failed) {
        dev_flag(a.hdr, CSRT_DEV_TIMEOUT);
        a.hdr->timeout_site = 2;
    }
    if (warp == 1) {
        __syncwarp();
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTcBN) : "memory");
    }
}


// ---------------------------------------------------------------------------
// Persistent variant (the default): one CTA per SM walks its share of the
// 128 x 256 tiles. The accumulator is double-buffered in tensor memory (512
// columns), so the epilogue of one tile overlaps the TMA loads and MMAs of the
// next. The epilogue goes through shared memory: each epilogue warp writes its
// 32 rows x 32 columns (128-byte swizzled, bank-conflict free) into one of two
// 4 KB staging buffers and one lane stores it with a TMA tensor store, so G
// leaves in full lines; rows and columns beyond the matrix are clipped by TMA.
// ---------------------------------------------------------------------------
constexpr int kPEpiBytes = 32 * 32 * 4;   // one 32 x 32 float staging buffer
constexpr int kPSmemBytes = kTcStages * kTcStageBytes + 4 * 2 * kPEpiBytes + 1024 + 256;

// Bounded wait that also gives up early once another role has aborted.
__device__ __forceinline__ bool mbar_wait_or_abort(uint64_t *bar, uint32_t parity, volatile int *abort_flag) {
    const uint32_t addr = smem_u32(bar);
    for (unsigned i = 0; i < kTcWaitLimit; ++i) {
        uint32_t done;
        asm volatile(
            "{\n .reg .pred p;\n mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n"
            " selp.u32 %0, 1, 0, p;\n}\n"
            : "=r"(done)
            : "r"(addr), "r"(parity)
            : "memory");
        if (done) return true;
        if ((i & 63) == 63 && *abort_flag) return false;
        if (i > 64) __nanosleep(32);
    }
    *abort_flag = 1;
    return false;
}

__device__ __forceinline__ void tma_store_2d(const CUtensorMap *map, int x, int y, const void *src) {
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];" ::"l"(
                     reinterpret_cast<uint64_t>(map)),
                 "r"(x), "r"(y), "r"(smem_u32(src))
                 : "memory");
    asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}

__global__ void __launch_bounds__(kTcThreads, 1)
    gemm_tf32_tc_persistent_kernel(const __grid_constant__ CUtensorMap map_a, const __grid_constant__ CUtensorMap map_b,
                                   const __grid_constant__ CUtensorMap map_g, TcArgs a, int32_t tiles_n,
                                   int32_t num_tiles) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sa = smem;
    uint8_t *sb = smem + kTcStages * kTcABytes;
    uint8_t *epi = smem + kTcStages * kTcStageBytes;                       // 1024-aligned
    uint64_t *full = reinterpret_cast<uint64_t *>(epi + 4 * 2 * kPEpiBytes);
    uint64_t *empty = full + kTcStages;
    uint64_t *accf = empty + kTcStages;    // [2] accumulator ready
    uint64_t *acce = accf + 2;             // [2] accumulator drained
    uint64_t *fin = acce + 2;              // all MMAs of this CTA complete
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(fin + 1);
    __shared__ volatile int s_abort;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int num_kb = (a.n + kTcBK - 1) / kTcBK;

    if (threadIdx.x == 0) {
        s_abort = 0;
        for (int s = 0; s < kTcStages; ++s) {
            mbar_init(full + s, 1);
            mbar_init(empty + s, 1);
        }
        mbar_init(accf, 1);
        mbar_init(accf + 1, 1);
        mbar_init(acce, 4);
        mbar_init(acce + 1, 4);
        mbar_init(fin, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&map_a)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&map_b)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&map_g)) : "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                     "r"(2 * kTcBN)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        if (lane == 0) {
            int it = 0;
            for (int t = blockIdx.x; t < num_tiles && !s_abort; t += gridDim.x) {
                const int m0 = (t / tiles_n) * kTcBM, n0 = (t % tiles_n) * kTcBN;
                for (int kb = 0; kb < num_kb; ++kb, ++it) {
                    const int s = it % kTcStages;
                    if (!mbar_wait_or_abort(empty + s, ((it / kTcStages) & 1) ^ 1, &s_abort)) break;
                    mbar_expect_tx(full + s, kTcStageBytes);
                    tma_load_2d(sa + s * kTcABytes, &map_a, kb * kTcBK, m0, full + s);
                    tma_load_2d(sb + s * kTcBBytes, &map_b, kb * kTcBK, n0, full + s);
                }
            }
            // every issued load must land before the CTA may exit
            for (int i = imax(0, it - kTcStages); i < it; ++i) mbar_wait(full + i % kTcStages, (i / kTcStages) & 1);
        }
    } else if (warp == 1) {
        if (lane == 0) {
            int it = 0, j = 0;
            for (int t = blockIdx.x; t < num_tiles && !s_abort; t += gridDim.x, ++j) {
                const int acc = j & 1;
                if (!mbar_wait_or_abort(acce + acc, ((j >> 1) & 1) ^ 1, &s_abort)) break;
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                const uint32_t d = tmem + (uint32_t)(acc * kTcBN);
                for (int kb = 0; kb < num_kb; ++kb, ++it) {
                    const int s = it % kTcStages;
                    if (!mbar_wait_or_abort(full + s, (it / kTcStages) & 1, &s_abort)) break;
                    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
#pragma unroll
                    for (int k = 0; k < kTcBK / 8; ++k) {
                        const uint64_t ad = smem_desc_sw128(sa + s * kTcABytes + k * 32);
                        const uint64_t bd = smem_desc_sw128(sb + s * kTcBBytes + k * 32);
                        mma_tf32(d, ad, bd, (kb > 0 || k > 0) ? 1u : 0u);
                    }
                    mma_commit(empty + s);
                }
                mma_commit(accf + acc);
            }
            mma_commit(fin);
            mbar_wait(fin, 0);   // nothing of ours still runs on the tensor core
        }
    } else {
        const int q = warp & 3;   // TMEM lanes 32q .. 32q+31 = tile rows 32q ..
        uint8_t *stage0 = epi + (q * 2) * kPEpiBytes;
        int chunk = 0, j = 0;
        for (int t = blockIdx.x; t < num_tiles; t += gridDim.x, ++j) {
            const int acc = j & 1;
            const bool ok = __all_sync(0xffffffffu, mbar_wait_or_abort(accf + acc, (j >> 1) & 1, &s_abort));
            if (!ok) break;
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const int m0 = (t / tiles_n) * kTcBM, n0 = (t % tiles_n) * kTcBN;
            for (int c = 0; c < kTcBN; c += 32, ++chunk) {
                uint8_t *buf = stage0 + (chunk & 1) * kPEpiBytes;
                if (lane == 0) asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
                __syncwarp();
                uint32_t r[32];
                tmem_ld_32cols(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * kTcBN + c), r);
                // row `lane` of the 32 x 32 block, 16-byte chunk i at (i ^ (lane & 7)) (128-byte swizzle)
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    float4 *dst = reinterpret_cast<float4 *>(buf + lane * 128 + ((i ^ (lane & 7)) << 4));
                    *dst = make_float4(__uint_as_float(r[4 * i]), __uint_as_float(r[4 * i + 1]),
                                       __uint_as_float(r[4 * i + 2]), __uint_as_float(r[4 * i + 3]));
                }
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                __syncwarp();
                if (lane == 0) tma_store_2d(&map_g, n0 + c, m0 + q * 32, buf);
            }
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            __syncwarp();
            if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(acce + acc)) : "memory");
        }
        if (lane == 0) asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
        __syncwarp();
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (threadIdx.x == 0 && s_abort) {
        dev_flag(a.hdr, CSRT_DEV_TIMEOUT);
        a.hdr->timeout_site = 4;
    }
    if (warp == 1) {
        __syncwarp();
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(2 * kTcBN) : "memory");
    }
}

static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static bool tried = false;
    if (!tried) {
        tried = true;
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    }
    return fn;
}

// Row-major rows x cols float32 matrix, box of `box_rows` rows x 32 columns, 128-byte swizzle
// (the operand stages and the 32 x 32 epilogue blocks share this layout).
static bool make_map(CUtensorMap *map, const float *base, int64_t rows, int64_t cols, int box_rows) {
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)cols * sizeof(float)};
    cuuint32_t box[2] = {32u, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float *>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

static bool device_is_sm10x() {
    static int cache[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return false;
    if (cache[dev] == 0) {
        int major = 0;
        cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
        cache[dev] = major == 10 ? 1 : 2;
    }
    return cache[dev] == 1;
}

int gemm_tc_tf32(const float *dy, const float *x, int32_t m, int32_t k, int32_t n, float *g, void *ws,
                 size_t ws_bytes, cudaStream_t s, bool *handled) {
    *handled = false;
    // TMA needs 16-byte aligned bases and row strides (n % 4 == 0).
    if (n % 4 != 0 || (reinterpret_cast<uintptr_t>(dy) & 15) || (reinterpret_cast<uintptr_t>(x) & 15)) return CSRT_OK;
    if (m < 64 || k < 64) return CSRT_OK;       // tiny outputs: the CUDA-core kernel is as fast
    CSRT_ARG(ws != nullptr && ws_bytes >= kWsHeaderBytes, "weight_grad_dense (tf32) needs the workspace");
    if (!device_is_sm10x()) return CSRT_OK;
    CUtensorMap ma, mb, mg;
    if (!make_map(&ma, dy, m, n, kTcBM) || !make_map(&mb, x, k, n, kTcBN)) return CSRT_OK;
    // the TMA-store epilogue needs a 16-byte aligned G with rows a multiple of 16 bytes
    const bool tma_out = k % 4 == 0 && (reinterpret_cast<uintptr_t>(g) & 15) == 0 && make_map(&mg, g, m, k, 32);
    static bool attr_set[64] = {false};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !attr_set[dev]) {
        CSRT_CHECK_CUDA(cudaFuncSetAttribute(gemm_tf32_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             kTcSmemBytes));
        CSRT_CHECK_CUDA(cudaFuncSetAttribute(gemm_tf32_tc_persistent_kernel,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, kPSmemBytes));
        attr_set[dev] = true;
    }
    TcArgs a;
    a.g = g;
    a.m = m;
    a.k = k;
    a.n = n;
    a.hdr = static_cast<WsHeader *>(ws);
    const int tiles_m = (int)ceil_div<int64_t>(m, kTcBM), tiles_n = (int)ceil_div<int64_t>(k, kTcBN);
    if (tma_out) {
        const int tiles = tiles_m * tiles_n;
        const int grid = imin(tiles, num_sms());
        gemm_tf32_tc_persistent_kernel<<<grid, kTcThreads, kPSmemBytes, s>>>(ma, mb, mg, a, tiles_n, tiles);
        count_launch();
        *handled = true;
        return check_launch("gemm_tf32_tc_persistent_kernel");
    }
    dim3 grid((unsigned)tiles_n, (unsigned)tiles_m);
    gemm_tf32_tc_kernel<<<grid, kTcThreads, kTcSmemBytes, s>>>(ma, mb, a);
    count_launch();
    *handled = true;
    return check_launch("gemm_tf32_tc_kernel");
}

}  // namespace csrt
