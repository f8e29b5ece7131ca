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
#include "tc_common.cuh"

namespace csrt {

struct TcArgs {
    float *g;
    int32_t m, k, n;
    WsHeader *hdr;
};

__global__ void __launch_bounds__(kTcThreads, 1)
    gemm_tf32_tc_kernel(const __grid_constant__ CUtensorMap map_a, const __grid_constant__ CUtensorMap map_b,
                        TcArgs a) {
    pdl_enter();
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
__global__ void __launch_bounds__(kTcThreads, 1)
    gemm_tf32_tc_persistent_kernel(const __grid_constant__ CUtensorMap map_a, const __grid_constant__ CUtensorMap map_b,
                                   const __grid_constant__ CUtensorMap map_g, TcArgs a, int32_t tiles_n,
                                   int32_t num_tiles) {
    pdl_enter();
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
        launch_pdl(gemm_tf32_tc_persistent_kernel, dim3(grid), dim3(kTcThreads), kPSmemBytes, s, ma, mb, mg, a,
                   tiles_n, tiles);
        count_launch();
        *handled = true;
        return check_launch("gemm_tf32_tc_persistent_kernel");
    }
    dim3 grid((unsigned)tiles_n, (unsigned)tiles_m);
    launch_pdl(gemm_tf32_tc_kernel, dim3(grid), dim3(kTcThreads), kTcSmemBytes, s, ma, mb, a);
    count_launch();
    *handled = true;
    return check_launch("gemm_tf32_tc_kernel");
}

}  // namespace csrt
