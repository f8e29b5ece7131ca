// Fused weight gradient + proximal update + re-compaction (the dense gradient
// never reaches memory).
//
// The prox step (Eq. prox with the soft threshold of Section 2.2, applied to
// the dense w - eta*G as in Section 3.3, compacted after every update as in
// Section 4.4) needs G = dY X^T at every entry, but only once: here the
// tensor-core GEMM's epilogue applies it straight from the accumulator.
//
//  1. fp_oldbits_kernel: per row of W_in, a bitmask of the stored columns and,
//     per 256-column tile, the index of the row's first stored entry in it.
//  2. gemm_prox_tc_kernel: the persistent tcgen05 GEMM of gemm_tc.cu (same
//     tiles, same MMA order, so the same G bits as weight_grad_dense TF32).
//     Its epilogue thread owns one row of a 128 x 256 tile; for each entry it
//     takes w from W_in (through the bitmask: loads only where a weight is
//     stored), forms z = fl(w - fl(eta*G)), keeps |z| > fl(eta*lambda) and
//     stages the kept values of (row, tile) contiguously plus the tile's keep
//     bitmask and its count.
//  3. fp_rowscan_kernel + scan_single_block_kernel: per-row offsets of the
//     tiles and the new row pointers.
//  4. fp_place_kernel: one warp per (row, tile) writes the tile's kept entries
//     at their final positions, one coalesced run per 32-column word, and the
//     word positions used to build the transposed copy from the bitmask.
// The result is bit-identical to weight_grad_dense (TF32) followed by
// prox_update_compact.
#include "tc_common.cuh"

namespace csrt {

int transpose_from_bits_ext(csrt_csr *w, const uint32_t *keepbits, const int32_t *wordpos, void *scratch,
                            size_t scratch_bytes, cudaStream_t s);
size_t transpose_scratch_bytes(int32_t rows, int32_t cols);

// The placement works on 128-column segments: each GEMM tile (256 columns) is
// two segments, handled by two epilogue warps per TMEM lane quarter.
constexpr int kFpTileCols = 128;                 // columns per segment
constexpr int kFpTileWords = kFpTileCols / 32;   // 4
constexpr int kFpMaxK = 16384;
constexpr int kFpThreads = 64 + 8 * 32;          // producer, MMA, 8 epilogue warps

struct FpLayout {
    int32_t nt, wpr;
    size_t off_obits, off_ostart, off_kbits, off_counts, off_rowtot, off_stage, off_wordpos, off_tr, total;
};

static size_t align256(size_t x) { return (x + 255) / 256 * 256; }

static FpLayout fp_layout(int32_t m, int32_t k) {
    FpLayout L;
    L.nt = (int32_t)ceil_div<int64_t>(k, kFpTileCols);
    L.wpr = k / 32;
    size_t o = 0;
    L.off_obits = o;   o += align256((size_t)m * L.wpr * 4);
    L.off_ostart = o;  o += align256((size_t)m * (L.nt + 1) * 4);
    L.off_kbits = o;   o += align256((size_t)m * L.wpr * 4);
    L.off_counts = o;  o += align256((size_t)m * L.nt * 4);
    L.off_rowtot = o;  o += align256((size_t)m * 4);
    L.off_stage = o;   o += align256((size_t)m * L.nt * kFpTileCols * 4);
    L.off_wordpos = o; o += align256((size_t)m * L.wpr * 4);
    L.off_tr = o;      o += align256(transpose_scratch_bytes(m, k));
    L.total = o;
    return L;
}

size_t fused_prox_scratch_bytes(int32_t rows, int32_t cols) {
    if (rows <= 0 || cols <= 0 || cols % 32 != 0) return 0;
    return fp_layout(rows, cols).total;
}

// 1. Old-pattern bitmask per row and the first stored entry of each tile.
__global__ void __launch_bounds__(256) fp_oldbits_kernel(const int32_t *__restrict__ row_ptr,
                                                         const int32_t *__restrict__ col, int32_t m, int32_t wpr,
                                                         int32_t nt, uint32_t *__restrict__ obits,
                                                         int32_t *__restrict__ ostart) {
    __shared__ uint32_t sw[8][kFpMaxK / 32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t r = (int64_t)blockIdx.x * 8 + warp;
    if (r >= m) return;
    uint32_t *w = sw[warp];
    for (int i = lane; i < wpr; i += 32) w[i] = 0u;
    __syncwarp();
    const int32_t s = row_ptr[r], e = row_ptr[r + 1];
    for (int32_t k = s + lane; k < e; k += 32) {
        const int c = __ldg(col + k);
        atomicOr(&w[c >> 5], 1u << (c & 31));
    }
    __syncwarp();
    for (int i = lane; i < wpr; i += 32) obits[r * wpr + i] = w[i];
    // stored entries per segment, then a warp exclusive scan over the segments (32 at a time)
    int32_t *os = ostart + r * (nt + 1);
    int32_t run = s;
    for (int t0 = 0; t0 < nt; t0 += 32) {
        const int t = t0 + lane;
        uint32_t c = 0;
        if (t < nt)
            for (int q = 0; q < kFpTileWords && t * kFpTileWords + q < wpr; ++q) c += __popc(w[t * kFpTileWords + q]);
        uint32_t incl = c;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const uint32_t u = __shfl_up_sync(0xffffffffu, incl, off);
            if (lane >= off) incl += u;
        }
        if (t < nt) os[t] = run + (int32_t)(incl - c);
        run += (int32_t)__shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) os[nt] = e;
}

struct FpArgs {
    int32_t m, k, n, nt, wpr;
    float eta, thr;
    const uint32_t *obits;
    const int32_t *ostart;
    const float *old_val;
    uint32_t *kbits;
    int32_t *counts;
    float *stage;
    WsHeader *hdr;
};

// 2. Persistent TF32 GEMM whose epilogue applies the prox step.
__global__ void __launch_bounds__(kFpThreads, 1)
    gemm_prox_tc_kernel(const __grid_constant__ CUtensorMap map_a, const __grid_constant__ CUtensorMap map_b,
                        FpArgs a, int32_t tiles_n, int32_t num_tiles) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sa = smem;
    uint8_t *sb = smem + kTcStages * kTcABytes;
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + kTcStages * kTcStageBytes);
    uint64_t *empty = full + kTcStages;
    uint64_t *accf = empty + kTcStages;
    uint64_t *acce = accf + 2;
    uint64_t *fin = acce + 2;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(fin + 1);
    __shared__ volatile int s_abort;
    __shared__ int s_nonfinite;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int num_kb = (a.n + kTcBK - 1) / kTcBK;

    if (threadIdx.x == 0) {
        s_abort = 0;
        s_nonfinite = 0;
        for (int s = 0; s < kTcStages; ++s) {
            mbar_init(full + s, 1);
            mbar_init(empty + s, 1);
        }
        mbar_init(accf, 1);
        mbar_init(accf + 1, 1);
        mbar_init(acce, 8);
        mbar_init(acce + 1, 8);
        mbar_init(fin, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&map_a)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&map_b)) : "memory");
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
            mbar_wait(fin, 0);
        }
    } else {
        // epilogue: warp w (2..9) reads TMEM lanes 32*(w%4).. (tile rows) and
        // segment h = (w-2)/4 of the tile (columns 128h .. 128h+127)
        const int q = warp & 3;
        const int h = (warp - 2) >> 2;
        bool nonfinite = false;
        float zsum = 0.f;
        int j = 0;
        for (int t = blockIdx.x; t < num_tiles; t += gridDim.x, ++j) {
            const int acc = j & 1;
            const int mt = t / tiles_n, nt = t % tiles_n;
            const int seg = nt * 2 + h;                     // segment index within the row
            const int64_t row = (int64_t)mt * kTcBM + q * 32 + lane;
            const bool rv = row < a.m && seg < a.nt;
            // stored-weight bitmask and first stored entry of this segment: known before the MMA ends
            uint32_t ob[kFpTileWords];
            int32_t oidx = 0;
            const int wbase = seg * kFpTileWords;
#pragma unroll
            for (int c = 0; c < kFpTileWords; ++c)
                ob[c] = (rv && wbase + c < a.wpr) ? __ldg(a.obits + row * a.wpr + wbase + c) : 0u;
            if (rv) oidx = __ldg(a.ostart + row * (a.nt + 1) + seg);
            // old weights of word 0 in flight before waiting for the accumulator
            float wnext[32];
#pragma unroll
            for (int jj = 0; jj < 32; ++jj)
                wnext[jj] = ((ob[0] >> jj) & 1u) ? __ldg(a.old_val + oidx + __popc(ob[0] & ((1u << jj) - 1u))) : 0.f;
            const bool ok = __all_sync(0xffffffffu, mbar_wait_or_abort(accf + acc, (j >> 1) & 1, &s_abort));
            if (!ok) break;
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            float *stage = a.stage + (row * a.nt + seg) * kFpTileCols;
            uint32_t cnt = 0;
#pragma unroll
            for (int c = 0; c < kFpTileWords; ++c) {
                uint32_t r[32];
                tmem_ld_32cols(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * kTcBN + h * kFpTileCols + c * 32),
                               r);
                float w[32];
#pragma unroll
                for (int jj = 0; jj < 32; ++jj) w[jj] = wnext[jj];
                oidx += __popc(ob[c]);
                if (c + 1 < kFpTileWords) {   // next word's old weights in flight while this one is computed
                    const uint32_t on = ob[c + 1];
#pragma unroll
                    for (int jj = 0; jj < 32; ++jj)
                        wnext[jj] = ((on >> jj) & 1u) ? __ldg(a.old_val + oidx + __popc(on & ((1u << jj) - 1u))) : 0.f;
                }
                uint32_t kw = 0;
#pragma unroll
                for (int jj = 0; jj < 32; ++jj) {
                    const float z = __fsub_rn(w[jj], __fmul_rn(a.eta, __uint_as_float(r[jj])));
                    zsum += z;   // a NaN anywhere in z stays NaN in the sum
                    if (fabsf(z) > a.thr) {
                        kw |= 1u << jj;
                        if (rv) stage[cnt] = __fsub_rn(z, copysignf(a.thr, z));
                        ++cnt;
                    }
                }
                if (rv && wbase + c < a.wpr) a.kbits[row * a.wpr + wbase + c] = kw;
            }
            if (rv) a.counts[row * a.nt + seg] = (int32_t)cnt;
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            __syncwarp();
            if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(acce + acc)) : "memory");
        }
        nonfinite = zsum != zsum;
        if (__any_sync(0xffffffffu, nonfinite) && lane == 0) s_nonfinite = 1;
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (threadIdx.x == 0) {
        if (s_abort) {
            dev_flag(a.hdr, CSRT_DEV_TIMEOUT);
            a.hdr->timeout_site = 5;
        }
        if (s_nonfinite) dev_flag(a.hdr, CSRT_DEV_NONFINITE);
    }
    if (warp == 1) {
        __syncwarp();
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(2 * kTcBN) : "memory");
    }
}

// 3. Per row: exclusive offsets of the segments (in place) and the row total.
__global__ void __launch_bounds__(256) fp_rowscan_kernel(int32_t *__restrict__ counts, int32_t m, int32_t nt,
                                                         int32_t *__restrict__ rowtot) {
    const int lane = threadIdx.x & 31;
    const int64_t r = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    if (r >= m) return;
    int32_t *c = counts + r * nt;
    int32_t run = 0;
    for (int t0 = 0; t0 < nt; t0 += 32) {
        const int t = t0 + lane;
        const int32_t v = t < nt ? c[t] : 0;
        int32_t incl = v;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const int32_t u = __shfl_up_sync(0xffffffffu, incl, off);
            if (lane >= off) incl += u;
        }
        if (t < nt) c[t] = run + incl - v;
        run += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) rowtot[r] = run;
}

// 4. One warp per (row, tile): final positions, one coalesced run per word.
__global__ void __launch_bounds__(256) fp_place_kernel(int32_t m, int32_t k, int32_t nt, int32_t wpr,
                                                       const int32_t *__restrict__ row_ptr,
                                                       const int32_t *__restrict__ toff,
                                                       const uint32_t *__restrict__ kbits,
                                                       const float *__restrict__ stage, int32_t *__restrict__ out_col,
                                                       float *__restrict__ out_val, int32_t *__restrict__ wordpos,
                                                       int64_t capacity) {
    const int lane = threadIdx.x & 31;
    const int64_t gw = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    if (gw >= (int64_t)m * nt) return;
    const int64_t r = gw / nt;
    const int t = (int)(gw % nt);
    const int64_t base = (int64_t)row_ptr[r] + toff[r * nt + t];
    const float *sv = stage + (r * nt + t) * kFpTileCols;
    int32_t pre = 0;
    const unsigned lt = (1u << lane) - 1u;
    for (int c = 0; c < kFpTileWords; ++c) {
        const int wi = t * kFpTileWords + c;
        if (wi >= wpr) break;
        const uint32_t kw = __ldg(kbits + r * wpr + wi);
        if (wordpos && lane == 0) wordpos[r * wpr + wi] = (int32_t)imin<int64_t>(base + pre, capacity);
        if ((kw >> lane) & 1u) {
            const int32_t idx = pre + __popc(kw & lt);
            const int64_t p = base + idx;
            if (p < capacity) {
                out_col[p] = t * kFpTileCols + c * 32 + lane;
                out_val[p] = __ldg(sv + idx);
            }
        }
        pre += __popc(kw);
    }
}

__global__ void fp_finish_kernel(const int32_t *__restrict__ row_ptr, int32_t m, int64_t capacity,
                                 int32_t *__restrict__ out_row_ptr, WsHeader *hdr) {
    // row pointers clamped to the capacity, overflow reported
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i <= m; i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t v = row_ptr[i];
        out_row_ptr[i] = (int32_t)imin<int64_t>(v, capacity);
        if (i == m && v > capacity) {
            dev_flag(hdr, CSRT_DEV_CAPACITY);
            atomicMax(&hdr->required, (unsigned long long)v);
        }
    }
}

int scan_exclusive_i32(const int32_t *in, int32_t n, int32_t *out, cudaStream_t s);

}  // namespace csrt

using namespace csrt;

extern "C" int weight_grad_prox_update(const csrt_csr *w_in, const float *dy, const float *x, int32_t n, float eta,
                                       float lambda, int32_t precision, float *g_scratch, csrt_csr *w_out, void *ws,
                                       size_t ws_bytes, void *stream) {
    CSRT_ARG(w_in && w_out, "csr is NULL");
    const int32_t m = w_in->rows, k = w_in->cols;
    CSRT_ARG(w_out->rows == m && w_out->cols == k, "w_in and w_out shapes differ");
    CSRT_ARG(m >= 0 && k >= 0 && n >= 0, "negative size");
    CSRT_ARG((int64_t)m * k < ((int64_t)1 << 31), "rows*cols must be below 2^31");
    CSRT_ARG(precision == CSRT_PREC_FP32 || precision == CSRT_PREC_TF32, "unknown precision %d", precision);
    CSRT_ARG(eta >= 0.f && lambda >= 0.f && eta <= 3.0e38f && lambda <= 3.0e38f,
             "eta and lambda must be finite and >= 0");
    CSRT_ARG(w_in->row_ptr != w_out->row_ptr && w_in->col_idx != w_out->col_idx && w_in->val != w_out->val,
             "w_out must not alias w_in");
    CSRT_ARG(ws != nullptr, "workspace is NULL");
    cudaStream_t s = as_stream(stream);
    const bool want_t = w_out->t_row_ptr != nullptr;
    if (want_t) CSRT_ARG(w_out->t_col_idx && w_out->t_val && w_out->t_pos, "transposed arrays partly set");

    const bool fused = precision == CSRT_PREC_TF32 && device_is_sm10x() && n > 0 && n % 4 == 0 && m >= 64 &&
                       k >= 64 && k % 32 == 0 && k <= kFpMaxK && dy && x &&
                       ((reinterpret_cast<uintptr_t>(dy) | reinterpret_cast<uintptr_t>(x)) & 15) == 0 &&
                       ws_bytes >= kWsHeaderBytes + fused_prox_scratch_bytes(m, k);
    if (!fused) {
        CSRT_ARG(g_scratch != nullptr, "this shape/precision needs g_scratch (M x K floats) for the unfused path");
        int rc = weight_grad_dense(dy, x, m, k, n, g_scratch, precision, ws, ws_bytes, stream);
        if (rc) return rc;
        return prox_update_compact(w_in, g_scratch, eta, lambda, w_out, ws, ws_bytes, stream);
    }
    const float thr = eta * lambda;   // fl32(eta*lambda), the threshold of Eq. prox
    const FpLayout L = fp_layout(m, k);
    char *base = ws_scratch(ws);
    uint32_t *obits = reinterpret_cast<uint32_t *>(base + L.off_obits);
    int32_t *ostart = reinterpret_cast<int32_t *>(base + L.off_ostart);
    uint32_t *kbits = reinterpret_cast<uint32_t *>(base + L.off_kbits);
    int32_t *counts = reinterpret_cast<int32_t *>(base + L.off_counts);
    int32_t *rowtot = reinterpret_cast<int32_t *>(base + L.off_rowtot);
    float *stage = reinterpret_cast<float *>(base + L.off_stage);
    int32_t *wordpos = reinterpret_cast<int32_t *>(base + L.off_wordpos);

    CUtensorMap ma, mb;
    CSRT_ARG(make_map(&ma, dy, m, n, kTcBM) && make_map(&mb, x, k, n, kTcBN), "tensor map encoding failed");
    static bool attr_set[64] = {false};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !attr_set[dev]) {
        CSRT_CHECK_CUDA(
            cudaFuncSetAttribute(gemm_prox_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kTcSmemBytes));
        attr_set[dev] = true;
    }
    fp_oldbits_kernel<<<(unsigned)ceil_div<int64_t>(m, 8), 256, 0, s>>>(w_in->row_ptr, w_in->col_idx, m, L.wpr, L.nt,
                                                                        obits, ostart);
    FpArgs a;
    a.m = m;
    a.k = k;
    a.n = n;
    a.nt = L.nt;
    a.wpr = L.wpr;
    a.eta = eta;
    a.thr = thr;
    a.obits = obits;
    a.ostart = ostart;
    a.old_val = w_in->val;
    a.kbits = kbits;
    a.counts = counts;
    a.stage = stage;
    a.hdr = static_cast<WsHeader *>(ws);
    const int tiles_m = (int)ceil_div<int64_t>(m, kTcBM), tiles_n = (int)ceil_div<int64_t>(k, kTcBN);
    const int tiles = tiles_m * tiles_n;
    gemm_prox_tc_kernel<<<imin(tiles, num_sms()), kFpThreads, kTcSmemBytes, s>>>(ma, mb, a, tiles_n, tiles);
    fp_rowscan_kernel<<<(unsigned)ceil_div<int64_t>((int64_t)m * 32, 256), 256, 0, s>>>(counts, m, L.nt, rowtot);
    count_launch(3);
    // new row pointers: exclusive scan of the row totals (int32: nnz <= M*K < 2^31)
    int rc = scan_exclusive_i32(rowtot, m, w_out->row_ptr, s);
    if (rc) return rc;
    fp_place_kernel<<<(unsigned)ceil_div<int64_t>((int64_t)m * L.nt * 32, 256), 256, 0, s>>>(
        m, k, L.nt, L.wpr, w_out->row_ptr, counts, kbits, stage, w_out->col_idx, w_out->val, want_t ? wordpos : nullptr,
        w_out->capacity);
    fp_finish_kernel<<<1, 256, 0, s>>>(w_out->row_ptr, m, w_out->capacity, w_out->row_ptr, static_cast<WsHeader *>(ws));
    count_launch(2);
    rc = check_launch("fused weight-gradient + prox kernels");
    if (rc) return rc;
    if (want_t) rc = transpose_from_bits_ext(w_out, kbits, wordpos, base + L.off_tr, L.total - L.off_tr, s);
    return rc;
}
