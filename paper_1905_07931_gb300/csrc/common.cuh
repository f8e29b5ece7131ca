// Internal helpers shared by the CUDA translation units of libcsrtrain.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "csrtrain.h"

namespace csrt {

// ---------------------------------------------------------------------------
// Workspace header: the first 256 bytes of every workspace.
// ---------------------------------------------------------------------------
struct WsHeader {
    unsigned int flags;             // CSRT_DEV_* bits, OR-ed by kernels
    unsigned int invalid_row;       // csrt_validate_csr: 0xffffffff - first invalid row (0: none)
    unsigned long long required;    // largest nnz an overflowing output needed
    unsigned int ticket;            // tile ticket of the running compaction
    unsigned int timeout_site;      // last wait that gave up (diagnostics)
    unsigned int pad1[58];
};
static_assert(sizeof(WsHeader) == 256, "workspace header is 256 bytes");
constexpr size_t kWsHeaderBytes = 256;
// After the header, counters of the SpMM carry protocol (a unit that finishes
// a row shared with other units counts in; the last one completes the row).
// Zeroed by csrt_workspace_init and left zero by every call; no call uses
// them as scratch.
constexpr size_t kWsCounterInts = 16384;
constexpr size_t kWsReservedBytes = kWsHeaderBytes + kWsCounterInts * sizeof(int32_t);

inline char *ws_scratch(void *ws) { return static_cast<char *>(ws) + kWsReservedBytes; }
inline int32_t *ws_counters(void *ws) {
    return reinterpret_cast<int32_t *>(static_cast<char *>(ws) + kWsHeaderBytes);
}

// Bounded spin: a wait on another block's flag gives up after this many
// polls (with nanosleep back-off it is far above any legitimate wait) and
// reports CSRT_DEV_TIMEOUT instead of hanging.
constexpr unsigned int kSpinLimit = 1u << 22;

__device__ __forceinline__ void dev_flag(WsHeader *h, unsigned int bits) {
    atomicOr(&h->flags, bits);
}

// ---------------------------------------------------------------------------
// Host-side error reporting
// ---------------------------------------------------------------------------
int fail(int code, const char *fmt, ...);
int check_launch(const char *what);
void count_launch(int n = 1);
int num_sms();   // SMs of the current device (cached per device)

#define CSRT_CHECK_CUDA(call)                                                   \
    do {                                                                        \
        cudaError_t e_ = (call);                                                \
        if (e_ != cudaSuccess)                                                  \
            return ::csrt::fail(CSRT_ERR_CUDA, "%s: %s", #call,                 \
                                cudaGetErrorString(e_));                        \
    } while (0)

#define CSRT_ARG(cond, ...)                                                     \
    do {                                                                        \
        if (!(cond)) return ::csrt::fail(CSRT_ERR_ARG, __VA_ARGS__);            \
    } while (0)

inline cudaStream_t as_stream(void *s) { return static_cast<cudaStream_t>(s); }

// Programmatic dependent launch. A kernel launched with launch_pdl may be
// scheduled while the kernel before it on the stream is finishing (its last
// blocks exiting and its writes being flushed), which hides the launch
// latency between consecutive kernels of a step. Every kernel therefore
// starts with pdl_enter(): griddepcontrol.wait returns once the previous
// kernel has completed and its writes are visible. Launched without the
// attribute, the instruction does nothing. (An explicit early
// launch_dependents, which would let the next kernel's blocks wait on the
// SMs during this kernel's last wave, measured slower on the training step.)
__device__ __forceinline__ void pdl_enter() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

template <typename... P, typename... A>
inline cudaError_t launch_pdl(void (*kernel)(P...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                              A &&...args) {
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<P>(args)...);
}

// ---------------------------------------------------------------------------
// Workspace sizes of the individual operations (bytes after the header).
// ---------------------------------------------------------------------------
size_t compact_scratch_bytes(int32_t rows, int32_t cols);
size_t transpose_scratch_bytes(int32_t rows, int32_t cols);
size_t spmm_scratch_bytes(int32_t max_n);
size_t sddmm_scratch_bytes(int64_t capacity, int32_t max_n);
size_t gemm_scratch_bytes(int32_t m, int32_t k, int32_t max_n);
size_t fused_prox_scratch_bytes(int32_t rows, int32_t cols);

// Internal entry used by csr_from_dense / prox_update_compact.
int transpose_impl(csrt_csr *w, void *ws, size_t ws_bytes, cudaStream_t s);

// ---------------------------------------------------------------------------
// Device helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ unsigned long long ld_acquire_u64(const unsigned long long *p) {
    unsigned long long v;
    asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ void st_release_u64(unsigned long long *p, unsigned long long v) {
    asm volatile("st.release.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

__device__ __forceinline__ float4 ldg_f4(const float *p) {
    return __ldg(reinterpret_cast<const float4 *>(p));
}

__device__ __forceinline__ float4 ld_stream_f4(const float *p) {
    float4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.f32 {%0,%1,%2,%3}, [%4];"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "l"(p));
    return v;
}

template <typename T>
__host__ __device__ __forceinline__ T imin(T a, T b) {
    return a < b ? a : b;
}
template <typename T>
__host__ __device__ __forceinline__ T imax(T a, T b) {
    return a < b ? b : a;
}

template <typename T>
__host__ __device__ __forceinline__ T ceil_div(T a, T b) {
    return (a + b - 1) / b;
}

// Transpose of a 32 x 32 bit matrix held one word per lane (bit j of lane i
// is element (i, j)): on return bit i of lane j is element (i, j). Five rounds,
// each exchanging half-blocks with the lane whose index differs in one bit.
__device__ __forceinline__ uint32_t warp_transpose32(uint32_t x) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int sft = 16; sft >= 1; sft >>= 1) {
        const uint32_t lo = sft == 16 ? 0x0000FFFFu : sft == 8 ? 0x00FF00FFu : sft == 4 ? 0x0F0F0F0Fu
                          : sft == 2 ? 0x33333333u : 0x55555555u;
        const uint32_t other = __shfl_xor_sync(0xffffffffu, x, sft);
        if ((lane & sft) == 0) x = (x & lo) | ((other & lo) << sft);
        else x = (x & ~lo) | ((other & ~lo) >> sft);
    }
    return x;
}

// Exclusive scan of n int32 values into out[0..n] (out[n] = the total) by one
// block of 1024 threads, each taking a contiguous run; with out_clamped also
// the same values clamped to `capacity`, a total above it reported in hdr
// (CSRT_DEV_CAPACITY and the needed count).
__device__ __forceinline__ void scan_block_1024(const int32_t *__restrict__ in, int32_t n, int32_t *__restrict__ out,
                                                int32_t *__restrict__ out_clamped, int64_t capacity, WsHeader *hdr) {
    __shared__ int32_t s_warp[32];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int per = (n + 1023) / 1024;
    const int i0 = min(n, tid * per), i1 = min(n, i0 + per);
    int32_t local = 0;
    for (int i = i0; i < i1; ++i) local += in[i];
    int32_t incl = local;
    for (int off = 1; off < 32; off <<= 1) {
        int32_t y = __shfl_up_sync(0xffffffffu, incl, off);
        if (lane >= off) incl += y;
    }
    if (lane == 31) s_warp[warp] = incl;
    __syncthreads();
    int32_t wp = 0, total = 0;
    for (int w = 0; w < 32; ++w) {
        if (w < warp) wp += s_warp[w];
        total += s_warp[w];
    }
    int32_t run = incl - local + wp;
    for (int i = i0; i < i1; ++i) {
        out[i] = run;
        if (out_clamped) out_clamped[i] = (int32_t)(run < capacity ? run : capacity);
        run += in[i];
    }
    if (tid == 0) {
        out[n] = total;
        if (out_clamped) {
            out_clamped[n] = (int32_t)(total < capacity ? total : capacity);
            if (total > capacity) {
                dev_flag(hdr, CSRT_DEV_CAPACITY);
                atomicMax(&hdr->required, (unsigned long long)total);
            }
        }
    }
}

// Block bx of a column scan over 32-row blocks, 256 threads (8 warps x 32
// columns): for columns 32bx .. 32bx+31, the per-block counts cnt[b][j]
// (nb x cols) become their exclusive prefix down the column, coltot[j] the
// column's total.
__device__ __forceinline__ void colscan_block(int32_t *__restrict__ cnt, int32_t nb, int32_t cols,
                                              int32_t *__restrict__ coltot, int bx) {
    __shared__ int32_t seg[8][32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int j = bx * 32 + lane;
    const int b0 = (int)(((int64_t)nb * warp) / 8), b1 = (int)(((int64_t)nb * (warp + 1)) / 8);
    int32_t sum = 0;
    if (j < cols)
        for (int b = b0; b < b1; ++b) sum += cnt[(int64_t)b * cols + j];
    seg[warp][lane] = sum;
    __syncthreads();
    int32_t run = 0;
    for (int w = 0; w < warp; ++w) run += seg[w][lane];
    if (j < cols) {
        for (int b = b0; b < b1; ++b) {
            int32_t *p = cnt + (int64_t)b * cols + j;
            const int32_t v = *p;
            *p = run;
            run += v;
        }
        if (warp == 7) coltot[j] = run;
    }
}

// First index in [lo, hi) where the monotone predicate (true ... true,
// false ... false) is false, or hi. All 32 lanes of a warp call it and get the
// same answer after about log32(hi - lo) rounds of one probe per lane.
template <typename Pred>
__device__ __forceinline__ int64_t warp_first_false(int64_t lo, int64_t hi, Pred pred) {
    const int lane = threadIdx.x & 31;
    int64_t len = hi - lo;
    while (len > 32) {
        const int64_t idx = lo + ((int64_t)(lane + 1) * len) / 32 - 1;  // last of chunk `lane`
        const int l = __popc(__ballot_sync(0xffffffffu, pred(idx)));
        if (l == 32) return hi;
        const int64_t nlo = lo + ((int64_t)l * len) / 32;
        hi = lo + ((int64_t)(l + 1) * len) / 32;
        lo = nlo;
        len = hi - lo;
    }
    const int64_t idx = lo + lane;
    const bool p = idx < hi && pred(idx);
    return lo + __popc(__ballot_sync(0xffffffffu, p));
}

// Bounded wait for the phase with the given parity of an mbarrier in shared
// memory (a bulk copy's completion): false if it gave up after kSpinLimit
// polls, backing off after the first few. Callers flag CSRT_DEV_TIMEOUT.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t *bar, uint32_t parity) {
    const uint32_t addr = (uint32_t)__cvta_generic_to_shared(bar);
    for (unsigned i = 0; i < kSpinLimit; ++i) {
        uint32_t done;
        asm volatile(
            "{\n .reg .pred p;\n mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n"
            " selp.u32 %0, 1, 0, p;\n}\n"
            : "=r"(done)
            : "r"(addr), "r"(parity)
            : "memory");
        if (done) return true;
        if (i > 16) __nanosleep(32);
    }
    return false;
}

// Two independent searches of warp_first_false, run round by round together
// so that the latencies of their probes overlap (each round issues both
// probes before either ballot). Results in ra and rb.
template <typename PredA, typename PredB>
__device__ __forceinline__ void warp_first_false2(int64_t lo_a, int64_t hi_a, PredA pred_a, int64_t lo_b,
                                                  int64_t hi_b, PredB pred_b, int64_t &ra, int64_t &rb) {
    const int lane = threadIdx.x & 31;
    bool done_a = false, done_b = false;
    ra = hi_a;
    rb = hi_b;
    while (true) {
        const int64_t len_a = hi_a - lo_a, len_b = hi_b - lo_b;
        const bool wa = !done_a && len_a > 32, wb = !done_b && len_b > 32;   // warp-uniform
        if (!wa && !wb) break;
        const int64_t ia = lo_a + ((int64_t)(lane + 1) * len_a) / 32 - 1;
        const int64_t ib = lo_b + ((int64_t)(lane + 1) * len_b) / 32 - 1;
        const bool pa = wa && pred_a(ia);
        const bool pb = wb && pred_b(ib);
        const int la = __popc(__ballot_sync(0xffffffffu, pa));
        const int lb = __popc(__ballot_sync(0xffffffffu, pb));
        if (wa) {
            if (la == 32) {
                done_a = true;
            } else {
                const int64_t nlo = lo_a + ((int64_t)la * len_a) / 32;
                hi_a = lo_a + ((int64_t)(la + 1) * len_a) / 32;
                lo_a = nlo;
            }
        }
        if (wb) {
            if (lb == 32) {
                done_b = true;
            } else {
                const int64_t nlo = lo_b + ((int64_t)lb * len_b) / 32;
                hi_b = lo_b + ((int64_t)(lb + 1) * len_b) / 32;
                lo_b = nlo;
            }
        }
    }
    const bool pa = !done_a && lo_a + lane < hi_a && pred_a(lo_a + lane);
    const bool pb = !done_b && lo_b + lane < hi_b && pred_b(lo_b + lane);
    const int la = __popc(__ballot_sync(0xffffffffu, pa));
    const int lb = __popc(__ballot_sync(0xffffffffu, pb));
    if (!done_a) ra = lo_a + la;
    if (!done_b) rb = lo_b + lb;
}

// First position p in [s, e) with col[p] >= target (col ascending in [s, e)).
__device__ __forceinline__ int64_t warp_lower_bound(const int32_t *__restrict__ col, int64_t s, int64_t e,
                                                    int32_t target) {
    return warp_first_false(s, e, [&](int64_t p) { return __ldg(col + p) < target; });
}

}  // namespace csrt
