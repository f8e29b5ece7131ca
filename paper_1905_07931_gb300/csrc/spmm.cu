// Sparse x dense products of the training step.
//
// spmm_fwd   Y = W X         Section 3.2.1 (dense x compressed', forward)
// spmm_bwd_t dX = W^T dY     Section 3.2.2 (dense x compressed, backward),
//                            run as the same kernel over the transposed arrays
// weight_grad_sddmm          gradient at the stored entries (Section 2.4)
// debias_update              SGD on the stored entries (Section 2.4, 4.3)
//
// Design (GB300): one warp per work unit. The rows and nonzeros of the CSR
// are split evenly with a merge-path partition (row ends merged with nonzero
// indices, Merrill & Garland), so a unit owns the same amount of work whether
// rows are uniform or power-law. The n columns of the dense operand are cut
// into tiles of 32*VW*NV floats; each lane holds NV vectors of VW floats, so
// one nonzero costs every lane NV 16-byte loads of X and 4*NV FMAs, and a
// warp moves 512*NV contiguous bytes per nonzero. Column indices and values
// are loaded 32 at a time, coalesced, and broadcast with shuffles; four
// nonzeros are in flight per lane. A row cut by a unit boundary leaves a
// partial sum ("carry") in the workspace; the carries of each cut row are
// added in unit order (by the last of the row's units to finish, counted in
// the workspace, or by a fix-up kernel), so the result is deterministic and
// no float atomics are used. Narrow products (n <= 16 floats per vector width) put a
// group of G < 32 lanes on each nonzero instead (spmm_group_kernel), and the
// SDDMM uses the same grouped layout.
#include <mutex>

#include "common.cuh"

namespace csrt {

constexpr int kSpThreads = 256;
constexpr int kWarpsPerSM = 32;   // units requested per SM

template <int VW> struct Vec;
template <> struct Vec<1> { using T = float; };
template <> struct Vec<2> { using T = float2; };
template <> struct Vec<4> { using T = float4; };

template <int VW>
__device__ __forceinline__ typename Vec<VW>::T ldv(const float *p) {
    return __ldg(reinterpret_cast<const typename Vec<VW>::T *>(p));
}
template <int VW>
__device__ __forceinline__ void stv(float *p, const float (&a)[VW]) {
    if constexpr (VW == 4) *reinterpret_cast<float4 *>(p) = make_float4(a[0], a[1], a[2], a[3]);
    else if constexpr (VW == 2) *reinterpret_cast<float2 *>(p) = make_float2(a[0], a[1]);
    else *p = a[0];
}
template <int VW>
__device__ __forceinline__ void unpack(const typename Vec<VW>::T &v, float (&a)[VW]) {
    if constexpr (VW == 4) { a[0] = v.x; a[1] = v.y; a[2] = v.z; a[3] = v.w; }
    else if constexpr (VW == 2) { a[0] = v.x; a[1] = v.y; }
    else a[0] = v;
}

// Number of row ends the merge path has consumed at diagonal d: the smallest
// i in [lo, hi) with row_ptr[i+1] + i >= d, else hi (Merrill & Garland's
// merge-path search with row ends as one list and nonzero indices as the
// other).
__device__ __forceinline__ int merge_rows_before(const int32_t *__restrict__ row_ptr, int64_t d, int64_t lo,
                                                 int64_t hi) {
    return (int)warp_first_false(lo, hi, [&](int64_t i) { return (int64_t)__ldg(row_ptr + i + 1) + i < d; });
}
// The rows before diagonals d0 and d1 (a unit's start and end), both
// searches run together.
__device__ __forceinline__ void merge_rows_before2(const int32_t *__restrict__ row_ptr, int32_t rows, int64_t nnz,
                                                   int64_t d0, int64_t d1, int &i0, int &i1) {
    int64_t r0, r1;
    warp_first_false2(
        imax<int64_t>(0, d0 - nnz), imin<int64_t>(d0, rows),
        [&](int64_t i) { return (int64_t)__ldg(row_ptr + i + 1) + i < d0; }, imax<int64_t>(0, d1 - nnz),
        imin<int64_t>(d1, rows), [&](int64_t i) { return (int64_t)__ldg(row_ptr + i + 1) + i < d1; }, r0, r1);
    i0 = (int)r0;
    i1 = (int)r1;
}

struct SpmmArgs {
    const int32_t *row_ptr;
    const int32_t *col;
    const float *val;
    int32_t rows;
    const float *x;
    int32_t n;
    float *y;
    int32_t units;    // merge-path units per n-tile
    int32_t n_tiles;
    float *carry;     // [n_tiles][units][TN]
    int32_t *carry_row;  // [units]
    int32_t *cnt;     // [n_tiles][units] counters of the shared rows (zero between calls), or null: fix-up kernel
    // optional epilogue on each finished row i: + bias[i], then ReLU, then
    // zero where mask[i, c] <= 0 (the ReLU backward of the layer below)
    const float *bias;
    int32_t relu;
    const float *mask;
    WsHeader *hdr;    // status word for a bounded wait that gives up (null: not reported)
};

// The epilogue of one row segment held by a lane (VW floats at column c).
template <int VW>
__device__ __forceinline__ void spmm_epilogue(const SpmmArgs &a, int64_t row, int c, float (&v)[VW]) {
    if (a.bias) {
        const float b = __ldg(a.bias + row);
#pragma unroll
        for (int e = 0; e < VW; ++e) v[e] = __fadd_rn(v[e], b);
    }
    if (a.relu) {
#pragma unroll
        for (int e = 0; e < VW; ++e) v[e] = fmaxf(v[e], 0.f);
    }
    if (a.mask) {
        const float *mp = a.mask + row * a.n + c;
#pragma unroll
        for (int e = 0; e < VW; ++e)
            if (!(__ldg(mp + e) > 0.f)) v[e] = 0.f;
    }
}

template <int VW, int NV>
__device__ __forceinline__ void spmm_consume(const SpmmArgs &a, int64_t k, int64_t kend, int n0,
                                             float (&acc)[NV][VW]) {
    const int lane = threadIdx.x & 31;
    constexpr int kStride = 32 * VW;
    bool in_n[NV];
#pragma unroll
    for (int v = 0; v < NV; ++v) in_n[v] = n0 + v * kStride < a.n;
    for (int64_t kb = k; kb < kend; kb += 32) {
        const int cnt = (int)imin<int64_t>(32, kend - kb);
        int my_c = 0;
        float my_w = 0.f;
        if (lane < cnt) {
            my_c = __ldg(a.col + kb + lane);
            my_w = __ldg(a.val + kb + lane);
        }
        int q = 0;
        for (; q + 4 <= cnt; q += 4) {
            int c[4];
            float w[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                c[u] = __shfl_sync(0xffffffffu, my_c, q + u);
                w[u] = __shfl_sync(0xffffffffu, my_w, q + u);
            }
            typename Vec<VW>::T xv[4][NV];
#pragma unroll
            for (int u = 0; u < 4; ++u)
#pragma unroll
                for (int v = 0; v < NV; ++v)
                    if (in_n[v]) xv[u][v] = ldv<VW>(a.x + (int64_t)c[u] * a.n + n0 + v * kStride);
#pragma unroll
            for (int u = 0; u < 4; ++u)
#pragma unroll
                for (int v = 0; v < NV; ++v)
                    if (in_n[v]) {
                        float f[VW];
                        unpack<VW>(xv[u][v], f);
#pragma unroll
                        for (int e = 0; e < VW; ++e) acc[v][e] = fmaf(w[u], f[e], acc[v][e]);
                    }
        }
        for (; q < cnt; ++q) {
            const int c = __shfl_sync(0xffffffffu, my_c, q);
            const float w = __shfl_sync(0xffffffffu, my_w, q);
#pragma unroll
            for (int v = 0; v < NV; ++v)
                if (in_n[v]) {
                    float f[VW];
                    unpack<VW>(ldv<VW>(a.x + (int64_t)c * a.n + n0 + v * kStride), f);
#pragma unroll
                    for (int e = 0; e < VW; ++e) acc[v][e] = fmaf(w, f[e], acc[v][e]);
                }
        }
    }
}

// Row r, cut between units ua..ub of the merge path (its first nonzero lies
// in unit ua, its end in unit ub): every one of them counts in after writing
// its part (ub the partial row in Y, the others their carries); the last to
// arrive adds the carries in unit order to the partial row, applies the
// epilogue and resets the counter. The sum is the fix-up kernel's, in the
// same order; no unit waits for another.
// G is the number of lanes that hold one row segment (32, or the group width
// of the narrow kernel): lane gl < G holds the tile columns gl*VW + v*G*VW.
template <int VW, int NV, int G = 32>
__device__ __forceinline__ void spmm_complete_shared_row(const SpmmArgs &a, int r, int64_t per, int t, int n0) {
    constexpr int TN = G * VW * NV;
    constexpr int kStride = G * VW;
    const int lane = threadIdx.x & 31;
    const int gl = lane % G;
    const int64_t d0 = (int64_t)__ldg(a.row_ptr + r) + r, d1 = (int64_t)__ldg(a.row_ptr + r + 1) + r;
    const int ua = (int)(d0 / per), ub = (int)(d1 / per);
    __threadfence();   // this unit's part is visible before it counts in
    __syncwarp();
    int last = 0;
    if (lane == 0) last = atomicAdd(a.cnt + (int64_t)t * a.units + ua, 1) == ub - ua;
    if (!__shfl_sync(0xffffffffu, last, 0)) return;
    __threadfence();   // the others' parts are visible to the last one
#pragma unroll
    for (int v = 0; v < NV; ++v) {
        const int c = n0 + v * kStride;
        if (lane >= G || c >= a.n) continue;
        float sum[VW];
#pragma unroll
        for (int e = 0; e < VW; ++e) sum[e] = 0.f;
        for (int w = ua; w < ub; ++w) {
            const float *cp = a.carry + ((int64_t)t * a.units + w) * TN + gl * VW + v * kStride;
#pragma unroll
            for (int e = 0; e < VW; ++e) sum[e] += __ldcg(cp + e);
        }
        float *yp = a.y + (int64_t)r * a.n + c;
        float out[VW];
#pragma unroll
        for (int e = 0; e < VW; ++e) out[e] = __ldcg(yp + e) + sum[e];
        if (a.bias || a.relu || a.mask) spmm_epilogue<VW>(a, r, c, out);
        stv<VW>(yp, out);
    }
    if (lane == 0) a.cnt[(int64_t)t * a.units + ua] = 0;
}

template <int VW, int NV>
__global__ void __launch_bounds__(kSpThreads, 3) spmm_merge_kernel(SpmmArgs a) {
    pdl_enter();
    constexpr int TN = 32 * VW * NV;
    constexpr int kStride = 32 * VW;
    const int lane = threadIdx.x & 31;
    const int64_t gw = ((int64_t)blockIdx.x * kSpThreads + threadIdx.x) >> 5;
    if (gw >= (int64_t)a.units * a.n_tiles) return;
    const int u = (int)(gw % a.units);
    const int t = (int)(gw / a.units);
    const int64_t nnz = __ldg(a.row_ptr + a.rows);
    const int64_t items = (int64_t)a.rows + nnz;
    const int64_t per = ceil_div<int64_t>(items, a.units);
    const int64_t d0 = min((int64_t)u * per, items), d1 = min(d0 + per, items);
    const int i0 = merge_rows_before(a.row_ptr, d0, imax<int64_t>(0, d0 - nnz), imin<int64_t>(d0, a.rows));
    const int i1 = merge_rows_before(a.row_ptr, d1, imax<int64_t>(0, d1 - nnz), imin<int64_t>(d1, a.rows));
    const int64_t k0 = d0 - i0, k1 = d1 - i1;
    const int n0 = t * TN + lane * VW;

    float acc[NV][VW];
#pragma unroll
    for (int v = 0; v < NV; ++v)
#pragma unroll
        for (int e = 0; e < VW; ++e) acc[v][e] = 0.f;

    // a row that began in an earlier unit receives carries; the fix-up applies its epilogue
    const bool first_row_cut = i0 < a.rows && k0 > __ldg(a.row_ptr + i0);
    const bool epi = a.bias || a.relu || a.mask;
    int64_t k = k0;
    for (int i = i0; i < i1; ++i) {
        const int64_t kend = __ldg(a.row_ptr + i + 1);
        spmm_consume<VW, NV>(a, k, kend, n0, acc);
        k = kend;
        float *yrow = a.y + (int64_t)i * a.n + n0;
        const bool apply = epi && !(i == i0 && first_row_cut);
#pragma unroll
        for (int v = 0; v < NV; ++v) {
            if (n0 + v * kStride < a.n) {
                if (apply) spmm_epilogue<VW>(a, i, n0 + v * kStride, acc[v]);
                stv<VW>(yrow + v * kStride, acc[v]);
            }
#pragma unroll
            for (int e = 0; e < VW; ++e) acc[v][e] = 0.f;
        }
    }
    spmm_consume<VW, NV>(a, k, k1, n0, acc);
    const bool has_carry = k1 > k;
    if (a.units > 1) {
        if (t == 0 && lane == 0) a.carry_row[u] = has_carry ? i1 : -1;
        if (has_carry) {
            float *cp = a.carry + ((int64_t)t * a.units + u) * TN + lane * VW;
#pragma unroll
            for (int v = 0; v < NV; ++v) stv<VW>(cp + v * kStride, acc[v]);
        }
        if (a.cnt) {
            // the rows this unit shares with others: the first (begun in an
            // earlier unit) and the last (going on in a later one); one row
            // when the unit lies inside a single row
            const int ra = first_row_cut ? i0 : -1;
            const int rb = (has_carry && i1 != ra) ? i1 : -1;
            if (ra >= 0) spmm_complete_shared_row<VW, NV>(a, ra, per, t, n0);
            if (rb >= 0) spmm_complete_shared_row<VW, NV>(a, rb, per, t, n0);
        }
    }
}

// ---------------------------------------------------------------------------
// Narrow products (n <= 16*VW): G lanes per nonzero.
//
// With all 32 lanes on one nonzero, a narrow product leaves most lanes idle
// (n = 1: one lane in 32) and keeps only a few loads in flight, so it runs
// far below the HBM rate that its CSR stream could reach. Here a group of
// G lanes (G*VW >= n) takes one nonzero, so a warp step covers E = 32/G
// nonzeros and a batch of U steps B = U*E nonzeros, cut at row ends. The
// column indices and values arrive ahead of their use through a per-warp
// ring of chunks in shared memory filled by bulk asynchronous copies (see
// below). At the end of a row the groups' partial sums are
// combined by a butterfly over the lane bits above G. The unit split, the
// row-end window and the shared-row protocol are those of spmm_merge_kernel
// (carries of TN = G*VW floats).
// ---------------------------------------------------------------------------
template <int VW> struct NarrowSteps { static constexpr int value = VW == 1 ? 8 : 4; };
constexpr int kNarrowChunk = 256;   // entries per ring chunk
constexpr int kNarrowStages = 4;    // ring chunks per warp
constexpr int kNarrowRingInts = 2 * kNarrowStages * kNarrowChunk;   // per warp: indices, then values
constexpr int kNarrowSmem = (kSpThreads / 32) * (kNarrowRingInts * (int)sizeof(int32_t) + kNarrowStages * 8);

__device__ __forceinline__ uint32_t sp_smem_addr(const void *p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}
// One bulk asynchronous copy global -> shared (16-byte aligned, a multiple of
// 16 bytes) that completes on the mbarrier bar.
__device__ __forceinline__ void sp_bulk_copy(void *dst, const void *src, uint32_t bytes, uint64_t *bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                     sp_smem_addr(dst)),
                 "l"(src), "r"(bytes), "r"(sp_smem_addr(bar))
                 : "memory");
}

template <int VW, int G>
__global__ void __launch_bounds__(kSpThreads, 3) spmm_group_kernel(SpmmArgs a) {
    pdl_enter();
    constexpr int E = 32 / G;
    constexpr int U = NarrowSteps<VW>::value;
    constexpr int B = U * E;
    constexpr int TN = G * VW;
    const int lane = threadIdx.x & 31, grp = lane / G, gl = lane % G;
    const int64_t gw = ((int64_t)blockIdx.x * kSpThreads + threadIdx.x) >> 5;
    if (gw >= (int64_t)a.units * a.n_tiles) return;
    const int u = (int)(gw % a.units);
    const int t = (int)(gw / a.units);
    const int64_t nnz = __ldg(a.row_ptr + a.rows);
    const int64_t items = (int64_t)a.rows + nnz;
    const int64_t per = ceil_div<int64_t>(items, a.units);
    const int64_t d0 = min((int64_t)u * per, items), d1 = min(d0 + per, items);
    int i0, i1;
    merge_rows_before2(a.row_ptr, a.rows, nnz, d0, d1, i0, i1);
    const int64_t k0 = d0 - i0, k1 = d1 - i1;
    const int c0 = t * TN + gl * VW;
    const bool in_n = c0 < a.n;
    const bool first_row_cut = i0 < a.rows && k0 > __ldg(a.row_ptr + i0);
    const bool epi = a.bias || a.relu || a.mask;

    // ends of rows wb .. wb+31 (one per lane); rows from i1 on end at k1 here
    int wb = i0;
    int64_t rpl = wb + lane < i1 ? (int64_t)__ldg(a.row_ptr + wb + lane + 1) : k1;
    auto row_end = [&](int r) -> int64_t {
        if (r >= i1) return k1;
        if (r - wb >= 32) {
            wb = r;
            rpl = wb + lane < i1 ? (int64_t)__ldg(a.row_ptr + wb + lane + 1) : k1;
        }
        return __shfl_sync(0xffffffffu, rpl, r - wb);
    };

    float acc[VW];
#pragma unroll
    for (int e = 0; e < VW; ++e) acc[e] = 0.f;
    // the groups' partial sums of one row, summed over the lane bits above G
    auto combine = [&](float (&v)[VW]) {
#pragma unroll
        for (int e = 0; e < VW; ++e) {
            v[e] = acc[e];
#pragma unroll
            for (int off = G; off < 32; off <<= 1) v[e] += __shfl_xor_sync(0xffffffffu, v[e], off);
            acc[e] = 0.f;
        }
    };

    int i = i0;
    int64_t e_row = row_end(i);
    int64_t kr = k0;   // first entry of the current row inside this unit
    auto finish_rows = [&](int64_t kb) {   // rows that end at or before kb are complete
        while (i < i1 && e_row <= kb) {
            float v[VW];
            combine(v);
            if (grp == 0 && in_n) {
                if (epi && !(i == i0 && first_row_cut)) spmm_epilogue<VW>(a, i, c0, v);
                stv<VW>(a.y + (int64_t)i * a.n + c0, v);
            }
            kr = e_row;
            ++i;
            e_row = row_end(i);
        }
    };
    // The unit's column indices and values stream through a ring of
    // kNarrowStages chunks of kNarrowChunk entries in shared memory (this
    // warp's slice): lane 0 starts one bulk copy per array and chunk,
    // kNarrowStages - 1 chunks ahead of the one being consumed, so the bytes
    // in flight cost neither registers nor per-entry copy instructions.
    // Chunks start at 16-byte boundaries (abase = k0 rounded down to 4
    // entries); the last 0-3 entries of the unit past a boundary, which a
    // bulk copy of whole 16-byte units could only cover by reading beyond
    // k1, are loaded by plain loads.
    extern __shared__ __align__(16) int32_t narrow_smem[];
    const int wib = threadIdx.x >> 5;
    int32_t *ring_c = narrow_smem + wib * kNarrowRingInts;
    float *ring_v = reinterpret_cast<float *>(ring_c + kNarrowStages * kNarrowChunk);
    uint64_t *bars = reinterpret_cast<uint64_t *>(narrow_smem + (kSpThreads / 32) * kNarrowRingInts) +
                     wib * kNarrowStages;
    if (lane == 0) {
#pragma unroll
        for (int q = 0; q < kNarrowStages; ++q)
            asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(sp_smem_addr(bars + q)) : "memory");
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncwarp();
    const int64_t abase = k0 & ~int64_t(3);
    const int64_t k1a = k1 & ~int64_t(3);
    bool failed = false;
    auto issue = [&](int64_t j) {   // chunk j: entries abase + j*C .. + C, clipped to k1
        const int64_t A = abase + j * kNarrowChunk;
        if (A >= k1) return;
        const int slot = (int)(j % kNarrowStages) * kNarrowChunk;
        const int64_t fe = imin<int64_t>(A + kNarrowChunk, k1a);
        const uint32_t nb = fe > A ? (uint32_t)(fe - A) * 4u : 0u;
        const int64_t t0 = imax<int64_t>(A, k1a), t1 = imin<int64_t>(A + kNarrowChunk, k1);
        if (lane < t1 - t0) {
            ring_c[slot + (int)(t0 - A) + lane] = __ldg(a.col + t0 + lane);
            ring_v[slot + (int)(t0 - A) + lane] = __ldg(a.val + t0 + lane);
        }
        if (lane == 0) {
            uint64_t *bar = bars + j % kNarrowStages;
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(sp_smem_addr(bar)),
                         "r"(2u * nb)
                         : "memory");
            if (nb) {
                sp_bulk_copy(ring_c + slot, a.col + A, nb, bar);
                sp_bulk_copy(ring_v + slot, a.val + A, nb, bar);
            }
        }
    };
#pragma unroll
    for (int q = 0; q < kNarrowStages - 1; ++q) issue(q);
    for (int64_t j = 0;; ++j) {
        const int64_t A = abase + j * kNarrowChunk;
        if (A >= k1) break;
        issue(j + kNarrowStages - 1);
        if (!mbar_wait_bounded(bars + j % kNarrowStages, (uint32_t)((j / kNarrowStages) & 1))) failed = true;
        __syncwarp();
        const int slot = (int)(j % kNarrowStages) * kNarrowChunk;
        const int64_t ce = imin<int64_t>(A + kNarrowChunk, k1);
        for (int64_t kb = imax<int64_t>(A, k0); kb < ce;) {
            finish_rows(kb);
            const int64_t kn = imin<int64_t>(imin<int64_t>(kb + B, e_row), ce);
            const int rem = in_n ? (int)(kn - kb - grp) : 0;
            const int off = slot + (int)(kb - A) + grp;
            int c[U];
            float w[U];
#pragma unroll
            for (int st = 0; st < U; ++st)
                if (st * E < rem) {
                    c[st] = ring_c[off + st * E];
                    w[st] = ring_v[off + st * E];
                }
            typename Vec<VW>::T xv[U];
#pragma unroll
            for (int st = 0; st < U; ++st)
                if (st * E < rem) xv[st] = ldv<VW>(a.x + (int64_t)c[st] * a.n + c0);
#pragma unroll
            for (int st = 0; st < U; ++st)
                if (st * E < rem) {
                    float f[VW];
                    unpack<VW>(xv[st], f);
#pragma unroll
                    for (int e = 0; e < VW; ++e) acc[e] = fmaf(w[st], f[e], acc[e]);
                }
            kb = kn;
        }
        __syncwarp();   // the slot is read before the copy issued next refills it
    }
    finish_rows(k1);
    if (failed && lane == 0 && a.hdr) {
        dev_flag(a.hdr, CSRT_DEV_TIMEOUT);
        a.hdr->timeout_site = 10;
    }
    // the unit ends inside row i1: its part is a carry
    const bool has_carry = k1 > kr;
    float v[VW];
    combine(v);
    if (a.units > 1) {
        if (t == 0 && lane == 0) a.carry_row[u] = has_carry ? i1 : -1;
        if (has_carry && grp == 0) stv<VW>(a.carry + ((int64_t)t * a.units + u) * TN + gl * VW, v);
        if (a.cnt) {
            const int ra = first_row_cut ? i0 : -1;
            const int rb = (has_carry && i1 != ra) ? i1 : -1;
            if (ra >= 0) spmm_complete_shared_row<VW, 1, G>(a, ra, per, t, c0);
            if (rb >= 0) spmm_complete_shared_row<VW, 1, G>(a, rb, per, t, c0);
        }
    }
}

// Adds the carries of every cut row, in unit order, to that row of Y. One warp
// per (unit, n-tile): warps whose unit is not the first carry of its row leave
// at once; the first one sums the row's carries column by column.
template <int TN>
__global__ void __launch_bounds__(256) spmm_fixup_kernel(SpmmArgs a) {
    pdl_enter();
    const int64_t gw = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (gw >= (int64_t)a.units * a.n_tiles) return;
    const int t = (int)(gw / a.units);
    const int u = (int)(gw % a.units);
    const int r = a.carry_row[u];
    if (r < 0 || (u > 0 && a.carry_row[u - 1] == r)) return;  // not the first carry of its row
    int last = u;
    while (last + 1 < a.units && a.carry_row[last + 1] == r) ++last;
    const bool epi = a.bias || a.relu || a.mask;
    // lane j holds columns j, j+32, ...: every carry's loads for them are
    // independent, so they are issued together, carry by carry in unit order
    // (tiles narrower than a warp use lanes j < TN)
    constexpr int kPer = (TN + 31) / 32;
    float sum[kPer];
#pragma unroll
    for (int q = 0; q < kPer; ++q) sum[q] = 0.f;
    for (int v = u; v <= last; ++v) {
        const float *cp = a.carry + ((int64_t)t * a.units + v) * TN + lane;
#pragma unroll
        for (int q = 0; q < kPer; ++q)
            if (lane + 32 * q < TN) sum[q] += __ldg(cp + 32 * q);
    }
#pragma unroll
    for (int q = 0; q < kPer; ++q) {
        const int col = t * TN + lane + 32 * q;
        if (lane + 32 * q >= TN || col >= a.n) break;
        float *yp = a.y + (int64_t)r * a.n + col;
        float out[1] = {*yp + sum[q]};
        if (epi) spmm_epilogue<1>(a, r, col, out);
        *yp = out[0];
    }
}

struct SpmmShape {
    int vw, nv, g, tn, n_tiles, units;
};

// Resident warps per SM of a kernel with `smem` bytes of dynamic shared
// memory (cached per device); above 48 KB the kernel is first allowed that
// much, once per device, which its launches rely on.
template <typename K>
static int kernel_warps_per_sm(K kernel, int (&cache)[64], int cap, size_t smem = 0) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return cap;
    if (cache[dev] == 0) {
        if (smem > 48 * 1024) cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        int blocks = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&blocks, kernel, kSpThreads, smem) != cudaSuccess ||
            blocks <= 0)
            blocks = cap / (kSpThreads / 32);
        cache[dev] = imin(blocks * (kSpThreads / 32), cap);
    }
    return cache[dev];
}

template <int VW, int NV, int G>
static int spmm_warps_per_sm() {
    static int cache[64] = {0};
    if constexpr (G == 32) return kernel_warps_per_sm(spmm_merge_kernel<VW, NV>, cache, kWarpsPerSM);
    else return kernel_warps_per_sm(spmm_group_kernel<VW, G>, cache, kWarpsPerSM, (size_t)kNarrowSmem);
}

static int pow2_at_least(int v) {
    int p = 1;
    while (p < v) p <<= 1;
    return p;
}

// Tile shape of a product with n columns: 32 lanes on one nonzero with NV
// vectors of VW floats each (n >= 128 for float4, 64 for float2, 32 for
// scalars), else the narrow kernel with G = the smallest power of two with
// G*VW >= n lanes per nonzero. The narrow kernel streams the index and value
// arrays with bulk copies, which need them 16-byte aligned (csr16); without
// that the 32-lane kernel takes narrow products too.
static SpmmShape spmm_shape(int32_t n, int64_t max_items, bool vec4_ok, bool vec2_ok, bool csr16) {
    SpmmShape s;
    s.nv = 1;
    s.g = 32;
    if (vec4_ok && n >= 128) { s.vw = 4; s.nv = n >= 256 ? 2 : 1; }
    else if (vec4_ok && n <= 64) { s.vw = 4; s.g = pow2_at_least((n + 3) / 4); }
    else if (vec2_ok && n >= 64) { s.vw = 2; }
    else if (vec2_ok && n <= 32) { s.vw = 2; s.g = pow2_at_least((n + 1) / 2); }
    else if (n <= 16) { s.vw = 1; s.g = pow2_at_least(n); }
    else { s.vw = 1; }
    if (!csr16) s.g = 32;
    s.tn = s.g * s.vw * s.nv;
    s.n_tiles = (int)ceil_div<int64_t>(n, s.tn);
    // one full wave of resident warps (a partial second wave would run at low occupancy)
    int wps = kWarpsPerSM;
#define CSRT_SPMM_WPS(VW, NV, G) \
    if (s.vw == VW && s.nv == NV && s.g == G) wps = spmm_warps_per_sm<VW, NV, G>();
    CSRT_SPMM_WPS(4, 2, 32) CSRT_SPMM_WPS(4, 1, 32) CSRT_SPMM_WPS(2, 1, 32) CSRT_SPMM_WPS(1, 1, 32)
    CSRT_SPMM_WPS(4, 1, 1) CSRT_SPMM_WPS(4, 1, 2) CSRT_SPMM_WPS(4, 1, 4) CSRT_SPMM_WPS(4, 1, 8) CSRT_SPMM_WPS(4, 1, 16)
    CSRT_SPMM_WPS(2, 1, 1) CSRT_SPMM_WPS(2, 1, 2) CSRT_SPMM_WPS(2, 1, 4) CSRT_SPMM_WPS(2, 1, 8) CSRT_SPMM_WPS(2, 1, 16)
    CSRT_SPMM_WPS(1, 1, 1) CSRT_SPMM_WPS(1, 1, 2) CSRT_SPMM_WPS(1, 1, 4) CSRT_SPMM_WPS(1, 1, 8) CSRT_SPMM_WPS(1, 1, 16)
#undef CSRT_SPMM_WPS
    const int64_t target = (int64_t)num_sms() * wps;
    int64_t units = ceil_div<int64_t>(target, s.n_tiles);
    units = imax<int64_t>(1, imin<int64_t>(units, max_items));
    s.units = (int)units;
    return s;
}

size_t spmm_scratch_bytes(int32_t max_n) {
    // units * n_tiles <= target + n_tiles, TN <= 256: carries plus carry rows.
    const int64_t target = (int64_t)num_sms() * kWarpsPerSM;
    const int64_t floats = (target + 1) * 256 + (int64_t)max_n + 256;
    return (size_t)floats * sizeof(float) + (size_t)(target + 1) * sizeof(int32_t) + 512;
}

// Launches the product kernel of shape sh (and, for rows cut by units when
// a.cnt is null, the fix-up kernel); returns the number of launches, or -1
// for a shape without a kernel.
static int spmm_dispatch(const SpmmShape &sh, const SpmmArgs &a, cudaStream_t s) {
    const int64_t threads = (int64_t)sh.units * sh.n_tiles * 32;
    const unsigned grid = (unsigned)ceil_div<int64_t>(threads, kSpThreads);
    const bool fix = sh.units > 1 && a.cnt == nullptr;
    const unsigned fg = (unsigned)ceil_div<int64_t>(threads, 256);
#define CSRT_SPMM_CASE(VW, NV, G, KERNEL)                                                   \
    if (sh.vw == VW && sh.nv == NV && sh.g == G) {                                          \
        launch_pdl(KERNEL, dim3(grid), dim3(kSpThreads), G < 32 ? (size_t)kNarrowSmem : 0, s, a);           \
        if (fix) launch_pdl(spmm_fixup_kernel<G * VW * NV>, dim3(fg), dim3(256), 0, s, a); \
        return fix ? 2 : 1;                                                                 \
    }
    CSRT_SPMM_CASE(4, 2, 32, (spmm_merge_kernel<4, 2>))
    CSRT_SPMM_CASE(4, 1, 32, (spmm_merge_kernel<4, 1>))
    CSRT_SPMM_CASE(2, 1, 32, (spmm_merge_kernel<2, 1>))
    CSRT_SPMM_CASE(1, 1, 32, (spmm_merge_kernel<1, 1>))
    CSRT_SPMM_CASE(4, 1, 1, (spmm_group_kernel<4, 1>))
    CSRT_SPMM_CASE(4, 1, 2, (spmm_group_kernel<4, 2>))
    CSRT_SPMM_CASE(4, 1, 4, (spmm_group_kernel<4, 4>))
    CSRT_SPMM_CASE(4, 1, 8, (spmm_group_kernel<4, 8>))
    CSRT_SPMM_CASE(4, 1, 16, (spmm_group_kernel<4, 16>))
    CSRT_SPMM_CASE(2, 1, 1, (spmm_group_kernel<2, 1>))
    CSRT_SPMM_CASE(2, 1, 2, (spmm_group_kernel<2, 2>))
    CSRT_SPMM_CASE(2, 1, 4, (spmm_group_kernel<2, 4>))
    CSRT_SPMM_CASE(2, 1, 8, (spmm_group_kernel<2, 8>))
    CSRT_SPMM_CASE(2, 1, 16, (spmm_group_kernel<2, 16>))
    CSRT_SPMM_CASE(1, 1, 1, (spmm_group_kernel<1, 1>))
    CSRT_SPMM_CASE(1, 1, 2, (spmm_group_kernel<1, 2>))
    CSRT_SPMM_CASE(1, 1, 4, (spmm_group_kernel<1, 4>))
    CSRT_SPMM_CASE(1, 1, 8, (spmm_group_kernel<1, 8>))
    CSRT_SPMM_CASE(1, 1, 16, (spmm_group_kernel<1, 16>))
#undef CSRT_SPMM_CASE
    return -1;
}

static int spmm_launch(const int32_t *row_ptr, const int32_t *col, const float *val, int32_t rows,
                       int64_t capacity, const float *x, int32_t n, float *y, void *ws, size_t ws_bytes,
                       cudaStream_t s, const float *bias = nullptr, int32_t relu = 0, const float *mask = nullptr) {
    if (rows == 0 || n == 0) return CSRT_OK;
    const bool v4 = (n % 4 == 0) && ((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(y)) & 15) == 0;
    const bool v2 = (n % 2 == 0) && ((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(y)) & 7) == 0;
    const bool csr16 = ((reinterpret_cast<uintptr_t>(col) | reinterpret_cast<uintptr_t>(val)) & 15) == 0;
    const SpmmShape sh = spmm_shape(n, (int64_t)rows + capacity, v4, v2, csr16);
    SpmmArgs a;
    a.row_ptr = row_ptr;
    a.col = col;
    a.val = val;
    a.rows = rows;
    a.x = x;
    a.n = n;
    a.y = y;
    a.units = sh.units;
    a.n_tiles = sh.n_tiles;
    a.bias = bias;
    a.relu = relu;
    a.mask = mask;
    a.hdr = static_cast<WsHeader *>(ws);
    const size_t carry_floats = (size_t)sh.units * sh.n_tiles * sh.tn;
    a.carry = reinterpret_cast<float *>(ws_scratch(ws));
    a.carry_row = reinterpret_cast<int32_t *>(a.carry + ((carry_floats + 63) / 64) * 64);
    a.cnt = nullptr;
    if (sh.units > 1) {
        const size_t need = kWsReservedBytes + ((carry_floats + 63) / 64) * 64 * sizeof(float) +
                            (size_t)sh.units * sizeof(int32_t);
        CSRT_ARG(ws != nullptr && ws_bytes >= need, "workspace too small for spmm (%zu < %zu)", ws_bytes, need);
        // wide products: rows shared by units are completed in the kernel by
        // the last unit to finish its part (more units than counters fall back
        // to the fix-up kernel). Narrow products take the fix-up kernel: their
        // units are short and nearly all share rows, and the fences of the
        // in-kernel completion cost more than the extra launch (27.6 vs 30.7
        // us at n = 1, 1-2 us at n = 8 and 32, on 4096 x 4096 at 50%)
        if (sh.g == 32 && (int64_t)sh.units * sh.n_tiles <= (int64_t)kWsCounterInts) a.cnt = ws_counters(ws);
    }
    const int launched = spmm_dispatch(sh, a, s);
    CSRT_ARG(launched > 0, "spmm: no kernel for shape vw=%d nv=%d g=%d", sh.vw, sh.nv, sh.g);
    count_launch(launched);
    return check_launch("spmm_merge_kernel");
}

// Column-index ring of the narrow SDDMM: chunks of kSdChunk entries copied
// with 4-byte cp.async, kSdStages - 1 chunks ahead.
constexpr int kSdChunk = 256;
constexpr int kSdStages = 3;

__device__ __forceinline__ void cp_async4(void *dst, const void *src) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"((uint32_t)__cvta_generic_to_shared(dst)), "l"(src)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

// ---------------------------------------------------------------------------
// SDDMM: g[k] = <dY[i_k, :], X[j_k, :]>
// ---------------------------------------------------------------------------
// Layout as in the narrow SpMM kernel: a group of G lanes (G*VW >= n, or
// G = 32 with NV vectors per lane and the n range walked in tiles of
// TN = 32*VW*NV) takes one stored entry, a warp step covers E = 32/G entries,
// and U steps form a batch whose column indices are requested before the
// previous batch is consumed. Every entry of a batch lies in one row, whose
// dY slice stays in registers for the whole row when one tile covers n (else
// it is reloaded once per batch and tile), so per entry only its row of X is
// read. The U dot products of a lane are finished together: the first
// log2(min(U, G)) butterfly steps over the group's lanes exchange halves of
// the U partial sums (a transposed reduction), the remaining steps add one
// value, and lane r*(G/R) of each group holds entry r's result. No partial
// buffers: the whole n range of an entry is summed in one warp, so the
// result does not depend on the unit split.
struct SddmmArgs {
    const int32_t *row_ptr;
    const int32_t *col;
    int32_t rows;
    const float *dy;
    const float *x;
    int32_t n;
    float *out;
    int32_t units;
};

// The row holding entry k: the largest i in [0, rows) with row_ptr[i] <= k.
__device__ __forceinline__ int row_of_entry(const int32_t *__restrict__ row_ptr, int32_t rows, int64_t k) {
    return (int)warp_first_false(1, rows, [&](int64_t i) { return (int64_t)__ldg(row_ptr + i) <= k; }) - 1;
}

// Sums each of the U values of a lane over the G lanes of its group. Values
// are taken in blocks of R = min(U, G): after the call, p[b*R] of lane gl
// holds the group's sum of value b*R + gl / (G/R).
template <int U, int G>
__device__ __forceinline__ void group_reduce_multi(float (&p)[U], int gl) {
    constexpr int R = U < G ? U : G;
#pragma unroll
    for (int b = 0; b < U / R; ++b) {
#pragma unroll
        for (int h = R / 2, off = G / 2; h >= 1; h >>= 1, off >>= 1) {
            const bool upper = (gl & off) != 0;
#pragma unroll
            for (int j = 0; j < h; ++j) {
                const float lo = p[b * R + j], hi = p[b * R + j + h];
                const float send = upper ? lo : hi;
                const float keep = upper ? hi : lo;
                p[b * R + j] = keep + __shfl_xor_sync(0xffffffffu, send, off);
            }
        }
#pragma unroll
        for (int off = G / (2 * R); off >= 1; off >>= 1) p[b * R] += __shfl_xor_sync(0xffffffffu, p[b * R], off);
    }
}

template <int VW, int NV, int G>
__global__ void __launch_bounds__(kSpThreads, 3) sddmm_kernel(SddmmArgs a) {
    pdl_enter();
    constexpr int E = 32 / G;
    constexpr int U = VW * NV >= 4 ? 4 : 8;
    constexpr int B = U * E;
    constexpr int TN = G * VW * NV, kStride = G * VW;
    constexpr int R = U < G ? U : G;
    const int lane = threadIdx.x & 31, grp = lane / G, gl = lane % G;
    const int64_t gw = ((int64_t)blockIdx.x * kSpThreads + threadIdx.x) >> 5;
    if (gw >= (int64_t)a.units) return;
    const int64_t nnz = __ldg(a.row_ptr + a.rows);
    const int64_t per = ceil_div<int64_t>(nnz, a.units);
    const int64_t k0 = min(gw * per, nnz), k1 = min(k0 + per, nnz);
    if (k0 >= k1) return;
    const int n_tiles = (int)ceil_div<int64_t>(a.n, TN);

    int row = row_of_entry(a.row_ptr, a.rows, k0);
    int wb = row;
    int64_t rpl = wb + lane < a.rows ? (int64_t)__ldg(a.row_ptr + wb + lane + 1) : nnz;
    auto row_end = [&](int r) -> int64_t {
        if (r - wb >= 32) {
            wb = r;
            rpl = wb + lane < a.rows ? (int64_t)__ldg(a.row_ptr + wb + lane + 1) : nnz;
        }
        return __shfl_sync(0xffffffffu, rpl, r - wb);
    };
    float dyv[NV][VW];
    auto load_dy = [&](int r, int tt) {
#pragma unroll
        for (int v = 0; v < NV; ++v) {
            const int c = tt * TN + gl * VW + v * kStride;
            if (c < a.n) unpack<VW>(ldv<VW>(a.dy + (int64_t)r * a.n + c), dyv[v]);
            else {
#pragma unroll
                for (int e = 0; e < VW; ++e) dyv[v][e] = 0.f;
            }
        }
    };
    int cn[U];
    auto fetch = [&](int64_t kb) {
        const int32_t *cp = a.col + kb + grp;
        const int lim = (int)imin<int64_t>(k1 - kb - grp, B);
#pragma unroll
        for (int s = 0; s < U; ++s) cn[s] = s * E < lim ? __ldg(cp + s * E) : 0;
    };

    int64_t e_row = row_end(row);
    if (n_tiles == 1) load_dy(row, 0);
    if constexpr (G > 1 && G < 32) {
        // 2..16 lanes per entry (one tile covers n): the unit's column indices
        // stream through a per-warp cp.async ring of kSdStages chunks of
        // kSdChunk entries, two chunks ahead of the one being consumed
        extern __shared__ __align__(16) int32_t sddmm_smem[];
        int32_t *ring = sddmm_smem + (threadIdx.x >> 5) * (kSdStages * kSdChunk);
        auto issue = [&](int64_t cs) {
            if (cs < k1) {
                const int slot = (int)(((cs - k0) / kSdChunk) % kSdStages) * kSdChunk;
#pragma unroll
                for (int q = 0; q < kSdChunk / 32; ++q) {
                    const int64_t idx = cs + q * 32 + lane;
                    if (idx < k1) cp_async4(ring + slot + q * 32 + lane, a.col + idx);
                }
            }
            cp_async_commit();
        };
#pragma unroll
        for (int q = 0; q < kSdStages - 1; ++q) issue(k0 + (int64_t)q * kSdChunk);
        for (int64_t cs = k0; cs < k1; cs += kSdChunk) {
            issue(cs + (int64_t)(kSdStages - 1) * kSdChunk);
            cp_async_wait<kSdStages - 1>();
            __syncwarp();
            const int slot = (int)(((cs - k0) / kSdChunk) % kSdStages) * kSdChunk;
            const int64_t ce = imin<int64_t>(cs + kSdChunk, k1);
            for (int64_t kb = cs; kb < ce;) {
                while (e_row <= kb) {   // the row holding entry kb (empty rows are passed over)
                    ++row;
                    e_row = row_end(row);
                    load_dy(row, 0);
                }
                const int64_t kn = imin<int64_t>(imin<int64_t>(kb + B, e_row), ce);
                const int rem = (int)(kn - kb - grp);
                const int off = slot + (int)(kb - cs) + grp;
                bool ok[U];
                int c[U];
                float p[U];
#pragma unroll
                for (int st = 0; st < U; ++st) {
                    ok[st] = st * E < rem;
                    c[st] = ok[st] ? ring[off + st * E] : 0;
                    p[st] = 0.f;
                }
                typename Vec<VW>::T xv[U][NV];
#pragma unroll
                for (int st = 0; st < U; ++st)
#pragma unroll
                    for (int v = 0; v < NV; ++v) {
                        const int col = gl * VW + v * kStride;
                        if (ok[st] && col < a.n) xv[st][v] = ldv<VW>(a.x + (int64_t)c[st] * a.n + col);
                    }
#pragma unroll
                for (int st = 0; st < U; ++st)
#pragma unroll
                    for (int v = 0; v < NV; ++v) {
                        const int col = gl * VW + v * kStride;
                        if (ok[st] && col < a.n) {
                            float f[VW];
                            unpack<VW>(xv[st][v], f);
#pragma unroll
                            for (int e = 0; e < VW; ++e) p[st] = fmaf(dyv[v][e], f[e], p[st]);
                        }
                    }
                group_reduce_multi<U, G>(p, gl);
                if (gl % (G / R) == 0) {
                    float *op = a.out + kb + grp;
                    const int r = gl / (G / R);
#pragma unroll
                    for (int b = 0; b < U / R; ++b) {
                        const int st = b * R + r;
                        if (st * E < rem) op[st * E] = p[b * R];
                    }
                }
                kb = kn;
            }
            __syncwarp();   // the slot is read before the copy issued next refills it
        }
        cp_async_wait<0>();
        return;
    }
    int64_t kb = k0;
    fetch(kb);
    while (kb < k1) {
        while (e_row <= kb) {   // the row holding entry kb (empty rows are passed over)
            ++row;
            e_row = row_end(row);
            if (n_tiles == 1) load_dy(row, 0);
        }
        int c[U];
#pragma unroll
        for (int s = 0; s < U; ++s) c[s] = cn[s];
        // the batch ends at the row's end or at the unit's, whichever is first
        const int64_t e_cur = imin<int64_t>(e_row, k1);
        const int64_t kn = imin<int64_t>(kb + B, e_cur);
        if (kn < k1) fetch(kn);
        const int rem = (int)imin<int64_t>(e_cur - kb - grp, B);
        bool ok[U];
#pragma unroll
        for (int s = 0; s < U; ++s) ok[s] = s * E < rem;
        float p[U];
#pragma unroll
        for (int s = 0; s < U; ++s) p[s] = 0.f;
        for (int tt = 0; tt < n_tiles; ++tt) {
            if (n_tiles > 1) load_dy(row, tt);
            typename Vec<VW>::T xv[U][NV];
#pragma unroll
            for (int s = 0; s < U; ++s)
#pragma unroll
                for (int v = 0; v < NV; ++v) {
                    const int col = tt * TN + gl * VW + v * kStride;
                    if (ok[s] && col < a.n) xv[s][v] = ldv<VW>(a.x + (int64_t)c[s] * a.n + col);
                }
#pragma unroll
            for (int s = 0; s < U; ++s)
#pragma unroll
                for (int v = 0; v < NV; ++v) {
                    const int col = tt * TN + gl * VW + v * kStride;
                    if (ok[s] && col < a.n) {
                        float f[VW];
                        unpack<VW>(xv[s][v], f);
#pragma unroll
                        for (int e = 0; e < VW; ++e) p[s] = fmaf(dyv[v][e], f[e], p[s]);
                    }
                }
        }
        float *op = a.out + kb + grp;
        if constexpr (G == 1) {
#pragma unroll
            for (int s = 0; s < U; ++s)
                if (ok[s]) op[s * E] = p[s];
        } else {
            group_reduce_multi<U, G>(p, gl);
            if (gl % (G / R) == 0) {
                const int r = gl / (G / R);
#pragma unroll
                for (int b = 0; b < U / R; ++b) {
                    const int s = b * R + r;
                    if (s * E < rem) op[s * E] = p[b * R];
                }
            }
        }
        kb = kn;
    }
}

size_t sddmm_scratch_bytes(int64_t, int32_t) { return 0; }

}  // namespace csrt

using namespace csrt;

static int check_csr_basic(const csrt_csr *w) {
    CSRT_ARG(w != nullptr && w->row_ptr != nullptr, "csr or row_ptr is NULL");
    CSRT_ARG(w->rows >= 0 && w->cols >= 0, "negative shape");
    CSRT_ARG((int64_t)w->rows * w->cols < ((int64_t)1 << 31), "rows*cols must be below 2^31");
    CSRT_ARG(w->capacity >= 0 && w->capacity < ((int64_t)1 << 31), "capacity out of range");
    CSRT_ARG(w->capacity == 0 || (w->col_idx && w->val), "col_idx/val NULL");
    return CSRT_OK;
}

extern "C" {

int spmm_fwd(const csrt_csr *w, const float *x, int32_t n, float *y, void *ws, size_t ws_bytes, void *stream) {
    int rc = check_csr_basic(w);
    if (rc) return rc;
    CSRT_ARG(n >= 0, "n < 0");
    CSRT_ARG((x && y) || n == 0 || w->rows == 0, "X or Y is NULL");
    return spmm_launch(w->row_ptr, w->col_idx, w->val, w->rows, w->capacity, x, n, y, ws, ws_bytes,
                       as_stream(stream));
}

int spmm_bwd_t(const csrt_csr *w, const float *dy, int32_t n, float *dx, void *ws, size_t ws_bytes,
               void *stream) {
    int rc = check_csr_basic(w);
    if (rc) return rc;
    CSRT_ARG(w->t_row_ptr && w->t_col_idx && w->t_val, "transposed arrays not set");
    CSRT_ARG(n >= 0, "n < 0");
    CSRT_ARG((dy && dx) || n == 0 || w->cols == 0, "dY or dX is NULL");
    return spmm_launch(w->t_row_ptr, w->t_col_idx, w->t_val, w->cols, w->capacity, dy, n, dx, ws, ws_bytes,
                       as_stream(stream));
}

int spmm_fwd_bias_act(const csrt_csr *w, const float *x, int32_t n, const float *bias, int32_t relu, float *y,
                      void *ws, size_t ws_bytes, void *stream) {
    int rc = check_csr_basic(w);
    if (rc) return rc;
    CSRT_ARG(n >= 0, "n < 0");
    CSRT_ARG((x && y) || n == 0 || w->rows == 0, "X or Y is NULL");
    return spmm_launch(w->row_ptr, w->col_idx, w->val, w->rows, w->capacity, x, n, y, ws, ws_bytes,
                       as_stream(stream), bias, relu ? 1 : 0, nullptr);
}

int spmm_bwd_t_relu(const csrt_csr *w, const float *dy, int32_t n, const float *y_below, float *dx, void *ws,
                    size_t ws_bytes, void *stream) {
    int rc = check_csr_basic(w);
    if (rc) return rc;
    CSRT_ARG(w->t_row_ptr && w->t_col_idx && w->t_val, "transposed arrays not set");
    CSRT_ARG(n >= 0, "n < 0");
    CSRT_ARG((dy && dx && y_below) || n == 0 || w->cols == 0, "dY, dX or the mask is NULL");
    return spmm_launch(w->t_row_ptr, w->t_col_idx, w->t_val, w->cols, w->capacity, dy, n, dx, ws, ws_bytes,
                       as_stream(stream), nullptr, 0, y_below);
}

int weight_grad_sddmm(const csrt_csr *w, const float *dy, const float *x, int32_t n, float *g_nnz, void *ws,
                      size_t ws_bytes, void *stream) {
    int rc = check_csr_basic(w);
    if (rc) return rc;
    CSRT_ARG(n >= 0, "n < 0");
    if (w->rows == 0 || w->capacity == 0) return CSRT_OK;
    CSRT_ARG(g_nnz != nullptr, "g_nnz is NULL");
    cudaStream_t s = as_stream(stream);
    if (n == 0) {
        CSRT_CHECK_CUDA(cudaMemsetAsync(g_nnz, 0, sizeof(float) * (size_t)w->capacity, s));
        return CSRT_OK;
    }
    CSRT_ARG(dy && x, "dY or X is NULL");
    const bool v4 = (n % 4 == 0) && ((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(dy)) & 15) == 0;
    const bool v2 = (n % 2 == 0) && ((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(dy)) & 7) == 0;
    const int vw = v4 ? 4 : v2 ? 2 : 1;
    const int g = imin(32, pow2_at_least((n + vw - 1) / vw));
    const int nv = g == 32 && n > 32 * vw ? 2 : 1;
    SddmmArgs a;
    a.row_ptr = w->row_ptr;
    a.col = w->col_idx;
    a.rows = w->rows;
    a.dy = dy;
    a.x = x;
    a.n = n;
    a.out = g_nnz;
    static int cache[64][3][6][2];
    int dev = 0;
    CSRT_CHECK_CUDA(cudaGetDevice(&dev));
    CSRT_ARG(dev >= 0 && dev < 64, "device ordinal %d out of range", dev);
    int lg = 0;
    while ((1 << lg) < g) ++lg;
    int &wps = cache[dev][vw == 4 ? 2 : vw - 1][lg][nv - 1];
    void (*kern)(SddmmArgs) = nullptr;
#define CSRT_SDDMM_CASE(VW, NV, G) \
    if (vw == VW && nv == NV && g == G) kern = sddmm_kernel<VW, NV, G>;
    CSRT_SDDMM_CASE(4, 1, 1) CSRT_SDDMM_CASE(4, 1, 2) CSRT_SDDMM_CASE(4, 1, 4) CSRT_SDDMM_CASE(4, 1, 8)
    CSRT_SDDMM_CASE(4, 1, 16) CSRT_SDDMM_CASE(4, 1, 32) CSRT_SDDMM_CASE(4, 2, 32)
    CSRT_SDDMM_CASE(2, 1, 1) CSRT_SDDMM_CASE(2, 1, 2) CSRT_SDDMM_CASE(2, 1, 4) CSRT_SDDMM_CASE(2, 1, 8)
    CSRT_SDDMM_CASE(2, 1, 16) CSRT_SDDMM_CASE(2, 1, 32) CSRT_SDDMM_CASE(2, 2, 32)
    CSRT_SDDMM_CASE(1, 1, 1) CSRT_SDDMM_CASE(1, 1, 2) CSRT_SDDMM_CASE(1, 1, 4) CSRT_SDDMM_CASE(1, 1, 8)
    CSRT_SDDMM_CASE(1, 1, 16) CSRT_SDDMM_CASE(1, 1, 32) CSRT_SDDMM_CASE(1, 2, 32)
#undef CSRT_SDDMM_CASE
    CSRT_ARG(kern != nullptr, "sddmm: no kernel for vw=%d nv=%d g=%d", vw, nv, g);
    // 2..16 lanes per entry: the per-warp ring of column indices in shared memory
    const size_t smem = (g > 1 && g < 32) ? (size_t)(kSpThreads / 32) * kSdStages * kSdChunk * sizeof(int32_t) : 0;
    if (wps == 0) {
        int blocks = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&blocks, kern, kSpThreads, smem) != cudaSuccess ||
            blocks <= 0)
            blocks = kWarpsPerSM / (kSpThreads / 32);
        wps = imin(blocks * (kSpThreads / 32), kWarpsPerSM);
    }
    a.units = (int)imax<int64_t>(1, imin<int64_t>((int64_t)num_sms() * wps, w->capacity));
    const unsigned grid = (unsigned)ceil_div<int64_t>((int64_t)a.units * 32, kSpThreads);
    launch_pdl(kern, dim3(grid), dim3(kSpThreads), smem, s, a);
    count_launch();
    return check_launch("sddmm_kernel");
}

}  // extern "C"

namespace csrt {
__global__ void debias_kernel(const int32_t *__restrict__ row_ptr, int32_t rows, float *__restrict__ val,
                              const float *__restrict__ g, float eta, float *__restrict__ t_val,
                              const int32_t *__restrict__ t_pos) {
    pdl_enter();
    const int64_t nnz = __ldg(row_ptr + rows);
    for (int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; k < nnz; k += (int64_t)gridDim.x * blockDim.x) {
        const float nv = __fsub_rn(val[k], __fmul_rn(eta, __ldg(g + k)));
        val[k] = nv;
        if (t_val) t_val[__ldg(t_pos + k)] = nv;
    }
}
}  // namespace csrt

extern "C" int debias_update(csrt_csr *w, const float *g_nnz, float eta, void *stream) {
    int rc = check_csr_basic(w);
    if (rc) return rc;
    CSRT_ARG(!(eta < 0.f) && eta <= 3.0e38f, "eta must be finite and >= 0");
    if (w->rows == 0 || w->capacity == 0) return CSRT_OK;
    CSRT_ARG(g_nnz != nullptr, "g_nnz is NULL");
    CSRT_ARG(w->t_val == nullptr || w->t_pos != nullptr, "t_val set without t_pos");
    const unsigned grid = (unsigned)imax<int64_t>(1, imin<int64_t>(ceil_div<int64_t>(w->capacity, 256), (int64_t)num_sms() * 8));
    launch_pdl(debias_kernel, dim3(grid), dim3(256), 0, as_stream(stream), w->row_ptr, w->rows, w->val, g_nnz, eta,
               w->t_val, w->t_pos);
    count_launch();
    return check_launch("debias_kernel");
}

// ---------------------------------------------------------------------------
// spmm_fwd_noalloc: the forward product for callers that cannot allocate.
//
// spmm_fwd needs a caller-provided workspace for the partial sums of rows that
// straddle two merge-path units. Some callers cannot provide one: code that
// runs inside a host framework which owns every device allocation through its
// own pool and does not let plugins call cudaMalloc, or a tight serving loop
// where an allocation's latency and possible failure are not acceptable. This
// variant keeps that scratch in a fixed array in device global memory that the
// library declares itself, so the caller passes only inputs and outputs.
//
// Limits and rules:
//  * The product may have at most kNoAllocMaxN = 4096 columns (n); larger n
//    is rejected with CSRT_ERR_ARG. The array holds kNoAllocFloats = 2^21
//    floats of partial sums (8 MiB) and kNoAllocRows = 2^16 row slots
//    (256 KiB). A call needs (units x n_tiles) x tn floats, where units x
//    n_tiles is at most SMs x 32 + n_tiles and tn at most 256, so every
//    n <= 4096 fits on GPUs of up to 255 SMs (GB300 has 152); a shape that
//    does not fit is rejected the same way. Every GPU that loads the library
//    holds the array until the process exits.
//  * A 256-byte status word beside the array collects CSRT_DEV_TIMEOUT when a
//    bounded wait of the product gives up (the result is then invalid);
//    spmm_fwd_noalloc_status reads and optionally clears it.
//  * The first call of either entry point on a device looks up the device
//    addresses with cudaGetSymbolAddress (once per device, guarded by a
//    std::call_once, with that device current); make that first call before
//    any stream capture begins.
//  * All calls share the one array and it keeps the last call's contents.
//    The partial sums need no clearing: each launch writes every slot it
//    later reads. Calls whose kernels overlap on the GPU (two streams, or two
//    threads) race on the array and give wrong results; serialise them.
// ---------------------------------------------------------------------------
namespace csrt {
constexpr int32_t kNoAllocMaxN = 4096;
constexpr int64_t kNoAllocFloats = (int64_t)1 << 21;
constexpr int64_t kNoAllocRows = (int64_t)1 << 16;
constexpr int kNoAllocMaxDevices = 64;
static __device__ __align__(256) float g_noalloc_carry[kNoAllocFloats];
static __device__ __align__(256) int32_t g_noalloc_carry_row[kNoAllocRows];
static __device__ __align__(256) WsHeader g_noalloc_status;

struct NoAllocAddrs {
    float *carry = nullptr;
    int32_t *carry_row = nullptr;
    WsHeader *status = nullptr;
    cudaError_t err = cudaSuccess;
};
static NoAllocAddrs g_noalloc_addrs[kNoAllocMaxDevices];
static std::once_flag g_noalloc_once[kNoAllocMaxDevices];

// The device addresses of the static arrays on the current device, looked
// up once per device; returns nullptr (with the message set) on failure.
static const NoAllocAddrs *noalloc_addrs() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        fail(CSRT_ERR_CUDA, "cudaGetDevice failed");
        return nullptr;
    }
    if (dev < 0 || dev >= kNoAllocMaxDevices) {
        fail(CSRT_ERR_ARG, "device ordinal %d out of range", dev);
        return nullptr;
    }
    std::call_once(g_noalloc_once[dev], [dev] {
        NoAllocAddrs &a = g_noalloc_addrs[dev];
        void *p = nullptr, *q = nullptr, *r = nullptr;
        a.err = cudaGetSymbolAddress(&p, g_noalloc_carry);
        if (a.err == cudaSuccess) a.err = cudaGetSymbolAddress(&q, g_noalloc_carry_row);
        if (a.err == cudaSuccess) a.err = cudaGetSymbolAddress(&r, g_noalloc_status);
        if (a.err == cudaSuccess) {
            a.carry = static_cast<float *>(p);
            a.carry_row = static_cast<int32_t *>(q);
            a.status = static_cast<WsHeader *>(r);
        }
    });
    const NoAllocAddrs &a = g_noalloc_addrs[dev];
    if (a.err != cudaSuccess) {
        fail(CSRT_ERR_CUDA, "cudaGetSymbolAddress of the static scratch failed on device %d: %s", dev,
             cudaGetErrorString(a.err));
        return nullptr;
    }
    return &a;
}
}  // namespace csrt

extern "C" int spmm_fwd_noalloc(const csrt_csr *w, const float *x, int32_t n, float *y, void *stream) {
    int rc = check_csr_basic(w);
    if (rc) return rc;
    CSRT_ARG(n >= 0, "n < 0");
    CSRT_ARG(n <= kNoAllocMaxN, "spmm_fwd_noalloc: n = %d exceeds the maximum of %d columns of its static scratch",
             n, kNoAllocMaxN);
    CSRT_ARG((x && y) || n == 0 || w->rows == 0, "X or Y is NULL");
    if (w->rows == 0 || n == 0) return CSRT_OK;
    const NoAllocAddrs *na = noalloc_addrs();
    if (na == nullptr) return CSRT_ERR_CUDA;
    const bool v4 = (n % 4 == 0) && ((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(y)) & 15) == 0;
    const bool v2 = (n % 2 == 0) && ((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(y)) & 7) == 0;
    const bool csr16 =
        ((reinterpret_cast<uintptr_t>(w->col_idx) | reinterpret_cast<uintptr_t>(w->val)) & 15) == 0;
    const SpmmShape sh = spmm_shape(n, (int64_t)w->rows + w->capacity, v4, v2, csr16);
    const int64_t carry_floats = (int64_t)sh.units * sh.n_tiles * sh.tn;
    CSRT_ARG(sh.units == 1 || (carry_floats <= kNoAllocFloats && sh.units <= kNoAllocRows),
             "spmm_fwd_noalloc: n = %d needs %lld floats of static scratch, the maximum is %lld", n,
             (long long)carry_floats, (long long)kNoAllocFloats);
    SpmmArgs a;
    a.row_ptr = w->row_ptr;
    a.col = w->col_idx;
    a.val = w->val;
    a.rows = w->rows;
    a.x = x;
    a.n = n;
    a.y = y;
    a.units = sh.units;
    a.n_tiles = sh.n_tiles;
    a.carry = na->carry;
    a.carry_row = na->carry_row;
    a.cnt = nullptr;   // shared rows are completed by the fix-up kernel
    a.bias = nullptr;
    a.relu = 0;
    a.mask = nullptr;
    a.hdr = na->status;   // a bounded wait that gives up sets CSRT_DEV_TIMEOUT here
    const int launched = spmm_dispatch(sh, a, as_stream(stream));
    CSRT_ARG(launched > 0, "spmm_fwd_noalloc: no kernel for shape vw=%d nv=%d g=%d", sh.vw, sh.nv, sh.g);
    count_launch(launched);
    return check_launch("spmm_fwd_noalloc");
}

extern "C" int spmm_fwd_noalloc_status(int32_t *flags, int32_t clear, void *stream) {
    CSRT_ARG(flags != nullptr, "flags is NULL");
    const NoAllocAddrs *na = noalloc_addrs();
    if (na == nullptr) return CSRT_ERR_CUDA;
    cudaStream_t s = as_stream(stream);
    CSRT_CHECK_CUDA(cudaStreamSynchronize(s));
    unsigned int word = 0;
    CSRT_CHECK_CUDA(cudaMemcpy(&word, &na->status->flags, sizeof(word), cudaMemcpyDeviceToHost));
    *flags = (int32_t)word;
    if (clear) {
        CSRT_CHECK_CUDA(cudaMemsetAsync(na->status, 0, sizeof(WsHeader), s));
        CSRT_CHECK_CUDA(cudaStreamSynchronize(s));
    }
    return CSRT_OK;
}
