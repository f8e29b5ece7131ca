// CSR construction and the fused proximal update + re-compaction.
//
// csr_from_dense (Section 3.1) and prox_update_compact (Eq. prox with the
// soft threshold of Section 2.2, applied to the dense w - eta*G as in
// Section 3.3, compacted after every update as in Section 4.4) are the same
// stream compaction over the M*K entries in row-major order; they differ only
// in the predicate and the kept value.
//
// Design (GB300): the M*K matrix is viewed as one flat array cut into tiles
// of 4096 entries. One 256-thread block per tile streams its 16 KB of the
// dense input with 16-byte loads that bypass L1, evaluates the predicate,
// ranks the kept entries with a block scan, and learns the number of entries
// kept by all earlier tiles with a single-pass decoupled look-back
// (Merrill & Garland) over a per-tile status word. Tiles are numbered by an
// atomic ticket, so a block only ever waits on blocks that are already
// running; every wait is bounded and reports CSRT_DEV_TIMEOUT instead of
// hanging. The dense input is read once and the CSR written once, coalesced.
// For the prox step, the old CSR entries of the tile's flat range are
// contiguous in the old arrays; they are scattered into a shared-memory copy
// of the tile so that w is read once as well. The SGD prox on rows whose
// length is a multiple of 32 takes a variant in which only a tile keeping
// more than an eighth of its entries waits for its prefix: a sparser tile
// writes its entries to a stash and a later kernel copies them into place
// (see the row-tile kernels below).
//
// csr_transpose builds the column-wise copy of the pattern that Section 3.2.2
// asks for (entries ordered by column, then row) in four deterministic
// kernels: per 32-row block and column a bitmask of the rows present, a scan
// of the per-block counts down each column, a scan over the columns, and a
// scatter whose rank inside a block is a popcount of the bitmask.
#include <cmath>

#include "common.cuh"

namespace csrt {

constexpr int kCThreads = 256;
constexpr int kCQuads = 4;                           // float4 per thread
constexpr int kTile = kCThreads * kCQuads * 4;       // 4096 entries per tile
constexpr unsigned long long kFlagAgg = 1ull << 32;  // tile aggregate published
constexpr unsigned long long kFlagInc = 2ull << 32;  // inclusive prefix published

// Look-back status words: one per tile; flat tiles (4096 entries) are the
// smallest, so their count bounds every path.
static size_t status_bytes(int64_t elems) {
    return ((size_t)ceil_div<int64_t>(elems, kTile) * sizeof(unsigned long long) + 255) / 256 * 256;
}
// Keep-bitmask and word positions emitted by the prox kernel for the transposed copy.
static size_t bits_bytes(int32_t rows, int32_t cols) {
    return ((size_t)rows * (size_t)ceil_div<int32_t>(cols, 32) * sizeof(uint32_t) + 255) / 256 * 256;
}

size_t transpose_scratch_bytes(int32_t rows, int32_t cols);
static size_t prox_place_bytes(int32_t rows, int32_t cols);

// Scratch of csr_from_dense / prox_update_compact / csr_transpose.
size_t compact_scratch_bytes(int32_t rows, int32_t cols) {
    const int64_t elems = (int64_t)rows * cols;
    return status_bytes(elems) + 2 * bits_bytes(rows, cols) + transpose_scratch_bytes(rows, cols) +
           prox_place_bytes(rows, cols);
}

struct CompactArgs {
    const float *src;          // dense matrix (from-dense) or G (prox)
    int32_t rows, cols;
    int64_t elems;
    const int32_t *in_row_ptr;  // prox: old CSR
    const int32_t *in_col;
    const float *in_val;
    float eta, thr;
    int32_t *out_row_ptr;
    int32_t *out_col;
    float *out_val;
    int64_t capacity;
    WsHeader *hdr;
    unsigned long long *status;  // one word per tile
    int64_t num_tiles;
    // adaptive prox step (Algorithms 1 and 2): the gradient is replaced by a
    // search direction, the moment arrays (dense, like G) updated in place
    int32_t opt;                 // kOptSgd, kOptRmsprop, kOptAdam
    float *m, *v;
    float beta1, beta2, c1, c2, bc1, bc2, eps;
};

constexpr int32_t kOptSgd = 0, kOptRmsprop = 1, kOptAdam = 2;

// Moment updates and search direction of one adaptive step, every operation
// rounded once in the order of the definitions: RMSProp (Algorithm 1)
//   v' = fl(fl(beta2*v) + fl(c2*fl(g*g))),  d = fl(g / fl(fl(sqrt(v')) + eps));
// Adam (Algorithm 2) with c_i = fl(1 - beta_i), bc_i = fl(1 - beta_i^t)
//   m' = fl(fl(beta1*m) + fl(c1*g)),  v' as above,
//   d = fl(fl(m'/bc1) / fl(fl(sqrt(fl(v'/bc2))) + eps)).
__device__ __forceinline__ float opt_direction(const CompactArgs &a, float g, float &m, float &v) {
    v = __fadd_rn(__fmul_rn(a.beta2, v), __fmul_rn(a.c2, __fmul_rn(g, g)));
    if (a.opt == kOptRmsprop) return __fdiv_rn(g, __fadd_rn(__fsqrt_rn(v), a.eps));
    m = __fadd_rn(__fmul_rn(a.beta1, m), __fmul_rn(a.c1, g));
    return __fdiv_rn(__fdiv_rn(m, a.bc1), __fadd_rn(__fsqrt_rn(__fdiv_rn(v, a.bc2)), a.eps));
}

// Decoupled look-back for tile `tile`, run by one whole warp: publishes the
// tile's aggregate, sums predecessors' aggregates back to the nearest
// published inclusive prefix, publishes this tile's inclusive prefix and
// returns the exclusive prefix (the number of entries kept before the tile).
// Each round reads a window of 32 * kLbWays predecessors (kLbWays per lane),
// so inclusive prefixes propagate kLbWays times faster than with one word per
// lane. Every poll is bounded; a wait that runs out sets CSRT_DEV_TIMEOUT.
constexpr int kLbWays = 4;

__device__ __forceinline__ unsigned long long lookback_warp(unsigned long long *status, int64_t tile,
                                                            uint32_t count, WsHeader *hdr) {
    const int lane = threadIdx.x & 31;
    if (tile == 0) {
        if (lane == 0) st_release_u64(status, kFlagInc | count);
        return 0;
    }
    if (lane == 0) st_release_u64(status + tile, kFlagAgg | count);
    unsigned long long prefix = 0;
    int64_t pred = tile - 1;   // window entry (v, lane) is predecessor pred - 32 v - lane
    unsigned int spins = 0;
    bool timed_out = false;
    while (true) {
        unsigned long long st[kLbWays];
#pragma unroll
        for (int v = 0; v < kLbWays; ++v) {
            const int64_t idx = pred - 32 * v - lane;
            st[v] = idx >= 0 ? ld_acquire_u64(status + idx) : kFlagInc;
        }
        int first_v = kLbWays, first_lane = 32;   // nearest inclusive prefix in the window
        while (true) {
            first_v = kLbWays;
            first_lane = 32;
#pragma unroll
            for (int v = kLbWays - 1; v >= 0; --v) {
                const unsigned inc = __ballot_sync(0xffffffffu, (st[v] >> 32) == 2);
                if (inc) {
                    first_v = v;
                    first_lane = __ffs(inc) - 1;
                }
            }
            // every entry nearer than the inclusive one must have published its aggregate
            bool missing = false;
#pragma unroll
            for (int v = 0; v < kLbWays; ++v) {
                const bool nearer = v < first_v || (v == first_v && lane < first_lane);
                missing |= nearer && (st[v] >> 32) == 0;
            }
            if (!__any_sync(0xffffffffu, missing)) break;
            if (++spins > kSpinLimit) {
                timed_out = true;
                break;
            }
            __nanosleep(32);
#pragma unroll
            for (int v = 0; v < kLbWays; ++v) {
                const int64_t idx = pred - 32 * v - lane;
                if ((st[v] >> 32) == 0 && idx >= 0) st[v] = ld_acquire_u64(status + idx);
            }
        }
        if (timed_out) break;
        unsigned long long part = 0;
#pragma unroll
        for (int v = 0; v < kLbWays; ++v) {
            const bool take = v < first_v || (v == first_v && lane <= first_lane);
            if (take) part += st[v] & 0xffffffffull;
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) part += __shfl_xor_sync(0xffffffffu, part, off);
        prefix += part;
        if (first_v < kLbWays) break;
        pred -= 32 * kLbWays;
    }
    if (lane == 0) {
        if (timed_out) {
            dev_flag(hdr, CSRT_DEV_TIMEOUT);
            hdr->timeout_site = 1;
        }
        st_release_u64(status + tile, kFlagInc | (prefix + count));
    }
    return prefix;
}

template <bool kProx, bool kVec>
__global__ void __launch_bounds__(kCThreads) compact_kernel(CompactArgs a) {
    pdl_enter();
    __shared__ __align__(16) float w_tile[kProx ? kTile : 4];
    __shared__ int32_t s_rowptr[kProx ? kTile + 2 : 2];
    __shared__ unsigned long long s_warp[kCThreads / 32];
    __shared__ unsigned long long s_excl;
    __shared__ int64_t s_range[2];
    __shared__ unsigned int s_tile;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (tid == 0) s_tile = atomicAdd(&a.hdr->ticket, 1u);
    __syncthreads();
    const int64_t tile = s_tile;
    if (tile >= a.num_tiles) return;  // cannot happen: one block per tile
    const int64_t e0 = tile * kTile;
    const int64_t e1 = min(e0 + (int64_t)kTile, a.elems);
    const int64_t K = a.cols;

    // 1. Stream this thread's 16 entries: quad q covers e0 + 4*(q*256 + tid).
    float v[kCQuads][4];
#pragma unroll
    for (int q = 0; q < kCQuads; ++q) {
        const int64_t e = e0 + 4 * (int64_t)(q * kCThreads + tid);
        if (kVec && e + 3 < e1) {
            float4 f = ld_stream_f4(a.src + e);
            v[q][0] = f.x; v[q][1] = f.y; v[q][2] = f.z; v[q][3] = f.w;
        } else {
#pragma unroll
            for (int c = 0; c < 4; ++c) v[q][c] = (e + c < e1) ? a.src[e + c] : 0.f;
        }
    }

    // 1b. Adaptive prox: the gradient becomes the search direction, the
    // moments are updated in place.
    if (kProx && a.opt != kOptSgd) {
#pragma unroll
        for (int q = 0; q < kCQuads; ++q) {
            const int64_t e = e0 + 4 * (int64_t)(q * kCThreads + tid);
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                if (e + c < e1) {
                    float mm = a.opt == kOptAdam ? a.m[e + c] : 0.f, vv = a.v[e + c];
                    v[q][c] = opt_direction(a, v[q][c], mm, vv);
                    if (a.opt == kOptAdam) a.m[e + c] = mm;
                    a.v[e + c] = vv;
                }
            }
        }
    }

    // 2. Prox: the old weights of this flat range, scattered into w_tile.
    if (kProx) {
        for (int i = tid; i < kTile; i += kCThreads) w_tile[i] = 0.f;
        const int64_t r0 = e0 / K, r1 = (e1 - 1) / K;  // rows touched, inclusive
        const int nr = (int)(r1 - r0 + 2);              // row_ptr entries r0..r1+1
        for (int i = tid; i < nr; i += kCThreads) s_rowptr[i] = a.in_row_ptr[r0 + i];
        __syncthreads();
        if (warp == 0) {
            int64_t s0 = warp_lower_bound(a.in_col, s_rowptr[0], s_rowptr[1], (int32_t)(e0 - r0 * K));
            if (lane == 0) s_range[0] = s0;
        } else if (warp == 1) {
            int64_t s1;
            if (e1 == (r1 + 1) * K) s1 = s_rowptr[nr - 1];
            else s1 = warp_lower_bound(a.in_col, s_rowptr[nr - 2], s_rowptr[nr - 1], (int32_t)(e1 - r1 * K));
            if (lane == 0) s_range[1] = s1;
        }
        __syncthreads();
        const int64_t s0 = s_range[0], s1 = s_range[1];
        for (int64_t k = s0 + tid; k < s1; k += kCThreads) {
            int lo = 0, hi = nr - 2;  // last row whose start is <= k
            while (lo < hi) {
                int mid = (lo + hi + 1) >> 1;
                if (s_rowptr[mid] <= k) lo = mid; else hi = mid - 1;
            }
            const int64_t f = (r0 + lo) * K + __ldg(a.in_col + k);
            w_tile[f - e0] = __ldg(a.in_val + k);
        }
        __syncthreads();
    }

    // 3. Predicate and kept value per entry.
    unsigned int keep = 0;  // bit q*4+c
    bool nonfinite = false;
#pragma unroll
    for (int q = 0; q < kCQuads; ++q) {
        const int64_t e = e0 + 4 * (int64_t)(q * kCThreads + tid);
        float4 w4 = make_float4(0.f, 0.f, 0.f, 0.f);
        if (kProx) w4 = reinterpret_cast<const float4 *>(w_tile)[q * kCThreads + tid];
        const float wv[4] = {w4.x, w4.y, w4.z, w4.w};
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            const bool valid = e + c < e1;
            bool k;
            if (kProx) {
                const float t = __fmul_rn(a.eta, v[q][c]);
                const float z = __fsub_rn(wv[c], t);
                k = valid && fabsf(z) > a.thr;
                nonfinite |= valid && isnan(z);
                v[q][c] = z > 0.f ? __fsub_rn(z, a.thr) : __fadd_rn(z, a.thr);
            } else {
                k = valid && v[q][c] != 0.f;
            }
            keep |= (unsigned)k << (q * 4 + c);
        }
    }
    if (kProx) {
        if (__syncthreads_or(nonfinite) && tid == 0) dev_flag(a.hdr, CSRT_DEV_NONFINITE);
    }

    // 4. Block scan of the four per-quad counts, packed in 16-bit fields.
    unsigned long long packed = 0;
#pragma unroll
    for (int q = 0; q < kCQuads; ++q)
        packed |= (unsigned long long)__popc((keep >> (q * 4)) & 0xFu) << (16 * q);
    unsigned long long incl = packed;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        unsigned long long y = __shfl_up_sync(0xffffffffu, incl, off);
        if (lane >= off) incl += y;
    }
    if (lane == 31) s_warp[warp] = incl;
    __syncthreads();
    unsigned long long warp_prefix = 0, block_total = 0;
#pragma unroll
    for (int w = 0; w < kCThreads / 32; ++w) {
        const unsigned long long t = s_warp[w];
        if (w < warp) warp_prefix += t;
        block_total += t;
    }
    const unsigned long long excl = incl - packed + warp_prefix;
    uint32_t quad_total[kCQuads];
    uint32_t tile_count = 0;
#pragma unroll
    for (int q = 0; q < kCQuads; ++q) {
        quad_total[q] = (uint32_t)((block_total >> (16 * q)) & 0xFFFFu);
        tile_count += quad_total[q];
    }

    // 5. Decoupled look-back for the number of entries kept before this tile.
    if (warp == 0) {
        const unsigned long long prefix = lookback_warp(a.status, tile, tile_count, a.hdr);
        if (lane == 0) s_excl = prefix;
    }
    __syncthreads();
    const int64_t tile_base = (int64_t)s_excl;
    const int64_t cap = a.capacity;

    // 6. Write kept entries and the row starts that fall in this tile.
    int64_t quad_base = tile_base;
#pragma unroll
    for (int q = 0; q < kCQuads; ++q) {
        int64_t pos = quad_base + (int64_t)((excl >> (16 * q)) & 0xFFFFu);
        const int64_t e = e0 + 4 * (int64_t)(q * kCThreads + tid);
        if (e < e1) {
            int64_t r = e / K;
            int64_t col = e - r * K;
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                if (e + c < e1) {
                    if (col == 0) a.out_row_ptr[r] = (int32_t)min(pos, cap);
                    if ((keep >> (q * 4 + c)) & 1u) {
                        if (pos < cap) {
                            a.out_col[pos] = (int32_t)col;
                            a.out_val[pos] = v[q][c];
                        }
                        ++pos;
                    }
                    if (++col == K) { col = 0; ++r; }
                }
            }
        }
        quad_base += quad_total[q];
    }
    if (tile == a.num_tiles - 1 && tid == 0) {
        const int64_t total = tile_base + tile_count;
        a.out_row_ptr[a.rows] = (int32_t)min(total, cap);
        if (total > cap) {
            dev_flag(a.hdr, CSRT_DEV_CAPACITY);
            atomicMax(&a.hdr->required, (unsigned long long)total);
        }
    }
}


// ---------------------------------------------------------------------------
// Row-tile compaction (the fast path: K % 4 == 0, K <= kRowMaxK, G 16-byte
// aligned). A tile is R whole rows (R*K <= max(K, kRowBudget) entries), so the
// old CSR entries of a tile are the contiguous range row_ptr[r0] ..
// row_ptr[r0+R) and no search is needed: they are scattered into a
// shared-memory copy of the tile's old weights. Each of the 8 warps owns a
// contiguous segment of the tile and walks it 128 entries (one float4 per
// lane) at a time: pass 1 counts the kept entries with four ballots per step,
// the block learns its global offset by decoupled look-back, pass 2
// re-evaluates the entries (G comes back from L1/L2) and writes them at ranks
// taken from the same ballots, so a warp's output of one step is one
// contiguous run. Positions are 32-bit (nnz < 2^31). Small per-block state
// (the old-weight tile only) lets several blocks share an SM and hide the
// look-back latency.
// ---------------------------------------------------------------------------
constexpr int kRowBudget = 8192;     // entries per tile when rows are short
constexpr int kRowMaxK = 16384;      // longest row the row-tile path takes

// Count/place prox (SGD, K % 32 == 0): per-row counts, their scan, per-tile
// counts and a stash of an eighth of each tile's entries (column and value).
struct PlaceLayout {
    int32_t rows_per_tile, stash;
    int64_t tiles;
    size_t off_rowcnt, off_raw, off_tilecnt, off_stcol, off_stval, total;
};

static PlaceLayout place_layout(int32_t rows, int32_t cols) {
    auto al = [](size_t x) { return (x + 255) / 256 * 256; };
    PlaceLayout L{};
    if (rows <= 0 || cols <= 0 || cols % 32 != 0 || cols > kRowMaxK) return L;
    L.rows_per_tile = imax<int32_t>(1, kRowBudget / cols);
    L.tiles = ceil_div<int64_t>(rows, L.rows_per_tile);
    L.stash = imax((L.rows_per_tile * cols + 7) / 8, 2 * kCThreads);   // the place kernel reads 512 ahead
    size_t o = 0;
    L.off_rowcnt = o;  o += al((size_t)rows * 4);
    L.off_raw = o;     o += al(((size_t)rows + 1) * 4);
    L.off_tilecnt = o; o += al((size_t)L.tiles * 4);
    L.off_stcol = o;   o += al((size_t)L.tiles * L.stash * 4);
    L.off_stval = o;   o += al((size_t)L.tiles * L.stash * 4);
    L.total = o;
    return L;
}

static size_t prox_place_bytes(int32_t rows, int32_t cols) { return place_layout(rows, cols).total; }

__device__ __forceinline__ uint32_t cvta_smem(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// Bounded wait for the phase with the given parity of an mbarrier.
__device__ __forceinline__ bool row_mbar_wait(uint64_t *bar, uint32_t parity) {
    return mbar_wait_bounded(bar, parity);
}

// Thread 0 only: stream `bytes` (16-byte aligned source, multiple of 16) into
// shared memory with one bulk asynchronous copy that completes on `bar`.
__device__ __forceinline__ void bulk_load(float *dst, const float *src, uint32_t bytes, uint64_t *bar) {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(cvta_smem(bar)), "r"(bytes)
                 : "memory");
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                     cvta_smem(dst)),
                 "l"(src), "r"(bytes), "r"(cvta_smem(bar))
                 : "memory");
}

struct Keep4 {
    bool k[4];
    float v[4];
};

template <bool kProx>
__device__ __forceinline__ Keep4 eval4(const float4 g, const float4 w, float eta, float thr) {
    Keep4 r;
    const float gv[4] = {g.x, g.y, g.z, g.w};
    const float wv[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        if (kProx) {
            const float z = __fsub_rn(wv[j], __fmul_rn(eta, gv[j]));
            r.k[j] = fabsf(z) > thr;
            r.v[j] = z > 0.f ? __fsub_rn(z, thr) : __fadd_rn(z, thr);
        } else {
            r.k[j] = gv[j] != 0.f;
            r.v[j] = gv[j];
        }
    }
    return r;
}

template <bool kProx>
__global__ void __launch_bounds__(kCThreads, 4) compact_rows_kernel(CompactArgs a, int32_t rows_per_tile) {
    pdl_enter();
    extern __shared__ __align__(16) float row_smem[];
    float *wt = row_smem;                                                        // old weights (prox)
    int32_t *s_rp = reinterpret_cast<int32_t *>(row_smem + (kProx ? rows_per_tile * a.cols : 0));
    __shared__ uint32_t s_wtot[kCThreads / 32];
    __shared__ uint32_t s_excl;
    __shared__ unsigned int s_tile;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int K = a.cols;
    if (tid == 0) s_tile = atomicAdd(&a.hdr->ticket, 1u);
    __syncthreads();
    const int64_t tile = s_tile;
    if (tile >= a.num_tiles) return;   // cannot happen: one block per tile
    const int r0 = (int)(tile * rows_per_tile);
    const int nrows = imin(rows_per_tile, a.rows - r0);
    const int n_el = nrows * K;
    const float *g = a.src + (int64_t)r0 * K;
    bool nonfinite = false;

    if (kProx) {
        for (int i = tid; i <= nrows; i += kCThreads) s_rp[i] = a.in_row_ptr[r0 + i];
        float4 *w4 = reinterpret_cast<float4 *>(wt);
        for (int i = tid; i < n_el / 4; i += kCThreads) w4[i] = make_float4(0.f, 0.f, 0.f, 0.f);
        __syncthreads();
        const int32_t s0 = s_rp[0], s1 = s_rp[nrows];
        for (int32_t k = s0 + tid; k < s1; k += kCThreads) {
            int lo = 0, hi = nrows - 1;  // row of entry k: last row whose start is <= k
            while (lo < hi) {
                const int mid = (lo + hi + 1) >> 1;
                if (s_rp[mid] <= k) lo = mid; else hi = mid - 1;
            }
            wt[lo * K + __ldg(a.in_col + k)] = __ldg(a.in_val + k);
        }
        __syncthreads();
    }

    // warp segment [e_beg, e_end), a multiple of 128 entries except at the end
    const int seg = ((n_el + 8 * 128 - 1) / (8 * 128)) * 128;
    const int e_beg = imin(warp * seg, n_el), e_end = imin(e_beg + seg, n_el);

    // pass 1: count; four steps of loads in flight per lane
    uint32_t cnt = 0;
    for (int base = e_beg; base < e_end; base += 4 * 128) {
        float4 gv[4], wv[4];
        bool in[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int b = base + 128 * u + 4 * lane;
            in[u] = b < e_end;
            gv[u] = in[u] ? ldg_f4(g + b) : make_float4(0.f, 0.f, 0.f, 0.f);
            wv[u] = (kProx && in[u]) ? *reinterpret_cast<const float4 *>(wt + b) : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const Keep4 r = eval4<kProx>(gv[u], wv[u], a.eta, a.thr);
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                cnt += __popc(__ballot_sync(0xffffffffu, in[u] && r.k[j]));
                if (kProx) nonfinite |= in[u] && isnan(r.v[j]);
            }
        }
    }
    if (lane == 0) s_wtot[warp] = cnt;
    __syncthreads();
    uint32_t pos = 0, tile_count = 0;
#pragma unroll
    for (int w = 0; w < kCThreads / 32; ++w) {
        const uint32_t t = s_wtot[w];
        if (w < warp) pos += t;
        tile_count += t;
    }
    if (warp == 0) {
        const unsigned long long prefix = lookback_warp(a.status, tile, tile_count, a.hdr);
        if (lane == 0) s_excl = (uint32_t)prefix;
    }
    __syncthreads();
    pos += s_excl;
    const uint32_t cap = (uint32_t)imin<int64_t>(a.capacity, 0x7fffffff);

    // pass 2: write the kept entries and the row starts
    int row = e_beg / K;
    int col = e_beg - row * K + 4 * lane;
    while (col >= K) { col -= K; ++row; }
    const unsigned lt = (1u << lane) - 1u;
    for (int base = e_beg; base < e_end; base += 4 * 128) {
        float4 gv[4], wv[4];
        bool in[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int b = base + 128 * u + 4 * lane;
            in[u] = b < e_end;
            gv[u] = in[u] ? ldg_f4(g + b) : make_float4(0.f, 0.f, 0.f, 0.f);
            wv[u] = (kProx && in[u]) ? *reinterpret_cast<const float4 *>(wt + b) : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const Keep4 r = eval4<kProx>(gv[u], wv[u], a.eta, a.thr);
            uint32_t p = pos, step = 0;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const unsigned m = __ballot_sync(0xffffffffu, in[u] && r.k[j]);
                p += __popc(m & lt);
                step += __popc(m);
            }
            if (in[u] && col == 0) a.out_row_ptr[r0 + row] = (int32_t)min(p, cap);
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                if (in[u] && r.k[j]) {
                    if (p < cap) {
                        a.out_col[p] = col + j;
                        a.out_val[p] = r.v[j];
                    }
                    ++p;
                }
            }
            pos += step;
            col += 128;
            while (col >= K) { col -= K; ++row; }
        }
    }
    if (tile == a.num_tiles - 1 && tid == 0) {
        const int64_t total = (int64_t)s_excl + tile_count;
        a.out_row_ptr[a.rows] = (int32_t)imin<int64_t>(total, cap);
        if (total > (int64_t)cap) {
            dev_flag(a.hdr, CSRT_DEV_CAPACITY);
            atomicMax(&a.hdr->required, (unsigned long long)total);
        }
    }
    if (kProx && __syncthreads_or(nonfinite) && tid == 0) dev_flag(a.hdr, CSRT_DEV_NONFINITE);
}


// ---------------------------------------------------------------------------
// Prox row-tile kernels (the prox update's fast path). Same tiling as
// compact_rows_kernel, one read of G per evaluation: the tile's G is
// bulk-copied into shared memory, the old CSR entries of its rows folded in
// (z of a stored weight in place, its position marked in a bitmask), and pass
// 1 evaluates every entry once, counts the kept ones per lane and parks each
// result in the tile (the kept value, or NaN for a dropped entry: a kept value
// is never NaN). Pass 2 reads only shared memory and writes the kept entries
// of a warp's segment at consecutive positions.
//
// prox_rows_kernel (one pass; the adaptive steps and K % 32 != 0): a tile
// learns the number of entries kept before it by decoupled look-back, then
// runs pass 2 to the output. With kBits (K % 32 == 0 and a transposed copy
// wanted) pass 2 also emits, per 32-entry word of a row, the keep bitmask and
// the CSR position of the word's first entry, from which the transposed copy
// is built without re-reading the CSR.
//
// prox_count_kernel + row scan + prox_place_kernel (the SGD prox with K % 32
// == 0): no block waits on another. The count kernel evaluates each tile,
// writes the keep bitmask of every word and the kept count of every row, and
// a tile that keeps at most an eighth of its entries also writes them,
// compacted in CSR order, to the tile's stash. After the exclusive scan of
// the row counts (the new row pointers), the place kernel copies a stashed
// tile's run to its final position, or evaluates a denser tile again from G
// and writes it through pass 2.
// ---------------------------------------------------------------------------
constexpr int kPsSteps = 4;   // 32-entry steps per warp iteration of pass 2 (independent loads)

// Shared memory of a prox tile: the tile's G (then z, then the parked
// results), the bitmask of positions holding a stored weight, the tile's row
// pointers and (count kernel) its rows' kept counts.
__host__ __device__ constexpr size_t prox_smem_floats(int64_t tile_cap, int64_t rows_per_tile) {
    return (size_t)(tile_cap + (tile_cap + 31) / 32 + 2 * rows_per_tile + 1);
}

// Everything before pass 1, once thread 0 has started the bulk copy of the
// tile's G onto `bar`: the tile's row pointers, the cleared bitmask, the
// adaptive direction (Algorithms 1 and 2: the moments updated in place and G
// replaced by the search direction), and the old entries folded into the
// tile. Ends with the tile in shared memory and a barrier. A wait that runs
// out sets *fail.
__device__ __forceinline__ void prox_tile_prepare(const CompactArgs &a, int r0, int nrows, int n_el, float *tile_v,
                                                  uint32_t *onbits, int32_t *s_rp, uint64_t *bar, int *fail) {
    const int tid = threadIdx.x;
    const int K = a.cols;
    const float eta = a.eta;
    for (int i = tid; i <= nrows; i += kCThreads) s_rp[i] = a.in_row_ptr[r0 + i];
    for (int i = tid; i < (n_el + 31) / 32; i += kCThreads) onbits[i] = 0u;
    bool waited = false;
    if (a.opt != kOptSgd) {
        // adaptive prox: the tile's G becomes the search direction (moments
        // updated in place, 16-byte rows since K % 4 == 0) before the fold
        if (!row_mbar_wait(bar, 0)) *fail = 1;
        waited = true;
        float *mp = a.m + (int64_t)r0 * K, *vp = a.v + (int64_t)r0 * K;
        for (int b = 4 * tid; b < n_el; b += 4 * kCThreads) {
            const float4 g4 = *reinterpret_cast<const float4 *>(tile_v + b);
            float4 m4 = a.opt == kOptAdam ? *reinterpret_cast<const float4 *>(mp + b) : make_float4(0.f, 0.f, 0.f, 0.f);
            float4 v4 = *reinterpret_cast<const float4 *>(vp + b);
            float4 d4;
            d4.x = opt_direction(a, g4.x, m4.x, v4.x);
            d4.y = opt_direction(a, g4.y, m4.y, v4.y);
            d4.z = opt_direction(a, g4.z, m4.z, v4.z);
            d4.w = opt_direction(a, g4.w, m4.w, v4.w);
            if (a.opt == kOptAdam) *reinterpret_cast<float4 *>(mp + b) = m4;
            *reinterpret_cast<float4 *>(vp + b) = v4;
            *reinterpret_cast<float4 *>(tile_v + b) = d4;
        }
    }
    __syncthreads();
    const int32_t s0 = s_rp[0], s1 = s_rp[nrows];
    constexpr int kOld = 4;   // old entries held per thread per pass
    for (int32_t kb = s0; kb < s1; kb += kOld * kCThreads) {
        int32_t pos_e[kOld];
        float wv[kOld];
#pragma unroll
        for (int q = 0; q < kOld; ++q) {
            const int32_t k = kb + q * kCThreads + tid;
            pos_e[q] = -1;
            wv[q] = 0.f;
            if (k < s1) {
                int lo = 0, hi = nrows - 1;
                while (lo < hi) {
                    const int mid = (lo + hi + 1) >> 1;
                    if (s_rp[mid] <= k) lo = mid; else hi = mid - 1;
                }
                pos_e[q] = lo * K + __ldg(a.in_col + k);
                wv[q] = __ldg(a.in_val + k);
            }
        }
        if (!waited) {   // the first batch of old entries was loaded while G streamed in
            if (!row_mbar_wait(bar, 0)) *fail = 1;
            waited = true;
        }
#pragma unroll
        for (int q = 0; q < kOld; ++q) {
            if (pos_e[q] >= 0) {
                const int e = pos_e[q];
                tile_v[e] = __fsub_rn(wv[q], __fmul_rn(eta, tile_v[e]));   // z of a stored weight
                atomicOr(&onbits[e >> 5], 1u << (e & 31));
            }
        }
    }
    if (!waited && !row_mbar_wait(bar, 0)) *fail = 1;
    __syncthreads();
}

// The warp's segment of the tile: whole 128-entry groups, 8 warps.
__device__ __forceinline__ void prox_segment(int n_el, int &e_beg, int &e_end) {
    const int warp = threadIdx.x >> 5;
    const int seg = ((n_el + 8 * 128 - 1) / (8 * 128)) * 128;
    e_beg = imin(warp * seg, n_el);
    e_end = imin(e_beg + seg, n_el);
}

// Pass 1 over the warp's segment: z (-eta*G off the pattern), keep, kept value
// parked in place; returns the lane's kept count. With kWords (K % 32 == 0)
// it also writes the keep bitmask of every 32-entry word (lanes 8q .. 8q+7 of
// a 128-entry group hold word q) and adds each word's count to its row's
// counter in shared memory.
template <bool kWords>
__device__ __forceinline__ uint32_t prox_pass1(const CompactArgs &a, float *tile_v, const uint32_t *onbits, int e_beg,
                                               int e_end, int r0, uint32_t *__restrict__ keepbits, int32_t wpr,
                                               int32_t *s_rowcnt, bool &nonfinite) {
    const int lane = threadIdx.x & 31;
    const int K = a.cols;
    const float eta = a.eta, thr = a.thr;
    uint32_t cnt = 0;
    int row = 0, col = 0;   // of the lane's first entry (kWords)
    if (kWords) {
        row = e_beg / K;
        col = e_beg - row * K + 4 * lane;
        while (col >= K) { col -= K; ++row; }
    }
    for (int b = e_beg + 4 * lane; b - 4 * lane < e_end; b += 128) {
        unsigned nib = 0;
        if (b < e_end) {
            float4 *vp = reinterpret_cast<float4 *>(tile_v + b);
            const float4 t4 = *vp;
            const unsigned on = (onbits[b >> 5] >> (b & 31)) & 0xFu;
            const float tv[4] = {t4.x, t4.y, t4.z, t4.w};
            float o[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                // off the pattern w = +0: z = fl(0 - fl(eta*G)) (its sign is irrelevant: zero is dropped)
                const float z = ((on >> j) & 1u) ? tv[j] : -__fmul_rn(eta, tv[j]);
                const bool k = fabsf(z) > thr;
                nonfinite |= z != z;
                o[j] = k ? __fsub_rn(z, copysignf(thr, z)) : __int_as_float(0x7fc00000);
                cnt += k;
                nib |= (k ? 1u : 0u) << j;
            }
            *vp = make_float4(o[0], o[1], o[2], o[3]);
        }
        if (kWords) {
            uint32_t word = nib << (4 * (lane & 7));
            word |= __shfl_xor_sync(0xffffffffu, word, 1);
            word |= __shfl_xor_sync(0xffffffffu, word, 2);
            word |= __shfl_xor_sync(0xffffffffu, word, 4);
            if (b < e_end && (lane & 7) == 0) {
                keepbits[(int64_t)(r0 + row) * wpr + (col >> 5)] = word;
                if (word) atomicAdd(&s_rowcnt[row], (int32_t)__popc(word));
            }
            col += 128;
            while (col >= K) { col -= K; ++row; }
        }
    }
    return cnt;
}

// Pass 2, a tile that keeps most of its entries: lane = entry of a 32-entry
// step; one ballot gives the step's keep word and every lane's rank in it, so
// the kept entries go out as one coalesced run (measured 14-34% faster on
// dense outputs). With K % 32 == 0 a step (the segments are whole 128-entry
// groups) is exactly one 32-column word of one row: its ballot is the keep
// bitmask of the transposed copy (written to keepbits when given) and `pos` at
// the step the position of the word's first entry (written to wordpos when
// given). Row pointers are written where a row starts when row_ptr is given.
__device__ __forceinline__ void prox_pass2_dense(const float *tile_v, int e_beg, int e_end, int K, int r0,
                                                 uint32_t pos, uint32_t cap, bool fits, int32_t *__restrict__ out_col,
                                                 float *__restrict__ out_val, int32_t *__restrict__ row_ptr,
                                                 uint32_t *__restrict__ keepbits, int32_t *__restrict__ wordpos,
                                                 int32_t wpr) {
    const int lane = threadIdx.x & 31;
    const unsigned lt = (1u << lane) - 1u;
    const float qnan = __int_as_float(0x7fc00000);
    const bool wide = K >= 32;   // a step crosses at most one row end
    int row = e_beg / K;         // row and column of the step's first entry
    int c0 = e_beg - row * K;
    for (int base = e_beg; base < e_end; base += 32 * kPsSteps) {
        float v4[kPsSteps];
#pragma unroll
        for (int u = 0; u < kPsSteps; ++u) {
            const int e = base + 32 * u + lane;
            v4[u] = e < e_end ? tile_v[e] : qnan;
        }
#pragma unroll
        for (int u = 0; u < kPsSteps; ++u) {
            if (base + 32 * u >= e_end) break;   // warp-uniform
            const bool k = v4[u] == v4[u];
            const unsigned m = __ballot_sync(0xffffffffu, k);
            const uint32_t p = pos + __popc(m & lt);
            int col = c0 + lane, rowl = row;
            if (wide) {
                if (col >= K) {
                    col -= K;
                    ++rowl;
                }
            } else {
                while (col >= K) {
                    col -= K;
                    ++rowl;
                }
            }
            if (row_ptr && (c0 == 0 || c0 + 32 > K)) {   // a row starts in this step
                if (base + 32 * u + lane < e_end && col == 0) row_ptr[r0 + rowl] = (int32_t)min(p, cap);
            }
            if (lane == 0 && (keepbits || wordpos)) {
                const int64_t wi = (int64_t)(r0 + row) * wpr + (c0 >> 5);
                if (keepbits) keepbits[wi] = m;
                if (wordpos) wordpos[wi] = (int32_t)pos;
            }
            if (k && (fits || p < cap)) {
                out_col[p] = col;
                out_val[p] = v4[u];
            }
            pos += __popc(m);
            c0 += 32;
            if (wide) {
                if (c0 >= K) {
                    c0 -= K;
                    ++row;
                }
            } else {
                while (c0 >= K) {
                    c0 -= K;
                    ++row;
                }
            }
        }
    }
}

// Pass 2, a tile that keeps few of its entries: four consecutive entries per
// lane, ranks from a warp scan, whose shorter dependency chain per 128
// entries wins on sparse outputs. Same optional outputs as the dense form.
__device__ __forceinline__ void prox_pass2_sparse(const float *tile_v, int e_beg, int e_end, int K, int r0,
                                                  uint32_t pos, uint32_t cap, int32_t *__restrict__ out_col,
                                                  float *__restrict__ out_val, int32_t *__restrict__ row_ptr,
                                                  uint32_t *__restrict__ keepbits, int32_t *__restrict__ wordpos,
                                                  int32_t wpr) {
    const int lane = threadIdx.x & 31;
    int row = e_beg / K;
    int col = e_beg - row * K + 4 * lane;
    while (col >= K) { col -= K; ++row; }
    for (int base = e_beg; base < e_end; base += 128) {
        const int b = base + 4 * lane;
        const bool in = b < e_end;
        const float4 v = in ? *reinterpret_cast<const float4 *>(tile_v + b) : make_float4(__int_as_float(0x7fc00000),
                                                                                   __int_as_float(0x7fc00000),
                                                                                   __int_as_float(0x7fc00000),
                                                                                   __int_as_float(0x7fc00000));
        const float vv[4] = {v.x, v.y, v.z, v.w};
        // keep bits of this lane's four entries; warp scan of their counts gives the ranks
        const unsigned nib = (unsigned)(vv[0] == vv[0]) | ((unsigned)(vv[1] == vv[1]) << 1) |
                             ((unsigned)(vv[2] == vv[2]) << 2) | ((unsigned)(vv[3] == vv[3]) << 3);
        const uint32_t c = __popc(nib);
        uint32_t incl = c;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const uint32_t t = __shfl_up_sync(0xffffffffu, incl, off);
            if (lane >= off) incl += t;
        }
        uint32_t p = pos + incl - c;
        if (row_ptr && in && col == 0) row_ptr[r0 + row] = (int32_t)min(p, cap);
        if (keepbits || wordpos) {
            // 32-entry word of lanes 8q .. 8q+7 (four bits per lane, in order)
            uint32_t word = nib << (4 * (lane & 7));
            word |= __shfl_xor_sync(0xffffffffu, word, 1);
            word |= __shfl_xor_sync(0xffffffffu, word, 2);
            word |= __shfl_xor_sync(0xffffffffu, word, 4);
            if (in && (lane & 7) == 0) {
                const int64_t wi = (int64_t)(r0 + row) * wpr + (col >> 5);
                if (keepbits) keepbits[wi] = word;
                if (wordpos) wordpos[wi] = (int32_t)p;
            }
        }
        if (nib) {
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                if ((nib >> j) & 1u) {
                    if (p < cap) {
                        out_col[p] = col + j;
                        out_val[p] = vv[j];
                    }
                    ++p;
                }
            }
        }
        pos += __shfl_sync(0xffffffffu, incl, 31);
        col += 128;
        while (col >= K) { col -= K; ++row; }
    }
}

// Thread 0: claim a tile (by ticket when `ticket`, else the block index) and
// start the bulk copy of its G onto `bar`. Returns the tile to every thread.
__device__ __forceinline__ int64_t prox_tile_start(const CompactArgs &a, int rows_per_tile, bool ticket,
                                                   float *tile_v, uint64_t *bar, unsigned int *s_tile, int *s_fail) {
    if (threadIdx.x == 0) {
        *s_fail = 0;
        const unsigned t = ticket ? atomicAdd(&a.hdr->ticket, 1u) : blockIdx.x;
        *s_tile = t;
        asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(cvta_smem(bar)) : "memory");
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        if (t < a.num_tiles) {
            const int64_t r0 = (int64_t)t * rows_per_tile;
            const int64_t nrows = imin<int64_t>(rows_per_tile, a.rows - r0);
            bulk_load(tile_v, a.src + r0 * a.cols, (uint32_t)(nrows * a.cols * 4), bar);
        }
    }
    __syncthreads();
    return *s_tile;
}

__device__ __forceinline__ void prox_flags(const CompactArgs &a, bool nonfinite, int fail) {
    if (__syncthreads_or(nonfinite) && threadIdx.x == 0) dev_flag(a.hdr, CSRT_DEV_NONFINITE);
    if (threadIdx.x == 0 && fail) {
        dev_flag(a.hdr, CSRT_DEV_TIMEOUT);
        a.hdr->timeout_site = 3;
    }
}

template <bool kBits>
__global__ void __launch_bounds__(kCThreads, 6) prox_rows_kernel(CompactArgs a, int32_t rows_per_tile,
                                                                  uint32_t *__restrict__ keepbits,
                                                                  int32_t *__restrict__ wordpos, int32_t wpr) {
    pdl_enter();
    extern __shared__ __align__(128) float prox_smem[];
    float *tile_v = prox_smem;
    const int tile_cap = rows_per_tile * a.cols;
    uint32_t *onbits = reinterpret_cast<uint32_t *>(prox_smem + tile_cap);
    int32_t *s_rp = reinterpret_cast<int32_t *>(onbits + (tile_cap + 31) / 32);
    __shared__ __align__(8) uint64_t s_bar;
    __shared__ uint32_t s_wtot[kCThreads / 32];
    __shared__ uint32_t s_excl;
    __shared__ unsigned int s_tile;
    __shared__ int s_fail;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int K = a.cols;
    const int64_t tile = prox_tile_start(a, rows_per_tile, true, tile_v, &s_bar, &s_tile, &s_fail);
    if (tile >= a.num_tiles) return;
    const int r0 = (int)(tile * rows_per_tile);
    const int nrows = imin(rows_per_tile, a.rows - r0);
    const int n_el = nrows * K;
    prox_tile_prepare(a, r0, nrows, n_el, tile_v, onbits, s_rp, &s_bar, &s_fail);
    int e_beg, e_end;
    prox_segment(n_el, e_beg, e_end);
    bool nonfinite = false;
    uint32_t cnt = prox_pass1<false>(a, tile_v, onbits, e_beg, e_end, r0, nullptr, 0, nullptr, nonfinite);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, off);
    if (lane == 0) s_wtot[warp] = cnt;
    __syncthreads();
    uint32_t pos = 0, tile_count = 0;
#pragma unroll
    for (int w = 0; w < kCThreads / 32; ++w) {
        const uint32_t t = s_wtot[w];
        if (w < warp) pos += t;
        tile_count += t;
    }
    if (warp == 0) {
        const unsigned long long prefix = lookback_warp(a.status, tile, tile_count, a.hdr);
        if (lane == 0) s_excl = (uint32_t)prefix;
    }
    __syncthreads();
    pos += s_excl;
    const uint32_t cap = (uint32_t)imin<int64_t>(a.capacity, 0x7fffffff);
    if (2 * (int64_t)tile_count > n_el) {   // dense tile
        const bool fits = (uint64_t)s_excl + tile_count <= cap;   // no position of the tile reaches the capacity
        prox_pass2_dense(tile_v, e_beg, e_end, K, r0, pos, cap, fits, a.out_col, a.out_val, a.out_row_ptr,
                         kBits ? keepbits : nullptr, kBits ? wordpos : nullptr, wpr);
    } else {
        prox_pass2_sparse(tile_v, e_beg, e_end, K, r0, pos, cap, a.out_col, a.out_val, a.out_row_ptr,
                          kBits ? keepbits : nullptr, kBits ? wordpos : nullptr, wpr);
    }
    if (tile == a.num_tiles - 1 && tid == 0) {
        const int64_t total = (int64_t)s_excl + tile_count;
        a.out_row_ptr[a.rows] = (int32_t)imin<int64_t>(total, cap);
        if (total > (int64_t)cap) {
            dev_flag(a.hdr, CSRT_DEV_CAPACITY);
            atomicMax(&a.hdr->required, (unsigned long long)total);
        }
    }
    prox_flags(a, nonfinite, s_fail);
}

// Count/place SGD prox (K % 32 == 0). Shared memory of a tile: its G (z at
// the stored positions after the fold), per 32-entry word the bitmasks of the
// stored positions and of the stored entries kept, the kept words (count
// kernel), the row pointers and the rows' kept counts.
__host__ __device__ constexpr size_t prox_cp_smem_floats(int64_t tile_cap, int64_t rows_per_tile) {
    return (size_t)(tile_cap + 3 * (tile_cap / 32) + 2 * rows_per_tile + 1);
}

// The stored entries of the tile's rows folded into the tile: z = fl(w -
// fl(eta*G)) in place, the position marked in onbits and, when |z| > thr (the
// entry is kept), in skeep (if given). Waits for the tile's bulk copy before
// the first update. NaN z sets *nonfinite.
__device__ __forceinline__ void prox_cp_fold(const CompactArgs &a, int nrows, float *tile_v, uint32_t *onbits,
                                             uint32_t *skeep, const int32_t *s_rp, uint64_t *bar, uint32_t parity,
                                             int *fail, bool &nonfinite) {
    const int tid = threadIdx.x;
    const int K = a.cols;
    const float eta = a.eta, thr = a.thr;
    const int32_t s0 = s_rp[0], s1 = s_rp[nrows];
    bool waited = false;
    constexpr int kOld = 4;
    for (int32_t kb = s0; kb < s1; kb += kOld * kCThreads) {
        int32_t pos_e[kOld];
        float wv[kOld];
#pragma unroll
        for (int q = 0; q < kOld; ++q) {
            const int32_t k = kb + q * kCThreads + tid;
            pos_e[q] = -1;
            wv[q] = 0.f;
            if (k < s1) {
                int lo = 0, hi = nrows - 1;
                while (lo < hi) {
                    const int mid = (lo + hi + 1) >> 1;
                    if (s_rp[mid] <= k) lo = mid; else hi = mid - 1;
                }
                pos_e[q] = lo * K + __ldg(a.in_col + k);
                wv[q] = __ldg(a.in_val + k);
            }
        }
        if (!waited) {
            if (!row_mbar_wait(bar, parity)) *fail = 1;
            waited = true;
        }
#pragma unroll
        for (int q = 0; q < kOld; ++q) {
            if (pos_e[q] >= 0) {
                const int e = pos_e[q];
                const float z = __fsub_rn(wv[q], __fmul_rn(eta, tile_v[e]));
                tile_v[e] = z;
                atomicOr(&onbits[e >> 5], 1u << (e & 31));
                if (skeep && fabsf(z) > thr) atomicOr(&skeep[e >> 5], 1u << (e & 31));
                nonfinite |= z != z;
            }
        }
    }
    if (!waited && !row_mbar_wait(bar, parity)) *fail = 1;
}

__device__ __forceinline__ int nth_set_bit(uint32_t m, int k);
__device__ __forceinline__ int warp_last_le(int pre, int e);

// The kept value of the lane's entry of a 32-entry step: z - sign(z)*thr with
// z the folded value at a stored position and fl(0 - fl(eta*G)) elsewhere.
__device__ __forceinline__ float prox_cp_value(float tv, bool stored, float eta, float thr) {
    const float z = stored ? tv : -__fmul_rn(eta, tv);
    return __fsub_rn(z, copysignf(thr, z));
}

// Count kernel (eta > 0): one tile per block, taken by ticket (a persistent
// form whose blocks took their next ticket when they started a tile, to load
// its row pointers early, was slower: 73.7 vs 69.9 us at lambda* and 155.7 vs
// 140.5 us at a dense output on 4096 x 9216, tiles being handed out a tile's
// time before they start, which lengthens the look-back and the tail). The sweep
// reads four entries per lane (a 128-entry group per warp step): off the
// pattern an entry is kept iff |fl(eta*G)| > thr, on it the fold's decision
// counts, and, eta being positive, fl(eta*v) is NaN exactly where v (G, or z
// at a stored position) is. Lanes 8q .. 8q+7 of a group hold its word q,
// assembled by three shuffles (measured against a ballot per word, lane =
// column: 76 vs 96 us for the 4096 x 9216 prox at the density-preserving
// lambda). The keep words collect in shared memory and, when the transposed
// copy wants them, leave afterwards as coalesced stores; the kept count of
// every row is summed from them (a one-row tile's is the tile's), and the
// tile's count is published at once. A tile keeping
// at most `stash` entries then writes them in CSR order to its stash (each
// warp its segment's, lane = word, at the position a scan of the words'
// counts gives), and is done without waiting on any other
// block; the place kernel copies the stash to its final position. A denser
// tile learns the number of entries kept before it by decoupled look-back
// over the published counts (the ones of stashed tiles never become
// inclusive prefixes, so it may sum further back) and writes its kept entries
// itself, a 32-entry word at a time, G read only once.
template <bool kBits>
__global__ void __launch_bounds__(kCThreads, 6) prox_count_kernel(CompactArgs a, int32_t rows_per_tile,
                                                                   uint32_t *__restrict__ keepbits,
                                                                   int32_t *__restrict__ wordpos, int32_t wpr,
                                                                   int32_t *__restrict__ rowcnt,
                                                                   int32_t *__restrict__ tilecnt,
                                                                   int32_t *__restrict__ st_col,
                                                                   float *__restrict__ st_val, int32_t stash) {
    pdl_enter();
    extern __shared__ __align__(128) float prox_smem[];
    const int tile_cap = rows_per_tile * a.cols;
    const int nw = tile_cap / 32;
    float *tile_v = prox_smem;
    uint32_t *onbits = reinterpret_cast<uint32_t *>(prox_smem + tile_cap);
    uint32_t *skeep = onbits + nw;   // stored entries kept; after the sweep, the words' exclusive counts
    uint32_t *kwords = skeep + nw;
    int32_t *s_rp = reinterpret_cast<int32_t *>(kwords + nw);
    __shared__ __align__(8) uint64_t s_bar;
    __shared__ uint32_t s_wtot[kCThreads / 32];
    __shared__ uint32_t s_excl;
    __shared__ unsigned int s_tile;
    __shared__ int s_fail;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int K = a.cols;
    const float eta = a.eta, thr = a.thr;
    const int64_t tile = prox_tile_start(a, rows_per_tile, true, tile_v, &s_bar, &s_tile, &s_fail);
    if (tile >= a.num_tiles) return;
    const int r0 = (int)(tile * rows_per_tile);
    const int nrows = imin(rows_per_tile, a.rows - r0);
    const int n_el = nrows * K;
    const int nwt = n_el / 32;   // words of this tile
    for (int i = tid; i <= nrows; i += kCThreads) s_rp[i] = a.in_row_ptr[r0 + i];
    for (int i = tid; i < nwt; i += kCThreads) {
        onbits[i] = 0u;
        skeep[i] = 0u;
    }
    __syncthreads();
    bool nonfinite = false;
    prox_cp_fold(a, nrows, tile_v, onbits, skeep, s_rp, &s_bar, 0, &s_fail, nonfinite);
    __syncthreads();

    // sweep of the warp's segment, a 128-entry group per step
    int e_beg, e_end;
    prox_segment(n_el, e_beg, e_end);
    const int w0 = e_beg >> 5, w1 = e_end >> 5;
    const int sh = 4 * (lane & 7);
    const bool leader = (lane & 7) == 0;   // lane 8q: writes word q of the group
    uint32_t cnt = 0;
    for (int b = e_beg + 4 * lane; b - 4 * lane < e_end; b += 128) {
        const bool in = b < e_end;
        const float4 t4 = in ? *reinterpret_cast<const float4 *>(tile_v + b) : make_float4(0.f, 0.f, 0.f, 0.f);
        const float z0 = __fmul_rn(eta, t4.x), z1 = __fmul_rn(eta, t4.y);   // |fl(0 - fl(eta*G))| = fl(eta*|G|)
        const float z2 = __fmul_rn(eta, t4.z), z3 = __fmul_rn(eta, t4.w);
        nonfinite |= (z0 != z0) | (z1 != z1) | (z2 != z2) | (z3 != z3);
        uint32_t word = ((fabsf(z0) > thr ? 1u : 0u) | (fabsf(z1) > thr ? 2u : 0u) | (fabsf(z2) > thr ? 4u : 0u) |
                         (fabsf(z3) > thr ? 8u : 0u))
                        << sh;
        word |= __shfl_xor_sync(0xffffffffu, word, 1);
        word |= __shfl_xor_sync(0xffffffffu, word, 2);
        word |= __shfl_xor_sync(0xffffffffu, word, 4);
        if (leader && in) {
            const int wi = b >> 5;
            word = (word & ~onbits[wi]) | skeep[wi];
            kwords[wi] = word;
            cnt += __popc(word);
        }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, off);
    if (lane == 0) s_wtot[warp] = cnt;
    __syncthreads();
    uint32_t wbase = 0, tile_count = 0;   // kept entries before this warp's segment; in the tile
#pragma unroll
    for (int w = 0; w < kCThreads / 32; ++w) {
        const uint32_t t = s_wtot[w];
        if (w < warp) wbase += t;
        tile_count += t;
    }
    // keep words out for the transposed copy (the tile's rows are contiguous
    // in keepbits); rows' counts, a warp per row (a one-row tile's is the tile's)
    if (kBits) {
        uint32_t *kb_tile = keepbits + (int64_t)r0 * wpr;
        for (int i = tid; i < nwt; i += kCThreads) kb_tile[i] = kwords[i];
    }
    if (nrows == 1) {
        if (tid == 0) rowcnt[r0] = (int32_t)tile_count;
    } else {
        for (int r = warp; r < nrows; r += kCThreads / 32) {
            int32_t c = 0;
            for (int i = lane; i < wpr; i += 32) c += __popc(kwords[r * wpr + i]);
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) c += __shfl_xor_sync(0xffffffffu, c, off);
            if (lane == 0) rowcnt[r0 + r] = c;
        }
    }
    const bool stashed = tile_count <= (uint32_t)stash;
    if (tid == 0) {
        tilecnt[tile] = stashed ? (int32_t)tile_count : -1 - (int32_t)tile_count;
        if (stashed)   // published without waiting (tile 0's count is its inclusive prefix)
            st_release_u64(a.status + tile, (tile == 0 ? kFlagInc : kFlagAgg) | tile_count);
    }
    if (stashed) {
        // the warp's kept entries, 32 words at a time, lane = word: its position from a warp scan of the
        // words' counts, then its kept entries one per step (measured against lane = entry, each entry's
        // word and bit found by searches: 69.8 vs 73.2 us for the 4096 x 9216 prox at the
        // density-preserving lambda, whose words keep 1.6 entries on average)
        int32_t *sc = st_col + tile * (int64_t)stash;
        float *sv = st_val + tile * (int64_t)stash;
        uint32_t pos = wbase;
        for (int i0 = w0; i0 < w1; i0 += 32) {
            const int wl = i0 + lane;
            uint32_t bits = wl < w1 ? kwords[wl] : 0u;
            const int c = __popc(bits);
            int incl = c;
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const int t = __shfl_up_sync(0xffffffffu, incl, off);
                if (lane >= off) incl += t;
            }
            const uint32_t ob = wl < w1 ? onbits[wl] : 0u;
            const int row = nrows == 1 ? 0 : wl / wpr;
            const int cbase = 32 * wl - row * K;
            const float *tvw = tile_v + 32 * wl;
            uint32_t p = pos + (uint32_t)(incl - c);
            while (bits) {
                const int bit = __ffs(bits) - 1;
                bits &= bits - 1u;
                sc[p] = cbase + bit;
                sv[p] = prox_cp_value(tvw[bit], (ob >> bit) & 1u, eta, thr);
                ++p;
            }
            pos += __shfl_sync(0xffffffffu, incl, 31);
        }
    } else {
        if (warp == 0) {
            const unsigned long long prefix = lookback_warp(a.status, tile, tile_count, a.hdr);
            if (lane == 0) s_excl = (uint32_t)prefix;
        }
        __syncthreads();
        // the warp's words at their final positions, one run per word
        const uint32_t cap = (uint32_t)imin<int64_t>(a.capacity, 0x7fffffff);
        const bool fits = (uint64_t)s_excl + tile_count <= cap;   // no position of the tile reaches the capacity
        const uint32_t lt = (1u << lane) - 1u;
        uint32_t pos = s_excl + wbase;
        int row = w0 / wpr, wc = w0 - row * wpr;
        for (int wi = w0; wi < w1; ++wi) {
            const uint32_t word = kwords[wi];
            if (kBits && lane == 0) wordpos[(int64_t)(r0 + row) * wpr + wc] = (int32_t)pos;
            if ((word >> lane) & 1u) {
                const uint32_t p = pos + __popc(word & lt);
                if (fits || p < cap) {
                    a.out_col[p] = 32 * wc + lane;
                    a.out_val[p] = prox_cp_value(tile_v[32 * wi + lane], (onbits[wi] >> lane) & 1u, eta, thr);
                }
            }
            pos += __popc(word);
            if (++wc == wpr) {
                wc = 0;
                ++row;
            }
        }
    }
    prox_flags(a, nonfinite, s_fail);
}

// Place kernel: a stashed tile's run is copied to its final position, and
// with kBits the word positions of the transposed copy are written from the
// keep words. Tiles the count kernel wrote itself (tilecnt -1 - count) are
// skipped. A block takes kPlaceTiles consecutive tiles and loads, for each,
// its count and the first two entries per thread of its stash together (a
// stash holds at least 512 entries, so these reads stay inside it whatever
// the count): one round of loads for the usual stash. With kPrefix the block
// also finds where its rows start, the sum of the counts of every earlier
// tile (a reduction; the launch takes this form up to kPlaceMaxTiles tiles),
// and writes their row pointers (clamped to the capacity; the last block the
// total and the overflow report), which otherwise the scan before it wrote,
// with the unclamped starts in raw.
constexpr int kPlaceTiles = 4;
constexpr int64_t kPlaceMaxTiles = 4096;
constexpr int kPlaceMaxRows = kPlaceTiles * (kRowBudget / 32);   // rows of a block (K >= 32)
template <bool kBits, bool kPrefix>
__global__ void __launch_bounds__(kCThreads, 4) prox_place_kernel(CompactArgs a, int32_t rows_per_tile,
                                                                  const uint32_t *__restrict__ keepbits,
                                                                  int32_t *__restrict__ wordpos, int32_t wpr,
                                                                  const int32_t *__restrict__ rowcnt,
                                                                  const int32_t *__restrict__ raw,
                                                                  const int32_t *__restrict__ tilecnt,
                                                                  const int32_t *__restrict__ st_col,
                                                                  const float *__restrict__ st_val, int32_t stash) {
    pdl_enter();
    __shared__ int32_t s_pre[kPrefix ? kPlaceMaxRows + 1 : 1];
    __shared__ int32_t s_red[kCThreads / 32], s_part[kCThreads / 32];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int64_t tile0 = (int64_t)blockIdx.x * kPlaceTiles;
    int32_t count[kPlaceTiles], c0[kPlaceTiles], c1[kPlaceTiles];
    float v0[kPlaceTiles], v1[kPlaceTiles];
#pragma unroll
    for (int j = 0; j < kPlaceTiles; ++j) {
        const int64_t tile = tile0 + j;
        count[j] = -1;
        c0[j] = c1[j] = 0;
        v0[j] = v1[j] = 0.f;
        if (tile < a.num_tiles) {
            const int32_t *sc = st_col + tile * (int64_t)stash;
            const float *sv = st_val + tile * (int64_t)stash;
            count[j] = __ldg(tilecnt + tile);
            c0[j] = __ldg(sc + tid);
            c1[j] = __ldg(sc + tid + kCThreads);
            v0[j] = __ldg(sv + tid);
            v1[j] = __ldg(sv + tid + kCThreads);
        }
    }
    const int64_t r_begin = tile0 * rows_per_tile;
    const int nr = (int)imin<int64_t>((int64_t)kPlaceTiles * rows_per_tile, a.rows - r_begin);
    const uint32_t cap = (uint32_t)imin<int64_t>(a.capacity, 0x7fffffff);
    int32_t block_base = 0;
    if (kPrefix) {
        // entries kept before the block: the counts of tiles 0 .. tile0-1, four loads in flight per thread
        int32_t part = 0;
        for (int64_t t0 = 0; t0 < tile0; t0 += 4 * kCThreads) {
            int32_t c[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int64_t t = t0 + u * kCThreads + tid;
                c[u] = t < tile0 ? __ldg(tilecnt + t) : 0;
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) part += c[u] >= 0 ? c[u] : -1 - c[u];
        }
        // the block's rows, four per thread: exclusive counts within the block
        int32_t rc[4], own = 0;
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int i = 4 * tid + u;
            rc[u] = i < nr ? __ldg(rowcnt + r_begin + i) : 0;
            own += rc[u];
        }
        int32_t incl = own;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const int32_t y = __shfl_up_sync(0xffffffffu, incl, off);
            if (lane >= off) incl += y;
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) part += __shfl_xor_sync(0xffffffffu, part, off);
        if (lane == 31) s_red[warp] = incl;
        if (lane == 0) s_part[warp] = part;
        __syncthreads();
        int32_t wpre = 0;
#pragma unroll
        for (int w = 0; w < kCThreads / 32; ++w) {
            if (w < warp) wpre += s_red[w];
            block_base += s_part[w];
        }
        int32_t run = block_base + wpre + incl - own;   // the start of this thread's first row
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int i = 4 * tid + u;
            if (i < nr) {
                s_pre[i] = run;
                a.out_row_ptr[r_begin + i] = (int32_t)imin<uint32_t>((uint32_t)run, cap);
            }
            run += rc[u];
        }
        if (r_begin + nr == a.rows && tid == kCThreads - 1) {   // the last block: the total
            a.out_row_ptr[a.rows] = (int32_t)imin<uint32_t>((uint32_t)run, cap);
            if ((int64_t)run > a.capacity) {
                dev_flag(a.hdr, CSRT_DEV_CAPACITY);
                atomicMax(&a.hdr->required, (unsigned long long)run);
            }
        }
        __syncthreads();
    }
#pragma unroll
    for (int j = 0; j < kPlaceTiles; ++j) {
        const int64_t tile = tile0 + j;
        if (count[j] <= 0) continue;
        const int32_t *sc = st_col + tile * (int64_t)stash;
        const float *sv = st_val + tile * (int64_t)stash;
        const uint32_t base = kPrefix ? (uint32_t)s_pre[j * rows_per_tile] : (uint32_t)__ldg(raw + tile * rows_per_tile);
        for (int i = tid; i < count[j]; i += kCThreads) {
            const uint32_t p = base + (uint32_t)i;
            const int32_t c = i < kCThreads ? c0[j] : i < 2 * kCThreads ? c1[j] : __ldg(sc + i);
            const float v = i < kCThreads ? v0[j] : i < 2 * kCThreads ? v1[j] : __ldg(sv + i);
            if (p < cap) {
                a.out_col[p] = c;
                a.out_val[p] = v;
            }
        }
    }
    if (kBits) {   // word positions: a warp per row of the stashed tiles, a scan of the words' kept counts
        for (int i = warp; i < nr; i += kCThreads / 32) {
            const int64_t tile = tile0 + i / rows_per_tile;
            if (__ldg(tilecnt + tile) < 0) continue;
            const int64_t r = r_begin + i;
            const int64_t wi0 = r * wpr;
            int32_t run = kPrefix ? s_pre[i] : __ldg(raw + r);
            for (int i0 = 0; i0 < wpr; i0 += 32) {
                const int w = i0 + lane;
                const int32_t c = w < wpr ? __popc(__ldg(keepbits + wi0 + w)) : 0;
                int32_t incl = c;
#pragma unroll
                for (int off = 1; off < 32; off <<= 1) {
                    const int32_t t = __shfl_up_sync(0xffffffffu, incl, off);
                    if (lane >= off) incl += t;
                }
                if (w < wpr) wordpos[wi0 + w] = run + incl - c;
                run += __shfl_sync(0xffffffffu, incl, 31);
            }
        }
    }
}

// The library's bounded waits run against events that never happen (failure
// detection without a fault): (0) the decoupled look-back of tile 1 while
// tile 0 never publishes, (1) an mbarrier wait on a barrier nothing arrives
// on (mbar_wait_bounded: the waits for the prox kernel's tile copy and for
// the narrow SpMM's ring chunks). Each gives up after its iteration limit,
// sets CSRT_DEV_TIMEOUT (with the site of the wait) and the kernel returns
// normally.
__global__ void bounded_wait_check_kernel(unsigned long long *__restrict__ status, WsHeader *hdr, int which) {
    pdl_enter();
    __shared__ __align__(8) uint64_t bar;
    if (which == 0) {
        lookback_warp(status, 1, 0u, hdr);   // status[0] is zero and stays zero
        return;
    }
    if (threadIdx.x == 0) {
        asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(cvta_smem(&bar)) : "memory");
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncwarp();
    if (threadIdx.x == 0 && !row_mbar_wait(&bar, 0)) {
        dev_flag(hdr, CSRT_DEV_TIMEOUT);
        hdr->timeout_site = 9;
    }
}

// Returns through *bits_done whether the prox kernel emitted the keep bitmask
// (then the transposed copy is built from it).
struct OptParams {
    int32_t opt;
    float *m, *v;
    float beta1, beta2, eps;
    int32_t t;
};

int scan_exclusive_i32_clamped(const int32_t *in, int32_t n, int32_t *out, int32_t *out_clamped, int64_t capacity,
                               void *ws, cudaStream_t s);

static int compact_launch(bool prox, const float *src, int32_t rows, int32_t cols, const csrt_csr *in,
                          float eta, float thr, csrt_csr *out, void *ws, size_t ws_bytes,
                          cudaStream_t s, bool want_bits = false, bool *bits_done = nullptr,
                          const OptParams *op = nullptr) {
    if (bits_done) *bits_done = false;
    const int64_t elems = (int64_t)rows * cols;
    if (elems == 0) {
        CSRT_CHECK_CUDA(cudaMemsetAsync(out->row_ptr, 0, sizeof(int32_t) * ((size_t)rows + 1), s));
        return CSRT_OK;
    }
    const bool opt_aligned =
        op == nullptr || op->opt == kOptSgd ||
        ((reinterpret_cast<uintptr_t>(op->v) | reinterpret_cast<uintptr_t>(op->m)) & 15) == 0;
    const bool row_path = cols % 4 == 0 && cols <= kRowMaxK && (reinterpret_cast<uintptr_t>(src) & 15) == 0 &&
                          opt_aligned;
    const int32_t rows_per_tile = row_path ? imax<int32_t>(1, kRowBudget / cols) : 0;
    const int64_t tiles = row_path ? ceil_div<int64_t>(rows, rows_per_tile) : ceil_div<int64_t>(elems, kTile);
    CSRT_ARG(ws_bytes >= kWsReservedBytes + status_bytes(elems), "workspace too small for compaction");
    WsHeader *hdr = static_cast<WsHeader *>(ws);
    unsigned long long *status = reinterpret_cast<unsigned long long *>(ws_scratch(ws));
    CSRT_CHECK_CUDA(cudaMemsetAsync(&hdr->ticket, 0, sizeof(unsigned int), s));
    CSRT_CHECK_CUDA(cudaMemsetAsync(status, 0, sizeof(unsigned long long) * tiles, s));
    CompactArgs a;
    a.src = src;
    a.rows = rows;
    a.cols = cols;
    a.elems = elems;
    a.in_row_ptr = in ? in->row_ptr : nullptr;
    a.in_col = in ? in->col_idx : nullptr;
    a.in_val = in ? in->val : nullptr;
    a.eta = eta;
    a.thr = thr;
    a.out_row_ptr = out->row_ptr;
    a.out_col = out->col_idx;
    a.out_val = out->val;
    a.capacity = out->capacity;
    a.hdr = hdr;
    a.status = status;
    a.num_tiles = tiles;
    a.opt = op ? op->opt : kOptSgd;
    a.m = op ? op->m : nullptr;
    a.v = op ? op->v : nullptr;
    a.beta1 = a.beta2 = a.c1 = a.c2 = a.bc1 = a.bc2 = a.eps = 0.f;
    if (op && op->opt != kOptSgd) {
        a.beta1 = op->beta1;
        a.beta2 = op->beta2;
        a.c1 = 1.0f - op->beta1;   // fl32(1 - beta)
        a.c2 = 1.0f - op->beta2;
        a.bc1 = (float)(1.0 - pow((double)op->beta1, (double)op->t));   // fl32(1 - beta^t), power in float64
        a.bc2 = (float)(1.0 - pow((double)op->beta2, (double)op->t));
        a.eps = op->eps;
    }
    if (row_path) {
        const size_t tile_cap = (size_t)rows_per_tile * cols;
        const size_t smem = prox ? prox_smem_floats((int64_t)tile_cap, rows_per_tile) * sizeof(float) : 0;
        static bool attr_done[64] = {false};
        int dev = 0;
        cudaGetDevice(&dev);
        if (dev >= 0 && dev < 64 && !attr_done[dev]) {
            const int max_smem = (int)(imax(prox_smem_floats(kRowMaxK, kRowBudget),
                                            prox_cp_smem_floats(kRowMaxK, kRowBudget)) * sizeof(float));
            CSRT_CHECK_CUDA(cudaFuncSetAttribute(prox_rows_kernel<true>,
                                                 cudaFuncAttributeMaxDynamicSharedMemorySize, max_smem));
            CSRT_CHECK_CUDA(cudaFuncSetAttribute(prox_rows_kernel<false>,
                                                 cudaFuncAttributeMaxDynamicSharedMemorySize, max_smem));
            CSRT_CHECK_CUDA(cudaFuncSetAttribute(prox_count_kernel<true>,
                                                 cudaFuncAttributeMaxDynamicSharedMemorySize, max_smem));
            CSRT_CHECK_CUDA(cudaFuncSetAttribute(prox_count_kernel<false>,
                                                 cudaFuncAttributeMaxDynamicSharedMemorySize, max_smem));
            attr_done[dev] = true;
        }
        if (prox) {
            const bool bits = want_bits && cols % 32 == 0 &&
                              ws_bytes >= kWsReservedBytes + status_bytes(elems) + 2 * bits_bytes(rows, cols) +
                                              transpose_scratch_bytes(rows, cols);
            char *base = ws_scratch(ws);
            uint32_t *keepbits = reinterpret_cast<uint32_t *>(base + status_bytes(elems));
            int32_t *wordpos = reinterpret_cast<int32_t *>(base + status_bytes(elems) + bits_bytes(rows, cols));
            const size_t pre = status_bytes(elems) + 2 * bits_bytes(rows, cols) + transpose_scratch_bytes(rows, cols);
            const PlaceLayout P = place_layout(rows, cols);
            if (a.opt == kOptSgd && eta > 0.f && P.total > 0 && P.rows_per_tile == rows_per_tile &&
                ws_bytes >= kWsReservedBytes + pre + P.total) {
                // count, the new row pointers (clamped to the capacity, overflow reported), place
                char *pb = base + pre;
                int32_t *rowcnt = reinterpret_cast<int32_t *>(pb + P.off_rowcnt);
                int32_t *raw = reinterpret_cast<int32_t *>(pb + P.off_raw);
                int32_t *tilecnt = reinterpret_cast<int32_t *>(pb + P.off_tilecnt);
                int32_t *st_col = reinterpret_cast<int32_t *>(pb + P.off_stcol);
                float *st_val = reinterpret_cast<float *>(pb + P.off_stval);
                const size_t smem_cp = prox_cp_smem_floats((int64_t)tile_cap, rows_per_tile) * sizeof(float);
                const bool words = want_bits;
                if (words)
                    launch_pdl(prox_count_kernel<true>, dim3((unsigned)tiles), dim3(kCThreads), smem_cp, s, a,
                               rows_per_tile, keepbits, wordpos, cols / 32, rowcnt, tilecnt, st_col, st_val, P.stash);
                else
                    launch_pdl(prox_count_kernel<false>, dim3((unsigned)tiles), dim3(kCThreads), smem_cp, s, a,
                               rows_per_tile, keepbits, nullptr, cols / 32, rowcnt, tilecnt, st_col, st_val, P.stash);
                count_launch();
                int rc = check_launch("prox count kernel");
                if (rc) return rc;
                // the row pointers: in the place kernel (a reduction over the tiles' counts) up to
                // kPlaceMaxTiles tiles, else a scan of the row counts first
                const bool prefix = tiles <= kPlaceMaxTiles;
                if (!prefix) {
                    rc = scan_exclusive_i32_clamped(rowcnt, rows, raw, out->row_ptr, out->capacity, ws, s);
                    if (rc) return rc;
                }
                const dim3 pgrid((unsigned)ceil_div<int64_t>(tiles, kPlaceTiles));
                const uint32_t *kb = words ? keepbits : nullptr;
                int32_t *wp = words ? wordpos : nullptr;
                if (words && prefix)
                    launch_pdl(prox_place_kernel<true, true>, pgrid, dim3(kCThreads), 0, s, a, rows_per_tile, kb, wp,
                               cols / 32, rowcnt, raw, tilecnt, st_col, st_val, P.stash);
                else if (words)
                    launch_pdl(prox_place_kernel<true, false>, pgrid, dim3(kCThreads), 0, s, a, rows_per_tile, kb, wp,
                               cols / 32, rowcnt, raw, tilecnt, st_col, st_val, P.stash);
                else if (prefix)
                    launch_pdl(prox_place_kernel<false, true>, pgrid, dim3(kCThreads), 0, s, a, rows_per_tile, kb, wp,
                               cols / 32, rowcnt, raw, tilecnt, st_col, st_val, P.stash);
                else
                    launch_pdl(prox_place_kernel<false, false>, pgrid, dim3(kCThreads), 0, s, a, rows_per_tile, kb,
                               wp, cols / 32, rowcnt, raw, tilecnt, st_col, st_val, P.stash);
                if (bits_done) *bits_done = words;
                count_launch();
                return check_launch("prox place kernel");
            }
            if (bits)
                launch_pdl(prox_rows_kernel<true>, dim3((unsigned)tiles), dim3(kCThreads), smem, s, a,
                           rows_per_tile, keepbits, wordpos, cols / 32);
            else
                launch_pdl(prox_rows_kernel<false>, dim3((unsigned)tiles), dim3(kCThreads), smem, s, a,
                           rows_per_tile, nullptr, nullptr, 0);
            if (bits_done) *bits_done = bits;
        } else {
            launch_pdl(compact_rows_kernel<false>, dim3((unsigned)tiles), dim3(kCThreads), 0, s, a, rows_per_tile);
        }
        count_launch();
        return check_launch("row-tile compaction kernel");
    }
    const bool vec = (reinterpret_cast<uintptr_t>(src) & 15) == 0;
    dim3 grid((unsigned)tiles), block(kCThreads);
    if (prox) {
        if (vec) launch_pdl(compact_kernel<true, true>, dim3(grid), dim3(block), 0, s, a);
        else launch_pdl(compact_kernel<true, false>, dim3(grid), dim3(block), 0, s, a);
    } else {
        if (vec) launch_pdl(compact_kernel<false, true>, dim3(grid), dim3(block), 0, s, a);
        else launch_pdl(compact_kernel<false, false>, dim3(grid), dim3(block), 0, s, a);
    }
    count_launch();
    return check_launch("compact_kernel");
}

// ---------------------------------------------------------------------------
// Transposed pattern (column-wise copy), deterministic.
// ---------------------------------------------------------------------------
constexpr int kTrRows = 32;      // rows per block: one bit each in a 32-bit word
constexpr int kTrChunk = 4096;   // most columns per block (16 KB of bitmask words)

size_t transpose_scratch_bytes(int32_t rows, int32_t cols) {
    const int64_t nb = ceil_div<int64_t>(rows, kTrRows);
    return (size_t)(nb * cols + cols + 64) * sizeof(int32_t);
}

// Bitmask of the rows of block b present in each column of chunk [c0, c0+cw).
__device__ __forceinline__ void tr_build_bits(unsigned int *bits, const int32_t *__restrict__ row_ptr,
                                              const int32_t *__restrict__ col, int32_t rows, int b,
                                              int c0, int cw, bool chunked) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int j = threadIdx.x; j < cw; j += blockDim.x) bits[j] = 0u;
    __syncthreads();
    for (int rr = warp; rr < kTrRows; rr += blockDim.x / 32) {
        const int r = b * kTrRows + rr;
        if (r >= rows) break;
        int64_t s = row_ptr[r], e = row_ptr[r + 1];
        if (chunked) {
            s = warp_lower_bound(col, s, e, c0);
            e = warp_lower_bound(col, s, e, c0 + cw);
        }
        for (int64_t k = s + lane; k < e; k += 32) atomicOr(&bits[__ldg(col + k) - c0], 1u << rr);
    }
    __syncthreads();
}

__global__ void __launch_bounds__(256) tr_count_kernel(const int32_t *__restrict__ row_ptr,
                                                       const int32_t *__restrict__ col, int32_t rows,
                                                       int32_t cols, int32_t chunk, int32_t *__restrict__ cnt) {
    pdl_enter();
    __shared__ unsigned int bits[kTrChunk];
    const int b = blockIdx.x, c0 = blockIdx.y * chunk;
    const int cw = min(chunk, cols - c0);
    tr_build_bits(bits, row_ptr, col, rows, b, c0, cw, gridDim.y > 1);
    int32_t *out = cnt + (int64_t)b * cols + c0;
    for (int j = threadIdx.x; j < cw; j += blockDim.x) out[j] = __popc(bits[j]);
}

// Exclusive scan of cnt[b][j] over b for 32 columns per block; column totals.
__global__ void __launch_bounds__(256) tr_colscan_kernel(int32_t *__restrict__ cnt, int32_t nb,
                                                         int32_t cols, int32_t *__restrict__ coltot) {
    pdl_enter();
    colscan_block(cnt, nb, cols, coltot, blockIdx.x);
}

// Exclusive scan of n values into out[0..n] (out[n] = total); one block.
__global__ void __launch_bounds__(1024) scan_single_block_kernel(const int32_t *__restrict__ in, int32_t n,
                                                                 int32_t *__restrict__ out) {
    pdl_enter();
    scan_block_1024(in, n, out, nullptr, 0, nullptr);
}

// The same scan, also writing the row pointers clamped to a CSR's capacity
// (a no-op unless the output overflows, which is then reported with the
// needed nnz): `out` keeps the unclamped pointers for the kernel that places
// the entries (whose stores check the capacity themselves).
__global__ void __launch_bounds__(1024) scan_clamped_kernel(const int32_t *__restrict__ in, int32_t n,
                                                            int32_t *__restrict__ out,
                                                            int32_t *__restrict__ out_clamped, int64_t capacity,
                                                            WsHeader *hdr) {
    pdl_enter();
    scan_block_1024(in, n, out, out_clamped, capacity, hdr);
}

int scan_exclusive_i32_clamped(const int32_t *in, int32_t n, int32_t *out, int32_t *out_clamped, int64_t capacity,
                               void *ws, cudaStream_t s) {
    launch_pdl(scan_clamped_kernel, dim3(1), dim3(1024), 0, s, in, n, out, out_clamped, capacity,
               static_cast<WsHeader *>(ws));
    count_launch();
    return check_launch("scan_clamped_kernel");
}

// Write kernel: one block per (32-row block, 256-column chunk). Phase A
// gathers the block's entries into a shared 32 x 256 value tile and the row
// bitmask of each column; phase B walks the columns one warp each, lane = row,
// so each column's run of entries leaves as one coalesced store; phase C
// writes t_pos in CSR order.
constexpr int kTwCols = 256;

__global__ void __launch_bounds__(256) tr_write_kernel(const int32_t *__restrict__ row_ptr,
                                                       const int32_t *__restrict__ col,
                                                       const float *__restrict__ val, int32_t rows,
                                                       int32_t cols, const int32_t *__restrict__ off,
                                                       const int32_t *__restrict__ t_row_ptr,
                                                       int32_t *__restrict__ t_col, float *__restrict__ t_val,
                                                       int32_t *__restrict__ t_pos, int64_t capacity) {
    pdl_enter();
    __shared__ unsigned int bits[kTwCols];
    __shared__ int32_t base[kTwCols];            // first position of this block's run in each column
    __shared__ float vt[kTrRows][kTwCols + 1];   // values of the block's entries, padded
    const int b = blockIdx.x, c0 = blockIdx.y * kTwCols;
    const int cw = min(kTwCols, cols - c0);
    const bool chunked = gridDim.y > 1;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int j = threadIdx.x; j < cw; j += blockDim.x) {
        bits[j] = 0u;
        base[j] = t_row_ptr[c0 + j] + off[(int64_t)b * cols + c0 + j];
    }
    __syncthreads();
    // phase A
    for (int rr = warp; rr < kTrRows; rr += 8) {
        const int r = b * kTrRows + rr;
        if (r >= rows) break;
        int64_t s = row_ptr[r], e = row_ptr[r + 1];
        if (chunked) {
            s = warp_lower_bound(col, s, e, c0);
            e = warp_lower_bound(col, s, e, c0 + cw);
        }
        for (int64_t k = s + lane; k < e; k += 32) {
            const int j = __ldg(col + k) - c0;
            atomicOr(&bits[j], 1u << rr);
            vt[rr][j] = __ldg(val + k);
        }
    }
    __syncthreads();
    // phase B: lane = row within the block
    const int my_row = b * kTrRows + lane;
    const unsigned below = (1u << lane) - 1u;
    for (int j = warp; j < cw; j += 8) {
        const unsigned m = bits[j];
        if ((m >> lane) & 1u) {
            const int64_t p = (int64_t)base[j] + __popc(m & below);
            if (p < capacity) {
                t_col[p] = my_row;
                t_val[p] = vt[lane][j];
            }
        }
    }
    // phase C: t_pos in CSR order
    for (int rr = warp; rr < kTrRows; rr += 8) {
        const int r = b * kTrRows + rr;
        if (r >= rows) break;
        int64_t s = row_ptr[r], e = row_ptr[r + 1];
        if (chunked) {
            s = warp_lower_bound(col, s, e, c0);
            e = warp_lower_bound(col, s, e, c0 + cw);
        }
        const unsigned below_rr = (1u << rr) - 1u;
        for (int64_t k = s + lane; k < e; k += 32) {
            const int j = __ldg(col + k) - c0;
            const int64_t p = (int64_t)base[j] + __popc(bits[j] & below_rr);
            if (p < capacity) t_pos[k] = (int32_t)p;
        }
    }
}


// ---------------------------------------------------------------------------
// Transposed copy from the prox kernel's keep bitmask (K % 32 == 0). One warp
// per (32-row block b, 32-column word c).
//  count: lane r loads row r's word; a 32 x 32 bit transpose (five shuffle
//         stages) gives lane j the rows present in column 32c + j; its popcount
//         is the block's count for that column.
//  write: the block's kept entries are enumerated twice, 32 at a time, one
//         entry per lane. Row-major order (the CSR order): the entry's row is
//         found by a binary search over the rows' exclusive kept counts, its
//         column as the k-th set bit of the row's word; its CSR position is
//         the word position + k, so the value is read and t_pos written
//         coalesced, and the value goes to a 32 x 32 shared tile.
//         Column-major order (the transposed order): the same with the
//         columns' counts and masks; consecutive entries of a column are
//         consecutive positions of its transposed run, so t_col and t_val
//         are written coalesced as well. A pass costs ceil(kept / 32)
//         iterations instead of one per row (or column) of the block; a
//         block with more than kTrbWalkMin kept entries is instead walked
//         row by row (lane = column) and column by column (lane = row),
//         which is cheaper once most lanes hold an entry.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) trb_count_kernel(const uint32_t *__restrict__ keepbits, int32_t rows,
                                                        int32_t wpr, int32_t cols, int32_t *__restrict__ cnt) {
    pdl_enter();
    const int lane = threadIdx.x & 31;
    const int64_t gw = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nb = ceil_div<int64_t>(rows, 32);
    if (gw >= nb * wpr) return;
    const int b = (int)(gw / wpr), c = (int)(gw % wpr);
    const int row = b * 32 + lane;
    const uint32_t x = row < rows ? __ldg(keepbits + (int64_t)row * wpr + c) : 0u;
    const uint32_t colmask = warp_transpose32(x);
    cnt[(int64_t)b * cols + c * 32 + lane] = __popc(colmask);
}

// Position of the k-th (from 0) set bit of m, for k < popc(m); always 0..31.
__device__ __forceinline__ int nth_set_bit(uint32_t m, int k) {
    int pos = 0;
#pragma unroll
    for (int sft = 16; sft >= 1; sft >>= 1) {
        const int c = __popc(m & ((1u << sft) - 1u));
        if (k >= c) {
            k -= c;
            m >>= sft;
            pos += sft;
        }
    }
    return pos;
}

// Largest lane r with pre(r) <= e, for pre nondecreasing over the lanes and
// pre(0) = 0 <= e. Every lane of the warp must call it.
__device__ __forceinline__ int warp_last_le(int pre, int e) {
    int r = 0;
#pragma unroll
    for (int sft = 16; sft >= 1; sft >>= 1) {
        const int v = __shfl_sync(0xffffffffu, pre, r + sft);
        if (v <= e) r += sft;
    }
    return r;
}

__device__ __forceinline__ int warp_exclusive_sum(int x, int &total) {
    const int lane = threadIdx.x & 31;
    int inc = x;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, inc, d);
        if (lane >= d) inc += y;
    }
    total = __shfl_sync(0xffffffffu, inc, 31);
    return inc - x;
}

constexpr int kTrbWalkMin = 384;   // kept entries of a 32 x 32 block above which it is walked

__global__ void __launch_bounds__(256) trb_write_kernel(const uint32_t *__restrict__ keepbits,
                                                        const int32_t *__restrict__ wordpos, int32_t rows,
                                                        int32_t wpr, int32_t cols, const int32_t *__restrict__ off,
                                                        const int32_t *__restrict__ t_row_ptr,
                                                        const float *__restrict__ val, int32_t *__restrict__ t_col,
                                                        float *__restrict__ t_val, int32_t *__restrict__ t_pos,
                                                        int64_t capacity) {
    pdl_enter();
    __shared__ float tile[8][32 * 32];   // element (r, j) at r*32 + (j ^ r)
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t gw = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nb = ceil_div<int64_t>(rows, 32);
    if (gw >= nb * wpr) return;   // whole warps
    const int b = (int)(gw / wpr), c = (int)(gw % wpr);
    const int my_row = b * 32 + lane;
    const uint32_t rw_mine = my_row < rows ? __ldg(keepbits + (int64_t)my_row * wpr + c) : 0u;
    const int32_t rp_mine = my_row < rows ? __ldg(wordpos + (int64_t)my_row * wpr + c) : 0;
    const int col = c * 32 + lane;
    // start of this block's part of column `col`'s transposed run
    const int64_t cb_mine = (int64_t)__ldg(t_row_ptr + col) + __ldg(off + (int64_t)b * cols + col);
    const uint32_t cm_mine = warp_transpose32(rw_mine);   // lane j: the block's rows kept in column 32c + j
    int total;
    const int rpre = warp_exclusive_sum(__popc(rw_mine), total);
    const int cpre = warp_exclusive_sum(__popc(cm_mine), total);
    float *tl = tile[warp];
    if (total > kTrbWalkMin) {
        // a dense block: walk its rows (lane = column) and then its columns
        // (lane = row); a step per row or column costs less than the search
        // of the enumeration once most lanes hold an entry
        // The 32 rows' values are loaded first, all in flight at once, then
        // staged (loading and staging row by row waited once per row).
        const unsigned lt = (1u << lane) - 1u;
        float v[32];
#pragma unroll
        for (int r = 0; r < 32; ++r) {
            const uint32_t rw = __shfl_sync(0xffffffffu, rw_mine, r);
            const int64_t pr = (int64_t)__shfl_sync(0xffffffffu, rp_mine, r) + __popc(rw & lt);
            v[r] = ((rw >> lane) & 1u) && pr < capacity ? __ldg(val + pr) : 0.f;
        }
        int64_t pc = cb_mine;
#pragma unroll
        for (int r = 0; r < 32; ++r) {
            const uint32_t rw = __shfl_sync(0xffffffffu, rw_mine, r);
            const int64_t pr = (int64_t)__shfl_sync(0xffffffffu, rp_mine, r) + __popc(rw & lt);
            if ((rw >> lane) & 1u) {
                tl[r * 32 + (lane ^ r)] = v[r];
                if (pc < capacity && pr < capacity) t_pos[pr] = (int32_t)pc;
                ++pc;
            }
        }
        __syncwarp();
        for (int j = 0; j < 32; ++j) {
            const uint32_t cm = __shfl_sync(0xffffffffu, cm_mine, j);
            if (cm == 0u) continue;
            const int64_t base = __shfl_sync(0xffffffffu, cb_mine, j);
            if ((cm >> lane) & 1u) {
                const int64_t p = base + __popc(cm & lt);
                if (p < capacity) {
                    t_col[p] = b * 32 + lane;
                    t_val[p] = tl[lane * 32 + (j ^ lane)];
                }
            }
        }
        return;
    }
    constexpr int kRounds = 4;   // 32-entry rounds whose value loads are in flight together
    for (int e00 = 0; e00 < total; e00 += 32 * kRounds) {   // row-major (CSR) order
        float v[kRounds];
        int64_t pr[kRounds], pc[kRounds];
        int at[kRounds];
#pragma unroll
        for (int q = 0; q < kRounds; ++q) {
            at[q] = -1;
            if (e00 + 32 * q >= total) continue;   // the same for every lane
            const int e = e00 + 32 * q + lane;
            const int r = warp_last_le(rpre, e);
            const uint32_t rw = __shfl_sync(0xffffffffu, rw_mine, r);
            const int k = e - __shfl_sync(0xffffffffu, rpre, r);
            const int32_t rp = __shfl_sync(0xffffffffu, rp_mine, r);
            const int j = nth_set_bit(rw, k);
            const uint32_t cm = __shfl_sync(0xffffffffu, cm_mine, j);
            const int64_t cb = __shfl_sync(0xffffffffu, cb_mine, j);
            pr[q] = (int64_t)rp + k;
            pc[q] = cb + __popc(cm & ((1u << r) - 1u));
            at[q] = e < total ? r * 32 + (j ^ r) : -1;
            v[q] = e < total && pr[q] < capacity ? __ldg(val + pr[q]) : 0.f;
        }
#pragma unroll
        for (int q = 0; q < kRounds; ++q) {
            if (e00 + 32 * q < total && at[q] >= 0) {
                tl[at[q]] = v[q];
                if (pc[q] < capacity && pr[q] < capacity) t_pos[pr[q]] = (int32_t)pc[q];
            }
        }
    }
    __syncwarp();
    for (int e0 = 0; e0 < total; e0 += 32) {   // column-major (transposed) order
        const int e = e0 + lane;
        const int j = warp_last_le(cpre, e);
        const uint32_t cm = __shfl_sync(0xffffffffu, cm_mine, j);
        const int k = e - __shfl_sync(0xffffffffu, cpre, j);
        const int64_t cb = __shfl_sync(0xffffffffu, cb_mine, j);
        const int r = nth_set_bit(cm, k);
        if (e < total) {
            const int64_t p = cb + k;
            if (p < capacity) {
                t_col[p] = b * 32 + r;
                t_val[p] = tl[r * 32 + (j ^ r)];
            }
        }
    }
}

// Column pointers of the transposed copy (t_row_ptr) and, per 32-row block
// and column, the block's offset in the column's run (in `scratch`, nb x cols
// int32, followed by the column totals), from a keep bitmask (cols % 32 == 0).
static int transpose_bits_prepare(csrt_csr *w, const uint32_t *keepbits, void *scratch, size_t scratch_bytes,
                                  cudaStream_t s) {
    const int32_t rows = w->rows, cols = w->cols;
    const int32_t wpr = cols / 32;
    CSRT_ARG(scratch_bytes >= transpose_scratch_bytes(rows, cols), "scratch too small for the transposed copy");
    int32_t *cnt = static_cast<int32_t *>(scratch);
    const int nb = (int)ceil_div<int64_t>(rows, 32);
    int32_t *coltot = cnt + (int64_t)nb * cols;
    const int64_t warps = (int64_t)nb * wpr;
    const unsigned grid = (unsigned)ceil_div<int64_t>(warps * 32, 256);
    launch_pdl(trb_count_kernel, dim3(grid), dim3(256), 0, s, keepbits, rows, wpr, cols, cnt);
    launch_pdl(tr_colscan_kernel, dim3(ceil_div(cols, 32)), dim3(256), 0, s, cnt, nb, cols, coltot);
    launch_pdl(scan_single_block_kernel, dim3(1), dim3(1024), 0, s, coltot, cols, w->t_row_ptr);
    count_launch(3);
    return check_launch("transposed-copy count kernels");
}

// Transposed copy from a keep bitmask and word positions (cols % 32 == 0);
// `scratch` holds the per-block column counts and the column totals.
int transpose_from_bits_ext(csrt_csr *w, const uint32_t *keepbits, const int32_t *wordpos, void *scratch,
                            size_t scratch_bytes, cudaStream_t s) {
    int rc = transpose_bits_prepare(w, keepbits, scratch, scratch_bytes, s);
    if (rc) return rc;
    const int32_t rows = w->rows, cols = w->cols;
    const int32_t wpr = cols / 32;
    const int32_t *cnt = static_cast<const int32_t *>(scratch);
    const int nb = (int)ceil_div<int64_t>(rows, 32);
    const int64_t warps = (int64_t)nb * wpr;
    const unsigned grid = (unsigned)ceil_div<int64_t>(warps * 32, 256);
    launch_pdl(trb_write_kernel, dim3(grid), dim3(256), 0, s, keepbits, wordpos, rows, wpr, cols, cnt, w->t_row_ptr,
               w->val, w->t_col_idx, w->t_val, w->t_pos, w->capacity);
    count_launch(1);
    return check_launch("transpose-from-bits kernels");
}

// Prox-kernel layout of the workspace: [status][keepbits][wordpos][cnt][coltot].
static int transpose_from_bits(csrt_csr *w, void *ws, size_t ws_bytes, cudaStream_t s) {
    const int32_t rows = w->rows, cols = w->cols;
    const int64_t elems = (int64_t)rows * cols;
    char *base = ws_scratch(ws);
    const uint32_t *keepbits = reinterpret_cast<const uint32_t *>(base + status_bytes(elems));
    const int32_t *wordpos = reinterpret_cast<const int32_t *>(base + status_bytes(elems) + bits_bytes(rows, cols));
    char *scratch = base + status_bytes(elems) + 2 * bits_bytes(rows, cols);
    return transpose_from_bits_ext(w, keepbits, wordpos, scratch, transpose_scratch_bytes(rows, cols), s);
}

// Exclusive scan of n int32 values into out[0..n] (out[n] = total), one block.
int scan_exclusive_i32(const int32_t *in, int32_t n, int32_t *out, cudaStream_t s) {
    launch_pdl(scan_single_block_kernel, dim3(1), dim3(1024), 0, s, in, n, out);
    count_launch();
    return check_launch("scan_single_block_kernel");
}

int transpose_impl(csrt_csr *w, void *ws, size_t ws_bytes, cudaStream_t s) {
    CSRT_ARG(w->t_row_ptr && w->t_col_idx && w->t_val && w->t_pos, "transposed arrays not set");
    const int32_t rows = w->rows, cols = w->cols;
    if (cols == 0) return CSRT_OK;
    if (rows == 0) {
        CSRT_CHECK_CUDA(cudaMemsetAsync(w->t_row_ptr, 0, sizeof(int32_t) * ((size_t)cols + 1), s));
        return CSRT_OK;
    }
    CSRT_ARG(ws_bytes >= kWsReservedBytes + transpose_scratch_bytes(rows, cols), "workspace too small for transpose");
    const int nb = (int)ceil_div<int64_t>(rows, kTrRows);
    // Enough blocks to fill the GPU: split the columns into chunks of at least
    // 256 (and at most kTrChunk) so that nb * nc reaches ~4 blocks per SM.
    int nc = (int)imax<int64_t>(ceil_div<int64_t>(cols, kTrChunk),
                                imin<int64_t>(ceil_div<int64_t>(4 * num_sms(), nb), ceil_div<int64_t>(cols, 256)));
    const int chunk = (int)ceil_div<int64_t>(ceil_div<int64_t>(cols, nc), 32) * 32;
    nc = (int)ceil_div<int64_t>(cols, chunk);
    int32_t *cnt = reinterpret_cast<int32_t *>(ws_scratch(ws));
    int32_t *coltot = cnt + (int64_t)nb * cols;
    launch_pdl(tr_count_kernel, dim3(dim3(nb, nc)), dim3(256), 0, s, w->row_ptr, w->col_idx, rows, cols, chunk, cnt);
    launch_pdl(tr_colscan_kernel, dim3(ceil_div(cols, 32)), dim3(256), 0, s, cnt, nb, cols, coltot);
    launch_pdl(scan_single_block_kernel, dim3(1), dim3(1024), 0, s, coltot, cols, w->t_row_ptr);
    launch_pdl(tr_write_kernel, dim3(dim3(nb, (unsigned)ceil_div<int64_t>(cols, kTwCols))), dim3(256), 0, s,
        w->row_ptr, w->col_idx, w->val, rows, cols, cnt, w->t_row_ptr, w->t_col_idx, w->t_val, w->t_pos,
        w->capacity);
    count_launch(4);
    return check_launch("csr_transpose kernels");
}

}  // namespace csrt

using namespace csrt;

static int check_csr(const csrt_csr *w, bool need_t) {
    CSRT_ARG(w != nullptr, "csr is NULL");
    CSRT_ARG(w->rows >= 0 && w->cols >= 0, "negative shape");
    CSRT_ARG((int64_t)w->rows * w->cols < ((int64_t)1 << 31), "rows*cols must be below 2^31");
    CSRT_ARG(w->row_ptr != nullptr, "row_ptr is NULL");
    CSRT_ARG(w->capacity >= 0 && w->capacity < ((int64_t)1 << 31), "capacity out of range");
    CSRT_ARG(w->capacity == 0 || (w->col_idx && w->val), "col_idx/val NULL");
    if (need_t) CSRT_ARG(w->t_row_ptr && w->t_col_idx && w->t_val && w->t_pos, "transposed arrays not set");
    return CSRT_OK;
}

extern "C" {

int csr_from_dense(const float *dense, int32_t rows, int32_t cols, csrt_csr *out, void *ws, size_t ws_bytes,
                   void *stream) {
    int rc = check_csr(out, false);
    if (rc) return rc;
    CSRT_ARG(out->rows == rows && out->cols == cols, "out shape differs from rows/cols");
    CSRT_ARG(dense != nullptr || (int64_t)rows * cols == 0, "dense is NULL");
    CSRT_ARG(ws != nullptr, "workspace is NULL");
    cudaStream_t s = as_stream(stream);
    rc = compact_launch(false, dense, rows, cols, nullptr, 0.f, 0.f, out, ws, ws_bytes, s);
    if (rc) return rc;
    if (out->t_row_ptr) rc = transpose_impl(out, ws, ws_bytes, s);
    return rc;
}

int csr_transpose(csrt_csr *w, void *ws, size_t ws_bytes, void *stream) {
    int rc = check_csr(w, true);
    if (rc) return rc;
    CSRT_ARG(ws != nullptr, "workspace is NULL");
    return transpose_impl(w, ws, ws_bytes, as_stream(stream));
}

static int prox_impl(const csrt_csr *w_in, const float *g, float eta, float lambda, csrt_csr *w_out, void *ws,
                     size_t ws_bytes, void *stream, const OptParams *op) {
    int rc = check_csr(w_in, false);
    if (rc) return rc;
    rc = check_csr(w_out, false);
    if (rc) return rc;
    CSRT_ARG(w_in->rows == w_out->rows && w_in->cols == w_out->cols, "w_in and w_out shapes differ");
    CSRT_ARG(w_in->row_ptr != w_out->row_ptr && w_in->col_idx != w_out->col_idx && w_in->val != w_out->val,
             "w_out must not alias w_in");
    CSRT_ARG(g != nullptr || (int64_t)w_in->rows * w_in->cols == 0, "G is NULL");
    CSRT_ARG(eta >= 0.f && lambda >= 0.f && eta <= 3.0e38f && lambda <= 3.0e38f,
             "eta and lambda must be finite and >= 0");
    CSRT_ARG(ws != nullptr, "workspace is NULL");
    const float thr = eta * lambda;  // fl32(eta*lambda), the threshold of Eq. prox
    cudaStream_t s = as_stream(stream);
    const bool want_t = w_out->t_row_ptr != nullptr;
    if (want_t) CSRT_ARG(w_out->t_col_idx && w_out->t_val && w_out->t_pos, "transposed arrays partly set");
    bool bits = false;
    rc = compact_launch(true, g, w_in->rows, w_in->cols, w_in, eta, thr, w_out, ws, ws_bytes, s, want_t, &bits, op);
    if (rc) return rc;
    if (want_t) rc = bits ? transpose_from_bits(w_out, ws, ws_bytes, s) : transpose_impl(w_out, ws, ws_bytes, s);
    return rc;
}

int prox_update_compact(const csrt_csr *w_in, const float *g, float eta, float lambda, csrt_csr *w_out,
                        void *ws, size_t ws_bytes, void *stream) {
    return prox_impl(w_in, g, eta, lambda, w_out, ws, ws_bytes, stream, nullptr);
}

int csrt_check_bounded_waits(void *ws, size_t ws_bytes, void *stream) {
    CSRT_ARG(ws != nullptr && ws_bytes >= kWsReservedBytes + 2 * sizeof(unsigned long long), "workspace too small");
    cudaStream_t s = as_stream(stream);
    unsigned long long *status = reinterpret_cast<unsigned long long *>(ws_scratch(ws));
    CSRT_CHECK_CUDA(cudaMemsetAsync(status, 0, 2 * sizeof(unsigned long long), s));
    launch_pdl(bounded_wait_check_kernel, dim3(1), dim3(32), 0, s, status, static_cast<WsHeader *>(ws), 0);
    launch_pdl(bounded_wait_check_kernel, dim3(1), dim3(32), 0, s, status, static_cast<WsHeader *>(ws), 1);
    count_launch(2);
    return check_launch("bounded_wait_check_kernel");
}

static int check_moments(const csrt_csr *w, const float *g, const float *m, const float *v, float eps) {
    const bool empty = w == nullptr || (int64_t)w->rows * w->cols == 0;
    CSRT_ARG(empty || v != nullptr, "v is NULL");
    CSRT_ARG(v == nullptr || (v != g && v != m), "v must not alias G or m");
    CSRT_ARG(m == nullptr || m != g, "m must not alias G");
    CSRT_ARG(eps > 0.f && eps <= 3.0e38f, "eps must be finite and > 0");
    return CSRT_OK;
}

int prox_rmsprop_update_compact(const csrt_csr *w_in, const float *g, float *v, float eta, float lambda,
                                float beta, float eps, csrt_csr *w_out, void *ws, size_t ws_bytes, void *stream) {
    int rc = check_moments(w_in, g, nullptr, v, eps);
    if (rc) return rc;
    CSRT_ARG(beta >= 0.f && beta < 1.f, "beta must be in [0, 1)");
    OptParams op;
    op.opt = kOptRmsprop;
    op.m = nullptr;
    op.v = v;
    op.beta1 = 0.f;
    op.beta2 = beta;
    op.eps = eps;
    op.t = 1;
    return prox_impl(w_in, g, eta, lambda, w_out, ws, ws_bytes, stream, &op);
}

int prox_adam_update_compact(const csrt_csr *w_in, const float *g, float *m, float *v, int32_t t, float eta,
                             float lambda, float beta1, float beta2, float eps, csrt_csr *w_out, void *ws,
                             size_t ws_bytes, void *stream) {
    int rc = check_moments(w_in, g, m, v, eps);
    if (rc) return rc;
    const bool empty = w_in == nullptr || (int64_t)w_in->rows * w_in->cols == 0;
    CSRT_ARG(empty || m != nullptr, "m is NULL");
    CSRT_ARG(t >= 1, "the step counter t starts at 1 (got %d)", t);
    CSRT_ARG(beta1 >= 0.f && beta1 < 1.f && beta2 >= 0.f && beta2 < 1.f, "beta1 and beta2 must be in [0, 1)");
    OptParams op;
    op.opt = kOptAdam;
    op.m = m;
    op.v = v;
    op.beta1 = beta1;
    op.beta2 = beta2;
    op.eps = eps;
    op.t = t;
    return prox_impl(w_in, g, eta, lambda, w_out, ws, ws_bytes, stream, &op);
}

}  // extern "C"
