// Fused weight gradient + proximal update + re-compaction (the dense gradient
// never reaches memory).
//
// The prox step (Eq. prox with the soft threshold of Section 2.2, applied to
// the dense w - eta*G as in Section 3.3, compacted after every update as in
// Section 4.4) needs G = dY X^T at every entry, but only once: here the
// tensor-core GEMM's epilogue applies it straight from the accumulator. The
// output position of an entry depends on the kept counts of every earlier row,
// so the GEMM runs twice; the accumulator of a tile is the same in both passes
// (same tiles, same MMA order), hence so are the keep decisions.
//
//  1. fp_oldbits_kernel: per row of W_in, a bitmask of the stored columns and,
//     per 128-column segment, the index of the row's first stored entry in it.
//  2. gemm_prox_tc_kernel<count>: the persistent tcgen05 GEMM of gemm_tc.cu
//     (same tiles, same MMA order, so the same G bits as weight_grad_dense
//     TF32). Each epilogue thread owns one row of a 128-column segment of a
//     128 x 256 tile; per entry it takes w from W_in (through the bitmask:
//     loads only where a weight is stored), forms z = fl(w - fl(eta*G)), keeps
//     |z| > fl(eta*lambda), and writes the keep bitmask and the kept count of
//     the segment.
//  3. fp_rowscan_kernel + scan_clamped_kernel: per-row offsets of the
//     segments and the new row pointers (clamped to the capacity in w_out).
//  4. With a transposed copy wanted: the count pass also writes its column
//     counts per 32-row block (a 32 x 32 bit transpose of the rows' keep
//     words); their scan down each column and the column pointers are taken
//     in the same two launches as step 3 (fp_rows_cols_scan_kernel,
//     fp_two_scans_kernel).
//  5. gemm_prox_tc_kernel<write>: the same GEMM again; the epilogue recomputes
//     z, passes each 32 x 32 block through shared memory and writes the kept
//     entries of one row at a time at their final positions (a coalesced run
//     per row and 32 columns). With the transposed copy (kT) the same staged
//     block is then walked column by column (lane = row): each column's kept
//     rows form one run of the transposed arrays, and each kept entry's
//     transposed position goes to t_pos during the row walk.
// The result is bit-identical to weight_grad_dense (TF32) followed by
// prox_update_compact.
#include "tc_common.cuh"

namespace csrt {

size_t transpose_scratch_bytes(int32_t rows, int32_t cols);

// Segments (the unit of the per-row offsets) are 64 columns, two 32-column
// words; a GEMM tile (256 columns) is four of them.
constexpr int kFpTileCols = 64;                  // columns per segment
constexpr int kFpTileWords = kFpTileCols / 32;   // 2
constexpr int kFpMaxK = 16384;

// Launch shape of each pass: epilogue warps and pipeline stages. Both passes
// are bound by the latency of their epilogues, so both run 16 epilogue warps
// (two per SM sub-partition and TMEM lane quarter, each owning 64 columns of
// a tile) with 3 pipeline stages; measured on the classifier-head step, 16
// warps beat 8 by 1.2% (count pass) and 1.4% (write pass, where the register
// cap of 18 warps asks for 4 prefetched weights and 4-row groups).
#ifndef CSRT_FP_COUNT_EPI
#define CSRT_FP_COUNT_EPI 16
#endif
#ifndef CSRT_FP_WRITE_EPI
#define CSRT_FP_WRITE_EPI 16
#endif
#ifndef CSRT_FP_WRITE_PRE
#define CSRT_FP_WRITE_PRE 4
#endif
#ifndef CSRT_FP_WRITE_GROUP
#define CSRT_FP_WRITE_GROUP 4
#endif
// kPre: stored old weights per word prefetched into registers; kGroup: rows
// of a word handled together in the write pass's column domain.
template <bool kWrite> struct FpShape;
template <> struct FpShape<false> {
    // kPre 4 rather than 8: 15% fewer instructions, the count pass of the
    // 4096 x 9216 layer 45.4 -> 44.4 us (at 5% density 2% of the rows' words
    // hold more than four stored weights, half the warps' words one such row;
    // the loop after the prefetched ones takes them)
    static constexpr int kEpi = CSRT_FP_COUNT_EPI, kStages = CSRT_FP_COUNT_EPI > 8 ? 3 : 4, kPre = 4, kGroup = 8;
};
#ifndef CSRT_FP_WRITE_STAGE_WORDS
#define CSRT_FP_WRITE_STAGE_WORDS 1
#endif
template <> struct FpShape<true> {
    // kStageWords: words of the span staged before they are written row by
    // row (the shared memory they take leaves 2 pipeline stages at 4 words,
    // 3 at 1 or 2). Staging 4 words completes each output sector within one
    // warp's consecutive stores (196 -> 186 us on a dense 4096 x 9216 output)
    // but costs the classifier-head step 5% (its outputs are 17-25% dense and
    // its MMA pipeline needs the third stage): 1 is the default.
    static constexpr int kEpi = CSRT_FP_WRITE_EPI, kPre = CSRT_FP_WRITE_PRE, kGroup = CSRT_FP_WRITE_GROUP,
                         kStageWords = CSRT_FP_WRITE_STAGE_WORDS, kStages = kStageWords > 2 ? 2 : 3;
};
// Threads of a pass: the producer warps (TMA, MMA; with kSplit a whole
// warpgroup of four, two of them idle) and the epilogue warps.
template <bool kWrite, bool kSplit = false> constexpr int fp_threads() {
    return (kSplit ? 128 : 64) + FpShape<kWrite>::kEpi * 32;
}
// kSplit (write pass): the producer warpgroup gives up registers, the four
// epilogue warpgroups take them (setmaxnreg), within the launch's allocation
// of 640 threads x 96 registers: 128 x 32 + 512 x 112 = 61,440. The 18-warp
// launch caps every thread at 96 registers, where the write pass spills
// (48-60 bytes); split, it does not (4096 x 9216 layer 136.2 -> 132.4 us,
// 4096 x 4096 with the transposed copy 114.5 -> 109.6 us). A cap of 112 for
// all 18 warps does not launch: registers are allocated for whole groups of
// four warps.
constexpr int kFpProdRegs = 32, kFpEpiRegs = 112;
static_assert(128 * kFpProdRegs + FpShape<true>::kEpi * 32 * kFpEpiRegs <= fp_threads<true, true>() * 96,
              "register split above the launch's allocation");
// Per epilogue warp: 32 x 32 float buffers, row r's 16-byte chunk c at float
// offset r*32 + ((c ^ (r & 7)) << 2), so that a row written as eight 16-byte
// stores and a column read one element per lane are both free of bank
// conflicts. The count pass needs one; the write pass one per word of its
// span (it stages the whole span before writing).
template <bool kWrite> __host__ __device__ constexpr int fp_span_words() {
    return kTcBN / (FpShape<kWrite>::kEpi / 4) / 32;
}
template <bool kWrite> __host__ __device__ constexpr int fp_xfloats() {
    return 32 * 32 * (kWrite ? FpShape<true>::kStageWords : 1);
}
// The write pass also keeps, per epilogue warp, a 32 x 32 byte buffer of the
// column offsets of each row's kept entries (sparse words, fp_write_compact).
template <bool kWrite> constexpr int fp_cbytes() { return kWrite ? 32 * 32 : 0; }
template <bool kWrite> constexpr int fp_smem_bytes() {
    return FpShape<kWrite>::kStages * kTcStageBytes + 1024 + 256 +
           FpShape<kWrite>::kEpi * (fp_xfloats<kWrite>() * 4 + fp_cbytes<kWrite>());
}
static_assert(fp_smem_bytes<false>() <= 232448 && fp_smem_bytes<true>() <= 232448, "shared memory per block");

struct FpLayout {
    int32_t nt, wpr;
    size_t off_obits, off_ostart, off_kbits, off_counts, off_rowtot, off_rawptr, off_wordpos, off_tr, total;
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
    L.off_rawptr = o;  o += align256((size_t)(m + 1) * 4);
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
    pdl_enter();
    __shared__ uint32_t sw[8][kFpMaxK / 32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t r = (int64_t)blockIdx.x * 8 + warp;
    if (r >= m) return;
    uint32_t *w = sw[warp];
    const int32_t s = row_ptr[r], e = row_ptr[r + 1];
    for (int i = lane; i < wpr; i += 32) w[i] = 0u;
    __syncwarp();
    // sixteen independent column loads in flight per lane: a row of up to 512
    // stored entries in one round (the kernel is bound by their latency: one
    // warp per row, few rows per SM)
    for (int32_t k = s + lane; k < e; k += 512) {
        int c[16];
#pragma unroll
        for (int u = 0; u < 16; ++u) c[u] = k + 32 * u < e ? __ldg(col + k + 32 * u) : -1;
#pragma unroll
        for (int u = 0; u < 16; ++u)
            if (c[u] >= 0) atomicOr(&w[c[u] >> 5], 1u << (c[u] & 31));
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
    uint32_t *kbits;     // count pass: keep bitmask per 32-column word
    int32_t *counts;     // count pass: kept entries per (row, segment); write pass: their offsets in the row
    const int32_t *row_ptr_out;   // write pass: new row pointers (not yet clamped to the capacity)
    int32_t *out_col;
    float *out_val;
    int32_t *wordpos;    // write pass: position of each word's first kept entry (or null)
    int64_t capacity;
    WsHeader *hdr;
};

// Write pass with the transposed copy: the start of each column's run (t_rp)
// and, per 32-row block and column, the block's offset in it (t_off), from the
// count pass's keep bits; the transposed arrays.
struct FpTArgs {
    const int32_t *t_rp, *t_off;
    int32_t *t_col;
    float *t_val;
    int32_t *t_pos;
    int32_t *t_cnt;   // count pass: kept rows per (32-row block, column)
};


// Per-tile inputs of an epilogue thread (its row of the tile's column span):
// the stored-weight bitmask of each word, the index of the span's first stored
// weight and, in the write pass, the position of its first kept entry and
// (transposed copy) the start of the run of column 32 * word + lane in the
// warp's 32-row block.
template <int W, bool kT>
struct FpMeta {
    uint32_t ob[W];
    uint32_t kb[W];   // write pass: the keep bitmask the count pass wrote
    int32_t cb[kT ? W : 1];
    int32_t o0, pos;
};

template <bool kWrite, bool kT, int W>
__device__ __forceinline__ void fp_load_meta(const FpArgs &a, const FpTArgs &ta, int t, int num_tiles, int tiles_n,
                                             int h, int64_t rowq, FpMeta<W, kT> &m) {
    const int mt = t / tiles_n, nt = t % tiles_n;
    const int64_t row = (int64_t)mt * kTcBM + rowq;
    const bool rv = t < num_tiles && row < a.m;
    const int word0 = nt * (kTcBN / 32) + h * W;
    const int seg0 = word0 / kFpTileWords;
    const bool sv = rv && seg0 < a.nt;
#pragma unroll
    for (int c = 0; c < W; ++c) m.ob[c] = (rv && word0 + c < a.wpr) ? __ldg(a.obits + row * a.wpr + word0 + c) : 0u;
#pragma unroll
    for (int c = 0; c < W; ++c)
        m.kb[c] = (kWrite && rv && word0 + c < a.wpr) ? __ldg(a.kbits + row * a.wpr + word0 + c) : 0u;
    m.o0 = sv ? __ldg(a.ostart + row * (a.nt + 1) + seg0) : 0;
    m.pos = (kWrite && sv) ? __ldg(a.row_ptr_out + row) + __ldg(a.counts + row * a.nt + seg0) : 0;
    if constexpr (kT) {
        const int64_t brow = (int64_t)mt * kTcBM + (rowq & ~(int64_t)31);   // the warp's 32-row block
        const bool bv = t < num_tiles && brow < a.m;
#pragma unroll
        for (int c = 0; c < W; ++c) {
            const int64_t col = (int64_t)(word0 + c) * 32 + (rowq & 31);
            m.cb[c] = (bv && word0 + c < a.wpr) ? __ldg(ta.t_rp + col) + __ldg(ta.t_off + (brow >> 5) * a.k + col) : 0;
        }
    }
}

// The first N stored weights of a word (its bitmask ob, first index o).
template <int N>
__device__ __forceinline__ void fp_load_words(const float *__restrict__ old_val, uint32_t ob, int32_t o,
                                              float (&wv)[N]) {
    const int nc = __popc(ob);
#pragma unroll
    for (int u = 0; u < N; ++u) wv[u] = u < nc ? __ldg(old_val + o + u) : 0.f;
}

// Transposed copy of one staged 32 x 32 word (element (r, j) at r*32 + (j ^
// ((r & 7) << 2))), lane = row: each column j's kept rows form one run in row
// order starting at cb_j, the start of column j's run in this 32-row block
// (cm: lane j's column mask, bit r = row r kept; cbl: lane j's cb_j).
template <bool kCheck>
__device__ __forceinline__ void fp_write_transposed(const float *xb, uint32_t cm, int32_t cbl, int64_t row0,
                                                    float thr, int32_t cap32, int32_t *__restrict__ t_col,
                                                    float *__restrict__ t_val) {
    const int lane = threadIdx.x & 31;
    const uint32_t lt = (1u << lane) - 1u;
    const int sw = (lane & 7) << 2;
#pragma unroll 4
    for (int j = 0; j < 32; ++j) {
        const uint32_t cmj = __shfl_sync(0xffffffffu, cm, j);
        const int32_t cbj = __shfl_sync(0xffffffffu, cbl, j);
        if ((cmj >> lane) & 1u) {
            const int32_t pc = cbj + __popc(cmj & lt);
            if (!kCheck || pc < cap32) {
                const float z = xb[lane * 32 + (j ^ sw)];
                t_col[pc] = (int32_t)(row0 + lane);
                t_val[pc] = __fsub_rn(z, copysignf(thr, z));
            }
        }
    }
}

// Write pass, column domain: lane = column within a word. Rows are taken in
// groups of G (independent, so their loads overlap); each row's kept entries
// of the W words of the span form one run of consecutive positions, written
// word after word with no other store in between, so the 32-byte sector shared
// by two words' runs is completed at once (a sector left half-written while
// other rows' stores go by is fetched back from DRAM to be merged).
// With kT (W = 1) each kept entry's transposed position goes to t_pos: the
// start of its column's run in the block (cbl) plus the kept rows above it.
template <bool kCheck, int G, int W, bool kT = false>
__device__ __forceinline__ void fp_write_span(const float *xb, const int (&lx)[8], uint32_t lt,
                                              const uint32_t (&kb)[W], int32_t pos, int32_t col0, float thr,
                                              int32_t cap32, int32_t *__restrict__ out_col,
                                              float *__restrict__ out_val, int32_t cbl = 0,
                                              int32_t *__restrict__ t_pos = nullptr) {
    const int lane = threadIdx.x & 31;
    static_assert(!kT || W == 1, "the transposed positions are written one word at a time");
    int32_t pc = cbl;   // kT: this column's next transposed position
#pragma unroll
    for (int i0 = 0; i0 < 32; i0 += G) {
        uint32_t kw[G][W];
        float z[G][W];
        int32_t p[G];
#pragma unroll
        for (int u = 0; u < G; ++u) {
            p[u] = __shfl_sync(0xffffffffu, pos, i0 + u);
#pragma unroll
            for (int c = 0; c < W; ++c) {
                kw[u][c] = __shfl_sync(0xffffffffu, kb[c], i0 + u);
                z[u][c] = xb[c * 1024 + (i0 + u) * 32 + lx[(i0 + u) & 7]];
            }
        }
#pragma unroll
        for (int u = 0; u < G; ++u) {
            int32_t pw = p[u];
#pragma unroll
            for (int c = 0; c < W; ++c) {
                const uint32_t kwi = kw[u][c];
                const int32_t q = pw + __popc(kwi & lt);
                const bool keep = (kwi >> lane) & 1u;
                if (keep && (!kCheck || q < cap32)) {
                    out_col[q] = col0 + c * 32 + lane;
                    out_val[q] = __fsub_rn(z[u][c], copysignf(thr, z[u][c]));
                    if (kT && (!kCheck || pc < cap32)) t_pos[q] = pc;
                }
                if (kT) pc += keep ? 1 : 0;
                pw += __popc(kwi);
            }
        }
    }
}

// Write pass, a word of the span whose 32 rows keep at most kFpWalkMax entries
// in all (9.4%): the row walk above would spend one step per row on mostly
// idle lanes. (Measured on the 4096 x 9216 layer: 6% output density 148.6 ->
// 118.6 us for the whole op; at 12% and above the row walk is faster, the
// compaction being a chain of dependent steps as long as the row's count.) Instead each thread compacts its own row in place (its kept values,
// soft-thresholded, to the first slots of its staged row, their column
// offsets to the byte buffer cb), and then lane = entry: the word's kept
// entries in row order, 32 at a time, each lane finding its row by a search
// over the rows' exclusive counts. The stores of one step form a few
// contiguous runs.
constexpr int kFpWalkMax = 96;

// With kT (cm, cbl, row0 as for fp_write_transposed): the word's transposed
// runs first, from the staged block, then each kept entry's transposed
// position to t_pos.
template <bool kCheck, bool kT = false>
__device__ __forceinline__ void fp_write_compact(const float *xb, uint8_t *cb, float *xr, int sw, uint32_t kw,
                                                 int32_t pos, int total, int32_t col0, float thr, int32_t cap32,
                                                 int32_t *__restrict__ out_col, float *__restrict__ out_val,
                                                 uint32_t cm = 0, int32_t cbl = 0, int64_t row0 = 0,
                                                 int32_t *__restrict__ t_col = nullptr,
                                                 float *__restrict__ t_val = nullptr,
                                                 int32_t *__restrict__ t_pos = nullptr) {
    const int lane = threadIdx.x & 31;
    if (kT) {
        fp_write_transposed<kCheck>(xb, cm, cbl, row0, thr, cap32, t_col, t_val);
        __syncwarp();   // the block's reads done before the rows are compacted in place
    }
    const int cnt = __popc(kw);
    const int maxc = (int)__reduce_max_sync(0xffffffffu, (unsigned)cnt);
    uint32_t bits = kw;
    uint8_t *cbr = cb + lane * 32;
    for (int u = 0; u < maxc; ++u) {
        if (u < cnt) {   // slot u <= column b: every slot below b was read before
            const int b = __ffs(bits) - 1;
            bits &= bits - 1u;
            const float z = xr[b ^ sw];
            xr[u ^ sw] = __fsub_rn(z, copysignf(thr, z));
            cbr[u] = (uint8_t)b;
        }
    }
    int inc = cnt;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, inc, d);
        if (lane >= d) inc += y;
    }
    const int rpre = inc - cnt;   // kept entries of the rows above this one
    __syncwarp();
    for (int e0 = 0; e0 < total; e0 += 32) {
        const int e = e0 + lane;
        int r = 0;   // the last row whose exclusive count is <= e
#pragma unroll
        for (int sft = 16; sft >= 1; sft >>= 1) {
            const int v = __shfl_sync(0xffffffffu, rpre, r + sft);
            if (v <= e) r += sft;
        }
        const int j = e - __shfl_sync(0xffffffffu, rpre, r);
        const int32_t q = __shfl_sync(0xffffffffu, pos, r) + j;
        const int jb = e < total ? cb[r * 32 + j] : 0;   // the entry's column in the word
        if (e < total && (!kCheck || q < cap32)) {
            out_val[q] = xb[r * 32 + (j ^ ((r & 7) << 2))];
            out_col[q] = col0 + jb;
        }
        if (kT) {
            const uint32_t cmj = __shfl_sync(0xffffffffu, cm, jb);
            const int32_t pc = __shfl_sync(0xffffffffu, cbl, jb) + __popc(cmj & ((1u << r) - 1u));
            if (e < total && (!kCheck || (q < cap32 && pc < cap32))) t_pos[q] = pc;
        }
    }
}

// 2./4. Persistent TF32 GEMM whose epilogue applies the prox step: counts and
// keep bits (kWrite = false) or the compacted entries (kWrite = true).
//
// Epilogue warp e reads TMEM lane quarter (e+2) % 4 (tile rows) and column span
// e / 4 of the tile (128 columns in the count pass, 64 in the write pass).
// Per 32-column word, in the row domain (thread = row): z = fl(-eta*G) for
// every entry (exact for an unstored weight: fl(0 - fl(eta*G)) = fl(-eta*G)),
// staged in the warp's buffer; entries with a stored weight are then fixed up
// to fl(w + z) = fl(w - fl(eta*G)). The count pass reads back only its own
// row. The write pass then switches to the column domain (lane = column): for
// each row of the 32 the kept entries form one run of consecutive positions,
// written with coalesced stores.
// kT: the transposed copy too (FpTArgs): its column counts per 32-row block
// (count pass) or its arrays (write pass).
template <bool kWrite, bool kT, bool kSplit = false>
__global__ void __launch_bounds__(fp_threads<kWrite, kSplit>(), 1)
    gemm_prox_tc_kernel(const __grid_constant__ CUtensorMap map_a, const __grid_constant__ CUtensorMap map_b,
                        FpArgs a, FpTArgs ta, int32_t tiles_n, int32_t num_tiles) {
    pdl_enter();
    constexpr int kEpi = FpShape<kWrite>::kEpi, kStages = FpShape<kWrite>::kStages;
    constexpr int kProd = kSplit ? 4 : 2;   // warps before the epilogue warps
    constexpr int kFpPre = FpShape<kWrite>::kPre, kGroup = FpShape<kWrite>::kGroup;
    constexpr int kSpanCols = kTcBN / (kEpi / 4);   // columns per epilogue warp
    constexpr int kSpanWords = kSpanCols / 32;
    static_assert(kSpanWords % kFpTileWords == 0, "a span holds whole segments");
    static_assert(!kWrite || kSpanWords % FpShape<true>::kStageWords == 0, "a span holds whole staged groups");
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sa = smem;
    uint8_t *sb = smem + kStages * kTcABytes;
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + kStages * kTcStageBytes);
    uint64_t *empty = full + kStages;
    uint64_t *accf = empty + kStages;
    uint64_t *acce = accf + 2;
    uint64_t *fin = acce + 2;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(fin + 1);
    float *xbuf = reinterpret_cast<float *>(smem + kStages * kTcStageBytes + 256);
    __shared__ volatile int s_abort;
    __shared__ int s_nonfinite;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int num_kb = (a.n + kTcBK - 1) / kTcBK;

    if (threadIdx.x == 0) {
        s_abort = 0;
        s_nonfinite = 0;
        for (int s = 0; s < kStages; ++s) {
            mbar_init(full + s, 1);
            mbar_init(empty + s, 1);
        }
        mbar_init(accf, 1);
        mbar_init(accf + 1, 1);
        mbar_init(acce, kEpi);
        mbar_init(acce + 1, kEpi);
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
    if (warp < kProd) {
    // every warp of a warpgroup runs the same setmaxnreg
    if constexpr (kSplit) asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(kFpProdRegs));
    if (warp == 0) {
        if (lane == 0) {
            int it = 0;
            for (int t = blockIdx.x; t < num_tiles && !s_abort; t += gridDim.x) {
                const int m0 = (t / tiles_n) * kTcBM, n0 = (t % tiles_n) * kTcBN;
                for (int kb = 0; kb < num_kb; ++kb, ++it) {
                    const int s = it % kStages;
                    if (!mbar_wait_or_abort(empty + s, ((it / kStages) & 1) ^ 1, &s_abort)) break;
                    mbar_expect_tx(full + s, kTcStageBytes);
                    tma_load_2d(sa + s * kTcABytes, &map_a, kb * kTcBK, m0, full + s);
                    tma_load_2d(sb + s * kTcBBytes, &map_b, kb * kTcBK, n0, full + s);
                }
            }
            for (int i = imax(0, it - kStages); i < it; ++i) mbar_wait(full + i % kStages, (i / kStages) & 1);
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
                    const int s = it % kStages;
                    if (!mbar_wait_or_abort(full + s, (it / kStages) & 1, &s_abort)) break;
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
    }
    } else {
        if constexpr (kSplit) asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(kFpEpiRegs));
        const int e = warp - kProd;
        const int q = warp & 3;   // the TMEM lane quarter this warp may read
        const int h = e >> 2;     // column span within the tile
        const int64_t rowq = q * 32 + lane;
        float *xb = xbuf + e * fp_xfloats<kWrite>();
        uint8_t *cb = reinterpret_cast<uint8_t *>(xbuf + kEpi * fp_xfloats<kWrite>()) + e * fp_cbytes<kWrite>();
        const int sw = (lane & 7) << 2;
        int lx[8];   // column-domain offsets: element (i, lane) at i*32 + lx[i & 7]
#pragma unroll
        for (int u = 0; u < 8; ++u) lx[u] = lane ^ (u << 2);
        const uint32_t lt = (1u << lane) - 1u;
        const int32_t cap32 = (int32_t)imin<int64_t>(a.capacity, 0x7fffffff);
        // every position is below the capacity unless the output overflows
        const bool fits = !kWrite || (int64_t)__ldg(a.row_ptr_out + a.m) <= a.capacity;
        float tsum = 0.f;
        // software pipeline: the next tile's metadata one tile ahead, the
        // next word's stored weights one word ahead
        FpMeta<kSpanWords, kT> cur, nxt;
        fp_load_meta<kWrite, kT>(a, ta, blockIdx.x, num_tiles, tiles_n, h, rowq, cur);
        fp_load_meta<kWrite, kT>(a, ta, blockIdx.x + gridDim.x, num_tiles, tiles_n, h, rowq, nxt);
        float wv_n[kFpPre];
        int32_t ow_n = cur.o0;
        fp_load_words(a.old_val, cur.ob[0], ow_n, wv_n);
        int j = 0;
        for (int t = blockIdx.x; t < num_tiles; t += gridDim.x, ++j) {
            const int acc = j & 1;
            const int mt = t / tiles_n, nt = t % tiles_n;
            const int64_t row = (int64_t)mt * kTcBM + rowq;
            const bool rv = row < a.m;
            const int word0 = nt * (kTcBN / 32) + h * kSpanWords;   // first word of the span
            const bool ok = __all_sync(0xffffffffu, mbar_wait_or_abort(accf + acc, (j >> 1) & 1, &s_abort));
            if (!ok) break;
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            int32_t pos = cur.pos;   // write pass: position of the row's next kept entry
            uint32_t cnt = 0;
            if (kWrite) __syncwarp();   // the previous tile's column reads are done
#pragma unroll
            for (int c = 0; c < kSpanWords; ++c) {
                const int word = word0 + c;
                const uint32_t obc = cur.ob[c];
                constexpr int kSW = kWrite ? FpShape<true>::kStageWords : 1;
                float *xr = xb + (kWrite ? (c % kSW) * 1024 : 0) + lane * 32;   // this thread's row of the word
                if (kWrite && c % kSW == 0 && c > 0) __syncwarp();   // the previous group's column reads are done
                float wv[kFpPre];
#pragma unroll
                for (int u = 0; u < kFpPre; ++u) wv[u] = wv_n[u];
                const int32_t ow = ow_n;
                if (c + 1 < kSpanWords) {
                    ow_n = ow + __popc(obc);
                    fp_load_words(a.old_val, cur.ob[c + 1 < kSpanWords ? c + 1 : c], ow_n, wv_n);
                } else {
                    ow_n = nxt.o0;
                    fp_load_words(a.old_val, nxt.ob[0], ow_n, wv_n);
                }
                uint32_t g[32];
                tmem_ld_32cols(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * kTcBN + h * kSpanCols + c * 32),
                               g);
                if (c == kSpanWords - 1) {   // accumulator fully read: hand it back to the MMA warp
                    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
                    __syncwarp();
                    if (lane == 0)
                        asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(acce + acc)) : "memory");
                }
                float zz[32];
#pragma unroll
                for (int jj = 0; jj < 32; ++jj) zz[jj] = __fmul_rn(-a.eta, __uint_as_float(g[jj]));
                uint32_t kw = 0;
                if (!kWrite) {
                    // keep bits of the unstored entries and the NaN probe, as trees
                    uint32_t k4[4] = {0u, 0u, 0u, 0u};
                    float s8[8];
#pragma unroll
                    for (int jj = 0; jj < 32; ++jj) k4[jj >> 3] |= (fabsf(zz[jj]) > a.thr ? 1u : 0u) << jj;
#pragma unroll
                    for (int u = 0; u < 8; ++u) s8[u] = (zz[u] + zz[u + 8]) + (zz[u + 16] + zz[u + 24]);
                    tsum += ((s8[0] + s8[1]) + (s8[2] + s8[3])) + ((s8[4] + s8[5]) + (s8[6] + s8[7]));
                    kw = (k4[0] | k4[1]) | (k4[2] | k4[3]);
                }
#pragma unroll
                for (int cc = 0; cc < 8; ++cc)
                    *reinterpret_cast<float4 *>(xr + ((cc << 2) ^ sw)) =
                        make_float4(zz[4 * cc], zz[4 * cc + 1], zz[4 * cc + 2], zz[4 * cc + 3]);
                // entries with a stored weight: z = fl(w - fl(eta*G)) = fl(w + zz)
                uint32_t bits = obc;
                if (__any_sync(0xffffffffu, bits != 0u)) {
                    // the first kFpPre stored entries, independent of each other
                    int bpos[kFpPre];
#pragma unroll
                    for (int u = 0; u < kFpPre; ++u) {
                        bpos[u] = bits ? __ffs(bits) - 1 : -1;
                        bits &= bits - 1u;
                    }
                    float zs[kFpPre];
#pragma unroll
                    for (int u = 0; u < kFpPre; ++u)
                        if (bpos[u] >= 0) zs[u] = __fadd_rn(wv[u], xr[bpos[u] ^ sw]);
#pragma unroll
                    for (int u = 0; u < kFpPre; ++u) {
                        if (bpos[u] < 0) continue;
                        const int b = bpos[u];
                        if (kWrite) {
                            xr[b ^ sw] = zs[u];
                        } else {
                            tsum += zs[u];
                            kw = fabsf(zs[u]) > a.thr ? (kw | (1u << b)) : (kw & ~(1u << b));
                        }
                    }
                }
                for (int u = kFpPre; bits; ++u) {   // rows with more stored weights in this word
                    const int b = __ffs(bits) - 1;
                    bits &= bits - 1u;
                    float *xe = xr + (b ^ sw);
                    const float z = __fadd_rn(__ldg(a.old_val + ow + u), *xe);
                    if (kWrite) {
                        *xe = z;
                    } else {
                        tsum += z;
                        kw = fabsf(z) > a.thr ? (kw | (1u << b)) : (kw & ~(1u << b));
                    }
                }
                if (!kWrite) {
                    if (rv && word < a.wpr) a.kbits[row * a.wpr + word] = kw;
                    if constexpr (kT) {   // lane j: kept rows of column 32 * word + j in this 32-row block
                        const uint32_t cmc = warp_transpose32(kw);
                        const int64_t brow = row - lane;
                        if (brow < a.m && word < a.wpr) ta.t_cnt[(brow >> 5) * a.k + word * 32 + lane] = __popc(cmc);
                    }
                    cnt += __popc(kw);
                    if (c % kFpTileWords == kFpTileWords - 1) {   // segment complete
                        const int seg = word / kFpTileWords;
                        if (rv && seg < a.nt) a.counts[row * a.nt + seg] = (int32_t)cnt;
                        cnt = 0;
                    }
                } else {
                    if (!kT && rv && word < a.wpr && a.wordpos) a.wordpos[row * a.wpr + word] = imin(pos, cap32);
                    pos += __popc(cur.kb[c]);
                    if (c % kSW == kSW - 1) {
                        // a group of words is staged: write it row by row. The
                        // keep bits come from the count pass, so the positions
                        // agree with the row pointers by construction.
                        __syncwarp();
                        uint32_t kbg[kSW];
                        int32_t pg = pos;   // position of the group's first entry
#pragma unroll
                        for (int u = 0; u < kSW; ++u) {
                            kbg[u] = cur.kb[c + 1 - kSW + u];
                            pg -= __popc(kbg[u]);
                        }
                        const int total =
                            kSW == 1 ? (int)__reduce_add_sync(0xffffffffu, (unsigned)__popc(kbg[0])) : kFpWalkMax + 1;
                        if constexpr (kT && kSW == 1) {
                            // the transposed copy too: lane j's column mask and run start in this 32-row block
                            const uint32_t cm = warp_transpose32(kbg[0]);
                            const int32_t cbl = cur.cb[c];
                            const int64_t row0 = row - lane;
                            if (total <= kFpWalkMax) {
                                if (fits)
                                    fp_write_compact<false, true>(xb, cb, xr, sw, kbg[0], pg, total, word * 32, a.thr,
                                                                  cap32, a.out_col, a.out_val, cm, cbl, row0, ta.t_col,
                                                                  ta.t_val, ta.t_pos);
                                else
                                    fp_write_compact<true, true>(xb, cb, xr, sw, kbg[0], pg, total, word * 32, a.thr,
                                                                 cap32, a.out_col, a.out_val, cm, cbl, row0, ta.t_col,
                                                                 ta.t_val, ta.t_pos);
                            } else {
                                if (fits) {
                                    fp_write_span<false, kGroup, 1, true>(xb, lx, lt, kbg, pg, word * 32, a.thr, cap32,
                                                                          a.out_col, a.out_val, cbl, ta.t_pos);
                                    fp_write_transposed<false>(xb, cm, cbl, row0, a.thr, cap32, ta.t_col, ta.t_val);
                                } else {
                                    fp_write_span<true, kGroup, 1, true>(xb, lx, lt, kbg, pg, word * 32, a.thr, cap32,
                                                                         a.out_col, a.out_val, cbl, ta.t_pos);
                                    fp_write_transposed<true>(xb, cm, cbl, row0, a.thr, cap32, ta.t_col, ta.t_val);
                                }
                            }
                        } else {
                          if (total <= kFpWalkMax) {
                            if (fits)
                                fp_write_compact<false>(xb, cb, xr, sw, kbg[0], pg, total, word * 32, a.thr, cap32,
                                                        a.out_col, a.out_val);
                            else
                                fp_write_compact<true>(xb, cb, xr, sw, kbg[0], pg, total, word * 32, a.thr, cap32,
                                                       a.out_col, a.out_val);
                          } else if (fits) {
                            fp_write_span<false, kGroup, kSW>(xb, lx, lt, kbg, pg, (word + 1 - kSW) * 32, a.thr, cap32,
                                                              a.out_col, a.out_val);
                          } else {
                            fp_write_span<true, kGroup, kSW>(xb, lx, lt, kbg, pg, (word + 1 - kSW) * 32, a.thr, cap32,
                                                             a.out_col, a.out_val);
                          }
                        }
                    }
                }
            }
            cur = nxt;
            fp_load_meta<kWrite, kT>(a, ta, t + 2 * gridDim.x, num_tiles, tiles_n, h, rowq, nxt);
        }
        if (!kWrite && __any_sync(0xffffffffu, tsum != tsum) && lane == 0) s_nonfinite = 1;
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (threadIdx.x == 0) {
        if (s_abort) {
            dev_flag(a.hdr, CSRT_DEV_TIMEOUT);
            a.hdr->timeout_site = kWrite ? 6 : 5;
        }
        if (s_nonfinite) dev_flag(a.hdr, CSRT_DEV_NONFINITE);
    }
    if (warp == 1) {
        __syncwarp();
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(2 * kTcBN) : "memory");
    }
}

// 3. Per row: exclusive offsets of the segments (in place) and the row total
// (warp r of the grid takes row r).
__device__ __forceinline__ void fp_rowscan_row(int32_t *__restrict__ counts, int32_t m, int32_t nt,
                                               int32_t *__restrict__ rowtot, int64_t r) {
    const int lane = threadIdx.x & 31;
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

__global__ void __launch_bounds__(256) fp_rowscan_kernel(int32_t *__restrict__ counts, int32_t m, int32_t nt,
                                                         int32_t *__restrict__ rowtot) {
    pdl_enter();
    fp_rowscan_row(counts, m, nt, rowtot, ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5);
}

// With a transposed copy the two scans between the passes share launches:
// blocks [0, rb) scan the rows' segment counts, the others the transposed
// copy's column counts down each column; then block 0 of the second kernel
// scans the row totals (the row pointers), block 1 the column totals (the
// transposed copy's column pointers).
__global__ void __launch_bounds__(256) fp_rows_cols_scan_kernel(int32_t *__restrict__ counts, int32_t m, int32_t nt,
                                                                int32_t *__restrict__ rowtot, int32_t rb,
                                                                int32_t *__restrict__ cnt, int32_t nb, int32_t cols,
                                                                int32_t *__restrict__ coltot) {
    pdl_enter();
    if ((int)blockIdx.x < rb)   // block-uniform
        fp_rowscan_row(counts, m, nt, rowtot, ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5);
    else
        colscan_block(cnt, nb, cols, coltot, (int)blockIdx.x - rb);
}

__global__ void __launch_bounds__(1024) fp_two_scans_kernel(const int32_t *__restrict__ rowtot, int32_t m,
                                                            int32_t *__restrict__ rawptr,
                                                            int32_t *__restrict__ row_ptr_out, int64_t capacity,
                                                            WsHeader *hdr, const int32_t *__restrict__ coltot,
                                                            int32_t cols, int32_t *__restrict__ t_row_ptr) {
    pdl_enter();
    if (blockIdx.x == 0)
        scan_block_1024(rowtot, m, rawptr, row_ptr_out, capacity, hdr);
    else
        scan_block_1024(coltot, cols, t_row_ptr, nullptr, 0, nullptr);
}

int scan_exclusive_i32_clamped(const int32_t *in, int32_t n, int32_t *out, int32_t *out_clamped, int64_t capacity,
                               void *ws, cudaStream_t s);

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
                       ws_bytes >= kWsReservedBytes + fused_prox_scratch_bytes(m, k);
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
    int32_t *rawptr = reinterpret_cast<int32_t *>(base + L.off_rawptr);
    int32_t *wordpos = reinterpret_cast<int32_t *>(base + L.off_wordpos);

    CUtensorMap ma, mb;
    CSRT_ARG(make_map(&ma, dy, m, n, kTcBM) && make_map(&mb, x, k, n, kTcBN), "tensor map encoding failed");
    static bool attr_set[64] = {false}, split_ok[64] = {false};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !attr_set[dev]) {
        CSRT_CHECK_CUDA(cudaFuncSetAttribute(gemm_prox_tc_kernel<false, false>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, fp_smem_bytes<false>()));
        CSRT_CHECK_CUDA(cudaFuncSetAttribute(gemm_prox_tc_kernel<true, false>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, fp_smem_bytes<true>()));
        CSRT_CHECK_CUDA(cudaFuncSetAttribute(gemm_prox_tc_kernel<true, true>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, fp_smem_bytes<true>()));
        CSRT_CHECK_CUDA(cudaFuncSetAttribute(gemm_prox_tc_kernel<false, true>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, fp_smem_bytes<false>()));
        CSRT_CHECK_CUDA(cudaFuncSetAttribute(gemm_prox_tc_kernel<true, false, true>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, fp_smem_bytes<true>()));
        CSRT_CHECK_CUDA(cudaFuncSetAttribute(gemm_prox_tc_kernel<true, true, true>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, fp_smem_bytes<true>()));
        // the register split needs the launch to hold what it hands out (ptxas gives 96 per thread at
        // 640 threads; the 18-warp write pass otherwise)
        cudaFuncAttributes fa0{}, fa1{};
        CSRT_CHECK_CUDA(cudaFuncGetAttributes(&fa0, gemm_prox_tc_kernel<true, false, true>));
        CSRT_CHECK_CUDA(cudaFuncGetAttributes(&fa1, gemm_prox_tc_kernel<true, true, true>));
        const int need = 128 * kFpProdRegs + FpShape<true>::kEpi * 32 * kFpEpiRegs;
        split_ok[dev] = fa0.numRegs * fp_threads<true, true>() >= need &&
                        fa1.numRegs * fp_threads<true, true>() >= need;
        attr_set[dev] = true;
    }
    const bool split = dev >= 0 && dev < 64 && split_ok[dev];
    launch_pdl(fp_oldbits_kernel, dim3((unsigned)ceil_div<int64_t>(m, 8)), dim3(256), 0, s, w_in->row_ptr,
               w_in->col_idx, m, L.wpr, L.nt, obits, ostart);
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
    a.row_ptr_out = rawptr;
    a.out_col = w_out->col_idx;
    a.out_val = w_out->val;
    a.wordpos = want_t ? wordpos : nullptr;
    FpTArgs ta{};   // the transposed copy: the count pass's column counts here, the write pass's arrays below
    if (want_t) ta.t_cnt = reinterpret_cast<int32_t *>(base + L.off_tr);
    a.capacity = w_out->capacity;
    a.hdr = static_cast<WsHeader *>(ws);
    const int tiles_m = (int)ceil_div<int64_t>(m, kTcBM), tiles_n = (int)ceil_div<int64_t>(k, kTcBN);
    const int tiles = tiles_m * tiles_n;
    const unsigned grid = (unsigned)imin(tiles, num_sms());
    if (want_t)
        launch_pdl(gemm_prox_tc_kernel<false, true>, dim3(grid), dim3(fp_threads<false>()), fp_smem_bytes<false>(), s,
                   ma, mb, a, ta, tiles_n, tiles);
    else
        launch_pdl(gemm_prox_tc_kernel<false, false>, dim3(grid), dim3(fp_threads<false>()), fp_smem_bytes<false>(), s,
                   ma, mb, a, ta, tiles_n, tiles);
    count_launch(2);
    const unsigned rb = (unsigned)ceil_div<int64_t>((int64_t)m * 32, 256);
    int rc = 0;
    if (!want_t) {
        launch_pdl(fp_rowscan_kernel, dim3(rb), dim3(256), 0, s, counts, m, L.nt, rowtot);
        count_launch(1);
        // new row pointers: exclusive scan of the row totals (int32: nnz <= M*K < 2^31), unclamped for the
        // write pass and clamped to the capacity in w_out (overflow reported)
        rc = scan_exclusive_i32_clamped(rowtot, m, rawptr, w_out->row_ptr, w_out->capacity, ws, s);
        if (rc) return rc;
    } else {
        // the same, paired with the transposed copy's scans of the count pass's column counts (its per-block
        // offsets down each column and its column pointers); the write pass writes its arrays
        int32_t *tcnt = reinterpret_cast<int32_t *>(base + L.off_tr);
        const int32_t nb = (int32_t)ceil_div<int64_t>(m, 32);
        int32_t *coltot = tcnt + (int64_t)nb * k;
        launch_pdl(fp_rows_cols_scan_kernel, dim3(rb + (unsigned)ceil_div(k, 32)), dim3(256), 0, s, counts, m, L.nt,
                   rowtot, (int32_t)rb, tcnt, nb, k, coltot);
        launch_pdl(fp_two_scans_kernel, dim3(2), dim3(1024), 0, s, rowtot, m, rawptr, w_out->row_ptr,
                   w_out->capacity, static_cast<WsHeader *>(ws), coltot, k, w_out->t_row_ptr);
        count_launch(2);
        ta.t_rp = w_out->t_row_ptr;
        ta.t_off = reinterpret_cast<const int32_t *>(base + L.off_tr);
        ta.t_col = w_out->t_col_idx;
        ta.t_val = w_out->t_val;
        ta.t_pos = w_out->t_pos;
    }
    if (want_t && split)
        launch_pdl(gemm_prox_tc_kernel<true, true, true>, dim3(grid), dim3(fp_threads<true, true>()),
                   fp_smem_bytes<true>(), s, ma, mb, a, ta, tiles_n, tiles);
    else if (want_t)
        launch_pdl(gemm_prox_tc_kernel<true, true>, dim3(grid), dim3(fp_threads<true>()), fp_smem_bytes<true>(), s,
                   ma, mb, a, ta, tiles_n, tiles);
    else if (split)
        launch_pdl(gemm_prox_tc_kernel<true, false, true>, dim3(grid), dim3(fp_threads<true, true>()),
                   fp_smem_bytes<true>(), s, ma, mb, a, ta, tiles_n, tiles);
    else
        launch_pdl(gemm_prox_tc_kernel<true, false>, dim3(grid), dim3(fp_threads<true>()), fp_smem_bytes<true>(), s,
                   ma, mb, a, ta, tiles_n, tiles);
    count_launch(1);
    return check_launch("fused weight-gradient + prox kernels");
}
