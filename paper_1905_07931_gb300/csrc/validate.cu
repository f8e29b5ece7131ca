// Structural validation of a CSR (and of its transposed copy): the invariants
// every call of the library assumes. There is no sanitizer on the GPUs this
// library targets, so a caller that builds or edits CSR arrays itself checks
// them here instead. Every read is bounded before it is made: a row's range
// is checked against the capacity before any column index of it is read, a
// column against the matrix width before t_row_ptr is indexed with it, a
// transposed position against the capacity before the transposed arrays are
// read there. A corrupted CSR therefore only sets a status bit.
#include "common.cuh"

namespace csrt {

constexpr int kVdThreads = 256;

__device__ __forceinline__ void vd_report(WsHeader *hdr, int64_t row) {
    atomicOr(&hdr->flags, (unsigned)CSRT_DEV_INVALID);
    atomicMax(&hdr->invalid_row, 0xffffffffu - (unsigned)row);
}

// One warp per row (grid-stride): row_ptr[0] == 0, 0 <= row_ptr[r] <=
// row_ptr[r+1] <= capacity, and within the row 0 <= col < cols, strictly
// ascending. `tag` offsets the reported row (the transposed pass reports
// rows + column).
__global__ void __launch_bounds__(kVdThreads) validate_rows_kernel(const int32_t *__restrict__ row_ptr,
                                                                   const int32_t *__restrict__ col, int32_t rows,
                                                                   int32_t cols, int64_t capacity, int64_t tag,
                                                                   WsHeader *hdr) {
    pdl_enter();
    const int lane = threadIdx.x & 31;
    const int64_t w0 = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    if (w0 == 0 && lane == 0 && __ldg(row_ptr) != 0) vd_report(hdr, tag);
    for (int64_t r = w0; r < rows; r += nw) {
        const int64_t s = __ldg(row_ptr + r), e = __ldg(row_ptr + r + 1);
        if (!(s >= 0 && s <= e && e <= capacity)) {
            if (lane == 0) vd_report(hdr, tag + r);
            continue;
        }
        bool bad = false;
        for (int64_t k = s + lane; k < e; k += 32) {
            const int32_t c = __ldg(col + k);
            const int32_t prev = k > s ? __ldg(col + k - 1) : -1;
            bad |= c < 0 || c >= cols || c <= prev;
        }
        if (__any_sync(0xffffffffu, bad) && lane == 0) vd_report(hdr, tag + r);
    }
}

// The transposed copy against the CSR: for every entry k of row r with
// column c, p = t_pos[k] lies in column c's range of the transposed arrays,
// t_col_idx[p] == r and t_val[p] has the bits of val[k]. Together with the
// row checks of both patterns and equal entry counts this makes t_pos a
// bijection. Rows whose own range is invalid are left to the row check.
__global__ void __launch_bounds__(kVdThreads) validate_transpose_kernel(const csrt_csr w, WsHeader *hdr) {
    pdl_enter();
    const int lane = threadIdx.x & 31;
    const int64_t w0 = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    if (w0 == 0 && lane == 0 && __ldg(w.row_ptr + w.rows) != __ldg(w.t_row_ptr + w.cols)) vd_report(hdr, w.rows);
    for (int64_t r = w0; r < w.rows; r += nw) {
        const int64_t s = __ldg(w.row_ptr + r), e = __ldg(w.row_ptr + r + 1);
        if (!(s >= 0 && s <= e && e <= w.capacity)) continue;
        bool bad = false;
        for (int64_t k = s + lane; k < e; k += 32) {
            const int32_t c = __ldg(w.col_idx + k);
            if (c < 0 || c >= w.cols) continue;   // reported by the row check
            const int64_t p = __ldg(w.t_pos + k);
            const int64_t ts = __ldg(w.t_row_ptr + c), te = __ldg(w.t_row_ptr + c + 1);
            if (!(p >= ts && p < te && p >= 0 && p < w.capacity)) {
                bad = true;
                continue;
            }
            bad |= __ldg(w.t_col_idx + p) != (int32_t)r;
            bad |= __float_as_uint(__ldg(w.t_val + p)) != __float_as_uint(__ldg(w.val + k));
        }
        if (__any_sync(0xffffffffu, bad) && lane == 0) vd_report(hdr, w.rows + w.cols + 1 + r);
    }
}

}  // namespace csrt

using namespace csrt;

extern "C" {

int csrt_validate_csr(const csrt_csr *w, void *ws, size_t ws_bytes, void *stream) {
    CSRT_ARG(w != nullptr && w->row_ptr != nullptr, "csr or row_ptr is NULL");
    CSRT_ARG(w->rows >= 0 && w->cols >= 0, "negative shape");
    CSRT_ARG(w->capacity >= 0 && w->capacity < ((int64_t)1 << 31), "capacity out of range");
    CSRT_ARG(w->capacity == 0 || w->col_idx != nullptr, "col_idx is NULL");
    CSRT_ARG(ws != nullptr && ws_bytes >= kWsHeaderBytes, "workspace too small");
    const bool t = w->t_row_ptr != nullptr;
    CSRT_ARG(!t || w->capacity == 0 || (w->t_col_idx && w->t_val && w->t_pos && w->val), "transposed arrays partly set");
    cudaStream_t s = as_stream(stream);
    WsHeader *hdr = static_cast<WsHeader *>(ws);
    auto grid = [](int64_t rows) {
        return dim3((unsigned)imax<int64_t>(1, imin<int64_t>(ceil_div<int64_t>(rows, kVdThreads / 32),
                                                             (int64_t)num_sms() * 8)));
    };
    launch_pdl(validate_rows_kernel, grid(w->rows), dim3(kVdThreads), 0, s, (const int32_t *)w->row_ptr,
               (const int32_t *)w->col_idx, w->rows, w->cols, w->capacity, (int64_t)0, hdr);
    count_launch();
    if (t) {
        launch_pdl(validate_rows_kernel, grid(w->cols), dim3(kVdThreads), 0, s, (const int32_t *)w->t_row_ptr,
                   (const int32_t *)w->t_col_idx, w->cols, w->rows, w->capacity, (int64_t)w->rows + 1, hdr);
        launch_pdl(validate_transpose_kernel, grid(w->rows), dim3(kVdThreads), 0, s, *w, hdr);
        count_launch(2);
    }
    return check_launch("validate kernels");
}

int csrt_get_invalid_row(const void *ws, int64_t *row, void *stream) {
    CSRT_ARG(ws != nullptr && row != nullptr, "workspace or row is NULL");
    WsHeader h;
    CSRT_CHECK_CUDA(cudaMemcpyAsync(&h, ws, sizeof(h), cudaMemcpyDeviceToHost, as_stream(stream)));
    CSRT_CHECK_CUDA(cudaStreamSynchronize(as_stream(stream)));
    *row = h.invalid_row == 0 ? -1 : (int64_t)(0xffffffffu - h.invalid_row);
    return CSRT_OK;
}

}  // extern "C"
