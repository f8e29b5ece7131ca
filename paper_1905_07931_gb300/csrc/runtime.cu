// Workspace, status word, error reporting and launch accounting.
#include <cstdarg>
#include <cstdio>
#include <cstring>

#include "common.cuh"

namespace csrt {

static thread_local char g_msg[512] = "";
static thread_local int64_t g_launches = 0;

int fail(int code, const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_msg, sizeof(g_msg), fmt, ap);
    va_end(ap);
    return code;
}

int check_launch(const char *what) {
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return fail(CSRT_ERR_CUDA, "%s launch: %s", what, cudaGetErrorString(e));
    return CSRT_OK;
}

void count_launch(int n) { g_launches += n; }

int num_sms() {
    static int cache[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
    if (cache[dev] == 0) {
        int v = 0;
        if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v <= 0)
            v = 148;
        cache[dev] = v;
    }
    return cache[dev];
}

}  // namespace csrt

using namespace csrt;

extern "C" {

int csrt_workspace_bytes(int32_t rows, int32_t cols, int32_t max_n, size_t *bytes) {
    CSRT_ARG(bytes != nullptr, "bytes is NULL");
    CSRT_ARG(rows >= 0 && cols >= 0 && max_n >= 0, "negative size");
    CSRT_ARG((int64_t)rows * cols < (int64_t)1 << 31, "rows*cols must be below 2^31");
    int64_t elems = (int64_t)rows * cols;
    size_t need = compact_scratch_bytes(rows, cols);
    size_t t = transpose_scratch_bytes(rows, cols);
    if (t > need) need = t;
    t = spmm_scratch_bytes(max_n);
    if (t > need) need = t;
    t = sddmm_scratch_bytes(elems, max_n);
    if (t > need) need = t;
    t = gemm_scratch_bytes(rows, cols, max_n);
    if (t > need) need = t;
    t = fused_prox_scratch_bytes(rows, cols);
    if (t > need) need = t;
    *bytes = kWsReservedBytes + ((need + 255) / 256) * 256;
    return CSRT_OK;
}

int csrt_workspace_init(void *ws, size_t ws_bytes, void *stream) {
    CSRT_ARG(ws != nullptr && ws_bytes >= kWsHeaderBytes, "workspace too small");
    CSRT_CHECK_CUDA(cudaMemsetAsync(ws, 0, ws_bytes, as_stream(stream)));
    return CSRT_OK;
}

int csrt_get_status(const void *ws, int32_t *flags, int64_t *required_nnz, void *stream) {
    CSRT_ARG(ws != nullptr, "workspace is NULL");
    WsHeader h;
    CSRT_CHECK_CUDA(cudaMemcpyAsync(&h, ws, sizeof(h), cudaMemcpyDeviceToHost, as_stream(stream)));
    CSRT_CHECK_CUDA(cudaStreamSynchronize(as_stream(stream)));
    if (flags) *flags = (int32_t)h.flags;
    if (required_nnz) *required_nnz = (int64_t)h.required;
    return CSRT_OK;
}

int csrt_clear_status(void *ws, void *stream) {
    CSRT_ARG(ws != nullptr, "workspace is NULL");
    CSRT_CHECK_CUDA(cudaMemsetAsync(ws, 0, 16, as_stream(stream)));
    return CSRT_OK;
}

const char *csrt_last_error(void) { return g_msg; }

int64_t csrt_launch_count(int reset) {
    int64_t v = g_launches;
    if (reset) g_launches = 0;
    return v;
}

}  // extern "C"
