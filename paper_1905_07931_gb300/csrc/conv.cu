// Convolution with a compressed (CSR) filter bank, without the unfolded input.
//
// Section 3.2 lowers a convolution to the product of the filter matrix W
// (C_out x C_in*k*k, here in CSR) with the unfolded input (the Caffe
// im2col matrix, C_in*k*k x B*Ho*Wo). The forward pass only needs, for each
// output pixel, the stored filter taps of its channel applied to the input
// window, so this kernel reads the input in place: the unfolded matrix, which
// is k*k times larger than the input, is never written or read.
//
// One block per (output channel m, tile of output pixels). The block stages
// the channel's stored taps in shared memory as (weight, input offset) pairs;
// tap k = (c*k + ky)*k + kx of the CSR row reads input pixel
// x[c][b][oy+ky][ox+kx], at offset c*B*H*W + ky*W + kx from the window's
// corner x[0][b][oy][ox]. Each thread accumulates kConvPer output pixels
// (consecutive pixels go to consecutive threads, so the input reads of a warp
// are contiguous along ox) over the taps in CSR order with one fused
// multiply-add per tap, then applies the bias and ReLU. The input window
// of a block is reused by every tap from L1.
#include "common.cuh"

namespace csrt {

constexpr int kConvThreads = 256;
constexpr int kConvPer = 4;          // output pixels per thread
constexpr int kConvTaps = 1024;      // taps staged per round

__global__ void __launch_bounds__(kConvThreads) conv_sparse_fwd_kernel(
    const int32_t *__restrict__ row_ptr, const int32_t *__restrict__ col, const float *__restrict__ val,
    const float *__restrict__ x, int32_t cin, int32_t b, int32_t h, int32_t w, int32_t k,
    const float *__restrict__ bias, int32_t relu, float *__restrict__ y) {
    pdl_enter();
    __shared__ float s_w[kConvTaps];
    __shared__ int64_t s_off[kConvTaps];
    const int ho = h - k + 1, wo = w - k + 1;
    const int64_t plane = (int64_t)b * h * w;             // one input channel
    const int64_t npix = (int64_t)b * ho * wo;            // output pixels per channel
    const int m = blockIdx.y;
    const int64_t p0 = (int64_t)blockIdx.x * kConvThreads * kConvPer + threadIdx.x;
    // window corner of each of this thread's pixels
    int64_t corner[kConvPer];
    bool valid[kConvPer];
#pragma unroll
    for (int q = 0; q < kConvPer; ++q) {
        const int64_t p = p0 + (int64_t)q * kConvThreads;
        valid[q] = p < npix;
        const int64_t pp = valid[q] ? p : 0;
        const int64_t s = pp / ((int64_t)ho * wo);
        const int rem = (int)(pp - s * ho * wo);
        const int oy = rem / wo, ox = rem - oy * wo;
        corner[q] = (s * h + oy) * w + ox;
    }
    float acc[kConvPer];
#pragma unroll
    for (int q = 0; q < kConvPer; ++q) acc[q] = 0.f;
    const int32_t t0 = __ldg(row_ptr + m), t1 = __ldg(row_ptr + m + 1);
    for (int32_t tb = t0; tb < t1; tb += kConvTaps) {
        const int nt = imin(kConvTaps, t1 - tb);
        __syncthreads();   // the previous round's taps are consumed
        for (int i = threadIdx.x; i < nt; i += kConvThreads) {
            const int tap = __ldg(col + tb + i);
            const int c = tap / (k * k), kk = tap - c * k * k;
            const int ky = kk / k, kx = kk - ky * k;
            s_off[i] = (int64_t)c * plane + (int64_t)ky * w + kx;
            s_w[i] = __ldg(val + tb + i);
        }
        __syncthreads();
        for (int i = 0; i < nt; ++i) {
            const float wt = s_w[i];
            const int64_t off = s_off[i];
#pragma unroll
            for (int q = 0; q < kConvPer; ++q)
                if (valid[q]) acc[q] = fmaf(wt, __ldg(x + corner[q] + off), acc[q]);
        }
    }
    const float bm = bias ? __ldg(bias + m) : 0.f;
#pragma unroll
    for (int q = 0; q < kConvPer; ++q) {
        if (!valid[q]) continue;
        float v = acc[q];
        if (bias) v = __fadd_rn(v, bm);
        if (relu) v = fmaxf(v, 0.f);
        y[(int64_t)m * npix + p0 + (int64_t)q * kConvThreads] = v;
    }
}

}  // namespace csrt

using namespace csrt;

extern "C" int csrt_conv2d_sparse_fwd(const csrt_csr *w, const float *x, int32_t c, int32_t b, int32_t h,
                                      int32_t wd, int32_t k, const float *bias, int32_t relu, float *y,
                                      void *stream) {
    CSRT_ARG(w != nullptr && w->row_ptr != nullptr, "csr is NULL");
    CSRT_ARG(c > 0 && b >= 0 && k > 0 && h >= k && wd >= k, "bad convolution shape");
    CSRT_ARG(w->cols == c * k * k, "filter matrix has %d columns, expected C*k*k = %d", w->cols, c * k * k);
    CSRT_ARG(w->rows > 0 && w->rows <= 65535, "output channels must be in 1..65535");
    const int64_t npix = (int64_t)b * (h - k + 1) * (wd - k + 1);
    if (npix == 0) return CSRT_OK;
    CSRT_ARG(x != nullptr && y != nullptr, "x or y is NULL");
    CSRT_ARG(w->capacity == 0 || (w->col_idx && w->val), "col_idx/val NULL");
    const int64_t blocks = ceil_div<int64_t>(npix, (int64_t)kConvThreads * kConvPer);
    CSRT_ARG(blocks < ((int64_t)1 << 31), "too many output pixels");
    launch_pdl(conv_sparse_fwd_kernel, dim3((unsigned)blocks, (unsigned)w->rows), dim3(kConvThreads), 0,
               as_stream(stream), w->row_ptr, w->col_idx, w->val, x, c, b, h, wd, k, bias, relu, y);
    count_launch();
    return check_launch("conv_sparse_fwd_kernel");
}
