// Network glue around the sparse layers: bias + ReLU, ReLU backward, bias
// gradient + SGD, softmax cross-entropy, im2col / col2im (the Caffe lowering
// of a convolution to a matrix product), 2x2 max pooling and the flatten
// permutation between convolution and fully connected layers. The paper uses
// these Caffe layers without describing them; they follow the textbook
// definitions. All are elementwise or row reductions, bound by HBM traffic;
// each thread handles one element (or one row for the reductions) with
// coalesced accesses along the sample index.
#include "common.cuh"

namespace csrt {

static unsigned grid_for(int64_t count, int threads = 256) {
    const int64_t cap = (int64_t)num_sms() * 16;
    return (unsigned)imax<int64_t>(1, imin<int64_t>(ceil_div<int64_t>(count, threads), cap));
}

__global__ void bias_act_kernel(float *__restrict__ y, const float *__restrict__ bias, int32_t m, int32_t n,
                                int relu) {
    pdl_enter();
    const int64_t total = (int64_t)m * n;
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
        float v = y[e];
        if (bias) v = __fadd_rn(v, __ldg(bias + e / n));
        if (relu) v = fmaxf(v, 0.f);
        y[e] = v;
    }
}

__global__ void relu_bwd_kernel(float *__restrict__ dy, const float *__restrict__ y, int64_t count) {
    pdl_enter();
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < count; e += (int64_t)gridDim.x * blockDim.x)
        if (!(__ldg(y + e) > 0.f)) dy[e] = 0.f;
}

// One warp per row: gb[i] = sum_c dy[i, c] in a fixed order; SGD on the bias.
__global__ void bias_grad_sgd_kernel(const float *__restrict__ dy, int32_t m, int32_t n, float *__restrict__ bias,
                                     float eta, float *__restrict__ gb_out) {
    pdl_enter();
    const int lane = threadIdx.x & 31;
    const int64_t row = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    if (row >= m) return;
    const float *p = dy + row * n;
    float s = 0.f;
    for (int c = lane; c < n; c += 32) s += __ldg(p + c);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
    if (lane == 0) {
        if (gb_out) gb_out[row] = s;
        if (bias) bias[row] = __fsub_rn(bias[row], __fmul_rn(eta, s));
    }
}

// Softmax cross-entropy: a block of 1024 threads takes 8 samples (columns);
// thread (class group g = 0..127, column c = 0..7) walks classes g, g+128, ...
// so every warp load covers 4 classes x 8 consecutive columns (32-byte
// segments). One pass keeps a running maximum and rescaled sum per thread;
// the four groups of a warp are combined by shuffles, then the 32 warps in
// shared memory, always in the same order; a second pass writes dz.
constexpr int kSmThreads = 1024;
constexpr int kSmGroups = kSmThreads / 8;   // class groups per block

__device__ __forceinline__ void softmax_merge(float &m, float &s, float m2, float s2) {
    const float mx = fmaxf(m, m2);
    float r = 0.f;
    if (m != -INFINITY) r += s * expf(m - mx);
    if (m2 != -INFINITY) r += s2 * expf(m2 - mx);
    m = mx;
    s = r;
}

__global__ void __launch_bounds__(kSmThreads) softmax_xent_kernel(const float *__restrict__ z,
                                                                  const int32_t *__restrict__ labels,
                                                                  int32_t classes, int32_t n, float *__restrict__ dz,
                                                                  float *__restrict__ per_sample) {
    pdl_enter();
    __shared__ float s_m[32][8], s_s[32][8];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int cl = lane & 7;
    const int grp = warp * 4 + (lane >> 3);
    const int64_t col = (int64_t)blockIdx.x * 8 + cl;
    const bool ok = col < n;
    float m = -INFINITY, sum = 0.f;
    constexpr int kBatch = 8;   // class values loaded together, then folded in order
    if (ok) {
        for (int c0 = grp; c0 < classes; c0 += kSmGroups * kBatch) {
            float xs[kBatch];
#pragma unroll
            for (int u = 0; u < kBatch; ++u) {
                const int c = c0 + kSmGroups * u;
                xs[u] = c < classes ? __ldg(z + (int64_t)c * n + col) : -INFINITY;
            }
#pragma unroll
            for (int u = 0; u < kBatch; ++u) {
                if (c0 + kSmGroups * u >= classes) break;
                const float x = xs[u];
                if (x > m) {
                    sum = sum * expf(m - x) + 1.f;
                    m = x;
                } else {
                    sum += expf(x - m);
                }
            }
        }
    }
    // the warp's four groups of each column (lanes cl, cl+8, cl+16, cl+24)
#pragma unroll
    for (int off = 8; off <= 16; off <<= 1) {
        const float m2 = __shfl_xor_sync(0xffffffffu, m, off);
        const float s2 = __shfl_xor_sync(0xffffffffu, sum, off);
        if (lane & off) softmax_merge(m, sum, m2, s2);   // same operands in both lanes, in a fixed order
        else {
            float mm = m2, ss = s2;
            softmax_merge(mm, ss, m, sum);
            m = mm;
            sum = ss;
        }
    }
    if (lane < 8) {
        s_m[warp][cl] = m;
        s_s[warp][cl] = sum;
    }
    __syncthreads();
    float mx = -INFINITY;
    for (int w = 0; w < 32; ++w) mx = fmaxf(mx, s_m[w][cl]);
    float se = 0.f;
    for (int w = 0; w < 32; ++w) {
        const float mw = s_m[w][cl];
        if (mw != -INFINITY) se += s_s[w][cl] * expf(mw - mx);
    }
    if (!ok) return;
    const float inv = 1.f / se;
    const float inv_n = 1.f / (float)n;
    const int lab = __ldg(labels + col);
    const bool lab_ok = lab >= 0 && lab < classes;   // an invalid label gives a NaN loss
    for (int c0 = grp; c0 < classes; c0 += kSmGroups * kBatch) {
        float xs[kBatch];
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
            const int c = c0 + kSmGroups * u;
            xs[u] = c < classes ? __ldg(z + (int64_t)c * n + col) : 0.f;
        }
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
            const int c = c0 + kSmGroups * u;
            if (c >= classes) break;
            const float p = expf(xs[u] - mx) * inv;
            dz[(int64_t)c * n + col] = (p - (c == lab ? 1.f : 0.f)) * inv_n;
        }
    }
    if (grp == 0)
        per_sample[col] = lab_ok ? -((__ldg(z + (int64_t)lab * n + col) - mx) - logf(se)) : __int_as_float(0x7fc00000);
}

// Mean of the per-sample losses in a fixed order (one block).
__global__ void __launch_bounds__(1024) mean_kernel(const float *__restrict__ v, int32_t n, float *__restrict__ out) {
    pdl_enter();
    __shared__ float s_warp[32];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    float s = 0.f;
    for (int i = tid; i < n; i += 1024) s += v[i];
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
    if (lane == 0) s_warp[warp] = s;
    __syncthreads();
    if (warp == 0) {
        s = s_warp[lane];
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
        if (lane == 0) out[0] = n ? s / (float)n : 0.f;
    }
}

__global__ void im2col_kernel(const float *__restrict__ x, int32_t c, int32_t b, int32_t h, int32_t w, int32_t k,
                              float *__restrict__ cols) {
    pdl_enter();
    const int ho = h - k + 1, wo = w - k + 1;
    const int64_t ncol = (int64_t)b * ho * wo;
    const int64_t total = (int64_t)c * k * k * ncol;
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
        const int64_t row = e / ncol, cc = e - row * ncol;
        const int ci = (int)(row / (k * k)), kk = (int)(row % (k * k));
        const int ky = kk / k, kx = kk % k;
        const int64_t s = cc / (ho * wo);
        const int rem = (int)(cc - s * ho * wo);
        const int oy = rem / wo, ox = rem % wo;
        cols[e] = __ldg(x + (((int64_t)ci * b + s) * h + (oy + ky)) * w + (ox + kx));
    }
}

__global__ void col2im_kernel(const float *__restrict__ dcols, int32_t c, int32_t b, int32_t h, int32_t w,
                              int32_t k, float *__restrict__ dx) {
    pdl_enter();
    const int ho = h - k + 1, wo = w - k + 1;
    const int64_t ncol = (int64_t)b * ho * wo;
    const int64_t total = (int64_t)c * b * h * w;
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
        const int xx = (int)(e % w);
        const int yy = (int)((e / w) % h);
        const int64_t s = (e / ((int64_t)w * h)) % b;
        const int ci = (int)(e / ((int64_t)w * h * b));
        float acc = 0.f;
        for (int ky = 0; ky < k; ++ky) {
            const int oy = yy - ky;
            if (oy < 0 || oy >= ho) continue;
            for (int kx = 0; kx < k; ++kx) {
                const int ox = xx - kx;
                if (ox < 0 || ox >= wo) continue;
                acc += __ldg(dcols + ((int64_t)ci * k * k + ky * k + kx) * ncol + s * ho * wo + oy * wo + ox);
            }
        }
        dx[e] = acc;
    }
}

__global__ void maxpool2_fwd_kernel(const float *__restrict__ x, int32_t c, int32_t b, int32_t h, int32_t w,
                                    float *__restrict__ y, int8_t *__restrict__ idx) {
    pdl_enter();
    const int ho = h / 2, wo = w / 2;
    const int64_t total = (int64_t)c * b * ho * wo;
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
        const int ox = (int)(e % wo);
        const int oy = (int)((e / wo) % ho);
        const int64_t plane = e / ((int64_t)wo * ho);   // ci*b + s
        const float *p = x + (plane * h + 2 * oy) * w + 2 * ox;
        const float v[4] = {__ldg(p), __ldg(p + 1), __ldg(p + w), __ldg(p + w + 1)};
        int best = 0;
        for (int q = 1; q < 4; ++q)
            if (v[q] > v[best]) best = q;   // first maximum in scan order wins
        y[e] = v[best];
        idx[e] = (int8_t)best;
    }
}

__global__ void maxpool2_bwd_kernel(const float *__restrict__ dy, const int8_t *__restrict__ idx, int32_t c,
                                    int32_t b, int32_t h, int32_t w, float *__restrict__ dx) {
    pdl_enter();
    const int ho = h / 2, wo = w / 2;
    const int64_t total = (int64_t)c * b * h * w;
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
        const int xx = (int)(e % w);
        const int yy = (int)((e / w) % h);
        const int64_t plane = e / ((int64_t)w * h);
        const int64_t o = (plane * ho + yy / 2) * wo + xx / 2;
        const int pos = (yy & 1) * 2 + (xx & 1);
        dx[e] = (__ldg(idx + o) == pos) ? __ldg(dy + o) : 0.f;
    }
}

// xf[ci*hw + s][bi] = x[ci][bi*hw + s] (forward); inverse if `inverse`.
__global__ void flatten_kernel(const float *__restrict__ in, int32_t c, int32_t b, int32_t hw, float *__restrict__ out,
                               int inverse) {
    pdl_enter();
    const int64_t total = (int64_t)c * b * hw;
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
        // e indexes the flattened layout: row f = ci*hw + s, column bi
        const int64_t f = e / b;
        const int bi = (int)(e % b);
        const int64_t ci = f / hw, s = f % hw;
        const int64_t src = (ci * b + bi) * hw + s;
        if (inverse) out[src] = __ldg(in + e);
        else out[e] = __ldg(in + src);
    }
}

// FP32 FMA throughput probe (the roof of the CUDA-core products): every
// thread runs kFmaChains independent fused multiply-add chains
// (x <- x*b + c with |b| < 1, so the values stay finite) for `iters` rounds
// and stores their sum, so nothing is optimised away.
constexpr int kFmaChains = 8;
constexpr int kFmaThreads = 512;
__global__ void __launch_bounds__(kFmaThreads) fma_peak_kernel(float *__restrict__ out, int32_t iters, float b,
                                                                float c) {
    pdl_enter();
    float x[kFmaChains];
#pragma unroll
    for (int k = 0; k < kFmaChains; ++k) x[k] = (float)(threadIdx.x + k) * 1e-3f;
    for (int i = 0; i < iters; ++i) {
#pragma unroll
        for (int k = 0; k < kFmaChains; ++k) x[k] = fmaf(x[k], b, c);
    }
    float sum = 0.f;
#pragma unroll
    for (int k = 0; k < kFmaChains; ++k) sum += x[k];
    out[(int64_t)blockIdx.x * blockDim.x + threadIdx.x] = sum;
}

}  // namespace csrt

using namespace csrt;

extern "C" {

int csrt_fma_peak_run(float *out, int32_t blocks, int32_t iters, double *flops, void *stream) {
    CSRT_ARG(out != nullptr && blocks > 0 && iters > 0, "bad probe arguments");
    if (flops) *flops = 2.0 * (double)blocks * kFmaThreads * kFmaChains * (double)iters;
    launch_pdl(fma_peak_kernel, dim3((unsigned)blocks), dim3(kFmaThreads), 0, as_stream(stream), out, iters,
               0.999999f, 1e-6f);
    count_launch();
    return check_launch("fma_peak_kernel");
}

int csrt_bias_act_fwd(float *y, const float *bias, int32_t m, int32_t n, int32_t relu, void *stream) {
    CSRT_ARG(m >= 0 && n >= 0, "negative size");
    if ((int64_t)m * n == 0) return CSRT_OK;
    CSRT_ARG(y != nullptr, "y is NULL");
    launch_pdl(bias_act_kernel, dim3(grid_for((int64_t)m * n)), dim3(256), 0, as_stream(stream), y, bias, m, n, relu);
    count_launch();
    return check_launch("bias_act_kernel");
}

int csrt_relu_bwd(float *dy, const float *y, int64_t count, void *stream) {
    CSRT_ARG(count >= 0, "negative count");
    if (count == 0) return CSRT_OK;
    CSRT_ARG(dy && y, "NULL pointer");
    launch_pdl(relu_bwd_kernel, dim3(grid_for(count)), dim3(256), 0, as_stream(stream), dy, y, count);
    count_launch();
    return check_launch("relu_bwd_kernel");
}

int csrt_bias_grad_sgd(const float *dy, int32_t m, int32_t n, float *bias, float eta, float *gb_out, void *stream) {
    CSRT_ARG(m >= 0 && n >= 0, "negative size");
    if (m == 0) return CSRT_OK;
    CSRT_ARG(dy != nullptr || n == 0, "dy is NULL");
    launch_pdl(bias_grad_sgd_kernel, dim3((unsigned)ceil_div<int64_t>((int64_t)m * 32, 256)), dim3(256), 0,
               as_stream(stream), dy, m, n, bias, eta, gb_out);
    count_launch();
    return check_launch("bias_grad_sgd_kernel");
}

int csrt_softmax_xent(const float *z, const int32_t *labels, int32_t classes, int32_t n, float *dz, float *loss,
                      void *stream) {
    CSRT_ARG(classes > 0 && n >= 0, "bad size");
    CSRT_ARG(z && labels && dz && loss, "NULL pointer");
    cudaStream_t s = as_stream(stream);
    if (n > 0) {
        launch_pdl(softmax_xent_kernel, dim3((unsigned)ceil_div<int64_t>(n, 8)), dim3(kSmThreads), 0, s, z, labels,
                   classes, n, dz, loss + 1);
        count_launch();
    }
    launch_pdl(mean_kernel, dim3(1), dim3(1024), 0, s, loss + 1, n, loss);
    count_launch();
    return check_launch("softmax_xent_kernel");
}

int csrt_im2col(const float *x, int32_t c, int32_t b, int32_t h, int32_t w, int32_t k, float *cols, void *stream) {
    CSRT_ARG(c >= 0 && b >= 0 && k >= 1 && h >= k && w >= k, "bad shape");
    const int64_t total = (int64_t)c * k * k * b * (h - k + 1) * (w - k + 1);
    if (total == 0) return CSRT_OK;
    CSRT_ARG(x && cols, "NULL pointer");
    launch_pdl(im2col_kernel, dim3(grid_for(total)), dim3(256), 0, as_stream(stream), x, c, b, h, w, k, cols);
    count_launch();
    return check_launch("im2col_kernel");
}

int csrt_col2im(const float *dcols, int32_t c, int32_t b, int32_t h, int32_t w, int32_t k, float *dx, void *stream) {
    CSRT_ARG(c >= 0 && b >= 0 && k >= 1 && h >= k && w >= k, "bad shape");
    const int64_t total = (int64_t)c * b * h * w;
    if (total == 0) return CSRT_OK;
    CSRT_ARG(dcols && dx, "NULL pointer");
    launch_pdl(col2im_kernel, dim3(grid_for(total)), dim3(256), 0, as_stream(stream), dcols, c, b, h, w, k, dx);
    count_launch();
    return check_launch("col2im_kernel");
}

int csrt_maxpool2_fwd(const float *x, int32_t c, int32_t b, int32_t h, int32_t w, float *y, int8_t *idx,
                      void *stream) {
    CSRT_ARG(c >= 0 && b >= 0 && h >= 0 && w >= 0 && h % 2 == 0 && w % 2 == 0, "bad shape");
    const int64_t total = (int64_t)c * b * (h / 2) * (w / 2);
    if (total == 0) return CSRT_OK;
    CSRT_ARG(x && y && idx, "NULL pointer");
    launch_pdl(maxpool2_fwd_kernel, dim3(grid_for(total)), dim3(256), 0, as_stream(stream), x, c, b, h, w, y, idx);
    count_launch();
    return check_launch("maxpool2_fwd_kernel");
}

int csrt_maxpool2_bwd(const float *dy, const int8_t *idx, int32_t c, int32_t b, int32_t h, int32_t w, float *dx,
                      void *stream) {
    CSRT_ARG(c >= 0 && b >= 0 && h >= 0 && w >= 0 && h % 2 == 0 && w % 2 == 0, "bad shape");
    const int64_t total = (int64_t)c * b * h * w;
    if (total == 0) return CSRT_OK;
    CSRT_ARG(dy && idx && dx, "NULL pointer");
    launch_pdl(maxpool2_bwd_kernel, dim3(grid_for(total)), dim3(256), 0, as_stream(stream), dy, idx, c, b, h, w, dx);
    count_launch();
    return check_launch("maxpool2_bwd_kernel");
}

int csrt_flatten(const float *x, int32_t c, int32_t b, int32_t hw, float *xf, void *stream) {
    CSRT_ARG(c >= 0 && b >= 0 && hw >= 0, "bad shape");
    const int64_t total = (int64_t)c * b * hw;
    if (total == 0) return CSRT_OK;
    CSRT_ARG(x && xf, "NULL pointer");
    launch_pdl(flatten_kernel, dim3(grid_for(total)), dim3(256), 0, as_stream(stream), x, c, b, hw, xf, 0);
    count_launch();
    return check_launch("flatten_kernel");
}

int csrt_unflatten(const float *xf, int32_t c, int32_t b, int32_t hw, float *x, void *stream) {
    CSRT_ARG(c >= 0 && b >= 0 && hw >= 0, "bad shape");
    const int64_t total = (int64_t)c * b * hw;
    if (total == 0) return CSRT_OK;
    CSRT_ARG(x && xf, "NULL pointer");
    launch_pdl(flatten_kernel, dim3(grid_for(total)), dim3(256), 0, as_stream(stream), xf, c, b, hw, x, 1);
    count_launch();
    return check_launch("flatten_kernel");
}

}  // extern "C"
