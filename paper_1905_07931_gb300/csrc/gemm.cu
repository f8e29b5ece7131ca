// Dense weight gradient G = dY X^T for the proximal phase.
//
// The prox step acts on the dense matrix w - eta*G (Section 3.3), so the
// gradient of every weight, zero or not, is needed: G[i, j] = sum_c dY[i, c]
// X[j, c], with both operands stored with the reduction index c contiguous.
//
// Two implementations:
//  * CSRT_PREC_FP32: a float32 FMA kernel on the CUDA cores (64 x 64 output
//    tile, 16-deep reduction slices staged in shared memory, 4 x 4 outputs per
//    thread). Shapes with few output tiles and a long reduction (the
//    convolution layers: 20 x 25 outputs summed over 73,728 columns) split the
//    reduction over blocks and add the partial tiles in a fixed order.
//  * CSRT_PREC_TF32: tcgen05 tensor cores (gemm_tc.cu).
#include "common.cuh"

namespace csrt {

constexpr int kGBM = 64, kGBN = 64, kGBK = 16;
constexpr int64_t kGemmScratchFloats = (int64_t)1 << 24;   // 64 MB cap on split-reduction partials

struct GemmSplit {
    int splits;
    int chunk;
};

static GemmSplit gemm_split(int32_t m, int32_t k, int32_t n) {
    const int64_t tiles = ceil_div<int64_t>(m, kGBM) * ceil_div<int64_t>(k, kGBN);
    const int64_t want_blocks = (int64_t)num_sms() * 4;
    int64_t splits = 1;
    if (tiles < want_blocks && n > 4 * kGBK * 8) {
        splits = imin<int64_t>(ceil_div<int64_t>(want_blocks, tiles), ceil_div<int64_t>(n, 512));
        splits = imin<int64_t>(splits, imax<int64_t>(1, kGemmScratchFloats / imax<int64_t>(1, (int64_t)m * k)));
        splits = imax<int64_t>(1, splits);
    }
    GemmSplit s;
    s.splits = (int)splits;
    s.chunk = (int)ceil_div<int64_t>(ceil_div<int64_t>(n, splits), kGBK) * kGBK;
    s.splits = (int)ceil_div<int64_t>(n, s.chunk);
    return s;
}

size_t gemm_scratch_bytes(int32_t m, int32_t k, int32_t max_n) {
    // A split is only taken for n > 512, and splits * m * k never exceeds
    // kGemmScratchFloats (nor ceil(n / 512) * m * k) for any m <= rows, k <= cols.
    if ((int64_t)m * k == 0 || max_n <= 4 * kGBK * 8) return 0;
    const int64_t floats = imin<int64_t>(kGemmScratchFloats, ceil_div<int64_t>(max_n, 512) * (int64_t)m * k);
    return (size_t)floats * sizeof(float) + 256;
}

__global__ void __launch_bounds__(256) gemm_nt_f32_kernel(const float *__restrict__ dy, const float *__restrict__ x,
                                                          int32_t m, int32_t k, int32_t n, int32_t chunk,
                                                          float *__restrict__ out) {
    pdl_enter();
    __shared__ float as[kGBK][kGBM + 4];
    __shared__ float bs[kGBK][kGBN + 4];
    const int tid = threadIdx.x;
    const int ty = tid / 16, tx = tid % 16;
    const int64_t i0 = (int64_t)blockIdx.y * kGBM, j0 = (int64_t)blockIdx.x * kGBN;
    const int split = blockIdx.z;
    const int nb = split * chunk, ne = min(n, nb + chunk);
    float acc[4][4] = {};
    for (int c0 = nb; c0 < ne; c0 += kGBK) {
#pragma unroll
        for (int l = 0; l < 4; ++l) {
            const int idx = tid + l * 256;
            const int r = idx / kGBK, kk = idx % kGBK;
            const int c = c0 + kk;
            as[kk][r] = (i0 + r < m && c < ne) ? __ldg(dy + (i0 + r) * n + c) : 0.f;
            bs[kk][r] = (j0 + r < k && c < ne) ? __ldg(x + (j0 + r) * n + c) : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < kGBK; ++kk) {
            float a[4], b[4];
#pragma unroll
            for (int t = 0; t < 4; ++t) {
                a[t] = as[kk][ty * 4 + t];
                b[t] = bs[kk][tx * 4 + t];
            }
#pragma unroll
            for (int p = 0; p < 4; ++p)
#pragma unroll
                for (int q = 0; q < 4; ++q) acc[p][q] = fmaf(a[p], b[q], acc[p][q]);
        }
        __syncthreads();
    }
    float *o = out + (int64_t)split * m * k;
#pragma unroll
    for (int p = 0; p < 4; ++p) {
        const int64_t i = i0 + ty * 4 + p;
        if (i >= m) continue;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int64_t j = j0 + tx * 4 + q;
            if (j < k) o[i * k + j] = acc[p][q];
        }
    }
}

__global__ void split_reduce_kernel(const float *__restrict__ part, int64_t count, int32_t splits,
                                    float *__restrict__ out) {
    pdl_enter();
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < count; e += (int64_t)gridDim.x * blockDim.x) {
        float s = 0.f;
        for (int p = 0; p < splits; ++p) s += part[(int64_t)p * count + e];
        out[e] = s;
    }
}

int gemm_tc_tf32(const float *dy, const float *x, int32_t m, int32_t k, int32_t n, float *g, void *ws,
                 size_t ws_bytes, cudaStream_t s, bool *handled);

}  // namespace csrt

using namespace csrt;

extern "C" int weight_grad_dense(const float *dy, const float *x, int32_t m, int32_t k, int32_t n, float *g,
                                 int32_t precision, void *ws, size_t ws_bytes, void *stream) {
    CSRT_ARG(m >= 0 && k >= 0 && n >= 0, "negative size");
    CSRT_ARG((int64_t)m * k < ((int64_t)1 << 31), "m*k must be below 2^31");
    CSRT_ARG(precision == CSRT_PREC_FP32 || precision == CSRT_PREC_TF32, "unknown precision %d", precision);
    if ((int64_t)m * k == 0) return CSRT_OK;
    CSRT_ARG(g != nullptr, "G is NULL");
    cudaStream_t s = as_stream(stream);
    if (n == 0) {
        CSRT_CHECK_CUDA(cudaMemsetAsync(g, 0, sizeof(float) * (size_t)m * k, s));
        return CSRT_OK;
    }
    CSRT_ARG(dy && x, "dY or X is NULL");
    if (precision == CSRT_PREC_TF32) {
        bool handled = false;
        int rc = gemm_tc_tf32(dy, x, m, k, n, g, ws, ws_bytes, s, &handled);
        if (rc || handled) return rc;
        // shapes the tensor-core kernel does not take fall through to FP32
    }
    const GemmSplit sp = gemm_split(m, k, n);
    float *out = g;
    if (sp.splits > 1) {
        const size_t need = kWsReservedBytes + (size_t)sp.splits * m * k * sizeof(float);
        CSRT_ARG(ws != nullptr && ws_bytes >= need, "workspace too small for split gemm (%zu < %zu)", ws_bytes, need);
        out = reinterpret_cast<float *>(ws_scratch(ws));
    }
    dim3 grid((unsigned)ceil_div<int64_t>(k, kGBN), (unsigned)ceil_div<int64_t>(m, kGBM), (unsigned)sp.splits);
    launch_pdl(gemm_nt_f32_kernel, dim3(grid), dim3(256), 0, s, dy, x, m, k, n, sp.chunk, out);
    count_launch();
    if (sp.splits > 1) {
        const int64_t count = (int64_t)m * k;
        const unsigned rg = (unsigned)imin<int64_t>(ceil_div<int64_t>(count, 256), (int64_t)num_sms() * 8);
        launch_pdl(split_reduce_kernel, dim3(rg), dim3(256), 0, s, out, count, sp.splits, g);
        count_launch();
    }
    return check_launch("gemm_nt_f32_kernel");
}
