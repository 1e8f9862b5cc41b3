// Token gate of the gated fusion (Sec. fusion; Alg. 1, "token-wise scalar gate"):
//   g_p = sigmoid(x_p . w_g + b_g),
// one scalar per token from the attention block's input hidden state x_p
// (d_model wide); it is the `gate` input of the fusion, Eq. (gate).
//
// HBM-bound GEMV (X is read once, 2 B per element in bf16): one warp per token
// row, 16-byte loads of x_p and w_g (w_g stays in L1), fp32 FMA, a shuffle
// reduction, then the sigmoid with the IEEE exp.
#include "common.cuh"

namespace rola {
namespace {

constexpr int kGateWarps = 8;

__device__ __forceinline__ void load8f(const __nv_bfloat16* p, float (&x)[8])
{
    const uint4 u = __ldg(reinterpret_cast<const uint4*>(p));
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float2 f = unpack_bf16(w[i]);
        x[2 * i] = f.x;
        x[2 * i + 1] = f.y;
    }
}
__device__ __forceinline__ void load8f(const float* p, float (&x)[8])
{
    const float4 a = __ldg(reinterpret_cast<const float4*>(p)), b = __ldg(reinterpret_cast<const float4*>(p) + 1);
    x[0] = a.x; x[1] = a.y; x[2] = a.z; x[3] = a.w;
    x[4] = b.x; x[5] = b.y; x[6] = b.z; x[7] = b.w;
}

template <typename T>
__global__ void __launch_bounds__(32 * kGateWarps) gate_kernel(long long rows, int D, const T* __restrict__ X,
                                                               const T* __restrict__ w, float b,
                                                               float* __restrict__ g)
{
    const int lane = threadIdx.x & 31;
    const long long stride = (long long)gridDim.x * kGateWarps;
    for (long long row = (long long)blockIdx.x * kGateWarps + (threadIdx.x >> 5); row < rows; row += stride) {
        const T* x = X + row * D;
        float acc = 0.0f;
        for (int c = lane * 8; c < D; c += 32 * 8) {
            float xv[8], wv[8];
            load8f(x + c, xv);
            load8f(w + c, wv);
#pragma unroll
            for (int i = 0; i < 8; ++i) acc = fmaf(xv[i], wv[i], acc);
        }
#pragma unroll
        for (int off = 16; off >= 1; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
        if (lane == 0) g[row] = 1.0f / (1.0f + expf(-(acc + b)));
    }
}

}  // namespace

cudaError_t launch_gate(rola_dtype_t dt, long long rows, int D, const void* X, const void* w, float b, float* g,
                        cudaStream_t st)
{
    int dev = 0, nsm = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    long long want = (rows + kGateWarps - 1) / kGateWarps;
    const long long cap = (long long)nsm * 8;            // 8 CTAs of 8 warps per SM, rows grid-strided
    const int grid = (int)(want < cap ? want : cap);
    if (dt == ROLA_BF16)
        gate_kernel<__nv_bfloat16><<<grid, 32 * kGateWarps, 0, st>>>(
            rows, D, static_cast<const __nv_bfloat16*>(X), static_cast<const __nv_bfloat16*>(w), b, g);
    else
        gate_kernel<float><<<grid, 32 * kGateWarps, 0, st>>>(rows, D, static_cast<const float*>(X),
                                                               static_cast<const float*>(w), b, g);
    return cudaGetLastError();
}

}  // namespace rola
