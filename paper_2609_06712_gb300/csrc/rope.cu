// 3D RoPE tables and the rotate + block-pool pass of the block mask.
//
// RoPE (Sec. 3, Eq. shiftinv; truncation Sec. 4.2): pair m acts on coordinates
// (2m, 2m+1); the first d_t/2 pairs turn with the temporal position, the next
// d_x/2 with the row, the rest with the column; within an axis the i-th pair
// turns by pos * theta^(-2i/d_axis).  The table holds (cos, sin) in fp32,
// evaluated in fp64 once per call.
#include "common.cuh"

namespace rola {

__global__ void rope_table_kernel(float2* __restrict__ tab, int T, int Hh, int Ww, int d_t, int d_x, int d_y,
                                  int off_t, int off_x, int off_y, double theta)
{
    int idx = blockIdx.x * blockDim.x + threadIdx.x;
    int rows = T + Hh + Ww;
    if (idx >= rows * kPairs) return;
    int row = idx / kPairs, m = idx % kPairs;
    int pt = d_t / 2, px = d_x / 2;
    int axis = m < pt ? 0 : (m < pt + px ? 1 : 2);
    int row_axis = row < T ? 0 : (row < T + Hh ? 1 : 2);
    float2 out = make_float2(1.0f, 0.0f);
    if (axis == row_axis) {
        int i = axis == 0 ? m : (axis == 1 ? m - pt : m - pt - px);
        int d_axis = axis == 0 ? d_t : (axis == 1 ? d_x : d_y);
        int pos = axis == 0 ? row + off_t : (axis == 1 ? row - T + off_x : row - T - Hh + off_y);
        double freq = pow(theta, -2.0 * (double)i / (double)d_axis);
        double s, c;
        sincos((double)pos * freq, &s, &c);
        out = make_float2((float)c, (float)s);
    }
    tab[idx] = out;
}

cudaError_t launch_rope_table(const rola_config_t& cfg, float2* tab, cudaStream_t st)
{
    int n = (cfg.T + cfg.Hh + cfg.Ww) * kPairs;
    rope_table_kernel<<<(n + 255) / 256, 256, 0, st>>>(tab, cfg.T, cfg.Hh, cfg.Ww, cfg.rope_split[0],
                                                       cfg.rope_split[1], cfg.rope_split[2], cfg.pos_offset[0],
                                                       cfg.pos_offset[1], cfg.pos_offset[2], cfg.rope_theta);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// rotate + pool: one CTA per (64-token block, head, q|k).  256 threads: 16 per
// token row (8 coordinates = 4 pairs each), 16 rows per pass, 4 passes.  Writes
// the rotated rows in the storage dtype and the fp32 block mean of the
// fp32-rotated (unrounded) values.  The block mean is the pairwise sum of the
// block's 64 slots in slot order (slots past the sequence hold +0), divided
// once by the token count: the evaluation order the block mask is defined
// with, so that every kernel computing it gives the same bits.

// Pairwise sum of the 64 values col[0], col[stride], ..., col[63 stride]:
// sum(x[0..n)) = sum(x[0..n/2)) + sum(x[n/2..n)), evaluated level by level.
__device__ __forceinline__ float pairwise64(const float* col, int stride)
{
    float v[kBlock];
#pragma unroll
    for (int i = 0; i < kBlock; ++i) v[i] = col[i * stride];
#pragma unroll
    for (int w = 1; w < kBlock; w *= 2)
#pragma unroll
        for (int i = 0; i < kBlock; i += 2 * w) v[i] = v[i] + v[i + w];
    return v[0];
}

template <typename T>
struct Vec8;
template <>
struct Vec8<__nv_bfloat16> {
    __device__ static void load(const __nv_bfloat16* p, float (&x)[8])
    {
        uint4 u = __ldg(reinterpret_cast<const uint4*>(p));
        uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            float2 f = unpack_bf16(w[i]);
            x[2 * i] = f.x;
            x[2 * i + 1] = f.y;
        }
    }
    __device__ static void store(__nv_bfloat16* p, const float (&x)[8])
    {
        uint4 u = make_uint4(pack_bf16(x[0], x[1]), pack_bf16(x[2], x[3]), pack_bf16(x[4], x[5]),
                             pack_bf16(x[6], x[7]));
        *reinterpret_cast<uint4*>(p) = u;
    }
};
template <>
struct Vec8<float> {
    __device__ static void load(const float* p, float (&x)[8])
    {
        float4 a = __ldg(reinterpret_cast<const float4*>(p));
        float4 b = __ldg(reinterpret_cast<const float4*>(p) + 1);
        x[0] = a.x; x[1] = a.y; x[2] = a.z; x[3] = a.w;
        x[4] = b.x; x[5] = b.y; x[6] = b.z; x[7] = b.w;
    }
    __device__ static void store(float* p, const float (&x)[8])
    {
        reinterpret_cast<float4*>(p)[0] = make_float4(x[0], x[1], x[2], x[3]);
        reinterpret_cast<float4*>(p)[1] = make_float4(x[4], x[5], x[6], x[7]);
    }
};

template <typename T>
__global__ void __launch_bounds__(256) rope_pool_kernel(Shape s, const T* __restrict__ q, const T* __restrict__ k,
                                                        const float2* __restrict__ tab, T* __restrict__ qr,
                                                        T* __restrict__ kr, float* __restrict__ qbar,
                                                        float* __restrict__ kbar)
{
    __shared__ __align__(16) float rot[kBlock][kDh];      // fp32 rotated rows, slot order
    const int blk = blockIdx.x, bh = blockIdx.y;
    const T* x = blockIdx.z == 0 ? q : k;
    T* xr = blockIdx.z == 0 ? qr : kr;
    float* xbar = blockIdx.z == 0 ? qbar : kbar;
    const int c8 = threadIdx.x & 15;        // coordinates 8*c8 .. 8*c8+7 (pairs 4*c8 .. 4*c8+3)
    const int rsub = threadIdx.x >> 4;      // row within a pass; rows rsub + 16 * pass
    const int n0 = blk * kBlock + rsub;
    constexpr int kPasses = kBlock / 16;
    // all loads first: four 16- or 32-byte vectors in flight per thread
    float v[kPasses][8];
#pragma unroll
    for (int pass = 0; pass < kPasses; ++pass) {
        const int n = n0 + 16 * pass;
        if (n < s.N) Vec8<T>::load(x + ((size_t)bh * s.N + n) * kDh + c8 * 8, v[pass]);
    }
    // grid position of the first row, then advanced by 16 tokens per pass
    const int hw = s.Hh * s.Ww;
    int t = n0 / hw, rem = n0 - t * hw;
    int xx = rem / s.Ww, yy = rem - xx * s.Ww;
    // table row base of each of this thread's 4 pairs: the pair's axis is fixed
    int axis[4];
#pragma unroll
    for (int p = 0; p < 4; ++p) {
        const int m = c8 * 4 + p;
        axis[p] = m < s.pt ? 0 : (m < s.pt + s.px ? 1 : 2);
    }
#pragma unroll
    for (int pass = 0; pass < kPasses; ++pass) {
        const int n = n0 + 16 * pass;
        float o[8] = {0, 0, 0, 0, 0, 0, 0, 0};
        if (n < s.N) {
#pragma unroll
            for (int p = 0; p < 4; ++p) {
                const int row = axis[p] == 0 ? t : (axis[p] == 1 ? s.T + xx : s.T + s.Hh + yy);
                const float2 cs = __ldg(tab + row * kPairs + c8 * 4 + p);
                const float2 y = rope_rotate(v[pass][2 * p], v[pass][2 * p + 1], cs);
                o[2 * p] = y.x;
                o[2 * p + 1] = y.y;
            }
            Vec8<T>::store(xr + ((size_t)bh * s.N + n) * kDh + c8 * 8, o);
        }
        float4* dst = reinterpret_cast<float4*>(&rot[rsub + 16 * pass][c8 * 8]);
        dst[0] = make_float4(o[0], o[1], o[2], o[3]);
        dst[1] = make_float4(o[4], o[5], o[6], o[7]);
        yy += 16;                           // advance to the token 16 further on
        while (yy >= s.Ww) {
            yy -= s.Ww;
            if (++xx == s.Hh) {
                xx = 0;
                ++t;
            }
        }
    }
    __syncthreads();
    if (threadIdx.x < kDh) {
        const int cnt = min(kBlock, s.N - blk * kBlock);
        const float sum = pairwise64(&rot[0][threadIdx.x], kDh);
        // with 128-token query blocks the query side keeps the sum (the 128-token tree's left or right half)
        xbar[((size_t)bh * s.nB + blk) * kDh + threadIdx.x] = (blockIdx.z == 0 && s.qb2) ? sum : sum / (float)cnt;
    }
}

// ---------------------------------------------------------------------------
// The same pass in cube geometry: one CTA per (cube, head, q|k|v).  Thread
// (rsub, c8) handles slot rsub + 16 dt of the cube for dt = 0..3, i.e. grid
// position (t0 + dt, x0 + rsub / 4, y0 + rsub % 4).  The rotated rows are
// written in block order (row 64 b + slot of the head's Np rows, zeros for
// slots outside the grid, so that the sparse kernels read finite values
// there); the v slice copies v into the same order without rotating it.

template <typename T>
__global__ void __launch_bounds__(256) rope_pool_cube_kernel(Shape s, const T* __restrict__ q,
                                                             const T* __restrict__ k, const T* __restrict__ v,
                                                             const float2* __restrict__ tab, T* __restrict__ qr,
                                                             T* __restrict__ kr, T* __restrict__ vp,
                                                             float* __restrict__ qbar, float* __restrict__ kbar)
{
    __shared__ __align__(16) float rot[kBlock][kDh];      // fp32 rotated rows, slot order
    const int blk = blockIdx.x, bh = blockIdx.y, z = blockIdx.z;
    const T* x = z == 0 ? q : (z == 1 ? k : v);
    T* xr = z == 0 ? qr : (z == 1 ? kr : vp);
    const int c8 = threadIdx.x & 15;
    const int rsub = threadIdx.x >> 4;
    constexpr int kPasses = kBlock / 16;
    const CubeOrigin o = cube_origin(s, blk);
    float v8[kPasses][8];
#pragma unroll
    for (int dt = 0; dt < kPasses; ++dt) {
        const int n = cube_token(s, o, rsub + 16 * dt);
        if (n >= 0) Vec8<T>::load(x + ((size_t)bh * s.N + n) * kDh + c8 * 8, v8[dt]);
    }
    int axis[4];
#pragma unroll
    for (int p = 0; p < 4; ++p) {
        const int m = c8 * 4 + p;
        axis[p] = m < s.pt ? 0 : (m < s.pt + s.px ? 1 : 2);
    }
    const int xx = o.x + (rsub >> 2), yy = o.y + (rsub & 3);
#pragma unroll
    for (int dt = 0; dt < kPasses; ++dt) {
        const int slot = rsub + 16 * dt;
        const int n = cube_token(s, o, slot);
        float out[8] = {0, 0, 0, 0, 0, 0, 0, 0};
        if (n >= 0) {
            if (z == 2) {
#pragma unroll
                for (int i = 0; i < 8; ++i) out[i] = v8[dt][i];
            } else {
                const int t = o.t + dt;
#pragma unroll
                for (int p = 0; p < 4; ++p) {
                    const int row = axis[p] == 0 ? t : (axis[p] == 1 ? s.T + xx : s.T + s.Hh + yy);
                    const float2 cs = __ldg(tab + row * kPairs + c8 * 4 + p);
                    const float2 y = rope_rotate(v8[dt][2 * p], v8[dt][2 * p + 1], cs);
                    out[2 * p] = y.x;
                    out[2 * p + 1] = y.y;
                }
            }
        }
        Vec8<T>::store(xr + ((size_t)bh * s.Np + (size_t)blk * kBlock + slot) * kDh + c8 * 8, out);
        if (z != 2) {
            float4* dst = reinterpret_cast<float4*>(&rot[slot][c8 * 8]);
            dst[0] = make_float4(out[0], out[1], out[2], out[3]);
            dst[1] = make_float4(out[4], out[5], out[6], out[7]);
        }
    }
    if (z == 2) return;
    __syncthreads();
    if (threadIdx.x < kDh) {
        const int cnt = min(4, s.T - o.t) * min(4, s.Hh - o.x) * min(4, s.Ww - o.y);
        (z == 0 ? qbar : kbar)[((size_t)bh * s.nB + blk) * kDh + threadIdx.x] =
            pairwise64(&rot[0][threadIdx.x], kDh) / (float)cnt;
    }
}

template <typename T>
cudaError_t launch_rope_pool_t(const Shape& s, const void* q, const void* k, const void* v, const float2* tab,
                               void* qr, void* kr, void* vp, float* qbar, float* kbar, cudaStream_t st)
{
    if (s.cube) {
        dim3 grid(s.nB, s.B * s.H, v ? 3 : 2);
        rope_pool_cube_kernel<T><<<grid, 256, 0, st>>>(s, (const T*)q, (const T*)k, (const T*)v, tab, (T*)qr,
                                                       (T*)kr, (T*)vp, qbar, kbar);
    } else {
        dim3 grid(s.nB, s.B * s.H, 2);
        rope_pool_kernel<T><<<grid, 256, 0, st>>>(s, (const T*)q, (const T*)k, tab, (T*)qr, (T*)kr, qbar, kbar);
    }
    return cudaGetLastError();
}

cudaError_t launch_rope_pool(const rola_config_t& cfg, const Shape& s, const void* q, const void* k, const void* v,
                             const float2* tab, void* qr, void* kr, void* vp, float* qbar, float* kbar,
                             cudaStream_t st)
{
    if (s.cube && v && !vp) return cudaErrorInvalidValue;
    return cfg.dtype == ROLA_BF16
               ? launch_rope_pool_t<__nv_bfloat16>(s, q, k, v, tab, qr, kr, vp, qbar, kbar, st)
               : launch_rope_pool_t<float>(s, q, k, v, tab, qr, kr, vp, qbar, kbar, st);
}

}  // namespace rola
