// Block-sparse softmax attention over the kept key blocks (kernel 2).
//
//   O^s_p = sum_{q in kept(i)} softmax_q(q^r_p . k^r_q / sqrt(d_h)) v_q,   p in block i
//
// (Sec. 3 softmax form restricted to the kept blocks, Alg. 1 sparse branch).
// q^r, k^r are the rotated copies written by the rotate + pool pass.  The
// bf16 path is a tcgen05 kernel: sparse_attn_rows.cu for contiguous key
// blocks (64-token query blocks or 128-token query chunks), sparse_attn_tc.cu
// for the cube geometry; this file holds the fp32 validation-mode kernel
// (online softmax in fp32) and the dispatch.
#include "common.cuh"

namespace rola {

// ===========================================================================
// fp32 validation mode: plain SIMT, one CTA per (query block, head), 256
// threads.  Shared memory: Q, K with padded rows (129 floats), V, S.
// q^r, k^r and v are read in block order (Np rows per head: the token order
// itself for contiguous chunks, cube slots for cubes); O^s rows go to their
// tokens.

constexpr int kF32Threads = 256;
constexpr int kPad = kDh + 1;

__global__ void __launch_bounds__(kF32Threads) sparse_attn_f32_kernel(Shape s, const float* __restrict__ qr,
                                                                      const float* __restrict__ kr,
                                                                      const float* __restrict__ v,
                                                                      const int32_t* __restrict__ kv_idx,
                                                                      float* __restrict__ o, float* __restrict__ lse)
{
    extern __shared__ float fsm[];
    float* Qs = fsm;                       // [64][129]
    float* Ks = Qs + kBlock * kPad;        // [64][129]
    float* Vs = Ks + kBlock * kPad;        // [64][128]
    float* Ss = Vs + kBlock * kDh;         // [64][65]
    const int qb = blockIdx.x, bh = blockIdx.y, tid = threadIdx.x;
    const size_t head = (size_t)bh * s.Np * kDh;
    const int32_t* kept = kv_idx + ((size_t)bh * s.nQ + (qb >> s.qb2)) * s.n_keep;   // the block's mask row
    for (int e = tid; e < kBlock * kDh; e += kF32Threads) {
        int r = e / kDh, d = e % kDh, n = qb * kBlock + r;
        Qs[r * kPad + d] = n < s.Np ? qr[head + (size_t)n * kDh + d] : 0.0f;
    }
    const int row = tid >> 2, quarter = tid & 3;
    float acc[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) acc[i] = 0.0f;
    float m_run = -INFINITY, l_run = 0.0f;
    const float scale = 0.08838834764831845f;   // 1/sqrt(128)
    for (int it = 0; it < s.n_keep; ++it) {
        const int j = kept[it];
        __syncthreads();
        for (int e = tid; e < kBlock * kDh; e += kF32Threads) {
            int r = e / kDh, d = e % kDh, n = j * kBlock + r;
            bool ok = n >= 0 && n < s.Np;
            Ks[r * kPad + d] = ok ? kr[head + (size_t)n * kDh + d] : 0.0f;
            Vs[r * kDh + d] = ok ? v[head + (size_t)n * kDh + d] : 0.0f;
        }
        __syncthreads();
        const int kvalid = s.N - j * kBlock;
        const CubeOrigin jo = cube_origin(s, j);
        float sv[16];
        float mx = m_run;
#pragma unroll 1
        for (int c = 0; c < 16; ++c) {
            int col = quarter * 16 + c;
            float dot = 0.0f;
            for (int d = 0; d < kDh; ++d) dot = fmaf(Qs[row * kPad + d], Ks[col * kPad + d], dot);
            const bool valid = s.cube ? cube_token(s, jo, col) >= 0 : col < kvalid;
            sv[c] = valid ? dot * scale : -INFINITY;
            mx = fmaxf(mx, sv[c]);
        }
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
        float alpha = expf(m_run - mx);
        float lsum = 0.0f;
#pragma unroll
        for (int c = 0; c < 16; ++c) {
            float p = expf(sv[c] - mx);
            Ss[row * 65 + quarter * 16 + c] = p;
            lsum += p;
        }
        lsum += __shfl_xor_sync(0xffffffffu, lsum, 1);
        lsum += __shfl_xor_sync(0xffffffffu, lsum, 2);
        l_run = l_run * alpha + lsum;
        m_run = mx;
        __syncwarp();
#pragma unroll
        for (int i = 0; i < 32; ++i) acc[i] *= alpha;
        for (int c = 0; c < kBlock; ++c) {
            float p = Ss[row * 65 + c];
#pragma unroll
            for (int i = 0; i < 32; ++i) acc[i] = fmaf(p, Vs[c * kDh + quarter + 4 * i], acc[i]);
        }
    }
    const int n = s.cube ? cube_token(s, cube_origin(s, qb), row) : qb * kBlock + row;
    if (n >= 0 && n < s.N) {
        float inv = 1.0f / l_run;
        if (lse && quarter == 0) lse[(size_t)bh * s.N + n] = m_run + logf(l_run);
        float* on = o + ((size_t)bh * s.N + n) * kDh;
#pragma unroll
        for (int i = 0; i < 32; ++i) on[quarter + 4 * i] = acc[i] * inv;
    }
}

// bf16 with contiguous key blocks (sparse_attn_rows.cu)
cudaError_t launch_sparse_attn_rows(const Shape& s, const void* qr, const void* kr, const void* v,
                                    const int32_t* kv_idx, void* o_s, float* lse, DeviceStatus* status,
                                    cudaStream_t st);

cudaError_t launch_sparse_attn(rola_dtype_t dt, const Shape& s, const void* qr, const void* kr, const void* v,
                               const int32_t* kv_idx, void* o_s, float* lse, DeviceStatus* status, cudaStream_t st)
{
    if (dt == ROLA_BF16 && !s.cube) return launch_sparse_attn_rows(s, qr, kr, v, kv_idx, o_s, lse, status, st);
    if (dt == ROLA_BF16) return launch_sparse_attn_tc(s, qr, kr, v, kv_idx, o_s, lse, status, st);
    dim3 grid(s.nB, s.B * s.H);
    size_t smem = sizeof(float) * (2 * kBlock * kPad + kBlock * kDh + kBlock * 65);
    cudaError_t e = cudaFuncSetAttribute(sparse_attn_f32_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    sparse_attn_f32_kernel<<<grid, kF32Threads, smem, st>>>(s, (const float*)qr, (const float*)kr, (const float*)v,
                                                            kv_idx, (float*)o_s, lse);
    return cudaGetLastError();
}

}  // namespace rola
