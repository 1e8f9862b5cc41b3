// Block-sparse softmax attention over the kept key blocks (kernel 2).
//
//   O^s_p = sum_{q in kept(i)} softmax_q(q^r_p . k^r_q / sqrt(d_h)) v_q,   p in block i
//
// (Sec. 3 softmax form restricted to the kept blocks, Alg. 1 sparse branch).
// q^r, k^r are the rotated copies written by the rotate + pool pass.  The
// softmax runs online in fp32 (running max and sum per query row), in base 2
// with log2(e)/sqrt(d_h) folded into the scores.
#include "common.cuh"

namespace rola {

// ===========================================================================
// bf16: one CTA per (query block, head), 4 warps x 16 query rows, warp-level
// m16n8k16 MMAs, K/V blocks double-buffered through cp.async.
// Shared memory: Q 16 KB | K 2 x 16 KB | V 2 x 16 KB, rows of 256 B with the
// 16-byte chunk index XOR-swizzled by (row & 7).

constexpr int kAttnThreads = 128;
constexpr int kTileBytes = kBlock * kDh * 2;   // 16 KB

__device__ __forceinline__ void load_tile_async(uint32_t sbase, const __nv_bfloat16* g, int row0, int N, int tid)
{
    // 64 rows x 16 chunks of 16 B = 1024 chunks, 8 per thread
#pragma unroll
    for (int it = 0; it < 8; ++it) {
        int e = tid + it * kAttnThreads;
        int r = e >> 4, c = e & 15;
        int n = row0 + r;
        bool ok = n >= 0 && n < N;   // rows outside [0, N) are zero-filled, never read
        const __nv_bfloat16* src = g + (size_t)(ok ? n : 0) * kDh + c * 8;
        cp_async16(sbase + sw128(r, c), src, ok ? 16 : 0);
    }
}

__global__ void __launch_bounds__(kAttnThreads) sparse_attn_bf16_kernel(
    Shape s, const __nv_bfloat16* __restrict__ qr, const __nv_bfloat16* __restrict__ kr,
    const __nv_bfloat16* __restrict__ v, const int32_t* __restrict__ kv_idx, __nv_bfloat16* __restrict__ o)
{
    extern __shared__ __align__(128) uint8_t smem[];
    const int qb = blockIdx.x, bh = blockIdx.y;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int g = lane >> 2, t4 = lane & 3;
    const uint32_t sQ = smem_u32(smem);
    const uint32_t sK = sQ + kTileBytes;
    const uint32_t sV = sK + 2 * kTileBytes;
    const size_t head = (size_t)bh * s.N * kDh;
    const int32_t* kept = kv_idx + ((size_t)bh * s.nB + qb) * s.n_keep;

    load_tile_async(sQ, qr + head, qb * kBlock, s.N, tid);
    int j0 = __ldg(kept);
    load_tile_async(sK, kr + head, j0 * kBlock, s.N, tid);
    load_tile_async(sV, v + head, j0 * kBlock, s.N, tid);
    cp_async_commit();

    float oacc[16][4];
#pragma unroll
    for (int i = 0; i < 16; ++i) oacc[i][0] = oacc[i][1] = oacc[i][2] = oacc[i][3] = 0.0f;
    float m_run[2] = {-INFINITY, -INFINITY}, l_run[2] = {0.0f, 0.0f};
    uint32_t qf[8][4];

    for (int it = 0; it < s.n_keep; ++it) {
        const int stage = it & 1;
        const int j = __ldg(kept + it);
        if (it + 1 < s.n_keep) {
            int jn = __ldg(kept + it + 1);
            load_tile_async(sK + (stage ^ 1) * kTileBytes, kr + head, jn * kBlock, s.N, tid);
            load_tile_async(sV + (stage ^ 1) * kTileBytes, v + head, jn * kBlock, s.N, tid);
        }
        cp_async_commit();
        cp_async_wait<1>();
        __syncthreads();
        if (it == 0) {
#pragma unroll
            for (int kc = 0; kc < 8; ++kc) {
                int mi = lane >> 3;
                int r = warp * 16 + (lane & 7) + (mi & 1) * 8;
                ldsm_x4(sQ + sw128(r, kc * 2 + (mi >> 1)), qf[kc][0], qf[kc][1], qf[kc][2], qf[kc][3]);
            }
        }
        const uint32_t kb = sK + stage * kTileBytes, vb = sV + stage * kTileBytes;
        // S = Q K^T : 16 rows x 64 keys per warp
        float sacc[8][4];
#pragma unroll
        for (int i = 0; i < 8; ++i) sacc[i][0] = sacc[i][1] = sacc[i][2] = sacc[i][3] = 0.0f;
#pragma unroll
        for (int kc = 0; kc < 8; ++kc) {
#pragma unroll
            for (int np = 0; np < 4; ++np) {
                int mi = lane >> 3;
                int key = np * 16 + (mi >> 1) * 8 + (lane & 7);
                uint32_t b0, b1, b2, b3;
                ldsm_x4(kb + sw128(key, kc * 2 + (mi & 1)), b0, b1, b2, b3);
                mma_bf16(sacc[2 * np], qf[kc][0], qf[kc][1], qf[kc][2], qf[kc][3], b0, b1);
                mma_bf16(sacc[2 * np + 1], qf[kc][0], qf[kc][1], qf[kc][2], qf[kc][3], b2, b3);
            }
        }
        // online softmax (base 2); keys past N are masked out
        const int kvalid = s.N - j * kBlock;
        float mx[2] = {m_run[0], m_run[1]};
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                int col = nt * 8 + t4 * 2 + (e & 1);
                float x = col < kvalid ? sacc[nt][e] * s.sm_scale_log2 : -INFINITY;
                sacc[nt][e] = x;
                mx[e >> 1] = fmaxf(mx[e >> 1], x);
            }
        }
        float alpha[2];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            mx[h] = fmaxf(mx[h], __shfl_xor_sync(0xffffffffu, mx[h], 1));
            mx[h] = fmaxf(mx[h], __shfl_xor_sync(0xffffffffu, mx[h], 2));
            alpha[h] = fast_exp2(m_run[h] - mx[h]);
            m_run[h] = mx[h];
            l_run[h] *= alpha[h];
        }
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            oacc[i][0] *= alpha[0]; oacc[i][1] *= alpha[0];
            oacc[i][2] *= alpha[1]; oacc[i][3] *= alpha[1];
        }
        uint32_t pf[8][2];
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) {
            float p0 = fast_exp2(sacc[nt][0] - mx[0]);
            float p1 = fast_exp2(sacc[nt][1] - mx[0]);
            float p2 = fast_exp2(sacc[nt][2] - mx[1]);
            float p3 = fast_exp2(sacc[nt][3] - mx[1]);
            pf[nt][0] = pack_bf16(p0, p1);
            pf[nt][1] = pack_bf16(p2, p3);
            // the row sums use the bf16-rounded weights the PV product sees
            float2 r0 = unpack_bf16(pf[nt][0]), r1 = unpack_bf16(pf[nt][1]);
            l_run[0] += r0.x + r0.y;
            l_run[1] += r1.x + r1.y;
        }
        // O += P V
#pragma unroll
        for (int kc = 0; kc < 4; ++kc) {
#pragma unroll
            for (int dp = 0; dp < 8; ++dp) {
                int mi = lane >> 3;
                int key = kc * 16 + (mi & 1) * 8 + (lane & 7);
                uint32_t b0, b1, b2, b3;
                ldsm_x4_t(vb + sw128(key, dp * 2 + (mi >> 1)), b0, b1, b2, b3);
                mma_bf16(oacc[2 * dp], pf[2 * kc][0], pf[2 * kc][1], pf[2 * kc + 1][0], pf[2 * kc + 1][1], b0, b1);
                mma_bf16(oacc[2 * dp + 1], pf[2 * kc][0], pf[2 * kc][1], pf[2 * kc + 1][0], pf[2 * kc + 1][1], b2,
                         b3);
            }
        }
        __syncthreads();   // this stage is refilled by the next iteration's prefetch
    }
    cp_async_wait<0>();
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        l_run[h] += __shfl_xor_sync(0xffffffffu, l_run[h], 1);
        l_run[h] += __shfl_xor_sync(0xffffffffu, l_run[h], 2);
    }
    const float inv0 = 1.0f / l_run[0], inv1 = 1.0f / l_run[1];
    const int r0 = qb * kBlock + warp * 16 + g;
#pragma unroll
    for (int dt = 0; dt < 16; ++dt) {
        int col = dt * 8 + t4 * 2;
        if (r0 < s.N)
            *reinterpret_cast<uint32_t*>(o + head + (size_t)r0 * kDh + col) =
                pack_bf16(oacc[dt][0] * inv0, oacc[dt][1] * inv0);
        if (r0 + 8 < s.N)
            *reinterpret_cast<uint32_t*>(o + head + (size_t)(r0 + 8) * kDh + col) =
                pack_bf16(oacc[dt][2] * inv1, oacc[dt][3] * inv1);
    }
}

// ===========================================================================
// fp32 validation mode: plain SIMT, one CTA per (query block, head), 256
// threads.  Shared memory: Q, K with padded rows (129 floats), V, S.

constexpr int kF32Threads = 256;
constexpr int kPad = kDh + 1;

__global__ void __launch_bounds__(kF32Threads) sparse_attn_f32_kernel(Shape s, const float* __restrict__ qr,
                                                                      const float* __restrict__ kr,
                                                                      const float* __restrict__ v,
                                                                      const int32_t* __restrict__ kv_idx,
                                                                      float* __restrict__ o)
{
    extern __shared__ float fsm[];
    float* Qs = fsm;                       // [64][129]
    float* Ks = Qs + kBlock * kPad;        // [64][129]
    float* Vs = Ks + kBlock * kPad;        // [64][128]
    float* Ss = Vs + kBlock * kDh;         // [64][65]
    const int qb = blockIdx.x, bh = blockIdx.y, tid = threadIdx.x;
    const size_t head = (size_t)bh * s.N * kDh;
    const int32_t* kept = kv_idx + ((size_t)bh * s.nB + qb) * s.n_keep;
    for (int e = tid; e < kBlock * kDh; e += kF32Threads) {
        int r = e / kDh, d = e % kDh, n = qb * kBlock + r;
        Qs[r * kPad + d] = n < s.N ? qr[head + (size_t)n * kDh + d] : 0.0f;
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
            bool ok = n >= 0 && n < s.N;
            Ks[r * kPad + d] = ok ? kr[head + (size_t)n * kDh + d] : 0.0f;
            Vs[r * kDh + d] = ok ? v[head + (size_t)n * kDh + d] : 0.0f;
        }
        __syncthreads();
        const int kvalid = s.N - j * kBlock;
        float sv[16];
        float mx = m_run;
#pragma unroll 1
        for (int c = 0; c < 16; ++c) {
            int col = quarter * 16 + c;
            float dot = 0.0f;
            for (int d = 0; d < kDh; ++d) dot = fmaf(Qs[row * kPad + d], Ks[col * kPad + d], dot);
            sv[c] = col < kvalid ? dot * scale : -INFINITY;
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
    const int n = qb * kBlock + row;
    if (n < s.N) {
        float inv = 1.0f / l_run;
#pragma unroll
        for (int i = 0; i < 32; ++i) o[head + (size_t)n * kDh + quarter + 4 * i] = acc[i] * inv;
    }
}

cudaError_t launch_sparse_attn(rola_dtype_t dt, const Shape& s, const void* qr, const void* kr, const void* v,
                               const int32_t* kv_idx, void* o_s, cudaStream_t st)
{
    dim3 grid(s.nB, s.B * s.H);
    if (dt == ROLA_BF16) {
        size_t smem = 5 * (size_t)kTileBytes;
        cudaError_t e = cudaFuncSetAttribute(sparse_attn_bf16_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)smem);
        if (e != cudaSuccess) return e;
        sparse_attn_bf16_kernel<<<grid, kAttnThreads, smem, st>>>(
            s, (const __nv_bfloat16*)qr, (const __nv_bfloat16*)kr, (const __nv_bfloat16*)v, kv_idx,
            (__nv_bfloat16*)o_s);
    } else {
        size_t smem = sizeof(float) * (2 * kBlock * kPad + kBlock * kDh + kBlock * 65 + kBlock);
        cudaError_t e = cudaFuncSetAttribute(sparse_attn_f32_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)smem);
        if (e != cudaSuccess) return e;
        sparse_attn_f32_kernel<<<grid, kF32Threads, smem, st>>>(s, (const float*)qr, (const float*)kr,
                                                                (const float*)v, kv_idx, (float*)o_s);
    }
    return cudaGetLastError();
}

}  // namespace rola
