// Block mask: pooled block scores and per-query-block top-n_keep (kernel 1).
//
// The paper's sparse engine selects key blocks by a "topk ratio" (Alg. 1)
// without stating the score.  This library scores block pairs by the mean-
// pooled ROTATED vectors, s_ij = q_bar_i . k_bar_j / sqrt(d_h), keeps the
// n_keep largest per row (ties to the lower block id) and lists them
// ascending.  All score arithmetic is fp32.
#include "common.cuh"

namespace rola {

// ---------------------------------------------------------------------------
// scores[bh][i][j] = (q_bar_i . k_bar_j) / sqrt(128): fp32 SIMT GEMM, one 128 x 128
// tile per CTA, 256 threads with 8 x 8 register tiles (rows ty + 16 u, columns
// tx + 16 w), d staged through shared memory in chunks of 16, transposed and
// double-buffered: the next chunk's global loads are in flight while the
// current chunk is multiplied.  Two neighbouring columns go through one packed
// fma.rn.f32x2 (each element an IEEE fma), so every score is the same
// ascending-d fp32 FMA chain whatever the tiling.

constexpr int kSTile = 128, kSChunk = 16;

// (two CTAs per SM: the 128-register budget keeps both resident)
__global__ void __launch_bounds__(256, 2) block_scores_kernel(Shape s, const float* __restrict__ qbar,
                                                              const float* __restrict__ kbar,
                                                              float* __restrict__ scores)
{
    __shared__ __align__(16) float qs[2][kSChunk][kSTile + 4];
    __shared__ __align__(16) float ks[2][kSChunk][kSTile + 4];
    const int bh = blockIdx.z, i0 = blockIdx.y * kSTile, j0 = blockIdx.x * kSTile;
    const float* Q = qbar + (size_t)bh * s.nQ * kDh;
    const float* K = kbar + (size_t)bh * s.nB * kDh;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    // loader: 128 rows x 16 d per operand = 512 float4, two per thread
    const int lrow = threadIdx.x >> 2, lq = threadIdx.x & 3;     // rows lrow, lrow + 64; d 4*lq .. 4*lq+3
    float4 ra[2], rb[2];
    auto fetch = [&](int d0) {
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int row = lrow + 64 * h;
            const int gi = i0 + row, gj = j0 + row;
            ra[h] = gi < s.nQ ? __ldg(reinterpret_cast<const float4*>(Q + (size_t)gi * kDh + d0) + lq)
                              : make_float4(0.f, 0.f, 0.f, 0.f);
            rb[h] = gj < s.nB ? __ldg(reinterpret_cast<const float4*>(K + (size_t)gj * kDh + d0) + lq)
                              : make_float4(0.f, 0.f, 0.f, 0.f);
        }
    };
    auto stash = [&](int buf) {
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int row = lrow + 64 * h;
            qs[buf][4 * lq][row] = ra[h].x; qs[buf][4 * lq + 1][row] = ra[h].y;
            qs[buf][4 * lq + 2][row] = ra[h].z; qs[buf][4 * lq + 3][row] = ra[h].w;
            ks[buf][4 * lq][row] = rb[h].x; ks[buf][4 * lq + 1][row] = rb[h].y;
            ks[buf][4 * lq + 2][row] = rb[h].z; ks[buf][4 * lq + 3][row] = rb[h].w;
        }
    };
    float acc[8][8] = {};
    fetch(0);
    stash(0);
    __syncthreads();
#pragma unroll 1
    for (int c = 0; c < kDh / kSChunk; ++c) {
        const int buf = c & 1;
        if (c + 1 < kDh / kSChunk) fetch((c + 1) * kSChunk);
#pragma unroll
        for (int d = 0; d < kSChunk; ++d) {
            const float4 a0 = *reinterpret_cast<const float4*>(&qs[buf][d][ty * 4]);
            const float4 a1 = *reinterpret_cast<const float4*>(&qs[buf][d][64 + ty * 4]);
            const float4 b0 = *reinterpret_cast<const float4*>(&ks[buf][d][tx * 4]);
            const float4 b1 = *reinterpret_cast<const float4*>(&ks[buf][d][64 + tx * 4]);
            const float av[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
            const float bv[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
            for (int u = 0; u < 8; ++u)
#pragma unroll
                for (int w = 0; w < 8; w += 2)
                    asm("{\n.reg .b64 ra, rb, rc;\n"
                        "mov.b64 ra, {%2, %2};\n"
                        "mov.b64 rb, {%3, %4};\n"
                        "mov.b64 rc, {%0, %1};\n"
                        "fma.rn.f32x2 rc, ra, rb, rc;\n"
                        "mov.b64 {%0, %1}, rc;\n}\n"
                        : "+f"(acc[u][w]), "+f"(acc[u][w + 1])
                        : "f"(av[u]), "f"(bv[w]), "f"(bv[w + 1]));
        }
        // the other buffer was last read in chunk c - 1, before the previous barrier
        if (c + 1 < kDh / kSChunk) stash(buf ^ 1);
        __syncthreads();
    }
    const float scale = 0.08838834764831845f;   // 1 / sqrt(128)
#pragma unroll
    for (int u = 0; u < 8; ++u) {
        const int gi = i0 + (u < 4 ? ty * 4 + u : 64 + ty * 4 + u - 4);
        if (gi >= s.nQ) continue;
        float* out = scores + ((size_t)bh * s.nQ + gi) * s.nB;
#pragma unroll
        for (int w = 0; w < 8; ++w) {
            const int gj = j0 + (w < 4 ? tx * 4 + w : 64 + tx * 4 + w - 4);
            if (gj < s.nB) out[gj] = acc[u][w] * scale;
        }
    }
}

// ---------------------------------------------------------------------------
// top-n_keep of each score row: one warp per row, 8 rows per CTA.  The row is
// mapped to order-preserving unsigned keys (+0 and -0 identified) and the
// n_keep-th largest key is found by a 4-pass 8-bit radix select over a
// per-warp histogram; the row is then scanned in ascending block order,
// taking every key above the threshold and the lowest-index keys equal to it.

__device__ __forceinline__ uint32_t order_key(float f)
{
    uint32_t u = __float_as_uint(f == 0.0f ? 0.0f : f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

constexpr int kTopkWarps = 8;

__global__ void __launch_bounds__(kTopkWarps * 32) block_topk_kernel(Shape s, const float* __restrict__ scores,
                                                                     int32_t* __restrict__ kv_idx)
{
    extern __shared__ uint32_t tk_smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    uint32_t* hist = tk_smem + warp * 256;
    uint32_t* keys = tk_smem + kTopkWarps * 256 + (size_t)warp * s.nB;
    const int row = blockIdx.x * kTopkWarps + warp;
    const int bh = blockIdx.y;
    if (row >= s.nQ) return;
    const float* srow = scores + ((size_t)bh * s.nQ + row) * s.nB;
    for (int j = lane; j < s.nB; j += 32) keys[j] = order_key(srow[j]);
    __syncwarp();

    uint32_t prefix = 0, pmask = 0;
    int need = s.n_keep;             // how many keys >= threshold are still to be placed
#pragma unroll 1
    for (int shift = 24; shift >= 0; shift -= 8) {
        for (int b = lane; b < 256; b += 32) hist[b] = 0;
        __syncwarp();
        for (int j = lane; j < s.nB; j += 32) {
            uint32_t key = keys[j];
            if ((key & pmask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1u);
        }
        __syncwarp();
        // lane owns bins 8*(31-lane) .. 8*(31-lane)+7 so that lane 0 holds the top bins
        int base = 8 * (31 - lane);
        uint32_t c[8];
        uint32_t tot = 0;
#pragma unroll
        for (int t = 0; t < 8; ++t) { c[t] = hist[base + t]; tot += c[t]; }
        // inclusive prefix over lanes (from the top bins down)
        uint32_t incl = tot;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += y;
        }
        uint32_t excl = incl - tot;
        // the lane whose range holds the need-th key from the top
        bool mine = excl < (uint32_t)need && incl >= (uint32_t)need;
        uint32_t ballot = __ballot_sync(0xffffffffu, mine);
        int src = ballot ? __ffs(ballot) - 1 : 0;
        int bin = 0, above = 0;
        if (lane == src) {
            uint32_t run = excl;
            for (int t = 7; t >= 0; --t) {
                if (run + c[t] >= (uint32_t)need) { bin = base + t; above = (int)run; break; }
                run += c[t];
            }
        }
        bin = __shfl_sync(0xffffffffu, bin, src);
        above = __shfl_sync(0xffffffffu, above, src);
        need -= above;
        prefix |= (uint32_t)bin << shift;
        pmask |= 255u << shift;
        __syncwarp();
    }
    // prefix is now the threshold key; `need` keys equal to it are kept (lowest j first)
    const uint32_t thr = prefix;
    int32_t* out = kv_idx + ((size_t)bh * s.nQ + row) * s.n_keep;
    int written = 0, eq_taken = 0;
    for (int j0 = 0; j0 < s.nB; j0 += 32) {
        int j = j0 + lane;
        uint32_t key = j < s.nB ? keys[j] : 0u;
        bool gt = j < s.nB && key > thr;
        bool eq = j < s.nB && key == thr;
        uint32_t eqb = __ballot_sync(0xffffffffu, eq);
        int eq_rank = eq_taken + __popc(eqb & ((1u << lane) - 1u));
        bool sel = gt || (eq && eq_rank < need);
        uint32_t selb = __ballot_sync(0xffffffffu, sel);
        int pos = written + __popc(selb & ((1u << lane) - 1u));
        if (sel && pos < s.n_keep) out[pos] = j;
        written += __popc(selb);
        eq_taken += __popc(eqb);
    }
}

cudaError_t launch_block_topk(const Shape& s, const float* qbar, const float* kbar, float* scores,
                              int32_t* kv_idx, cudaStream_t st)
{
    const int tj = (s.nB + kSTile - 1) / kSTile, ti = (s.nQ + kSTile - 1) / kSTile;
    block_scores_kernel<<<dim3(tj, ti, s.B * s.H), 256, 0, st>>>(s, qbar, kbar, scores);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    size_t smem = (size_t)kTopkWarps * 256 * 4 + (size_t)kTopkWarps * s.nB * 4;
    if (smem > 48 * 1024) {
        e = cudaFuncSetAttribute(block_topk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
    }
    dim3 grid((s.nQ + kTopkWarps - 1) / kTopkWarps, s.B * s.H);
    block_topk_kernel<<<grid, kTopkWarps * 32, smem, st>>>(s, scores, kv_idx);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// 128-token query means: the 64-token chunks' fp32 q sums S (each the pairwise
// tree over its 64 slots) give chunk c of 128 tokens the tree's top node
// S[2c] + S[2c+1] (an absent right half is the empty tree, +0), divided once by
// the chunk's token count -- the pairwise sum over 128 slots.
__global__ void qpool128_kernel(Shape s, const float* __restrict__ qsum, float* __restrict__ qbar)
{
    const int c = blockIdx.x, bh = blockIdx.y, d = threadIdx.x;
    const float* src = qsum + ((size_t)bh * s.nB + 2 * c) * kDh + d;
    const float right = 2 * c + 1 < s.nB ? src[kDh] : 0.0f;
    const int cnt = min(128, s.N - 128 * c);
    qbar[((size_t)bh * s.nQ + c) * kDh + d] = (src[0] + right) / (float)cnt;
}

cudaError_t launch_qpool128(const Shape& s, const float* qsum64, float* qbar128, cudaStream_t st)
{
    qpool128_kernel<<<dim3(s.nQ, s.B * s.H), kDh, 0, st>>>(s, qsum64, qbar128);
    return cudaGetLastError();
}

}  // namespace rola
