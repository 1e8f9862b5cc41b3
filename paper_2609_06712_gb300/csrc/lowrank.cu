// Low-rank branch of the fp32 validation mode: the summary (kernel 3) and the
// readout + gated fusion (kernel 4).  The bf16 path has them in prepass.cu and
// readout.cu.
//
// Eq. (qklr):  k~_q = R_r(q) SiLU(P_k k^n_q),   q~_p = R_r(p) SiLU(P_q q^n_p)
// Eq. (ctx):   C = sum_q k~_q v_q^T,            O^lr_p = RMSNorm(q~_p^T C)   (no gain)
// Eq. (gate):  r_p = sqrt(mean_i O^s_{p,i}^2 + eps),  O_p = (O^s_p / r_p + g_p O^lr_p) r_p
//
// R_r keeps the first r/2 rotary pairs of the native ordering (Sec. 4.2).  The
// fusion is evaluated as O^s_p + g_p r_p O^lr_p, which is the same expression
// with one rounding fewer.  The fp32 summary reduction over N is split across
// CTAs; each writes an fp32 partial to the workspace and a second kernel adds
// the partials in split order, so C is bitwise reproducible run to run.
#include "common.cuh"

namespace rola {

// The feature map in the fp32 validation mode: SiLU with the IEEE exp and
// divide, or one of the ablation's activations.
struct ActIeee {
    int kind;
    __device__ float operator()(float x) const
    {
        return kind == ROLA_LOWRANK_ACT_SILU ? x / (1.0f + expf(-x)) : ActAblation{kind}(x);
    }
};

// ===========================================================================
// Split-N partitioning of the fp32 summary: CTA = (split, head).

constexpr int kSumTile = 128;

int summary_splits(const Shape& s)
{
    int bh = s.B * s.H;
    int tiles = (s.N + kSumTile - 1) / kSumTile;
    int want = (4 * 152 + bh - 1) / bh;
    int per = (tiles + want - 1) / want;
    if (per < 1) per = 1;
    return (tiles + per - 1) / per;
}


// ===========================================================================
// summary, fp32 validation mode: CTA = (split, head), 256 threads, 64-token tiles.

constexpr int kF32Tile = 64;

__global__ void __launch_bounds__(256) summary_f32_kernel(Shape s, int tokens_per_split, const float* __restrict__ k,
                                                          const float* __restrict__ v, const float* __restrict__ Pk,
                                                          const float2* __restrict__ tab, float* __restrict__ partials)
{
    extern __shared__ float fsm[];
    const int R = s.r;
    float* Ps = fsm;                           // [R][129]
    float* Ks = Ps + R * (kDh + 1);            // [64][129]
    float* Vs = Ks + kF32Tile * (kDh + 1);     // [64][128]
    float* Us = Vs + kF32Tile * kDh;           // [64][R+1]
    const int split = blockIdx.x, bh = blockIdx.y, h = bh % s.H, tid = threadIdx.x;
    const size_t head = (size_t)bh * s.N * kDh;
    const int n_begin = split * tokens_per_split;
    const int n_end = min(s.N, n_begin + tokens_per_split);
    for (int e = tid; e < R * kDh; e += 256) Ps[(e / kDh) * (kDh + 1) + e % kDh] = Pk[(size_t)h * R * kDh + e];
    const int d = tid & 127, ahalf = tid >> 7;          // C[a][d] for a in this thread's half
    const int a0 = ahalf * (R / 2);
    float acc[64];
    float zacc = 0.0f;
#pragma unroll
    for (int i = 0; i < 64; ++i) acc[i] = 0.0f;
    for (int n0 = n_begin; n0 < n_end; n0 += kF32Tile) {
        __syncthreads();
        for (int e = tid; e < kF32Tile * kDh; e += 256) {
            int r = e / kDh, c = e % kDh, n = n0 + r;
            bool ok = n < n_end;
            Ks[r * (kDh + 1) + c] = ok ? k[head + (size_t)n * kDh + c] : 0.0f;
            Vs[r * kDh + c] = ok ? v[head + (size_t)n * kDh + c] : 0.0f;
        }
        __syncthreads();
        for (int e = tid; e < kF32Tile * (R / 2); e += 256) {
            int r = e / (R / 2), m = e % (R / 2), n = n0 + r;
            float u0 = 0.0f, u1 = 0.0f;
            for (int c = 0; c < kDh; ++c) {
                u0 = fmaf(Ks[r * (kDh + 1) + c], Ps[(2 * m) * (kDh + 1) + c], u0);
                u1 = fmaf(Ks[r * (kDh + 1) + c], Ps[(2 * m + 1) * (kDh + 1) + c], u1);
            }
            float2 cs = n < n_end ? rope_cs(tab, s, n, m) : make_float2(0.0f, 0.0f);
            const float2 f = lowrank_pair(u0, u1, cs, s.lr_rope, ActIeee{s.lr_act});
            Us[r * (R + 1) + 2 * m] = f.x;
            Us[r * (R + 1) + 2 * m + 1] = f.y;
        }
        __syncthreads();
        for (int r = 0; r < kF32Tile; ++r) {
            float vv = Vs[r * kDh + d];
#pragma unroll
            for (int i = 0; i < 64; ++i)
                if (i < R / 2) acc[i] = fmaf(Us[r * (R + 1) + a0 + i], vv, acc[i]);
        }
        if (tid < R)
            for (int r = 0; r < kF32Tile; ++r) zacc += Us[r * (R + 1) + tid];
    }
    float* part = partials + ((size_t)bh * gridDim.x + split) * (size_t)(R * kDh + R);
#pragma unroll
    for (int i = 0; i < 64; ++i)
        if (i < R / 2) part[(size_t)(a0 + i) * kDh + d] = acc[i];
    if (tid < R) part[(size_t)R * kDh + tid] = zacc;
}

// ===========================================================================
// fixed-order combine of the split partials -> C (fp32), z, and a bf16 copy of C

__global__ void summary_combine_kernel(Shape s, int nsplit, const float* __restrict__ partials, float* __restrict__ C,
                                       float* __restrict__ z, __nv_bfloat16* __restrict__ Cbf)
{
    const int bh = blockIdx.y;
    const int per = s.r * kDh + s.r;
    const int e = blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= per) return;
    const float* p = partials + (size_t)bh * nsplit * per + e;
    float x = 0.0f;
    for (int sp = 0; sp < nsplit; ++sp) x += p[(size_t)sp * per];
    if (e < s.r * kDh) {
        C[(size_t)bh * s.r * kDh + e] = x;
        if (Cbf) Cbf[(size_t)bh * s.r * kDh + e] = __float2bfloat16_rn(x);
    } else if (z) {
        z[(size_t)bh * s.r + (e - s.r * kDh)] = x;
    }
}

// C [B*H][r][128] fp32 -> bf16 [B*H][rp][128], rows r .. rp-1 zero
__global__ void c_to_bf16_kernel(int r, int rp, int n, const float* __restrict__ C, __nv_bfloat16* __restrict__ Cbf)
{
    const int e = blockIdx.x * blockDim.x + threadIdx.x;     // index into the padded copy
    if (e >= n) return;
    const int bh = e / (rp * kDh), rest = e - bh * rp * kDh, row = rest / kDh;
    Cbf[e] = row < r ? __float2bfloat16_rn(C[((size_t)bh * r) * kDh + rest]) : __float2bfloat16_rn(0.0f);
}

cudaError_t launch_c_to_bf16(const Shape& s, const float* C, __nv_bfloat16* Cbf, cudaStream_t st)
{
    int n = s.B * s.H * s.rp * kDh;
    c_to_bf16_kernel<<<(n + 255) / 256, 256, 0, st>>>(s.r, s.rp, n, C, Cbf);
    return cudaGetLastError();
}

cudaError_t launch_lowrank_summary(rola_dtype_t dt, const Shape& s, int nsplit, const void* k, const void* v,
                                   const void* P_k, const float2* tab, float* partials, float* C, float* z,
                                   __nv_bfloat16* Cbf, cudaStream_t st)
{
    if (dt != ROLA_FP32) return cudaErrorInvalidValue;      // bf16: launch_prepass
    int tiles = (s.N + kSumTile - 1) / kSumTile;
    int tps = ((tiles + nsplit - 1) / nsplit) * kSumTile;
    size_t smem = sizeof(float) * ((size_t)s.r * (kDh + 1) + kF32Tile * (kDh + 1) + kF32Tile * kDh +
                                   kF32Tile * (s.r + 1));
    cudaError_t e = cudaFuncSetAttribute(summary_f32_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    summary_f32_kernel<<<dim3(nsplit, s.B * s.H), 256, smem, st>>>(s, tps, (const float*)k, (const float*)v,
                                                                    (const float*)P_k, tab, partials);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    int per = s.r * kDh + s.r;
    summary_combine_kernel<<<dim3((per + 255) / 256, s.B * s.H), 256, 0, st>>>(s, nsplit, partials, C, z, Cbf);
    return cudaGetLastError();
}

// ===========================================================================
// apply, fp32 validation mode: CTA = (64-token block, head), 256 threads.

__global__ void __launch_bounds__(256) apply_f32_kernel(Shape s, const float* __restrict__ q,
                                                        const float* __restrict__ Pq, const float* __restrict__ C,
                                                        const float* __restrict__ gate, const float* o_s, float* o,
                                                        const float2* __restrict__ tab)
{
    extern __shared__ float fsm[];
    const int R = s.r;
    float* Ps = fsm;                        // [R][129]
    float* Cs = Ps + R * (kDh + 1);         // [R][128]
    float* Qs = Cs + R * kDh;               // [64][129]
    float* Us = Qs + kBlock * (kDh + 1);    // [64][R+1]
    const int blk = blockIdx.x, bh = blockIdx.y, h = bh % s.H, b = bh / s.H, tid = threadIdx.x;
    const size_t head = (size_t)bh * s.N * kDh;
    for (int e = tid; e < R * kDh; e += 256) {
        Ps[(e / kDh) * (kDh + 1) + e % kDh] = Pq[(size_t)h * R * kDh + e];
        Cs[e] = C[(size_t)bh * R * kDh + e];
    }
    for (int e = tid; e < kBlock * kDh; e += 256) {
        int r = e / kDh, c = e % kDh, n = blk * kBlock + r;
        Qs[r * (kDh + 1) + c] = n < s.N ? q[head + (size_t)n * kDh + c] : 0.0f;
    }
    __syncthreads();
    for (int e = tid; e < kBlock * (R / 2); e += 256) {
        int r = e / (R / 2), m = e % (R / 2), n = min(blk * kBlock + r, s.N - 1);
        float u0 = 0.0f, u1 = 0.0f;
        for (int c = 0; c < kDh; ++c) {
            u0 = fmaf(Qs[r * (kDh + 1) + c], Ps[(2 * m) * (kDh + 1) + c], u0);
            u1 = fmaf(Qs[r * (kDh + 1) + c], Ps[(2 * m + 1) * (kDh + 1) + c], u1);
        }
        float2 cs = rope_cs(tab, s, n, m);
        const float2 f = lowrank_pair(u0, u1, cs, s.lr_rope, ActIeee{s.lr_act});
        Us[r * (R + 1) + 2 * m] = f.x;
        Us[r * (R + 1) + 2 * m + 1] = f.y;
    }
    __syncthreads();
    const int row = tid >> 2, quarter = tid & 3;
    const int n = blk * kBlock + row, nc = min(n, s.N - 1);
    float y[32], os[32];
    float ssy = 0.0f, sso = 0.0f;
#pragma unroll
    for (int i = 0; i < 32; ++i) {
        int d = quarter + 4 * i;
        float acc = 0.0f;
        for (int a = 0; a < R; ++a) acc = fmaf(Us[row * (R + 1) + a], Cs[a * kDh + d], acc);
        y[i] = acc;
        os[i] = o_s[head + (size_t)nc * kDh + d];
        ssy += acc * acc;
        sso += os[i] * os[i];
    }
    ssy += __shfl_xor_sync(0xffffffffu, ssy, 1);
    ssy += __shfl_xor_sync(0xffffffffu, ssy, 2);
    sso += __shfl_xor_sync(0xffffffffu, sso, 1);
    sso += __shfl_xor_sync(0xffffffffu, sso, 2);
    float gp = gate ? gate[(size_t)b * s.N + nc] : s.default_gate;
    float rp = sqrtf(sso / kDh + s.eps_fuse);
    float coef = gp * rp / sqrtf(ssy / kDh + s.eps_lr);
    __syncthreads();   // every thread has read its O^s before any (possibly aliased) write
    if (n < s.N)
#pragma unroll
        for (int i = 0; i < 32; ++i) o[head + (size_t)n * kDh + quarter + 4 * i] = os[i] + coef * y[i];
}

cudaError_t launch_lowrank_apply(rola_dtype_t dt, const Shape& s, const void* q, const void* P_q, const float* C,
                                 const __nv_bfloat16* Cbf, const float* gate, const void* o_s, void* o,
                                 const float2* tab, DeviceStatus* status, cudaStream_t st)
{
    if (dt == ROLA_BF16) return launch_readout(s, q, P_q, Cbf, gate, o_s, o, tab, status, st);
    size_t smem = sizeof(float) * ((size_t)s.r * (kDh + 1) + (size_t)s.r * kDh + kBlock * (kDh + 1) +
                                   kBlock * (s.r + 1));
    cudaError_t e = cudaFuncSetAttribute(apply_f32_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    apply_f32_kernel<<<dim3(s.nC, s.B * s.H), 256, smem, st>>>(s, (const float*)q, (const float*)P_q, C, gate,
                                                              (const float*)o_s, (float*)o, tab);
    return cudaGetLastError();
}

}  // namespace rola
