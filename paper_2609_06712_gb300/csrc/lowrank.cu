// Low-rank branch: the fp32 summary of the validation mode (the bf16 summary
// is part of the pre-pass, prepass.cu) and readout + gated fusion (kernel 4).
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

// SiLU evaluations: IEEE exp and divide (fp32 validation mode) and the
// MUFU-based one of the bf16 readout
struct SiluIeee {
    __device__ float operator()(float x) const { return x / (1.0f + expf(-x)); }
};
struct SiluMufu {
    __device__ float operator()(float x) const { return silu(x); }
};
__device__ constexpr SiluIeee silu_ieee{};
__device__ constexpr SiluMufu silu_mufu{};

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

__device__ __forceinline__ void load_rows_async(uint32_t sbase, const __nv_bfloat16* g, int row0, int nrows,
                                                int limit, int tid, int nthreads)
{
    for (int e = tid; e < nrows * 16; e += nthreads) {
        int r = e >> 4, c = e & 15;
        int n = row0 + r;
        const __nv_bfloat16* src = g + (size_t)min(n, limit - 1) * kDh + c * 8;
        cp_async16(sbase + sw128(r, c), src, n < limit ? 16 : 0);
    }
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
            const float2 f = lowrank_pair(u0, u1, cs, s.lr_rope, silu_ieee);
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
// apply, bf16: CTA = (64-token block, head), 4 warps x 16 tokens.
//   U = Q P_q^T -> q~ = R_r SiLU(U) (registers, never stored) -> y = q~ C (MMA,
//   C in bf16) -> O^lr = y / sqrt(mean y^2 + eps_lr) -> fuse with O^s.
// Shared memory: P_q r x 256 B | C r x 256 B | Q 16 KB | O^s 16 KB, all 256-byte
// rows, swizzled.  O^s comes in and O goes out through the shared tile with
// 16-byte accesses.

template <int R>
__global__ void __launch_bounds__(128, 4) apply_bf16_kernel(Shape s, const __nv_bfloat16* __restrict__ q,
                                                         const __nv_bfloat16* __restrict__ Pq,
                                                         const __nv_bfloat16* __restrict__ Cbf,
                                                         const float* __restrict__ gate,
                                                         const __nv_bfloat16* o_s, __nv_bfloat16* o,
                                                         const float2* __restrict__ tab)
{
    extern __shared__ __align__(128) uint8_t smem[];
    constexpr int NT = R / 8;
    const int blk = blockIdx.x, bh = blockIdx.y, h = bh % s.H, b = bh / s.H;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, g = lane >> 2, t4 = lane & 3;
    const uint32_t sP = smem_u32(smem);
    const uint32_t sC = sP + R * 256;
    const uint32_t sQ = sC + R * 256;
    const uint32_t sO = sQ + kBlock * 256;
    uint8_t* o_gen = smem + 2 * R * 256 + kBlock * 256;
    const size_t head = (size_t)bh * s.N * kDh;
    load_rows_async(sP, Pq + (size_t)h * s.r * kDh, 0, R, s.r, tid, 128);     // rows past r read as zero
    load_rows_async(sC, Cbf + (size_t)bh * R * kDh, 0, R, R, tid, 128);       // rp rows, zero-padded
    load_rows_async(sQ, q + head, blk * kBlock, kBlock, s.N, tid, 128);
    load_rows_async(sO, o_s + head, blk * kBlock, kBlock, s.N, tid, 128);
    cp_async_commit();
    cp_async_wait<0>();
    __syncthreads();
    const int mi = lane >> 3;
    float u[NT][4];
#pragma unroll
    for (int a = 0; a < NT; ++a) u[a][0] = u[a][1] = u[a][2] = u[a][3] = 0.0f;
#pragma unroll
    for (int kc = 0; kc < 8; ++kc) {
        uint32_t a0, a1, a2, a3;
        ldsm_x4(sQ + sw128(warp * 16 + (lane & 7) + (mi & 1) * 8, kc * 2 + (mi >> 1)), a0, a1, a2, a3);
#pragma unroll
        for (int np = 0; np < NT / 2; ++np) {
            uint32_t b0, b1, b2, b3;
            ldsm_x4(sP + sw128(np * 16 + (mi >> 1) * 8 + (lane & 7), kc * 2 + (mi & 1)), b0, b1, b2, b3);
            mma_bf16(u[2 * np], a0, a1, a2, a3, b0, b1);
            mma_bf16(u[2 * np + 1], a0, a1, a2, a3, b2, b3);
        }
    }
    const int n_lo = blk * kBlock + warp * 16 + g, n_hi = n_lo + 8;
    const int n_lo_c = min(n_lo, s.N - 1), n_hi_c = min(n_hi, s.N - 1);
    uint32_t qf[NT][2];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
        const int m = nt * 4 + t4;
        float2 c0 = rope_cs(tab, s, n_lo_c, m), c1 = rope_cs(tab, s, n_hi_c, m);
        const float2 f0 = lowrank_pair(u[nt][0], u[nt][1], c0, s.lr_rope, silu_mufu);
        const float2 f1 = lowrank_pair(u[nt][2], u[nt][3], c1, s.lr_rope, silu_mufu);
        qf[nt][0] = pack_bf16(f0.x, f0.y);
        qf[nt][1] = pack_bf16(f1.x, f1.y);
    }
    float y[16][4];
#pragma unroll
    for (int i = 0; i < 16; ++i) y[i][0] = y[i][1] = y[i][2] = y[i][3] = 0.0f;
#pragma unroll
    for (int kc = 0; kc < R / 16; ++kc) {
#pragma unroll
        for (int dp = 0; dp < 8; ++dp) {
            uint32_t b0, b1, b2, b3;
            ldsm_x4_t(sC + sw128(kc * 16 + (mi & 1) * 8 + (lane & 7), dp * 2 + (mi >> 1)), b0, b1, b2, b3);
            mma_bf16(y[2 * dp], qf[2 * kc][0], qf[2 * kc][1], qf[2 * kc + 1][0], qf[2 * kc + 1][1], b0, b1);
            mma_bf16(y[2 * dp + 1], qf[2 * kc][0], qf[2 * kc][1], qf[2 * kc + 1][0], qf[2 * kc + 1][1], b2, b3);
        }
    }
    // per-row RMS of y and of O^s (the 4 lanes of a quad share a row); O^s stays
    // in shared memory and is read again for the fusion
    const int r_lo = warp * 16 + g, r_hi = r_lo + 8;                 // rows within the tile
    float ssy[2] = {0.0f, 0.0f}, sso[2] = {0.0f, 0.0f};
#pragma unroll
    for (int dt = 0; dt < 16; ++dt) {
        const uint32_t lo_off = sw128(r_lo, dt) + t4 * 4, hi_off = sw128(r_hi, dt) + t4 * 4;
        float2 lo = unpack_bf16(*reinterpret_cast<const uint32_t*>(o_gen + lo_off));
        float2 hi = unpack_bf16(*reinterpret_cast<const uint32_t*>(o_gen + hi_off));
        ssy[0] += y[dt][0] * y[dt][0] + y[dt][1] * y[dt][1];
        ssy[1] += y[dt][2] * y[dt][2] + y[dt][3] * y[dt][3];
        sso[0] += lo.x * lo.x + lo.y * lo.y;
        sso[1] += hi.x * hi.x + hi.y * hi.y;
    }
    float coef[2];
#pragma unroll
    for (int hr = 0; hr < 2; ++hr) {
        ssy[hr] += __shfl_xor_sync(0xffffffffu, ssy[hr], 1);
        ssy[hr] += __shfl_xor_sync(0xffffffffu, ssy[hr], 2);
        sso[hr] += __shfl_xor_sync(0xffffffffu, sso[hr], 1);
        sso[hr] += __shfl_xor_sync(0xffffffffu, sso[hr], 2);
        int n = hr ? n_hi_c : n_lo_c;
        float gp = gate ? __ldg(gate + (size_t)b * s.N + n) : s.default_gate;
        float rp = sqrtf(sso[hr] * (1.0f / kDh) + s.eps_fuse);
        coef[hr] = gp * rp * rsqrtf(ssy[hr] * (1.0f / kDh) + s.eps_lr);
    }
    // fused rows back into the shared tile (each thread rewrites what it read), then 16-byte stores
#pragma unroll
    for (int dt = 0; dt < 16; ++dt) {
        uint32_t* lo_p = reinterpret_cast<uint32_t*>(o_gen + sw128(r_lo, dt) + t4 * 4);
        uint32_t* hi_p = reinterpret_cast<uint32_t*>(o_gen + sw128(r_hi, dt) + t4 * 4);
        const float2 lo = unpack_bf16(*lo_p), hi = unpack_bf16(*hi_p);
        *lo_p = pack_bf16(lo.x + coef[0] * y[dt][0], lo.y + coef[0] * y[dt][1]);
        *hi_p = pack_bf16(hi.x + coef[1] * y[dt][2], hi.y + coef[1] * y[dt][3]);
    }
    __syncthreads();
#pragma unroll
    for (int it = 0; it < 8; ++it) {
        const int e = it * 128 + tid;
        const int row = e >> 4, c = e & 15;
        const int n = blk * kBlock + row;
        if (n < s.N)
            *reinterpret_cast<uint4*>(o + head + (size_t)n * kDh + c * 8) =
                *reinterpret_cast<const uint4*>(o_gen + sw128(row, c));
    }
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
        const float2 f = lowrank_pair(u0, u1, cs, s.lr_rope, silu_ieee);
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

template <int R>
static cudaError_t launch_apply_bf16_r(const Shape& s, const void* q, const void* P_q, const __nv_bfloat16* Cbf,
                                       const float* gate, const void* o_s, void* o, const float2* tab, cudaStream_t st)
{
    size_t smem = (size_t)R * 512 + 2 * kBlock * 256;
    cudaError_t e = cudaFuncSetAttribute(apply_bf16_kernel<R>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    apply_bf16_kernel<R><<<dim3(s.nB, s.B * s.H), 128, smem, st>>>(
        s, (const __nv_bfloat16*)q, (const __nv_bfloat16*)P_q, Cbf, gate, (const __nv_bfloat16*)o_s,
        (__nv_bfloat16*)o, tab);
    return cudaGetLastError();
}

cudaError_t launch_lowrank_apply(rola_dtype_t dt, const Shape& s, const void* q, const void* P_q, const float* C,
                                 const __nv_bfloat16* Cbf, const float* gate, const void* o_s, void* o,
                                 const float2* tab, DeviceStatus* status, cudaStream_t st)
{
    if (dt == ROLA_BF16) {
        // small r: one CTA per block, four per SM (P_q and C re-read from L2 are cheap);
        // large r: the persistent kernel, which loads P_q and C once per head
        switch (s.rp) {
            case 16: return launch_apply_bf16_r<16>(s, q, P_q, Cbf, gate, o_s, o, tab, st);
            case 32: return launch_apply_bf16_r<32>(s, q, P_q, Cbf, gate, o_s, o, tab, st);
            case 48: return launch_apply_bf16_r<48>(s, q, P_q, Cbf, gate, o_s, o, tab, st);
            default: return launch_readout(s, q, P_q, Cbf, gate, o_s, o, tab, status, st);
        }
    }
    size_t smem = sizeof(float) * ((size_t)s.r * (kDh + 1) + (size_t)s.r * kDh + kBlock * (kDh + 1) +
                                   kBlock * (s.r + 1));
    cudaError_t e = cudaFuncSetAttribute(apply_f32_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    apply_f32_kernel<<<dim3(s.nB, s.B * s.H), 256, smem, st>>>(s, (const float*)q, (const float*)P_q, C, gate,
                                                              (const float*)o_s, (float*)o, tab);
    return cudaGetLastError();
}

}  // namespace rola
