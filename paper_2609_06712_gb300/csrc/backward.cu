// Backward pass of the module: the gradients the single-stage fine-tune needs
// (Sec. impl, post-training: the backbone's q, k, v and the new P_q, P_k and
// gate are all trained).  Each kernel undoes forward steps in reverse order:
//
//   fusion     O = O^s + g r_p O^lr,  r_p = sqrt(mean (O^s)^2 + eps_f)     Eq. (gate)
//              dO^s = dO + g (O^lr . dO) O^s / (d r_p),  dg_p = r_p (O^lr . dO)
//   readout    O^lr = y / rho,  y = q~^T C                                  Eq. (ctx)
//              dy = (dO^lr - O^lr (O^lr . dO^lr) / d) / rho,  dq~ = C dy,  dC += q~ dy^T
//   features   q~ = R_r phi(P_q q) (or the placement / map cfg selects)     Eq. (qklr)
//              du = phi'(u) R_r^T dq~,  dq += P_q^T du,  dP_q += du q^T
//   summary    C = sum_j k~_j v_j^T:  dk~_j = dC v_j,  dv_j += dC^T k~_j    Eq. (ctx)
//   sparse     P = softmax(q^r k^r / sqrt d) over the kept blocks, O^s = P v
//              dS = P (dO^s v^T - D),  D_p = dO^s_p . O^s_p,
//              dq^r = dS k^r / sqrt d,  dk^r = dS^T q^r / sqrt d,  dv += P^T dO^s
//   RoPE       dq += R(p)^T dq^r,  dk += R(p)^T dk^r                        Sec. 3
//
// bf16: the low-rank gradients run on mma.sync (this file) and the sparse ones
// on tcgen05 (sparse_bwd_tc.cu), with fp32 accumulation; the fp32 validation
// mode runs fp32 SIMT kernels throughout (this file).  The low-rank parts of
// dq, dk, dv are fp32 workspace rows that the sparse kernels' epilogues add
// before the single conversion to the storage type.  Reductions over tokens
// (dC, dP_q, dP_k) go through per-chunk partials summed in a fixed order, and
// the key-side sparse gradients walk, for each key block, the query blocks
// that kept it in ascending order, so results are bitwise reproducible.
#include <type_traits>

#include "common.cuh"

namespace rola {
namespace {

constexpr int kBT = 256;                   // threads of the per-block kernels
constexpr int kLd = kDh + 1;               // padded fp32 row of a 128-wide tile

__device__ __forceinline__ float to_f(float x) { return x; }
__device__ __forceinline__ float to_f(__nv_bfloat16 x) { return __bfloat162float(x); }
template <typename T>
__device__ __forceinline__ T from_f(float x);
template <>
__device__ __forceinline__ float from_f<float>(float x) { return x; }
template <>
__device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float x) { return __float2bfloat16_rn(x); }

// The feature map in the backward pass: phi (IEEE evaluations) and phi'.
struct ActBwd {
    int kind;
    __device__ float operator()(float x) const
    {
        return kind == ROLA_LOWRANK_ACT_SILU ? x / (1.0f + expf(-x)) : ActAblation{kind}(x);
    }
    __device__ float grad(float x) const
    {
        switch (kind) {
            case ROLA_LOWRANK_ACT_IDENTITY: return 1.0f;
            case ROLA_LOWRANK_ACT_TANH: {
                const float t = tanhf(x);
                return 1.0f - t * t;
            }
            case ROLA_LOWRANK_ACT_RELU: return x > 0.0f ? 1.0f : 0.0f;
            case ROLA_LOWRANK_ACT_GELU:    // Phi(x) + x Phi'(x), Phi' the standard normal density
                return 0.5f * (1.0f + erff(x * 0.7071067811865476f)) + x * expf(-0.5f * x * x) * 0.3989422804014327f;
            default: {
                const float sg = 1.0f / (1.0f + expf(-x));
                return sg * (1.0f + x * (1.0f - sg));
            }
        }
    }
};

// R^T on one pair: rotation by the opposite angle.
__device__ __forceinline__ float2 rope_rotate_t(float x0, float x1, float2 cs)
{
    return make_float2(__fmaf_rn(x0, cs.x, __fmul_rn(x1, cs.y)), __fmaf_rn(x1, cs.x, -__fmul_rn(x0, cs.y)));
}

// Backward of one pair of low-rank features: (u0, u1) = the pair's rows of P x,
// (g0, g1) = dL/d(feature pair) -> dL/d(u0, u1), for the placement `mode`.
__device__ __forceinline__ float2 lowrank_pair_bwd(float u0, float u1, float g0, float g1, float2 cs, int mode,
                                                   ActBwd act)
{
    if (mode == ROLA_LOWRANK_ROPE_INSIDE) {          // f = phi(R u): du = R^T (phi'(R u) df)
        const float2 w = rope_rotate(u0, u1, cs);
        return rope_rotate_t(act.grad(w.x) * g0, act.grad(w.y) * g1, cs);
    }
    if (mode == ROLA_LOWRANK_ROPE_NONE) return make_float2(act.grad(u0) * g0, act.grad(u1) * g1);
    const float2 d = rope_rotate_t(g0, g1, cs);      // f = R phi(u): du = phi'(u) R^T df
    return make_float2(act.grad(u0) * d.x, act.grad(u1) * d.y);
}

// ---------------------------------------------------------------------------
// Low-rank branch, query side: one CTA per (64-token chunk, head).  Shared
// memory (fp32): X [64][129] q rows, Y [64][129] dy rows, F and G [64][r+1]
// (features, then u / du), W [r][129] (P_q, then C, then P_q).  A thread owns
// row t = tid / 4 and the columns quarter + 4 i of 128-wide rows, or the
// columns quarter + 4 i of r-wide rows.

struct LrSmem {
    float* X;
    float* Y;
    float* F;
    float* G;
    float* W;
    int rl;     // r + 1
};

__device__ __forceinline__ LrSmem lr_smem(float* base, int r)
{
    LrSmem m;
    m.rl = r + 1;
    m.X = base;
    m.Y = m.X + 64 * kLd;
    m.F = m.Y + 64 * kLd;
    m.G = m.F + 64 * m.rl;
    m.W = m.G + 64 * m.rl;
    return m;
}

size_t lr_smem_bytes(int r) { return sizeof(float) * (2 * 64 * kLd + 2 * 64 * (r + 1) + (size_t)r * kLd); }

template <typename T>
__device__ void load_rows(float* dst, const T* src, int n0, int N)
{
    for (int e = threadIdx.x; e < 64 * kDh; e += kBT) {
        const int t = e / kDh, d = e - t * kDh;
        dst[t * kLd + d] = n0 + t < N ? to_f(src[(size_t)(n0 + t) * kDh + d]) : 0.0f;
    }
}

template <typename T>
__device__ void load_weight(float* W, const T* src, int r)
{
    for (int e = threadIdx.x; e < r * kDh; e += kBT) {
        const int a = e / kDh, d = e - a * kDh;
        W[a * kLd + d] = to_f(src[e]);
    }
}

// U = X W^T (u[t][a] = sum_d X[t][d] W[a][d]) into G, then the features into F.
__device__ void features_fwd(const Shape& s, const LrSmem& m, const float2* tab, int n0, ActBwd act)
{
    const int t = threadIdx.x >> 2, quarter = threadIdx.x & 3;
    for (int a = quarter; a < s.r; a += 4) {
        float acc = 0.0f;
        for (int d = 0; d < kDh; ++d) acc = fmaf(m.X[t * kLd + d], m.W[a * kLd + d], acc);
        m.G[t * m.rl + a] = acc;
    }
    __syncthreads();
    for (int e = threadIdx.x; e < 64 * (s.r / 2); e += kBT) {
        const int tt = e / (s.r / 2), pm = e - tt * (s.r / 2);
        const int n = n0 + tt;
        float2 f = make_float2(0.0f, 0.0f);
        if (n < s.N) f = lowrank_pair(m.G[tt * m.rl + 2 * pm], m.G[tt * m.rl + 2 * pm + 1], rope_cs(tab, s, n, pm),
                                      s.lr_rope, act);
        m.F[tt * m.rl + 2 * pm] = f.x;
        m.F[tt * m.rl + 2 * pm + 1] = f.y;
    }
    __syncthreads();
}

// du from df (held by this thread for columns quarter + 4 i) and u (in G);
// the pair partner column is held by the neighbouring lane (quarter ^ 1).
// Writes du over u in G.
__device__ void features_bwd(const Shape& s, const LrSmem& m, const float2* tab, int n0, ActBwd act,
                             const float* df)
{
    const int t = threadIdx.x >> 2, quarter = threadIdx.x & 3;
    const int n = n0 + t;
    float du[kDh / 4];
#pragma unroll
    for (int i = 0; i < kDh / 4; ++i) {
        const int a = quarter + 4 * i;
        const float other = __shfl_xor_sync(0xffffffffu, df[i], 1);
        du[i] = 0.0f;
        if (a < s.r && n < s.N) {
            const int a0 = a & ~1;
            const float g0 = (a & 1) ? other : df[i], g1 = (a & 1) ? df[i] : other;
            const float2 d = lowrank_pair_bwd(m.G[t * m.rl + a0], m.G[t * m.rl + a0 + 1], g0, g1,
                                              rope_cs(tab, s, n, a0 >> 1), s.lr_rope, act);
            du[i] = (a & 1) ? d.y : d.x;
        }
    }
    __syncthreads();
#pragma unroll
    for (int i = 0; i < kDh / 4; ++i) {
        const int a = quarter + 4 * i;
        if (a < s.r) m.G[t * m.rl + a] = du[i];
    }
    __syncthreads();
}

// part[a][d] = sum_t A[t][a] B[t][d] over the chunk's 64 rows (A r-wide, B 128-wide).
__device__ void chunk_outer(const Shape& s, const float* A, int lda, const float* B, float* part)
{
    const int d = threadIdx.x & (kDh - 1);
    for (int a = threadIdx.x >> 7; a < s.r; a += kBT / kDh) {
        float acc = 0.0f;
        for (int t = 0; t < 64; ++t) acc = fmaf(A[t * lda + a], B[t * kLd + d], acc);
        part[(size_t)a * kDh + d] = acc;
    }
}

template <typename T>
__global__ void __launch_bounds__(kBT) lr_bwd_q_kernel(Shape s, const T* __restrict__ q, const T* __restrict__ Pq,
                                                       const float* __restrict__ C, const float* __restrict__ gate,
                                                       const T* __restrict__ o_s, const T* __restrict__ dO,
                                                       const float2* __restrict__ tab, T* __restrict__ dOs,
                                                       float* __restrict__ Dv, float* __restrict__ dq_acc,
                                                       float* __restrict__ dg_h, float* __restrict__ partC,
                                                       float* __restrict__ partPq)
{
    extern __shared__ float lsm[];
    const LrSmem m = lr_smem(lsm, s.r);
    const int chunk = blockIdx.x, bh = blockIdx.y, h = bh % s.H, b = bh / s.H;
    const int n0 = chunk * 64;
    const int t = threadIdx.x >> 2, quarter = threadIdx.x & 3;
    const int n = n0 + t;
    const size_t head = (size_t)bh * s.N * kDh;
    const ActBwd act{s.lr_act};
    load_rows(m.X, q + head, n0, s.N);
    load_weight(m.W, Pq + (size_t)h * s.r * kDh, s.r);
    __syncthreads();
    features_fwd(s, m, tab, n0, act);
    // W <- C of this head
    for (int e = threadIdx.x; e < s.r * kDh; e += kBT) m.W[(e / kDh) * kLd + e % kDh] = C[(size_t)bh * s.r * kDh + e];
    __syncthreads();
    // y, then the fusion and RMSNorm backward per row (4 threads per row)
    float y[32], os[32], go[32];
    float syy = 0.0f, sos = 0.0f;
#pragma unroll
    for (int i = 0; i < 32; ++i) {
        const int d = quarter + 4 * i;
        float acc = 0.0f;
        for (int a = 0; a < s.r; ++a) acc = fmaf(m.F[t * m.rl + a], m.W[a * kLd + d], acc);
        y[i] = acc;
        os[i] = n < s.N ? to_f(o_s[head + (size_t)n * kDh + d]) : 0.0f;
        go[i] = n < s.N ? to_f(dO[head + (size_t)n * kDh + d]) : 0.0f;
        syy = fmaf(acc, acc, syy);
        sos = fmaf(os[i], os[i], sos);
    }
    syy += __shfl_xor_sync(0xffffffffu, syy, 1);
    syy += __shfl_xor_sync(0xffffffffu, syy, 2);
    sos += __shfl_xor_sync(0xffffffffu, sos, 1);
    sos += __shfl_xor_sync(0xffffffffu, sos, 2);
    const float rho = sqrtf(syy / (float)kDh + s.eps_lr), irho = 1.0f / rho;
    const float rp = sqrtf(sos / (float)kDh + s.eps_fuse);
    const float g = n < s.N ? (gate ? gate[(size_t)b * s.N + n] : s.default_gate) : 0.0f;
    float a_dot = 0.0f;
#pragma unroll
    for (int i = 0; i < 32; ++i) a_dot = fmaf(y[i] * irho, go[i], a_dot);
    a_dot += __shfl_xor_sync(0xffffffffu, a_dot, 1);
    a_dot += __shfl_xor_sync(0xffffffffu, a_dot, 2);
    const float coef = g * a_dot / ((float)kDh * rp);
    float dsum = 0.0f, od = 0.0f;
#pragma unroll
    for (int i = 0; i < 32; ++i) {
        const float gs = fmaf(coef, os[i], go[i]);           // dL/dO^s
        if (n < s.N) dOs[head + (size_t)n * kDh + quarter + 4 * i] = from_f<T>(gs);
        dsum = fmaf(gs, os[i], dsum);
        od = fmaf(y[i] * irho, g * rp * go[i], od);
    }
    dsum += __shfl_xor_sync(0xffffffffu, dsum, 1);
    dsum += __shfl_xor_sync(0xffffffffu, dsum, 2);
    od += __shfl_xor_sync(0xffffffffu, od, 1);
    od += __shfl_xor_sync(0xffffffffu, od, 2);
    if (quarter == 0 && n < s.N) {
        Dv[(size_t)bh * s.N + n] = dsum;
        dg_h[(size_t)bh * s.N + n] = rp * a_dot;
    }
#pragma unroll
    for (int i = 0; i < 32; ++i)
        m.Y[t * kLd + quarter + 4 * i] = n < s.N ? (g * rp * go[i] - y[i] * irho * od / (float)kDh) * irho : 0.0f;
    __syncthreads();
    // dq~ = C dy (columns quarter + 4 i of the r features), then du
    float df[kDh / 4];
#pragma unroll
    for (int i = 0; i < kDh / 4; ++i) {
        const int a = quarter + 4 * i;
        float acc = 0.0f;
        if (a < s.r)
            for (int d = 0; d < kDh; ++d) acc = fmaf(m.Y[t * kLd + d], m.W[a * kLd + d], acc);
        df[i] = acc;
    }
    features_bwd(s, m, tab, n0, act, df);
    // dC partial = F^T dY, dP_q partial = dU^T X
    const size_t slot = ((size_t)bh * s.nC + chunk) * s.r * kDh;
    chunk_outer(s, m.F, m.rl, m.Y, partC + slot);
    chunk_outer(s, m.G, m.rl, m.X, partPq + slot);
    __syncthreads();
    load_weight(m.W, Pq + (size_t)h * s.r * kDh, s.r);
    __syncthreads();
    // dq (low-rank part) = P_q^T du, initialising the fp32 accumulator
    if (n < s.N) {
#pragma unroll 4
        for (int i = 0; i < 32; ++i) {
            const int d = quarter + 4 * i;
            float acc = 0.0f;
            for (int a = 0; a < s.r; ++a) acc = fmaf(m.G[t * m.rl + a], m.W[a * kLd + d], acc);
            dq_acc[head + (size_t)n * kDh + d] = acc;
        }
    }
}

// Key side: one CTA per (chunk, head); X = k rows, Y = v rows, W = P_k / dC.
template <typename T>
__global__ void __launch_bounds__(kBT) lr_bwd_k_kernel(Shape s, const T* __restrict__ k, const T* __restrict__ v,
                                                       const T* __restrict__ Pk, const float* __restrict__ dC,
                                                       const float2* __restrict__ tab, float* __restrict__ dk_acc,
                                                       float* __restrict__ dv_acc, float* __restrict__ partPk)
{
    extern __shared__ float lsm[];
    const LrSmem m = lr_smem(lsm, s.r);
    const int chunk = blockIdx.x, bh = blockIdx.y, h = bh % s.H;
    const int n0 = chunk * 64;
    const int t = threadIdx.x >> 2, quarter = threadIdx.x & 3;
    const int n = n0 + t;
    const size_t head = (size_t)bh * s.N * kDh;
    const ActBwd act{s.lr_act};
    load_rows(m.X, k + head, n0, s.N);
    load_rows(m.Y, v + head, n0, s.N);
    load_weight(m.W, Pk + (size_t)h * s.r * kDh, s.r);
    __syncthreads();
    features_fwd(s, m, tab, n0, act);
    for (int e = threadIdx.x; e < s.r * kDh; e += kBT) m.W[(e / kDh) * kLd + e % kDh] = dC[(size_t)bh * s.r * kDh + e];
    __syncthreads();
    // dk~ = dC v_j (r columns), dv (low-rank part) = dC^T k~_j
    float df[kDh / 4];
#pragma unroll
    for (int i = 0; i < kDh / 4; ++i) {
        const int a = quarter + 4 * i;
        float acc = 0.0f;
        if (a < s.r)
            for (int d = 0; d < kDh; ++d) acc = fmaf(m.Y[t * kLd + d], m.W[a * kLd + d], acc);
        df[i] = acc;
    }
    if (n < s.N) {
#pragma unroll 4
        for (int i = 0; i < 32; ++i) {
            const int d = quarter + 4 * i;
            float acc = 0.0f;
            for (int a = 0; a < s.r; ++a) acc = fmaf(m.F[t * m.rl + a], m.W[a * kLd + d], acc);
            dv_acc[head + (size_t)n * kDh + d] = acc;
        }
    }
    features_bwd(s, m, tab, n0, act, df);
    chunk_outer(s, m.G, m.rl, m.X, partPk + ((size_t)bh * s.nC + chunk) * s.r * kDh);
    __syncthreads();
    load_weight(m.W, Pk + (size_t)h * s.r * kDh, s.r);
    __syncthreads();
    if (n < s.N) {
#pragma unroll 4
        for (int i = 0; i < 32; ++i) {
            const int d = quarter + 4 * i;
            float acc = 0.0f;
            for (int a = 0; a < s.r; ++a) acc = fmaf(m.G[t * m.rl + a], m.W[a * kLd + d], acc);
            dk_acc[head + (size_t)n * kDh + d] = acc;
        }
    }
}

// out[g][e] = sum over the groups' slots in order: slot (b, h, chunk) for
// out[h] (per_batch = true: P_q, P_k summed over the batch) or for out[bh].
__global__ void reduce_chunks_kernel(Shape s, const float* __restrict__ part, float* __restrict__ out,
                                     bool per_batch)
{
    const int per = s.r * kDh;
    const int e = blockIdx.x * blockDim.x + threadIdx.x;
    const int grp = blockIdx.y;
    if (e >= per) return;
    float acc = 0.0f;
    const int nb = per_batch ? s.B : 1;
    for (int b = 0; b < nb; ++b) {
        const int bh = per_batch ? b * s.H + grp : grp;
        const float* p = part + (size_t)bh * s.nC * per + e;
        for (int c = 0; c < s.nC; ++c) acc += p[(size_t)c * per];
    }
    out[(size_t)grp * per + e] = acc;
}

// ---------------------------------------------------------------------------
// Sparse branch, query side: one CTA per (query block, head).  Thread (row,
// quarter) owns dq^r[row][quarter + 4 i]; scores of a (row, 16-key) strip.

struct SpSmem {
    float* Q;
    float* O;      // dO^s rows (fp32)
    float* K;
    float* V;
    float* S;      // [64][65]
    float* S2;     // [64][65]
    float* lse;    // [64]
    float* D;      // [64]
};

__device__ __forceinline__ SpSmem sp_smem(float* base)
{
    SpSmem m;
    m.Q = base;
    m.O = m.Q + 64 * kLd;
    m.K = m.O + 64 * kLd;
    m.V = m.K + 64 * kLd;
    m.S = m.V + 64 * kLd;
    m.S2 = m.S + 64 * 65;
    m.lse = m.S2 + 64 * 65;
    m.D = m.lse + 64;
    return m;
}

constexpr size_t kSpSmemBytes = sizeof(float) * (4 * 64 * kLd + 2 * 64 * 65 + 2 * 64);

// Row-pair rotation back by R(p)^T of a thread's columns quarter + 4 i: the
// partner column of an even column is held by lane ^ 1.
__device__ __forceinline__ void rotate_back(const Shape& s, const float2* tab, int n, int quarter, float (&x)[32])
{
#pragma unroll
    for (int i = 0; i < 32; ++i) {
        const int d = quarter + 4 * i;
        const float other = __shfl_xor_sync(0xffffffffu, x[i], 1);
        const float x0 = (d & 1) ? other : x[i], x1 = (d & 1) ? x[i] : other;
        const float2 r = rope_rotate_t(x0, x1, rope_cs(tab, s, n < s.N ? n : 0, d >> 1));
        x[i] = (d & 1) ? r.y : r.x;
    }
}

template <typename T>
__global__ void __launch_bounds__(kBT) sparse_bwd_dq_kernel(Shape s, const T* __restrict__ qr,
                                                            const T* __restrict__ kr, const T* __restrict__ v,
                                                            const int32_t* __restrict__ kv_idx,
                                                            const float* __restrict__ lse,
                                                            const float* __restrict__ Dv,
                                                            const T* __restrict__ dOs,
                                                            const float2* __restrict__ tab,
                                                            float* __restrict__ dq_acc)
{
    extern __shared__ float ssm[];
    const SpSmem m = sp_smem(ssm);
    const int qb = blockIdx.x, bh = blockIdx.y;
    const int row = threadIdx.x >> 2, quarter = threadIdx.x & 3;
    // q^r, k^r, v, dO^s, lse and D in block order (Np rows per head); dq rows by token
    const size_t head = (size_t)bh * s.Np * kDh;
    const int n0 = qb * 64, n = slot_token(s, qb, row);
    load_rows(m.Q, qr + head, n0, s.Np);
    load_rows(m.O, dOs + head, n0, s.Np);
    if (threadIdx.x < 64) {
        const bool v = slot_token(s, qb, threadIdx.x) >= 0;
        m.lse[threadIdx.x] = v ? lse[(size_t)bh * s.Np + n0 + threadIdx.x] : 0.0f;
        m.D[threadIdx.x] = v ? Dv[(size_t)bh * s.Np + n0 + threadIdx.x] : 0.0f;
    }
    const float scale = 0.08838834764831845f;     // 1 / sqrt(128)
    float acc[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) acc[i] = 0.0f;
    const int32_t* kept = kv_idx + ((size_t)bh * s.nB + qb) * s.n_keep;
    for (int it = 0; it < s.n_keep; ++it) {
        const int j = kept[it];
        if (j < 0 || j >= s.nB) continue;            // not a block id (the same for the whole CTA)
        __syncthreads();
        load_rows(m.K, kr + head, j * 64, s.Np);
        load_rows(m.V, v + head, j * 64, s.Np);
        __syncthreads();
        for (int c = 0; c < 16; ++c) {
            const int col = quarter * 16 + c;
            float sc = 0.0f, dp = 0.0f;
            for (int d = 0; d < kDh; ++d) {
                sc = fmaf(m.Q[row * kLd + d], m.K[col * kLd + d], sc);
                dp = fmaf(m.O[row * kLd + d], m.V[col * kLd + d], dp);
            }
            const bool valid = n >= 0 && slot_token(s, j, col) >= 0;
            const float p = valid ? expf(fmaf(sc, scale, -m.lse[row])) : 0.0f;
            m.S[row * 65 + col] = p * (dp - m.D[row]);
        }
        __syncwarp();
#pragma unroll
        for (int i = 0; i < 32; ++i) {
            float a = acc[i];
            for (int c = 0; c < 64; ++c) a = fmaf(m.S[row * 65 + c], m.K[c * kLd + quarter + 4 * i], a);
            acc[i] = a;
        }
    }
#pragma unroll
    for (int i = 0; i < 32; ++i) acc[i] *= scale;
    rotate_back(s, tab, n >= 0 ? n : s.N, quarter, acc);
    if (n >= 0) {
        float* dst = dq_acc + ((size_t)bh * s.N + n) * kDh;
#pragma unroll
        for (int i = 0; i < 32; ++i) dst[quarter + 4 * i] += acc[i];
    }
}

// For every (head, key block): the query blocks that kept it, ascending.  One
// CTA per head: count, exclusive scan, then fill walking the query blocks in
// order (the kept ids of one row are distinct, so a row's entries never share
// a cursor).
__global__ void __launch_bounds__(1024) mask_transpose_kernel(Shape s, const int32_t* __restrict__ kv_idx,
                                                              int32_t* __restrict__ off, int32_t* __restrict__ list)
{
    extern __shared__ int cur[];
    const int bh = blockIdx.x;
    const int32_t* kv = kv_idx + (size_t)bh * s.nB * s.n_keep;
    for (int j = threadIdx.x; j < s.nB; j += blockDim.x) cur[j] = 0;
    __syncthreads();
    for (int e = threadIdx.x; e < s.nB * s.n_keep; e += blockDim.x)
        if (kv[e] >= 0 && kv[e] < s.nB) atomicAdd(&cur[kv[e]], 1);
    __syncthreads();
    int32_t* o = off + (size_t)bh * (s.nB + 1);
    if (threadIdx.x == 0) {
        int run = 0;
        for (int j = 0; j < s.nB; ++j) {
            const int c = cur[j];
            o[j] = run;
            cur[j] = run;
            run += c;
        }
        o[s.nB] = run;
    }
    __syncthreads();
    int32_t* l = list + (size_t)bh * s.nB * s.n_keep;
    for (int i = 0; i < s.nB; ++i) {
        for (int t = threadIdx.x; t < s.n_keep; t += blockDim.x) {
            const int j = kv[(size_t)i * s.n_keep + t];
            if (j >= 0 && j < s.nB) l[cur[j]++] = i;
        }
        __syncthreads();
    }
}

// Key side: one CTA per (key block, head) over the query blocks that kept it.
// Thread (key row, quarter) owns dk^r and dv of its key row, columns quarter + 4 i.
template <typename T>
__global__ void __launch_bounds__(kBT) sparse_bwd_dkdv_kernel(Shape s, const T* __restrict__ qr,
                                                              const T* __restrict__ kr, const T* __restrict__ v,
                                                              const int32_t* __restrict__ off,
                                                              const int32_t* __restrict__ list,
                                                              const float* __restrict__ lse,
                                                              const float* __restrict__ Dv,
                                                              const T* __restrict__ dOs,
                                                              const float2* __restrict__ tab,
                                                              float* __restrict__ dk_acc, float* __restrict__ dv_acc)
{
    extern __shared__ float ssm[];
    const SpSmem m = sp_smem(ssm);
    const int kb = blockIdx.x, bh = blockIdx.y;
    const int krow = threadIdx.x >> 2, quarter = threadIdx.x & 3;
    // q^r, k^r, v, dO^s, lse and D in block order (Np rows per head); dk, dv rows by token
    const size_t head = (size_t)bh * s.Np * kDh;
    const int n = slot_token(s, kb, krow);
    load_rows(m.K, kr + head, kb * 64, s.Np);
    load_rows(m.V, v + head, kb * 64, s.Np);
    const float scale = 0.08838834764831845f;
    float ak[32], av[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) ak[i] = av[i] = 0.0f;
    const int32_t* o = off + (size_t)bh * (s.nB + 1);
    const int32_t* l = list + (size_t)bh * s.nB * s.n_keep;
    const int e0 = o[kb], e1 = o[kb + 1];
    for (int e = e0; e < e1; ++e) {
        const int qb = l[e];
        __syncthreads();
        load_rows(m.Q, qr + head, qb * 64, s.Np);
        load_rows(m.O, dOs + head, qb * 64, s.Np);
        if (threadIdx.x < 64) {
            const bool v = slot_token(s, qb, threadIdx.x) >= 0;
            m.lse[threadIdx.x] = v ? lse[(size_t)bh * s.Np + qb * 64 + threadIdx.x] : 0.0f;
            m.D[threadIdx.x] = v ? Dv[(size_t)bh * s.Np + qb * 64 + threadIdx.x] : 0.0f;
        }
        __syncthreads();
        for (int c = 0; c < 16; ++c) {
            const int qc = quarter * 16 + c;
            float sc = 0.0f, dp = 0.0f;
            for (int d = 0; d < kDh; ++d) {
                sc = fmaf(m.Q[qc * kLd + d], m.K[krow * kLd + d], sc);
                dp = fmaf(m.O[qc * kLd + d], m.V[krow * kLd + d], dp);
            }
            const bool valid = n >= 0 && slot_token(s, qb, qc) >= 0;
            const float p = valid ? expf(fmaf(sc, scale, -m.lse[qc])) : 0.0f;
            m.S[krow * 65 + qc] = p;
            m.S2[krow * 65 + qc] = p * (dp - m.D[qc]);
        }
        __syncwarp();
#pragma unroll
        for (int i = 0; i < 32; ++i) {
            float a = av[i], b = ak[i];
            for (int c = 0; c < 64; ++c) {
                a = fmaf(m.S[krow * 65 + c], m.O[c * kLd + quarter + 4 * i], a);
                b = fmaf(m.S2[krow * 65 + c], m.Q[c * kLd + quarter + 4 * i], b);
            }
            av[i] = a;
            ak[i] = b;
        }
    }
#pragma unroll
    for (int i = 0; i < 32; ++i) ak[i] *= scale;
    rotate_back(s, tab, n >= 0 ? n : s.N, quarter, ak);
    if (n >= 0) {
        float* dk = dk_acc + ((size_t)bh * s.N + n) * kDh;
        float* dv = dv_acc + ((size_t)bh * s.N + n) * kDh;
#pragma unroll
        for (int i = 0; i < 32; ++i) {
            dk[quarter + 4 * i] += ak[i];
            dv[quarter + 4 * i] += av[i];
        }
    }
}

// ---------------------------------------------------------------------------
// Shared helpers of the bf16 mma.sync kernels below: tiles of 64 rows x 128
// bf16 in shared memory with 256-byte rows whose 16-byte chunks are
// XOR-swizzled by the row (sw128), filled by cp.async; m16n8k16 fragments
// through ldmatrix.  (The bf16 sparse gradients run on tcgen05, in
// sparse_bwd_tc.cu.)

constexpr int kMT = 128;                          // threads of the mma kernels
constexpr uint32_t kTile = 64 * 256;              // one 64 x 128 bf16 tile

// cp.async of rows [n0, n0 + 64) of a [N][128] bf16 array into a swizzled tile
// (rows past N zero-filled from a clamped, valid address).
__device__ __forceinline__ void tile_async(uint32_t dst, const __nv_bfloat16* src, int n0, int N)
{
    for (int e = threadIdx.x; e < 64 * 16; e += kMT) {
        const int r = e >> 4, c = e & 15;
        const bool ok = n0 + r < N;
        const __nv_bfloat16* g = src + (size_t)(ok ? n0 + r : 0) * kDh + c * 8;
        cp_async16(dst + sw128(r, c), g, ok ? 16 : 0);
    }
}

// ldmatrix lane addresses: an A operand (16 rows from r0, k chunks 2 kk, 2 kk + 1),
// B from [n][k] storage (n rows from n0, two n-tiles), B from [k][n] storage
// (.trans; k rows from k0, n chunks from c0, two n-tiles).
__device__ __forceinline__ uint32_t a_addr(uint32_t t, int r0, int kk, int lane)
{
    return t + sw128(r0 + (lane & 7) + ((lane >> 3) & 1) * 8, 2 * kk + (lane >> 4));
}
__device__ __forceinline__ uint32_t bn_addr(uint32_t t, int n0, int kk, int lane)
{
    return t + sw128(n0 + (lane & 7) + (lane >> 4) * 8, 2 * kk + ((lane >> 3) & 1));
}
__device__ __forceinline__ uint32_t bt_addr(uint32_t t, int k0, int c0, int lane)
{
    return t + sw128(k0 + (lane & 7) + ((lane >> 3) & 1) * 8, c0 + (lane >> 4));
}

// ---------------------------------------------------------------------------
// bf16 low-rank backward on the tensor cores: one CTA (4 warps, 16 tokens
// each) per (64-token chunk, head), R = r rounded up to 16 (rows r .. R-1 of
// P read as zero, so those features and their gradients are zero).  A
// thread's accumulator columns 8 nt + 2 tig, +1 are one feature pair (the
// layout the forward's readout uses), so the rotation, phi and phi' are
// thread-local.  Token-contracting products (dC = F^T dY, dP = dU^T X) read
// the bf16 copies the warps leave in shared memory, A through ldmatrix.trans.

// A = (a 16-row slice of a [k][m] tile)^T: ldmatrix.trans lane address for
// m rows from m0 (chunks m0/8, m0/8 + 1) and k rows from k0.
__device__ __forceinline__ uint32_t at_addr(uint32_t t, int k0, int m0, int lane)
{
    return t + sw128(k0 + (lane & 7) + (lane >> 4) * 8, (m0 >> 3) + ((lane >> 3) & 1));
}

// C-fragment pairs (rows g, g + 8) to A fragments over k = 16 ks .. 16 ks + 15: n-tiles 2 ks and
// 2 ks + 1 of the C layout are the two k halves of the A layout.
template <int NT>
__device__ __forceinline__ void frag_a(const float (&w)[NT][4], int ks, uint32_t& a0, uint32_t& a1, uint32_t& a2,
                                       uint32_t& a3)
{
    a0 = pack_bf16(w[2 * ks][0], w[2 * ks][1]);
    a1 = pack_bf16(w[2 * ks][2], w[2 * ks][3]);
    a2 = pack_bf16(w[2 * ks + 1][0], w[2 * ks + 1][1]);
    a3 = pack_bf16(w[2 * ks + 1][2], w[2 * ks + 1][3]);
}

// rows [0, rows) of a [rows][128] array (bf16 or fp32) into a swizzled bf16 tile;
// rows [rows, R) zero.
template <typename T>
__device__ void weight_tile(uint8_t* base, uint32_t off, const T* src, int rows, int R)
{
    for (int e = threadIdx.x; e < R * 64; e += kMT) {
        const int a = e >> 6, d = (e & 63) * 2;
        const float x0 = a < rows ? to_f(src[(size_t)a * kDh + d]) : 0.0f;
        const float x1 = a < rows ? to_f(src[(size_t)a * kDh + d + 1]) : 0.0f;
        *reinterpret_cast<uint32_t*>(base + off + sw128(a, d >> 3) + (d & 7) * 2) = pack_bf16(x0, x1);
    }
}

__device__ __forceinline__ void put_pair(uint8_t* base, uint32_t off, int row, int col, float x0, float x1)
{
    *reinterpret_cast<uint32_t*>(base + off + sw128(row, col >> 3) + (col & 7) * 2) = pack_bf16(x0, x1);
}

// acc[R/8][4] = A(16 x 128: rows r0 of tile ta) * (R rows of tile tb)^T
template <int R>
__device__ __forceinline__ void mma_rows_x_w(float (&acc)[R / 8][4], uint32_t ta, int r0, uint32_t tb, int lane)
{
#pragma unroll
    for (int kk = 0; kk < 8; ++kk) {
        uint32_t a0, a1, a2, a3;
        ldsm_x4(a_addr(ta, r0, kk, lane), a0, a1, a2, a3);
#pragma unroll
        for (int np = 0; np < R / 16; ++np) {
            uint32_t b0, b1, b2, b3;
            ldsm_x4(bn_addr(tb, 16 * np, kk, lane), b0, b1, b2, b3);
            mma_bf16(acc[2 * np], a0, a1, a2, a3, b0, b1);
            mma_bf16(acc[2 * np + 1], a0, a1, a2, a3, b2, b3);
        }
    }
}

// acc[16][4] = A(16 x R from fragments w) * (R rows x 128 of tile tb)
template <int R>
__device__ __forceinline__ void mma_wfrag_x_w(float (&acc)[16][4], const float (&w)[R / 8][4], uint32_t tb, int lane)
{
#pragma unroll
    for (int ks = 0; ks < R / 16; ++ks) {
        uint32_t a0, a1, a2, a3;
        frag_a(w, ks, a0, a1, a2, a3);
#pragma unroll
        for (int np = 0; np < 8; ++np) {
            uint32_t b0, b1, b2, b3;
            ldsm_x4_t(bt_addr(tb, 16 * ks, 2 * np, lane), b0, b1, b2, b3);
            mma_bf16(acc[2 * np], a0, a1, a2, a3, b0, b1);
            mma_bf16(acc[2 * np + 1], a0, a1, a2, a3, b2, b3);
        }
    }
}

// acc[R/8][4] = A(16 x 128 from fragments w[16][4]) * (R rows of tile tb)^T
template <int R>
__device__ __forceinline__ void mma_dfrag_x_wt(float (&acc)[R / 8][4], const float (&w)[16][4], uint32_t tb, int lane)
{
#pragma unroll
    for (int kk = 0; kk < 8; ++kk) {
        uint32_t a0, a1, a2, a3;
        frag_a(w, kk, a0, a1, a2, a3);
#pragma unroll
        for (int np = 0; np < R / 16; ++np) {
            uint32_t b0, b1, b2, b3;
            ldsm_x4(bn_addr(tb, 16 * np, kk, lane), b0, b1, b2, b3);
            mma_bf16(acc[2 * np], a0, a1, a2, a3, b0, b1);
            mma_bf16(acc[2 * np + 1], a0, a1, a2, a3, b2, b3);
        }
    }
}

// part[a][d] (R x 128, fp32, first r rows stored) = sum over the chunk's 64 tokens of
// A[t][a] B[t][d], A and B swizzled bf16 tiles; warp w takes the 16 x 32 output tiles w, w + 4, ...
template <int R>
__device__ void mma_outer(uint32_t tA, uint32_t tB, int r, float* part, int warp, int lane)
{
    const int g = lane >> 2, tig = lane & 3;
    for (int tile = warp; tile < (R / 16) * 4; tile += 4) {
        const int a0 = (tile >> 2) * 16, d0 = (tile & 3) * 32;
        float acc[4][4] = {};
#pragma unroll
        for (int ks = 0; ks < 4; ++ks) {
            uint32_t x0, x1, x2, x3;
            ldsm_x4_t(at_addr(tA, 16 * ks, a0, lane), x0, x1, x2, x3);
#pragma unroll
            for (int np = 0; np < 2; ++np) {
                uint32_t b0, b1, b2, b3;
                ldsm_x4_t(bt_addr(tB, 16 * ks, (d0 >> 3) + 2 * np, lane), b0, b1, b2, b3);
                mma_bf16(acc[2 * np], x0, x1, x2, x3, b0, b1);
                mma_bf16(acc[2 * np + 1], x0, x1, x2, x3, b2, b3);
            }
        }
#pragma unroll
        for (int nt = 0; nt < 4; ++nt) {
            const int d = d0 + 8 * nt + 2 * tig;
            if (a0 + g < r) *reinterpret_cast<float2*>(part + (size_t)(a0 + g) * kDh + d) = make_float2(acc[nt][0], acc[nt][1]);
            if (a0 + g + 8 < r)
                *reinterpret_cast<float2*>(part + (size_t)(a0 + g + 8) * kDh + d) = make_float2(acc[nt][2], acc[nt][3]);
        }
    }
}

// u (fragments) -> features (fragments) for rows t0, t0 + 8 of the chunk, tokens n0 + t.
template <int R>
__device__ __forceinline__ void frag_features(const Shape& s, const float2* tab, const float (&u)[R / 8][4],
                                              float (&f)[R / 8][4], int n0, int t0, int tig, ActBwd act)
{
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int n = n0 + t0 + 8 * h;
#pragma unroll
        for (int nt = 0; nt < R / 8; ++nt) {
            const int a = 8 * nt + 2 * tig;
            float2 y = make_float2(0.0f, 0.0f);
            if (n < s.N && a < s.r) y = lowrank_pair(u[nt][2 * h], u[nt][2 * h + 1], rope_cs(tab, s, n, a >> 1), s.lr_rope, act);
            f[nt][2 * h] = y.x;
            f[nt][2 * h + 1] = y.y;
        }
    }
}

// dL/du (fragments, over df) for rows t0, t0 + 8.
template <int R>
__device__ __forceinline__ void frag_features_bwd(const Shape& s, const float2* tab, const float (&u)[R / 8][4],
                                                  float (&df)[R / 8][4], int n0, int t0, int tig, ActBwd act)
{
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int n = n0 + t0 + 8 * h;
#pragma unroll
        for (int nt = 0; nt < R / 8; ++nt) {
            const int a = 8 * nt + 2 * tig;
            float2 d = make_float2(0.0f, 0.0f);
            if (n < s.N && a < s.r)
                d = lowrank_pair_bwd(u[nt][2 * h], u[nt][2 * h + 1], df[nt][2 * h], df[nt][2 * h + 1],
                                     rope_cs(tab, s, n, a >> 1), s.lr_rope, act);
            df[nt][2 * h] = d.x;
            df[nt][2 * h + 1] = d.y;
        }
    }
}

template <int R>
__global__ void __launch_bounds__(kMT, R <= 32 ? 3 : 1) lr_bwd_q_mma_kernel(Shape s, const __nv_bfloat16* __restrict__ q,
                                                           const __nv_bfloat16* __restrict__ Pq,
                                                           const float* __restrict__ C,
                                                           const float* __restrict__ gate,
                                                           const __nv_bfloat16* __restrict__ o_s,
                                                           const __nv_bfloat16* __restrict__ dO,
                                                           const float2* __restrict__ tab,
                                                           __nv_bfloat16* __restrict__ dOs, float* __restrict__ Dv,
                                                           float* __restrict__ dq_acc, float* __restrict__ dg_h,
                                                           float* __restrict__ partC, float* __restrict__ partPq)
{
    extern __shared__ __align__(128) uint8_t msm[];
    const uint32_t b0 = smem_u32(msm);
    // layout: X [64] | P [R rows] | C [R rows] | F [64] | dY [64] (rows of 256 B); dU takes F's place
    // once the dC partial (F^T dY) is taken
    const uint32_t sX = b0, sP = b0 + kTile, sC = b0 + kTile + R * 256, sF = sC + R * 256, sY = sF + kTile,
                   sU = sF;
    const int chunk = blockIdx.x, bh = blockIdx.y, h = bh % s.H, b = bh / s.H;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, tig = lane & 3;
    const int n0 = chunk * 64, t0 = 16 * warp + g;
    const size_t head = (size_t)bh * s.N * kDh;
    const ActBwd act{s.lr_act};
    tile_async(sX, q + head, n0, s.N);
    cp_async_commit();
    weight_tile(msm, sP - b0, Pq + (size_t)h * s.r * kDh, s.r, R);
    weight_tile(msm, sC - b0, C + (size_t)bh * s.r * kDh, s.r, R);
    cp_async_wait<0>();
    __syncthreads();
    // u = P_q q, features
    float u[R / 8][4] = {}, f[R / 8][4];
    mma_rows_x_w<R>(u, sX, 16 * warp, sP, lane);
    frag_features<R>(s, tab, u, f, n0, t0, tig, act);
#pragma unroll
    for (int nt = 0; nt < R / 8; ++nt) {
        put_pair(msm, sF - b0, t0, 8 * nt + 2 * tig, f[nt][0], f[nt][1]);
        put_pair(msm, sF - b0, t0 + 8, 8 * nt + 2 * tig, f[nt][2], f[nt][3]);
    }
    // y = q~^T C
    float y[16][4] = {};
    mma_wfrag_x_w<R>(y, f, sC, lane);
    // fusion and RMSNorm backward, rows t0 and t0 + 8 (the quad of a row holds its 128 columns)
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
        const int n = n0 + t0 + 8 * hh;
        const bool valid = n < s.N;
        float os[32], go[32];
        float syy = 0.0f, sos = 0.0f;
#pragma unroll
        for (int nt = 0; nt < 16; ++nt) {
            const int d = 8 * nt + 2 * tig;
            float2 ov = make_float2(0.0f, 0.0f), gv = make_float2(0.0f, 0.0f);
            if (valid) {
                ov = unpack_bf16(*reinterpret_cast<const uint32_t*>(o_s + head + (size_t)n * kDh + d));
                gv = unpack_bf16(*reinterpret_cast<const uint32_t*>(dO + head + (size_t)n * kDh + d));
            }
            os[2 * nt] = ov.x; os[2 * nt + 1] = ov.y;
            go[2 * nt] = gv.x; go[2 * nt + 1] = gv.y;
            syy = fmaf(y[nt][2 * hh], y[nt][2 * hh], fmaf(y[nt][2 * hh + 1], y[nt][2 * hh + 1], syy));
            sos = fmaf(ov.x, ov.x, fmaf(ov.y, ov.y, sos));
        }
        syy += __shfl_xor_sync(0xffffffffu, syy, 1);
        syy += __shfl_xor_sync(0xffffffffu, syy, 2);
        sos += __shfl_xor_sync(0xffffffffu, sos, 1);
        sos += __shfl_xor_sync(0xffffffffu, sos, 2);
        const float irho = 1.0f / sqrtf(syy / (float)kDh + s.eps_lr);
        const float rp = sqrtf(sos / (float)kDh + s.eps_fuse);
        const float gt = valid ? (gate ? gate[(size_t)b * s.N + n] : s.default_gate) : 0.0f;
        float a_dot = 0.0f;
#pragma unroll
        for (int nt = 0; nt < 16; ++nt)
            a_dot = fmaf(y[nt][2 * hh] * irho, go[2 * nt], fmaf(y[nt][2 * hh + 1] * irho, go[2 * nt + 1], a_dot));
        a_dot += __shfl_xor_sync(0xffffffffu, a_dot, 1);
        a_dot += __shfl_xor_sync(0xffffffffu, a_dot, 2);
        const float coef = gt * a_dot / ((float)kDh * rp);
        float dsum = 0.0f, od = 0.0f;
#pragma unroll
        for (int nt = 0; nt < 16; ++nt) {
            const int d = 8 * nt + 2 * tig;
            const float gs0 = fmaf(coef, os[2 * nt], go[2 * nt]), gs1 = fmaf(coef, os[2 * nt + 1], go[2 * nt + 1]);
            if (valid) *reinterpret_cast<uint32_t*>(dOs + head + (size_t)n * kDh + d) = pack_bf16(gs0, gs1);
            dsum = fmaf(gs0, os[2 * nt], fmaf(gs1, os[2 * nt + 1], dsum));
            od = fmaf(y[nt][2 * hh] * irho, gt * rp * go[2 * nt], fmaf(y[nt][2 * hh + 1] * irho, gt * rp * go[2 * nt + 1], od));
        }
        dsum += __shfl_xor_sync(0xffffffffu, dsum, 1);
        dsum += __shfl_xor_sync(0xffffffffu, dsum, 2);
        od += __shfl_xor_sync(0xffffffffu, od, 1);
        od += __shfl_xor_sync(0xffffffffu, od, 2);
        if (tig == 0 && valid) {
            Dv[(size_t)bh * s.N + n] = dsum;
            dg_h[(size_t)bh * s.N + n] = rp * a_dot;
        }
        // y <- dy (rows of invalid tokens zero)
#pragma unroll
        for (int nt = 0; nt < 16; ++nt) {
            const float dy0 = valid ? (gt * rp * go[2 * nt] - y[nt][2 * hh] * irho * od / (float)kDh) * irho : 0.0f;
            const float dy1 = valid ? (gt * rp * go[2 * nt + 1] - y[nt][2 * hh + 1] * irho * od / (float)kDh) * irho : 0.0f;
            y[nt][2 * hh] = dy0;
            y[nt][2 * hh + 1] = dy1;
            put_pair(msm, sY - b0, t0 + 8 * hh, 8 * nt + 2 * tig, dy0, dy1);
        }
    }
    // dq~ = C dy, then du
    float df[R / 8][4] = {};
    mma_dfrag_x_wt<R>(df, y, sC, lane);
    frag_features_bwd<R>(s, tab, u, df, n0, t0, tig, act);
    // dq (low-rank part) = P_q^T du, fp32 rows
    {
        float dq[16][4] = {};
        mma_wfrag_x_w<R>(dq, df, sP, lane);
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
            const int n = n0 + t0 + 8 * hh;
            if (n >= s.N) continue;
#pragma unroll
            for (int nt = 0; nt < 16; ++nt)
                *reinterpret_cast<float2*>(dq_acc + head + (size_t)n * kDh + 8 * nt + 2 * tig) =
                    make_float2(dq[nt][2 * hh], dq[nt][2 * hh + 1]);
        }
    }
    __syncthreads();
    const size_t slot = ((size_t)bh * s.nC + chunk) * s.r * kDh;
    mma_outer<R>(sF, sY, s.r, partC + slot, warp, lane);
    __syncthreads();                              // F consumed: du goes in its place
#pragma unroll
    for (int nt = 0; nt < R / 8; ++nt) {
        put_pair(msm, sU - b0, t0, 8 * nt + 2 * tig, df[nt][0], df[nt][1]);
        put_pair(msm, sU - b0, t0 + 8, 8 * nt + 2 * tig, df[nt][2], df[nt][3]);
    }
    __syncthreads();
    mma_outer<R>(sU, sX, s.r, partPq + slot, warp, lane);
}

template <int R>
__global__ void __launch_bounds__(kMT) lr_bwd_k_mma_kernel(Shape s, const __nv_bfloat16* __restrict__ k,
                                                           const __nv_bfloat16* __restrict__ v,
                                                           const __nv_bfloat16* __restrict__ Pk,
                                                           const float* __restrict__ dC,
                                                           const float2* __restrict__ tab,
                                                           float* __restrict__ dk_acc, float* __restrict__ dv_acc,
                                                           float* __restrict__ partPk)
{
    extern __shared__ __align__(128) uint8_t msm[];
    const uint32_t b0 = smem_u32(msm);
    // layout: X (k) [64] | V [64] | P [R rows] | dC [R rows]; dU takes V's place: a warp reads only its
    // own 16 rows of V (dk~ = dC v) and writes dU to the same rows, so 48 KB at r = 32 and four CTAs an SM
    const uint32_t sX = b0, sV = b0 + kTile, sP = b0 + 2 * kTile, sC = sP + R * 256, sU = sV;
    const int chunk = blockIdx.x, bh = blockIdx.y, h = bh % s.H;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, tig = lane & 3;
    const int n0 = chunk * 64, t0 = 16 * warp + g;
    const size_t head = (size_t)bh * s.N * kDh;
    const ActBwd act{s.lr_act};
    tile_async(sX, k + head, n0, s.N);
    tile_async(sV, v + head, n0, s.N);
    cp_async_commit();
    weight_tile(msm, sP - b0, Pk + (size_t)h * s.r * kDh, s.r, R);
    weight_tile(msm, sC - b0, dC + (size_t)bh * s.r * kDh, s.r, R);
    cp_async_wait<0>();
    __syncthreads();
    float u[R / 8][4] = {}, f[R / 8][4];
    mma_rows_x_w<R>(u, sX, 16 * warp, sP, lane);
    frag_features<R>(s, tab, u, f, n0, t0, tig, act);
    // dv (low-rank part) = dC^T k~ : rows of F times dC
    {
        float dv[16][4] = {};
        mma_wfrag_x_w<R>(dv, f, sC, lane);
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
            const int n = n0 + t0 + 8 * hh;
            if (n >= s.N) continue;
#pragma unroll
            for (int nt = 0; nt < 16; ++nt)
                *reinterpret_cast<float2*>(dv_acc + head + (size_t)n * kDh + 8 * nt + 2 * tig) =
                    make_float2(dv[nt][2 * hh], dv[nt][2 * hh + 1]);
        }
    }
    // dk~ = dC v, then du
    float df[R / 8][4] = {};
    mma_rows_x_w<R>(df, sV, 16 * warp, sC, lane);
    frag_features_bwd<R>(s, tab, u, df, n0, t0, tig, act);
    __syncwarp();                                 // this warp's V rows are read: dU goes in their place
#pragma unroll
    for (int nt = 0; nt < R / 8; ++nt) {
        put_pair(msm, sU - b0, t0, 8 * nt + 2 * tig, df[nt][0], df[nt][1]);
        put_pair(msm, sU - b0, t0 + 8, 8 * nt + 2 * tig, df[nt][2], df[nt][3]);
    }
    {
        float dk[16][4] = {};
        mma_wfrag_x_w<R>(dk, df, sP, lane);
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
            const int n = n0 + t0 + 8 * hh;
            if (n >= s.N) continue;
#pragma unroll
            for (int nt = 0; nt < 16; ++nt)
                *reinterpret_cast<float2*>(dk_acc + head + (size_t)n * kDh + 8 * nt + 2 * tig) =
                    make_float2(dk[nt][2 * hh], dk[nt][2 * hh + 1]);
        }
    }
    __syncthreads();
    mma_outer<R>(sU, sX, s.r, partPk + ((size_t)bh * s.nC + chunk) * s.r * kDh, warp, lane);
}

// 64-row tiles (three on the query side, two on the key side) and the two R-row weight tiles
template <int R>
size_t lr_mma_smem(bool key_side) { return (key_side ? 2 : 3) * (size_t)kTile + 2 * (size_t)R * 256; }

template <int R>
cudaError_t launch_lr_mma_r(const Shape& s, const BackwardArgs& a, bool key_side, cudaStream_t st)
{
    const dim3 chunks(s.nC, s.B * s.H);
    const size_t smem = lr_mma_smem<R>(key_side);
    using bf = __nv_bfloat16;
    if (!key_side) {
        cudaError_t e = cudaFuncSetAttribute(lr_bwd_q_mma_kernel<R>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)smem);
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(lr_bwd_q_mma_kernel<R>, cudaFuncAttributePreferredSharedMemoryCarveout,
                                     cudaSharedmemCarveoutMaxShared);
        if (e != cudaSuccess) return e;
        lr_bwd_q_mma_kernel<R><<<chunks, kMT, smem, st>>>(
            s, static_cast<const bf*>(a.q), static_cast<const bf*>(a.P_q), a.C, a.gate, static_cast<const bf*>(a.o_s),
            static_cast<const bf*>(a.dO), a.tab, static_cast<bf*>(a.dOs), a.Dv, a.dq_acc, a.dg_h, a.partC, a.partPq);
    } else {
        cudaError_t e = cudaFuncSetAttribute(lr_bwd_k_mma_kernel<R>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)smem);
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(lr_bwd_k_mma_kernel<R>, cudaFuncAttributePreferredSharedMemoryCarveout,
                                     cudaSharedmemCarveoutMaxShared);
        if (e != cudaSuccess) return e;
        lr_bwd_k_mma_kernel<R><<<chunks, kMT, smem, st>>>(s, static_cast<const bf*>(a.k), static_cast<const bf*>(a.v),
                                                          static_cast<const bf*>(a.P_k), a.dC, a.tab, a.dk_acc,
                                                          a.dv_acc, a.partPk);
    }
    return cudaGetLastError();
}

cudaError_t launch_lr_mma(const Shape& s, const BackwardArgs& a, bool key_side, cudaStream_t st)
{
    switch (s.rp) {
        case 16: return launch_lr_mma_r<16>(s, a, key_side, st);
        case 32: return launch_lr_mma_r<32>(s, a, key_side, st);
        case 48: return launch_lr_mma_r<48>(s, a, key_side, st);
        case 64: return launch_lr_mma_r<64>(s, a, key_side, st);
        case 80: return launch_lr_mma_r<80>(s, a, key_side, st);
        case 96: return launch_lr_mma_r<96>(s, a, key_side, st);
        case 112: return launch_lr_mma_r<112>(s, a, key_side, st);
        case 128: return launch_lr_mma_r<128>(s, a, key_side, st);
        default: return cudaErrorInvalidValue;
    }
}

// dO^s rows, lse and D from token order into block order (cube geometry):
// row 64 b + i of the head's Np rows is slot i of block b (zeros for slots
// outside the grid).  One CTA per (block, head).
template <typename T>
__global__ void __launch_bounds__(kBT) block_order_kernel(Shape s, const T* __restrict__ dOs,
                                                          const float* __restrict__ lse, const float* __restrict__ Dv,
                                                          T* __restrict__ dOs_b, float* __restrict__ lse_b,
                                                          float* __restrict__ Dv_b)
{
    const int b = blockIdx.x, bh = blockIdx.y;
    for (int e = threadIdx.x; e < 64 * kDh; e += kBT) {
        const int i = e / kDh, d = e - i * kDh;
        const int n = slot_token(s, b, i);
        dOs_b[((size_t)bh * s.Np + (size_t)b * 64 + i) * kDh + d] =
            n >= 0 ? dOs[((size_t)bh * s.N + n) * kDh + d] : from_f<T>(0.0f);
    }
    if (threadIdx.x < 64) {
        const int n = slot_token(s, b, threadIdx.x);
        const size_t r = (size_t)bh * s.Np + (size_t)b * 64 + threadIdx.x;
        lse_b[r] = n >= 0 ? lse[(size_t)bh * s.N + n] : 0.0f;
        Dv_b[r] = n >= 0 ? Dv[(size_t)bh * s.N + n] : 0.0f;
    }
}

template <typename T>
__global__ void store_grad_kernel(size_t n, const float* __restrict__ acc, T* __restrict__ out)
{
    for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n; e += (size_t)gridDim.x * blockDim.x)
        out[e] = from_f<T>(acc[e]);
}

__global__ void gate_grad_kernel(Shape s, const float* __restrict__ dg_h, float* __restrict__ dgate)
{
    const int p = blockIdx.x * blockDim.x + threadIdx.x, b = blockIdx.y;
    if (p >= s.N) return;
    float acc = 0.0f;
    for (int h = 0; h < s.H; ++h) acc += dg_h[((size_t)b * s.H + h) * s.N + p];
    dgate[(size_t)b * s.N + p] = acc;
}

template <typename T>
cudaError_t launch_backward_t(const Shape& s, const BackwardArgs& a, cudaStream_t st)
{
    const dim3 chunks(s.nC, s.B * s.H), blocks(s.nB, s.B * s.H);
    const size_t lsm = lr_smem_bytes(s.r);
    cudaError_t e;
    e = cudaFuncSetAttribute(lr_bwd_q_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)lsm);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(lr_bwd_k_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)lsm);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(sparse_bwd_dq_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSpSmemBytes);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(sparse_bwd_dkdv_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)kSpSmemBytes);
    if (e != cudaSuccess) return e;
    const T* q = static_cast<const T*>(a.q);
    const T* k = static_cast<const T*>(a.k);
    const T* v = static_cast<const T*>(a.v);
    const T* qr = static_cast<const T*>(a.qr);
    const T* kr = static_cast<const T*>(a.kr);
    constexpr bool kMma = std::is_same<T, __nv_bfloat16>::value;
    if constexpr (kMma) {
        e = launch_lr_mma(s, a, false, st);
    } else {
        lr_bwd_q_kernel<T><<<chunks, kBT, lsm, st>>>(s, q, static_cast<const T*>(a.P_q), a.C, a.gate,
                                                     static_cast<const T*>(a.o_s), static_cast<const T*>(a.dO), a.tab,
                                                     static_cast<T*>(a.dOs), a.Dv, a.dq_acc, a.dg_h, a.partC,
                                                     a.partPq);
        e = cudaGetLastError();
    }
    if (e != cudaSuccess) return e;
    const dim3 red((s.r * kDh + 255) / 256, s.B * s.H), red_h((s.r * kDh + 255) / 256, s.H);
    reduce_chunks_kernel<<<red, 256, 0, st>>>(s, a.partC, a.dC, false);
    reduce_chunks_kernel<<<red_h, 256, 0, st>>>(s, a.partPq, a.dP_q, true);
    if constexpr (kMma) {
        e = launch_lr_mma(s, a, true, st);
        if (e != cudaSuccess) return e;
    } else {
        lr_bwd_k_kernel<T><<<chunks, kBT, lsm, st>>>(s, k, v, static_cast<const T*>(a.P_k), a.dC, a.tab, a.dk_acc,
                                                     a.dv_acc, a.partPk);
    }
    reduce_chunks_kernel<<<red_h, 256, 0, st>>>(s, a.partPk, a.dP_k, true);
    // the sparse kernels read v, dO^s, lse and D in block order (copies for cube blocks)
    if (s.cube)
        block_order_kernel<T><<<blocks, kBT, 0, st>>>(s, static_cast<const T*>(a.dOs), a.lse, a.Dv,
                                                      static_cast<T*>(a.dOs_blk), a.lse_blk, a.Dv_blk);
    const T* vb = static_cast<const T*>(s.cube ? a.v_blk : a.v);
    const T* dOb = static_cast<const T*>(s.cube ? a.dOs_blk : a.dOs);
    const float* lseb = s.cube ? a.lse_blk : a.lse;
    const float* Dvb = s.cube ? a.Dv_blk : a.Dv;
    if constexpr (kMma) {
        e = launch_sparse_bwd_dq_tc(s, qr, kr, vb, dOb, a.kv_idx, lseb, Dvb, a.tab, a.dq_acc, a.dq, a.status, st);
        if (e != cudaSuccess) return e;
    } else {
        sparse_bwd_dq_kernel<T><<<blocks, kBT, kSpSmemBytes, st>>>(s, qr, kr, vb, a.kv_idx, lseb, Dvb, dOb, a.tab,
                                                                  a.dq_acc);
    }
    const size_t tsm = sizeof(int) * (size_t)s.nB;
    if (tsm > 48 * 1024) {
        e = cudaFuncSetAttribute(mask_transpose_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)tsm);
        if (e != cudaSuccess) return e;
    }
    mask_transpose_kernel<<<s.B * s.H, 1024, tsm, st>>>(s, a.kv_idx, a.tr_off, a.tr_list);
    if constexpr (kMma) {
        e = launch_sparse_bwd_dkdv_tc(s, qr, kr, vb, dOb, a.tr_off, a.tr_list, lseb, Dvb, a.tab, a.dk_acc, a.dv_acc,
                                      a.dk, a.dv, a.status, st);
        if (e != cudaSuccess) return e;
    } else {
        sparse_bwd_dkdv_kernel<T><<<blocks, kBT, kSpSmemBytes, st>>>(s, qr, kr, vb, a.tr_off, a.tr_list, lseb, Dvb,
                                                                    dOb, a.tab, a.dk_acc, a.dv_acc);
        const size_t nel = (size_t)s.B * s.H * s.N * kDh;
        const int sg = 152 * 8;
        store_grad_kernel<T><<<sg, 256, 0, st>>>(nel, a.dq_acc, static_cast<T*>(a.dq));
        store_grad_kernel<T><<<sg, 256, 0, st>>>(nel, a.dk_acc, static_cast<T*>(a.dk));
        store_grad_kernel<T><<<sg, 256, 0, st>>>(nel, a.dv_acc, static_cast<T*>(a.dv));
    }
    if (a.dgate) gate_grad_kernel<<<dim3((s.N + 255) / 256, s.B), 256, 0, st>>>(s, a.dg_h, a.dgate);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_backward(rola_dtype_t dt, const Shape& s, const BackwardArgs& a, cudaStream_t st)
{
    return dt == ROLA_BF16 ? launch_backward_t<__nv_bfloat16>(s, a, st) : launch_backward_t<float>(s, a, st);
}

}  // namespace rola
