// Internal declarations shared by the RoLA CUDA translation units.
//
// Layout conventions (all tensors dense):
//   q, k, v, o          [B][H][N][128]      bf16 (ROLA_BF16) or fp32 (ROLA_FP32)
//   P_q, P_k            [H][r][128]
//   rotated q^r, k^r    [B][H][N][128]      workspace, storage dtype
//   pooled q_bar, k_bar [B][H][nB][128]     workspace, fp32
//   RoPE table          [T + Hh + Ww][64]   float2 (cos, sin) per grid row and pair;
//                                           row t for temporal pairs, T + x for height
//                                           pairs, T + Hh + y for width pairs
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/rola.h"

namespace rola {

constexpr int kDh = 128;      // head dimension supported by the kernels
constexpr int kBlock = 64;    // token block of the mask and of the sparse branch
constexpr int kPairs = kDh / 2;

// Status words at the start of the workspace (one 256-byte line).
struct DeviceStatus {
    int32_t code;             // rola_status_t of the last failing device-side check
    int32_t where;            // kernel-specific site id
    int32_t pad[62];
};

// Kernel-side view of a validated configuration.
struct Shape {
    int B, H, N, nB, n_keep, r;   // nB: key blocks of the sparse branch (chunks or cubes)
    int nQ;                   // query blocks (rows of the mask): nB, or ceil(N / 128) with 128-token queries
    int qb2;                  // 1 with 128-token query blocks: the mask row of 64-token block i is i >> 1
    int nC;                   // 64-token chunks ceil(N / 64): the units of the low-rank kernels
    int rp;                   // r rounded up to a multiple of 16: the width the bf16 kernels run at
                              // (rows r .. rp-1 of P are read as zero, so those features are zero)
    int T, Hh, Ww;
    int pt, px;               // pairs on the temporal / height axis (rest: width)
    float eps_lr, eps_fuse;
    float default_gate;       // sigmoid(gate_bias)
    float sm_scale_log2;      // log2(e) / sqrt(128)
    uint64_t wait_limit_ns;   // bound of every device-side wait
    int debug_flags;          // ROLA_DEBUG_* test hooks
    int lr_rope;              // rola_lowrank_rope_t
    int lr_act;               // rola_lowrank_act_t
    int cube;                 // block geometry: 0 contiguous 64-token chunks, 1 4x4x4 cubes
    int nCh, nCw;             // cubes along the row / column axis (cube geometry)
    int Np;                   // rows per head of the block-ordered copies q^r, k^r (and v):
                              // N, or nB * 64 in cube geometry (a cube's slots, padded)
    float rcp_plane, rcp_nCw; // fp32 1 / (nCh * nCw) and 1 / nCw (cube_origin_rcp)
};

// Most blocks per sequence: the top-k kernel keeps one row of nB 32-bit keys per
// warp (8 warps) beside 8 KB of scratch in 227 KB of shared memory.
constexpr int kMaxBlocks = 7008;

// Cube geometry: block b is the cube (ct, cx, cy) = t-major index b over the
// cube grid; its slot i = 16 dt + 4 dx + dy holds token (4ct+dt, 4cx+dx, 4cy+dy)
// when that lies inside the grid.
struct CubeOrigin {
    int t, x, y;
};
__host__ __device__ __forceinline__ CubeOrigin cube_origin(const Shape& s, int b)
{
    const int per_t = s.nCh * s.nCw;
    const int ct = b / per_t, rem = b - ct * per_t, cx = rem / s.nCw;
    return {4 * ct, 4 * cx, 4 * (rem - cx * s.nCw)};
}
// cube_origin with both divisions done as a multiply by the fp32 reciprocal:
// floor((a + 0.5) * fl(1/d)) equals a / d exactly whenever a < 2^22, because the
// product's error, below (a + 0.5) / d * 2^-23, stays under the distance 0.5 / d
// from (a + 0.5) / d to the nearest integer (block ids are below kMaxBlocks).
__device__ __forceinline__ CubeOrigin cube_origin_rcp(const Shape& s, int b)
{
    const int ct = __float2int_rz(__fmul_rn((float)b + 0.5f, s.rcp_plane));
    const int rem = b - ct * (s.nCh * s.nCw);
    const int cx = __float2int_rz(__fmul_rn((float)rem + 0.5f, s.rcp_nCw));
    return {4 * ct, 4 * cx, 4 * (rem - cx * s.nCw)};
}
// Flat index of the token in slot i of the cube at o, or -1 outside the grid.
__host__ __device__ __forceinline__ int cube_token(const Shape& s, CubeOrigin o, int i)
{
    const int t = o.t + (i >> 4), x = o.x + ((i >> 2) & 3), y = o.y + (i & 3);
    return (t < s.T && x < s.Hh && y < s.Ww) ? (t * s.Hh + x) * s.Ww + y : -1;
}

// Either geometry: the token of slot i of block b (-1 for a slot past the
// sequence or outside the grid), and the validity of the 32 slots [c0, c0 + 32)
// of block b as a bit mask.
// (The template forms fix the geometry at compile time.)
template <bool kCube>
__device__ __forceinline__ int slot_token_g(const Shape& s, int b, int i)
{
    if constexpr (!kCube) return b * 64 + i < s.N ? b * 64 + i : -1;
    else return cube_token(s, cube_origin_rcp(s, b), i);
}
__device__ __forceinline__ int slot_token(const Shape& s, int b, int i)
{
    return s.cube ? slot_token_g<true>(s, b, i) : slot_token_g<false>(s, b, i);
}
template <bool kCube>
__device__ __forceinline__ uint32_t slot_mask32_g(const Shape& s, int b, int c0)
{
    if constexpr (!kCube) {
        const int rem = s.N - b * 64 - c0;
        return rem >= 32 ? 0xffffffffu : (rem <= 0 ? 0u : (1u << rem) - 1u);
    }
    else {
        const CubeOrigin o = cube_origin_rcp(s, b);
        uint32_t m = 0;
        for (int i = 0; i < 32; ++i)
            if (cube_token(s, o, c0 + i) >= 0) m |= 1u << i;
        return m;
    }
}
__device__ __forceinline__ uint32_t slot_mask32(const Shape& s, int b, int c0)
{
    return s.cube ? slot_mask32_g<true>(s, b, c0) : slot_mask32_g<false>(s, b, c0);
}

// Rotation (cos, sin) of pair m for the token at flat index n.
__device__ __forceinline__ float2 rope_cs(const float2* __restrict__ tab, const Shape& s, int n, int m)
{
    int hw = s.Hh * s.Ww;
    int row;
    if (m < s.pt) row = n / hw;
    else if (m < s.pt + s.px) row = s.T + (n / s.Ww) % s.Hh;
    else row = s.T + s.Hh + n % s.Ww;
    return tab[row * kPairs + m];
}

// One RoPE pair rotation (x0, x1) -> (x0 cos - x1 sin, x0 sin + x1 cos) with
// its roundings spelled out, so that every kernel that rotates gets the same
// bits for the same inputs.
__device__ __forceinline__ float2 rope_rotate(float x0, float x1, float2 cs)
{
    return make_float2(__fmaf_rn(x0, cs.x, -__fmul_rn(x1, cs.y)), __fmaf_rn(x0, cs.y, __fmul_rn(x1, cs.x)));
}

// One pair of low-rank features from the projected pair (u0, u1) = the pair's
// two rows of P x: R_r after SiLU (Eq. qklr, ROLA_LOWRANK_ROPE_OUTSIDE), before
// it (Prop. inside, ROLA_LOWRANK_ROPE_INSIDE) or not at all (ROLA_LOWRANK_ROPE_NONE).
// `act` is the feature-map evaluation the caller uses (SiLU, or ActAblation).
template <typename Act>
__device__ __forceinline__ float2 lowrank_pair(float u0, float u1, float2 cs, int mode, Act act)
{
    if (mode == ROLA_LOWRANK_ROPE_INSIDE) {
        const float2 r = rope_rotate(u0, u1, cs);
        return make_float2(act(r.x), act(r.y));
    }
    const float a0 = act(u0), a1 = act(u1);
    return mode == ROLA_LOWRANK_ROPE_NONE ? make_float2(a0, a1) : rope_rotate(a0, a1, cs);
}

// ---------------------------------------------------------------- host side

// Workspace carve-up for one configuration.
struct Workspace {
    size_t status, table, qr, kr, vp, qbar, kbar, qbar2, scores, kv_idx, C, z, Cbf, partials, total;
    int nsplit;               // fp32 summary splits
    size_t prepass_slots;     // bf16 pre-pass partial slots
};

// Host launchers, one per kernel family.  All return cudaGetLastError().
cudaError_t launch_rope_table(const rola_config_t& cfg, float2* tab, cudaStream_t st);
// q^r, k^r (rows in block order, Np per head) and the block means; in cube
// geometry also v copied into block order (vp) when v is given.  With
// 128-token query blocks (s.qb2) qbar receives the 64-token blocks' q SUMS,
// which launch_qpool128 turns into the 128-token means.
cudaError_t launch_rope_pool(const rola_config_t& cfg, const Shape& s, const void* q, const void* k,
                             const void* v, const float2* tab, void* qr, void* kr, void* vp, float* qbar,
                             float* kbar, cudaStream_t st);
// qbar [B*H][nQ][128] (query means), kbar [B*H][nB][128]: scores [B*H][nQ][nB], kv_idx [B*H][nQ][n_keep].
cudaError_t launch_block_topk(const Shape& s, const float* qbar, const float* kbar, float* scores,
                              int32_t* kv_idx, cudaStream_t st);
// 128-token query means from the 64-token q sums: (S[2c] + S[2c+1]) / tokens of chunk c.
cudaError_t launch_qpool128(const Shape& s, const float* qsum64, float* qbar128, cudaStream_t st);
// lse (nullable): fp32 [B][H][N], log sum_j exp(s_pj) of each query row (natural log).
cudaError_t launch_sparse_attn(rola_dtype_t dt, const Shape& s, const void* qr, const void* kr,
                               const void* v, const int32_t* kv_idx, void* o_s, float* lse, DeviceStatus* status,
                               cudaStream_t st);
cudaError_t launch_sparse_attn_tc(const Shape& s, const void* qr, const void* kr, const void* v,
                                  const int32_t* kv_idx, void* o_s, float* lse, DeviceStatus* status,
                                  cudaStream_t st);
cudaError_t launch_lowrank_summary(rola_dtype_t dt, const Shape& s, int nsplit, const void* k,
                                   const void* v, const void* P_k, const float2* tab, float* partials,
                                   float* C, float* z, __nv_bfloat16* Cbf, cudaStream_t st);
cudaError_t launch_c_to_bf16(const Shape& s, const float* C, __nv_bfloat16* Cbf, cudaStream_t st);
cudaError_t launch_lowrank_apply(rola_dtype_t dt, const Shape& s, const void* q, const void* P_q,
                                 const float* C, const __nv_bfloat16* Cbf, const float* gate,
                                 const void* o_s, void* o, const float2* tab, DeviceStatus* status,
                                 cudaStream_t st);
// bf16 readout + fusion (readout.cu): persistent, TMA in and out, P_q and C once per head
cudaError_t launch_readout(const Shape& s, const void* q, const void* P_q, const __nv_bfloat16* Cbf,
                           const float* gate, const void* o_s, void* o, const float2* tab, DeviceStatus* status,
                           cudaStream_t st);

// Token gate g = sigmoid(X w_g + b) over `rows` rows of D features (gate.cu).
// Everything the backward pass reads and writes (device pointers; the fp32
// scratch rows live in the backward workspace).
struct BackwardArgs {
    const void *q, *k, *v, *P_q, *P_k, *o_s, *dO;     // storage dtype
    const float *C, *gate, *lse;
    const int32_t* kv_idx;
    const float2* tab;
    const void *qr, *kr;                                // rotated copies
    void* dOs;                                          // dL/dO^s, storage dtype
    const void* v_blk;                                  // cube blocks: v, dO^s, lse, D in block order
    void* dOs_blk;
    float *lse_blk, *Dv_blk;
    float *Dv, *dq_acc, *dk_acc, *dv_acc, *dg_h;        // fp32 scratch
    float *partC, *partPq, *partPk, *dC;                // per-chunk partials, reduced dC
    int32_t *tr_off, *tr_list;                          // transposed mask
    void *dq, *dk, *dv;                                 // outputs, storage dtype
    float *dP_q, *dP_k, *dgate;                         // outputs, fp32 (dgate nullable)
    DeviceStatus* status;                               // the backward workspace's status word
};
cudaError_t launch_backward(rola_dtype_t dt, const Shape& s, const BackwardArgs& a, cudaStream_t st);
// The bf16 query-side sparse gradient on tcgen05: dq = dq_lr + R^T (dS K / sqrt d), bf16.
cudaError_t launch_sparse_bwd_dq_tc(const Shape& s, const void* qr, const void* kr, const void* v, const void* dOs,
                                    const int32_t* kv_idx, const float* lse, const float* Dv, const float2* tab,
                                    const float* dq_lr, void* dq, DeviceStatus* status, cudaStream_t st);
// The bf16 key-side sparse gradients on tcgen05 over the transposed mask (off, list):
// dk = dk_lr + R^T (dS^T Q / sqrt d), dv = dv_lr + P^T dO^s, bf16.
cudaError_t launch_sparse_bwd_dkdv_tc(const Shape& s, const void* qr, const void* kr, const void* v, const void* dOs,
                                      const int32_t* off, const int32_t* list, const float* lse, const float* Dv,
                                      const float2* tab, const float* dk_lr, const float* dv_lr, void* dk, void* dv,
                                      DeviceStatus* status, cudaStream_t st);

cudaError_t launch_gate(rola_dtype_t dt, long long rows, int D, const void* X, const void* w, float b, float* g,
                        cudaStream_t st);

// Number of N-splits of the summary reduction for this shape (fp32 kernel).
int summary_splits(const Shape& s);

// The bf16 pre-pass (prepass.cu): `ctas` persistent CTAs each walk a
// contiguous range of (head, 64-token block) units.  Given q (fused form) it
// writes q^r, k^r and the pooled means exactly as launch_rope_pool does; it
// always writes the summary partials, one slot per (CTA c, head bh) at index
// c + bh, which launch_prepass_combine adds in CTA order.  With `ctas` CTAs
// the partial buffer needs ctas + B*H - 1 slots of r*128 + r floats.
constexpr int kMaxPrepassCtas = 512;
int prepass_ctas(const Shape& s, int max_ctas);     // its CTAs per SM x the SMs of the current device, at most max_ctas
cudaError_t launch_prepass(const Shape& s, int ctas, const void* q, const void* k, const void* v,
                           const void* P_k, const float2* tab, void* qr, void* kr, float* qbar, float* kbar,
                           float* partials, DeviceStatus* status, cudaStream_t st);
cudaError_t launch_prepass_combine(const Shape& s, int ctas, const float* partials, float* C, float* z,
                                   __nv_bfloat16* Cbf, cudaStream_t st);

// Host-side configuration checks shared by the entry points (api.cu).
rola_status_t validate(const rola_config_t* cfg);   // ROLA_OK if the kernels handle cfg
Shape make_shape(const rola_config_t& cfg);          // cfg must be valid
int num_blocks_of(const rola_config_t& cfg);
int num_keep_of(const rola_config_t& cfg);

// ---------------------------------------------------------------- device PTX helpers

__device__ __forceinline__ uint32_t smem_u32(const void* p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// 16-byte async copy global -> shared; src_bytes < 16 zero-fills the rest.
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, int src_bytes)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src), "r"(src_bytes)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory"); }

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& a, uint32_t& b, uint32_t& c, uint32_t& d)
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(a), "=r"(b), "=r"(c), "=r"(d) : "r"(addr));
}
__device__ __forceinline__ void ldsm_x2(uint32_t addr, uint32_t& a, uint32_t& b)
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0,%1}, [%2];\n" : "=r"(a), "=r"(b) : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& a, uint32_t& b, uint32_t& c, uint32_t& d)
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(a), "=r"(b), "=r"(c), "=r"(d) : "r"(addr));
}

// D += A(16x16 bf16, row) * B(16x8 bf16, col), fp32 accumulate.
__device__ __forceinline__ void mma_bf16(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1)
{
    asm volatile("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
                 "{%8,%9}, {%0,%1,%2,%3};\n"
                 : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
                 : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi)
{
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}
__device__ __forceinline__ float2 unpack_bf16(uint32_t u)
{
    __nv_bfloat162 v = *reinterpret_cast<__nv_bfloat162*>(&u);
    return __bfloat1622float2(v);
}

__device__ __forceinline__ float fast_exp2(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;\n" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ float silu(float x) { return x / (1.0f + __expf(-x)); }

// The feature maps of the activation ablation other than SiLU (Tab. abl_activation),
// chosen at run time by `kind` (a rola_lowrank_act_t).  tanhf and erff are CUDA's
// accurate functions; GELU is the exact x Phi(x) form.
struct ActAblation {
    int kind;
    __device__ float operator()(float x) const
    {
        switch (kind) {
            case ROLA_LOWRANK_ACT_IDENTITY: return x;
            case ROLA_LOWRANK_ACT_TANH: return tanhf(x);
            case ROLA_LOWRANK_ACT_RELU: return fmaxf(x, 0.0f);
            default: return 0.5f * x * (1.0f + erff(x * 0.7071067811865476f));
        }
    }
};

// Byte offset of 16-byte chunk c of row r in a [rows][128 bf16] tile with the
// chunk index XOR-swizzled by the row (conflict-free ldmatrix on 8-row groups).
__device__ __forceinline__ uint32_t sw128(int r, int c) { return r * 256 + ((c ^ (r & 7)) << 4); }

// Byte offset of 16-byte chunk c (0..15) of row r in a 64-row block tile as a
// [chunk][row][64] TMA box with 128-byte swizzle writes it: the two 64-wide
// halves of a row are 8 KB apart, and within 1024-byte atoms chunk c & 7 of
// row r sits at (c & 7) ^ (r & 7).
__device__ __forceinline__ uint32_t tsw(int r, int c)
{
    return (c >> 3) * 8192 + r * 128 + (((c & 7) ^ (r & 7)) << 4);
}

}  // namespace rola
