// C ABI entry points of include/rola.h: validation, workspace layout, launches.
#include <math.h>
#include <string.h>

#include "common.cuh"

using namespace rola;

namespace rola {

// The output projection (out_proj.cu).
cudaError_t launch_out_proj(int B, int N, int H, int d_model, const void* O, const void* W, const float* bias,
                            void* Y, DeviceStatus* status, uint64_t wait_limit_ns, cudaStream_t st);
cudaError_t launch_out_proj_f32(int B, int N, int H, int d_model, const float* O, const float* W, const float* bias,
                                float* Y, cudaStream_t st);

int num_blocks_of(const rola_config_t& c)
{
    if (c.block_geometry == ROLA_BLOCK_CUBE)
        return ((c.T + 3) / 4) * ((c.Hh + 3) / 4) * ((c.Ww + 3) / 4);
    return (int)(((int64_t)c.N + c.block - 1) / c.block);
}

// Rows per head of the block-ordered copies q^r, k^r (and v in cube geometry).
int64_t block_rows_of(const rola_config_t& c)
{
    return c.block_geometry == ROLA_BLOCK_CUBE ? (int64_t)num_blocks_of(c) * c.block : c.N;
}

int num_qblocks_of(const rola_config_t& c)
{
    if (c.query_block == 128) return (int)(((int64_t)c.N + 127) / 128);
    return num_blocks_of(c);
}

int num_keep_of(const rola_config_t& c)
{
    int nkb = num_blocks_of(c);
    double x = floor((double)c.keep_ratio * (double)nkb + 0.5);
    int n = (int)x;
    if (n < 1) n = 1;
    if (n > nkb) n = nkb;
    return n;
}

rola_status_t validate(const rola_config_t* c)
{
    if (!c) return ROLA_ERR_INVALID_ARG;
    if (c->B < 1 || c->H < 1 || c->N < 1 || c->T < 1 || c->Hh < 1 || c->Ww < 1) return ROLA_ERR_INVALID_ARG;
    if ((int64_t)c->T * c->Hh * c->Ww != c->N) return ROLA_ERR_INVALID_ARG;
    if (c->dtype != ROLA_BF16 && c->dtype != ROLA_FP32) return ROLA_ERR_INVALID_ARG;
    if (c->d_h != kDh) return c->d_h > 0 ? ROLA_ERR_UNSUPPORTED : ROLA_ERR_INVALID_ARG;
    if (c->block != kBlock) return c->block > 0 ? ROLA_ERR_UNSUPPORTED : ROLA_ERR_INVALID_ARG;
    for (int a = 0; a < 3; ++a)
        if (c->rope_split[a] < 0 || (c->rope_split[a] & 1)) return ROLA_ERR_INVALID_ARG;
    if (c->rope_split[0] + c->rope_split[1] + c->rope_split[2] != c->d_h) return ROLA_ERR_INVALID_ARG;
    if (!(c->rope_theta > 0.0) || !isfinite(c->rope_theta)) return ROLA_ERR_INVALID_ARG;
    if (!(c->keep_ratio >= 0.0f && c->keep_ratio <= 1.0f)) return ROLA_ERR_INVALID_ARG;
    if (c->r < 2 || (c->r & 1) || c->r > c->d_h) return ROLA_ERR_INVALID_ARG;
    if (c->r % 8 != 0) return ROLA_ERR_UNSUPPORTED;
    if (!(c->eps_lr >= 0.0f) || !(c->eps_fuse >= 0.0f) || !isfinite(c->eps_lr) || !isfinite(c->eps_fuse))
        return ROLA_ERR_INVALID_ARG;
    if (!isfinite(c->gate_bias)) return ROLA_ERR_INVALID_ARG;
    for (int a = 0; a < 3; ++a)
        if (c->pos_offset[a] < -(1 << 20) || c->pos_offset[a] > (1 << 20)) return ROLA_ERR_INVALID_ARG;
    if (c->wait_limit_ms < 0 || c->wait_limit_ms > 60000) return ROLA_ERR_INVALID_ARG;
    if (c->debug_flags & ~ROLA_DEBUG_SKIP_FIRST_K_COPY) return ROLA_ERR_INVALID_ARG;
    if (c->lowrank_rope < ROLA_LOWRANK_ROPE_OUTSIDE || c->lowrank_rope > ROLA_LOWRANK_ROPE_NONE)
        return ROLA_ERR_INVALID_ARG;
    if (c->lowrank_act < ROLA_LOWRANK_ACT_SILU || c->lowrank_act > ROLA_LOWRANK_ACT_GELU) return ROLA_ERR_INVALID_ARG;
    if (c->block_geometry != ROLA_BLOCK_FLAT && c->block_geometry != ROLA_BLOCK_CUBE) return ROLA_ERR_INVALID_ARG;
    if (c->query_block != 0 && c->query_block != kBlock && c->query_block != 128) return ROLA_ERR_INVALID_ARG;
    if (c->query_block == 128 && c->block_geometry != ROLA_BLOCK_FLAT) return ROLA_ERR_UNSUPPORTED;
    // grid / index limits of the kernels
    if ((int64_t)c->B * c->H > 65535) return ROLA_ERR_UNSUPPORTED;
    // the top-k kernel holds a row of nB keys per warp in shared memory (8 warps, 227 KB)
    if (num_blocks_of(*c) > kMaxBlocks) return ROLA_ERR_UNSUPPORTED;
    // the sparse kernel counts a CTA's kept blocks in 32 bits (ring slots and phases)
    if ((int64_t)c->B * c->H * num_blocks_of(*c) * num_keep_of(*c) >= ((int64_t)1 << 31)) return ROLA_ERR_UNSUPPORTED;
    if ((int64_t)c->B * c->H * c->N * c->d_h > ((int64_t)1 << 40)) return ROLA_ERR_UNSUPPORTED;
    // cube geometry: the padded block-ordered rows of a head stay addressable in int
    if (block_rows_of(*c) > ((int64_t)1 << 30)) return ROLA_ERR_UNSUPPORTED;
    return ROLA_OK;
}

Shape make_shape(const rola_config_t& c)
{
    Shape s;
    s.B = c.B; s.H = c.H; s.N = c.N; s.r = c.r;
    s.rp = (c.r + 15) & ~15;
    s.nB = num_blocks_of(c);
    s.nQ = num_qblocks_of(c);
    s.qb2 = c.query_block == 128 ? 1 : 0;
    s.nC = (int)(((int64_t)c.N + kBlock - 1) / kBlock);
    s.n_keep = num_keep_of(c);
    s.T = c.T; s.Hh = c.Hh; s.Ww = c.Ww;
    s.pt = c.rope_split[0] / 2;
    s.px = c.rope_split[1] / 2;
    s.eps_lr = c.eps_lr;
    s.eps_fuse = c.eps_fuse;
    s.default_gate = (float)(1.0 / (1.0 + exp(-(double)c.gate_bias)));
    s.sm_scale_log2 = (float)(1.4426950408889634 / sqrt((double)kDh));
    s.wait_limit_ns = (uint64_t)(c.wait_limit_ms > 0 ? c.wait_limit_ms : 2000) * 1000000ull;
    s.debug_flags = c.debug_flags;
    s.lr_rope = c.lowrank_rope;
    s.lr_act = c.lowrank_act;
    s.cube = c.block_geometry == ROLA_BLOCK_CUBE;
    s.nCh = (c.Hh + 3) / 4;
    s.nCw = (c.Ww + 3) / 4;
    s.Np = (int)block_rows_of(c);
    s.rcp_plane = (float)(1.0 / ((double)s.nCh * s.nCw));
    s.rcp_nCw = (float)(1.0 / (double)s.nCw);
    return s;
}

}  // namespace rola

namespace {

constexpr size_t kAlign = 256;

size_t align_up(size_t x) { return (x + kAlign - 1) & ~(kAlign - 1); }

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

Workspace layout(const rola_config_t& c)
{
    Shape s = make_shape(c);
    size_t esz = c.dtype == ROLA_BF16 ? 2 : 4;
    size_t bh = (size_t)c.B * c.H;
    Workspace w;
    w.nsplit = summary_splits(s);
    size_t off = 0;
    w.status = off; off = align_up(off + sizeof(DeviceStatus));
    w.table = off; off = align_up(off + sizeof(float2) * (size_t)(c.T + c.Hh + c.Ww) * kPairs);
    w.qr = off; off = align_up(off + esz * bh * s.Np * kDh);
    w.kr = off; off = align_up(off + esz * bh * s.Np * kDh);
    w.vp = off; off = align_up(off + (s.cube ? esz * bh * s.Np * kDh : 0));   // v in block order (cube)
    w.qbar = off; off = align_up(off + 4 * bh * s.nB * kDh);
    w.kbar = off; off = align_up(off + 4 * bh * s.nB * kDh);
    w.qbar2 = off; off = align_up(off + (s.qb2 ? 4 * bh * s.nQ * kDh : 0));   // 128-token query means
    w.scores = off; off = align_up(off + 4 * bh * s.nQ * s.nB);
    w.kv_idx = off; off = align_up(off + 4 * bh * s.nQ * s.n_keep);
    w.C = off; off = align_up(off + 4 * bh * c.r * kDh);
    w.z = off; off = align_up(off + 4 * bh * c.r);
    w.Cbf = off; off = align_up(off + 2 * bh * s.rp * kDh);           // zero-padded to rp rows
    // summary partials: fp32 split-N slots, or the bf16 pre-pass's per-(CTA, head) slots
    const size_t units = bh * s.nC;          // the pre-pass works on 64-token chunks
    w.prepass_slots = (units < (size_t)kMaxPrepassCtas ? units : (size_t)kMaxPrepassCtas) + bh - 1;
    const size_t slots = c.dtype == ROLA_BF16 ? w.prepass_slots : bh * w.nsplit;
    w.partials = off; off = align_up(off + 4 * slots * ((size_t)s.rp * kDh + s.rp));
    w.total = off;
    return w;
}

template <typename T>
T* at(void* ws, size_t off) { return reinterpret_cast<T*>(static_cast<uint8_t*>(ws) + off); }

rola_status_t check_ws(const rola_config_t& c, const void* ws, size_t ws_bytes)
{
    if (!ws || (reinterpret_cast<uintptr_t>(ws) & (kAlign - 1))) return ROLA_ERR_WORKSPACE;
    if (ws_bytes < layout(c).total) return ROLA_ERR_WORKSPACE;
    return ROLA_OK;
}

#define ROLA_TRY(expr)                                  \
    do {                                                \
        cudaError_t e_ = (expr);                        \
        if (e_ != cudaSuccess) return ROLA_ERR_CUDA;    \
    } while (0)

#define ROLA_CHECK(expr)                                \
    do {                                                \
        rola_status_t st_ = (expr);                     \
        if (st_ != ROLA_OK) return st_;                 \
    } while (0)

// Start of every entry point: clear the status word, build the RoPE table.
rola_status_t prologue(const rola_config_t& c, void* ws, const Workspace& w, cudaStream_t st)
{
    ROLA_TRY(cudaMemsetAsync(at<uint8_t>(ws, w.status), 0, sizeof(DeviceStatus), st));
    ROLA_TRY(launch_rope_table(c, at<float2>(ws, w.table), st));
    return ROLA_OK;
}

// The low-rank summary alone: C (fp32), z (nullable) and, when Cbf is given, C in bf16.
rola_status_t run_summary(const rola_config_t& c, const Shape& s, const Workspace& w, const void* k, const void* v,
                          const void* P_k, float* C, float* z, __nv_bfloat16* Cbf, void* ws, cudaStream_t st)
{
    if (c.dtype == ROLA_BF16) {
        const int ctas = prepass_ctas(s, kMaxPrepassCtas);
        if (ctas <= 0) return ROLA_ERR_CUDA;
        ROLA_TRY(launch_prepass(s, ctas, nullptr, k, v, P_k, at<float2>(ws, w.table), nullptr, nullptr, nullptr,
                                nullptr, at<float>(ws, w.partials), at<DeviceStatus>(ws, w.status), st));
        ROLA_TRY(launch_prepass_combine(s, ctas, at<float>(ws, w.partials), C, z, Cbf, st));
    } else {
        ROLA_TRY(launch_lowrank_summary(c.dtype, s, w.nsplit, k, v, P_k, at<float2>(ws, w.table),
                                        at<float>(ws, w.partials), C, z, Cbf, st));
    }
    return ROLA_OK;
}

// q^r, k^r and the block means; v in block order too when v is given and the geometry is cubes.
cudaError_t rope_pool(const rola_config_t& c, const Shape& s, const Workspace& w, const void* q, const void* k,
                      const void* v, void* ws, cudaStream_t st)
{
    return launch_rope_pool(c, s, q, k, s.cube ? v : nullptr, at<float2>(ws, w.table), at<void>(ws, w.qr),
                            at<void>(ws, w.kr), at<void>(ws, w.vp), at<float>(ws, w.qbar), at<float>(ws, w.kbar), st);
}

// The v rows the sparse kernels read: the caller's v, or its block-ordered copy in cube geometry.
const void* sparse_v(const Shape& s, const Workspace& w, const void* v, void* ws)
{
    return s.cube ? at<void>(ws, w.vp) : v;
}

// Block scores and top-k from the pooled means (128-token query means first, when configured).
cudaError_t select_blocks(const Shape& s, const Workspace& w, int32_t* kv_idx, void* ws, cudaStream_t st)
{
    const float* qm = at<float>(ws, w.qbar);
    if (s.qb2) {
        cudaError_t e = launch_qpool128(s, at<float>(ws, w.qbar), at<float>(ws, w.qbar2), st);
        if (e != cudaSuccess) return e;
        qm = at<float>(ws, w.qbar2);
    }
    return launch_block_topk(s, qm, at<float>(ws, w.kbar), at<float>(ws, w.scores), kv_idx, st);
}

rola_status_t run_mask(const rola_config_t& c, const Shape& s, const Workspace& w, const void* q, const void* k,
                       const void* v, int32_t* kv_idx, void* ws, cudaStream_t st)
{
    ROLA_TRY(rope_pool(c, s, w, q, k, v, ws, st));
    ROLA_TRY(select_blocks(s, w, kv_idx, ws, st));
    return ROLA_OK;
}

// Backward workspace: the status word and RoPE table as in the forward
// workspace, the rotated copies, fp32 gradient rows and partials.
struct BwdWorkspace {
    size_t status, table, qr, kr, vp, qbar, kbar, dOs, Dv, dq, dk, dv, dg, partC, partPq, partPk, dC, tr_off, tr_list,
        dOs_b, lse_b, Dv_b, total;
};

BwdWorkspace bwd_layout(const rola_config_t& c)
{
    const Shape s = make_shape(c);
    const size_t esz = c.dtype == ROLA_BF16 ? 2 : 4;
    const size_t bh = (size_t)c.B * c.H, rows = bh * c.N, brows = bh * s.Np;   // token rows, block-ordered rows
    const size_t part = 4 * bh * s.nC * (size_t)c.r * kDh;
    const size_t cube = s.cube ? 1 : 0;
    BwdWorkspace w;
    size_t off = 0;
    w.status = off; off = align_up(off + sizeof(DeviceStatus));
    w.table = off; off = align_up(off + sizeof(float2) * (size_t)(c.T + c.Hh + c.Ww) * kPairs);
    w.qr = off; off = align_up(off + esz * brows * kDh);
    w.kr = off; off = align_up(off + esz * brows * kDh);
    w.vp = off; off = align_up(off + cube * esz * brows * kDh);
    w.qbar = off; off = align_up(off + 4 * bh * s.nB * kDh);
    w.kbar = off; off = align_up(off + 4 * bh * s.nB * kDh);
    w.dOs = off; off = align_up(off + esz * rows * kDh);
    w.Dv = off; off = align_up(off + 4 * rows);
    w.dq = off; off = align_up(off + 4 * rows * kDh);
    w.dk = off; off = align_up(off + 4 * rows * kDh);
    w.dv = off; off = align_up(off + 4 * rows * kDh);
    w.dg = off; off = align_up(off + 4 * rows);
    w.partC = off; off = align_up(off + part);
    w.partPq = off; off = align_up(off + part);
    w.partPk = off; off = align_up(off + part);
    w.dC = off; off = align_up(off + 4 * bh * (size_t)c.r * kDh);
    w.tr_off = off; off = align_up(off + 4 * bh * (s.nB + 1));
    w.tr_list = off; off = align_up(off + 4 * bh * (size_t)s.nB * s.n_keep);
    w.dOs_b = off; off = align_up(off + cube * esz * brows * kDh);
    w.lse_b = off; off = align_up(off + cube * 4 * brows);
    w.Dv_b = off; off = align_up(off + cube * 4 * brows);
    w.total = off;
    return w;
}

// The forward pass.  With o_s_out the sparse output is kept there (and O written
// to o), with lse_out the log-sum-exp of every query row, with C_out the summary:
// what the backward pass reads.
rola_status_t forward_impl(const rola_config_t* cfg, const void* q, const void* k, const void* v, const void* P_q,
                           const void* P_k, const float* gate, void* o, int32_t* kv_idx_out, void* o_s_out,
                           float* lse_out, float* C_out, void* ws, size_t ws_bytes, void* stream,
                           void* const* stage_events)
{
    ROLA_CHECK(validate(cfg));
    if (!q || !k || !v || !P_q || !P_k || !o) return ROLA_ERR_INVALID_ARG;
    if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(P_q) || !aligned16(P_k) || !aligned16(o) ||
        (kv_idx_out && !aligned16(kv_idx_out)) || (gate && (reinterpret_cast<uintptr_t>(gate) & 3u)) ||
        (o_s_out && (!aligned16(o_s_out) || o_s_out == o)) || (lse_out && !aligned16(lse_out)) ||
        (C_out && !aligned16(C_out)))
        return ROLA_ERR_INVALID_ARG;
    ROLA_CHECK(check_ws(*cfg, ws, ws_bytes));
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    auto mark = [&](int i) -> cudaError_t {
        return stage_events ? cudaEventRecord(static_cast<cudaEvent_t>(stage_events[i]), st) : cudaSuccess;
    };
    Workspace w = layout(*cfg);
    Shape s = make_shape(*cfg);
    int32_t* kv = kv_idx_out ? kv_idx_out : at<int32_t>(ws, w.kv_idx);
    ROLA_TRY(mark(0));
    ROLA_CHECK(prologue(*cfg, ws, w, st));
    if (cfg->dtype == ROLA_BF16 && s.cube) {
        // stage 1: q^r, k^r, v in cube order and the cube means, then the summary
        // partials (the fused pre-pass pools contiguous chunks only);
        // stage 2: block scores + top-k, and the summary combine
        const int ctas = prepass_ctas(s, kMaxPrepassCtas);
        if (ctas <= 0) return ROLA_ERR_CUDA;
        ROLA_TRY(rope_pool(*cfg, s, w, q, k, v, ws, st));
        ROLA_TRY(launch_prepass(s, ctas, nullptr, k, v, P_k, at<float2>(ws, w.table), nullptr, nullptr, nullptr,
                                nullptr, at<float>(ws, w.partials), at<DeviceStatus>(ws, w.status), st));
        ROLA_TRY(mark(1));
        ROLA_TRY(select_blocks(s, w, kv, ws, st));
        ROLA_TRY(launch_prepass_combine(s, ctas, at<float>(ws, w.partials), at<float>(ws, w.C), at<float>(ws, w.z),
                                        at<__nv_bfloat16>(ws, w.Cbf), st));
    } else if (cfg->dtype == ROLA_BF16) {
        // stage 1: one pass over q, k, v -> q^r, k^r, block means, summary partials;
        // stage 2: block scores + top-k, and the summary combine
        const int ctas = prepass_ctas(s, kMaxPrepassCtas);
        if (ctas <= 0) return ROLA_ERR_CUDA;
        ROLA_TRY(launch_prepass(s, ctas, q, k, v, P_k, at<float2>(ws, w.table), at<void>(ws, w.qr),
                                at<void>(ws, w.kr), at<float>(ws, w.qbar), at<float>(ws, w.kbar),
                                at<float>(ws, w.partials), at<DeviceStatus>(ws, w.status), st));
        ROLA_TRY(mark(1));
        ROLA_TRY(select_blocks(s, w, kv, ws, st));
        ROLA_TRY(launch_prepass_combine(s, ctas, at<float>(ws, w.partials), at<float>(ws, w.C), at<float>(ws, w.z),
                                        at<__nv_bfloat16>(ws, w.Cbf), st));
    } else {
        // stage 1: the block mask; stage 2: the summary
        ROLA_CHECK(run_mask(*cfg, s, w, q, k, v, kv, ws, st));
        ROLA_TRY(mark(1));
        ROLA_CHECK(run_summary(*cfg, s, w, k, v, P_k, at<float>(ws, w.C), at<float>(ws, w.z),
                               at<__nv_bfloat16>(ws, w.Cbf), ws, st));
    }
    if (C_out)
        ROLA_TRY(cudaMemcpyAsync(C_out, at<float>(ws, w.C), sizeof(float) * (size_t)s.B * s.H * s.r * kDh,
                                 cudaMemcpyDeviceToDevice, st));
    void* os = o_s_out ? o_s_out : o;
    ROLA_TRY(mark(2));
    ROLA_TRY(launch_sparse_attn(cfg->dtype, s, at<void>(ws, w.qr), at<void>(ws, w.kr), sparse_v(s, w, v, ws), kv, os,
                                lse_out, at<DeviceStatus>(ws, w.status), st));
    ROLA_TRY(mark(3));
    ROLA_TRY(launch_lowrank_apply(cfg->dtype, s, q, P_q, at<float>(ws, w.C), at<__nv_bfloat16>(ws, w.Cbf), gate, os,
                                  o, at<float2>(ws, w.table), at<DeviceStatus>(ws, w.status), st));
    ROLA_TRY(mark(4));
    return ROLA_OK;
}


// Y = concat_h(O) W_o^T (+ b_o); `clear` clears the status word first (every entry point
// does; the block entry point keeps the forward's).
rola_status_t out_proj_impl(const rola_config_t* cfg, const void* O, const void* W_o, const float* b_o,
                            int32_t d_model, void* Y, void* ws, size_t ws_bytes, cudaStream_t st, bool clear)
{
    ROLA_CHECK(validate(cfg));
    if (!O || !W_o || !Y || d_model < 64 || d_model % 64 != 0) return ROLA_ERR_INVALID_ARG;
    if (!aligned16(O) || !aligned16(W_o) || !aligned16(Y) || (b_o && !aligned16(b_o))) return ROLA_ERR_INVALID_ARG;
    if ((int64_t)cfg->B * cfg->N * d_model > ((int64_t)1 << 40)) return ROLA_ERR_UNSUPPORTED;
    if (!ws || (reinterpret_cast<uintptr_t>(ws) & (kAlign - 1)) || ws_bytes < sizeof(DeviceStatus))
        return ROLA_ERR_WORKSPACE;
    if (clear) ROLA_TRY(cudaMemsetAsync(ws, 0, sizeof(DeviceStatus), st));
    const Shape s = make_shape(*cfg);
    if (cfg->dtype == ROLA_BF16)
        ROLA_TRY(launch_out_proj(cfg->B, cfg->N, cfg->H, d_model, O, W_o, b_o, Y, static_cast<DeviceStatus*>(ws),
                                 s.wait_limit_ns, st));
    else
        ROLA_TRY(launch_out_proj_f32(cfg->B, cfg->N, cfg->H, d_model, static_cast<const float*>(O),
                                     static_cast<const float*>(W_o), b_o, static_cast<float*>(Y), st));
    return ROLA_OK;
}

}  // namespace

extern "C" {

rola_status_t rola_config_init(rola_config_t* cfg)
{
    if (!cfg) return ROLA_ERR_INVALID_ARG;
    memset(cfg, 0, sizeof(*cfg));
    cfg->d_h = kDh;
    cfg->rope_split[0] = 44;
    cfg->rope_split[1] = 42;
    cfg->rope_split[2] = 42;
    cfg->rope_theta = 10000.0;
    cfg->block = kBlock;
    cfg->keep_ratio = 0.1f;
    cfg->r = 32;
    cfg->eps_lr = 1e-6f;
    cfg->eps_fuse = 1e-6f;
    cfg->gate_bias = -1.946f;
    cfg->dtype = ROLA_BF16;
    return ROLA_OK;
}

int32_t rola_num_blocks(const rola_config_t* cfg)
{
    if (validate(cfg) != ROLA_OK) return 0;
    return num_blocks_of(*cfg);
}

int32_t rola_num_query_blocks(const rola_config_t* cfg)
{
    if (validate(cfg) != ROLA_OK) return 0;
    return num_qblocks_of(*cfg);
}

int32_t rola_num_keep(const rola_config_t* cfg)
{
    if (validate(cfg) != ROLA_OK) return 0;
    return num_keep_of(*cfg);
}

size_t rola_workspace_bytes(const rola_config_t* cfg)
{
    if (validate(cfg) != ROLA_OK) return 0;
    return layout(*cfg).total;
}

rola_status_t rola_block_mask(const rola_config_t* cfg, const void* q, const void* k, int32_t* kv_idx, void* ws,
                              size_t ws_bytes, void* stream)
{
    ROLA_CHECK(validate(cfg));
    if (!q || !k || !kv_idx || !aligned16(q) || !aligned16(k) || !aligned16(kv_idx)) return ROLA_ERR_INVALID_ARG;
    ROLA_CHECK(check_ws(*cfg, ws, ws_bytes));
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    Workspace w = layout(*cfg);
    Shape s = make_shape(*cfg);
    ROLA_CHECK(prologue(*cfg, ws, w, st));
    return run_mask(*cfg, s, w, q, k, nullptr, kv_idx, ws, st);
}

rola_status_t rola_sparse_attn(const rola_config_t* cfg, const void* q, const void* k, const void* v,
                               const int32_t* kv_idx, void* o_s, void* ws, size_t ws_bytes, void* stream)
{
    ROLA_CHECK(validate(cfg));
    if (!q || !k || !v || !kv_idx || !o_s) return ROLA_ERR_INVALID_ARG;
    if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(kv_idx) || !aligned16(o_s))
        return ROLA_ERR_INVALID_ARG;
    ROLA_CHECK(check_ws(*cfg, ws, ws_bytes));
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    Workspace w = layout(*cfg);
    Shape s = make_shape(*cfg);
    ROLA_CHECK(prologue(*cfg, ws, w, st));
    // rotated copies in block order (the pooled means are a by-product here)
    ROLA_TRY(rope_pool(*cfg, s, w, q, k, v, ws, st));
    ROLA_TRY(launch_sparse_attn(cfg->dtype, s, at<void>(ws, w.qr), at<void>(ws, w.kr), sparse_v(s, w, v, ws), kv_idx,
                                o_s, nullptr, at<DeviceStatus>(ws, w.status), st));
    return ROLA_OK;
}

rola_status_t rola_lowrank_summary(const rola_config_t* cfg, const void* k, const void* v, const void* P_k, float* C,
                                   float* z, void* ws, size_t ws_bytes, void* stream)
{
    ROLA_CHECK(validate(cfg));
    if (!k || !v || !P_k || !C) return ROLA_ERR_INVALID_ARG;
    if (!aligned16(k) || !aligned16(v) || !aligned16(P_k) || !aligned16(C) || (z && !aligned16(z)))
        return ROLA_ERR_INVALID_ARG;
    ROLA_CHECK(check_ws(*cfg, ws, ws_bytes));
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    Workspace w = layout(*cfg);
    Shape s = make_shape(*cfg);
    ROLA_CHECK(prologue(*cfg, ws, w, st));
    return run_summary(*cfg, s, w, k, v, P_k, C, z, nullptr, ws, st);
}

rola_status_t rola_lowrank_apply(const rola_config_t* cfg, const void* q, const void* P_q, const float* C,
                                 const float* gate, const void* o_s, void* o, void* ws, size_t ws_bytes, void* stream)
{
    ROLA_CHECK(validate(cfg));
    if (!q || !P_q || !C || !o_s || !o) return ROLA_ERR_INVALID_ARG;
    if (!aligned16(q) || !aligned16(P_q) || !aligned16(C) || !aligned16(o_s) || !aligned16(o) ||
        (gate && (reinterpret_cast<uintptr_t>(gate) & 3u)))
        return ROLA_ERR_INVALID_ARG;
    ROLA_CHECK(check_ws(*cfg, ws, ws_bytes));
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    Workspace w = layout(*cfg);
    Shape s = make_shape(*cfg);
    ROLA_CHECK(prologue(*cfg, ws, w, st));
    __nv_bfloat16* Cbf = at<__nv_bfloat16>(ws, w.Cbf);
    if (cfg->dtype == ROLA_BF16) ROLA_TRY(launch_c_to_bf16(s, C, Cbf, st));
    ROLA_TRY(launch_lowrank_apply(cfg->dtype, s, q, P_q, C, Cbf, gate, o_s, o, at<float2>(ws, w.table),
                                  at<DeviceStatus>(ws, w.status), st));
    return ROLA_OK;
}

rola_status_t rola_forward_timed(const rola_config_t* cfg, const void* q, const void* k, const void* v,
                                 const void* P_q, const void* P_k, const float* gate, void* o, int32_t* kv_idx_out,
                                 void* ws, size_t ws_bytes, void* stream, void* const* stage_events)
{
    return forward_impl(cfg, q, k, v, P_q, P_k, gate, o, kv_idx_out, nullptr, nullptr, nullptr, ws, ws_bytes, stream,
                        stage_events);
}

rola_status_t rola_forward_train(const rola_config_t* cfg, const void* q, const void* k, const void* v,
                                 const void* P_q, const void* P_k, const float* gate, void* o, int32_t* kv_idx_out,
                                 void* o_s, float* lse, float* C, void* ws, size_t ws_bytes, void* stream)
{
    if (!kv_idx_out || !o_s || !lse || !C) return validate(cfg) == ROLA_OK ? ROLA_ERR_INVALID_ARG : validate(cfg);
    if (validate(cfg) == ROLA_OK && cfg->query_block == 128) return ROLA_ERR_UNSUPPORTED;   // no backward for it
    return forward_impl(cfg, q, k, v, P_q, P_k, gate, o, kv_idx_out, o_s, lse, C, ws, ws_bytes, stream, nullptr);
}

rola_status_t rola_forward(const rola_config_t* cfg, const void* q, const void* k, const void* v, const void* P_q,
                           const void* P_k, const float* gate, void* o, int32_t* kv_idx_out, void* ws,
                           size_t ws_bytes, void* stream)
{
    return rola_forward_timed(cfg, q, k, v, P_q, P_k, gate, o, kv_idx_out, ws, ws_bytes, stream, nullptr);
}

size_t rola_backward_workspace_bytes(const rola_config_t* cfg)
{
    if (validate(cfg) != ROLA_OK) return 0;
    return bwd_layout(*cfg).total;
}

rola_status_t rola_backward(const rola_config_t* cfg, const void* q, const void* k, const void* v, const void* P_q,
                            const void* P_k, const float* gate, const int32_t* kv_idx, const void* o_s,
                            const float* lse, const float* C, const void* dO, void* dq, void* dk, void* dv,
                            float* dP_q, float* dP_k, float* dgate, void* ws, size_t ws_bytes, void* stream)
{
    ROLA_CHECK(validate(cfg));
    if (cfg->query_block == 128) return ROLA_ERR_UNSUPPORTED;
    const void* in[] = {q, k, v, P_q, P_k, kv_idx, o_s, lse, C, dO, dq, dk, dv, dP_q, dP_k};
    for (const void* p : in)
        if (!p || !aligned16(p)) return ROLA_ERR_INVALID_ARG;
    if ((gate && (reinterpret_cast<uintptr_t>(gate) & 3u)) || (dgate && (reinterpret_cast<uintptr_t>(dgate) & 3u)))
        return ROLA_ERR_INVALID_ARG;
    const BwdWorkspace w = bwd_layout(*cfg);
    if (!ws || (reinterpret_cast<uintptr_t>(ws) & (kAlign - 1)) || ws_bytes < w.total) return ROLA_ERR_WORKSPACE;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const Shape s = make_shape(*cfg);
    ROLA_TRY(cudaMemsetAsync(at<uint8_t>(ws, w.status), 0, sizeof(DeviceStatus), st));
    ROLA_TRY(launch_rope_table(*cfg, at<float2>(ws, w.table), st));
    ROLA_TRY(launch_rope_pool(*cfg, s, q, k, s.cube ? v : nullptr, at<float2>(ws, w.table), at<void>(ws, w.qr),
                              at<void>(ws, w.kr), s.cube ? at<void>(ws, w.vp) : nullptr, at<float>(ws, w.qbar),
                              at<float>(ws, w.kbar), st));
    BackwardArgs a;
    a.q = q; a.k = k; a.v = v; a.P_q = P_q; a.P_k = P_k; a.o_s = o_s; a.dO = dO;
    a.C = C; a.gate = gate; a.lse = lse; a.kv_idx = kv_idx;
    a.tab = at<float2>(ws, w.table);
    a.qr = at<void>(ws, w.qr); a.kr = at<void>(ws, w.kr);
    a.dOs = at<void>(ws, w.dOs); a.Dv = at<float>(ws, w.Dv);
    a.dq_acc = at<float>(ws, w.dq); a.dk_acc = at<float>(ws, w.dk); a.dv_acc = at<float>(ws, w.dv);
    a.dg_h = at<float>(ws, w.dg);
    a.partC = at<float>(ws, w.partC); a.partPq = at<float>(ws, w.partPq); a.partPk = at<float>(ws, w.partPk);
    a.dC = at<float>(ws, w.dC);
    a.tr_off = at<int32_t>(ws, w.tr_off); a.tr_list = at<int32_t>(ws, w.tr_list);
    a.dq = dq; a.dk = dk; a.dv = dv; a.dP_q = dP_q; a.dP_k = dP_k; a.dgate = dgate;
    a.status = at<DeviceStatus>(ws, w.status);
    a.v_blk = s.cube ? at<void>(ws, w.vp) : v;
    a.dOs_blk = s.cube ? at<void>(ws, w.dOs_b) : nullptr;
    a.lse_blk = s.cube ? at<float>(ws, w.lse_b) : nullptr;
    a.Dv_blk = s.cube ? at<float>(ws, w.Dv_b) : nullptr;
    ROLA_TRY(launch_backward(cfg->dtype, s, a, st));
    return ROLA_OK;
}

rola_status_t rola_gate(const rola_config_t* cfg, const void* X, const void* w_g, float b_g, int32_t d_model,
                        float* gate, void* stream)
{
    ROLA_CHECK(validate(cfg));
    if (!X || !w_g || !gate || d_model < 8 || d_model % 8 != 0 || !isfinite(b_g)) return ROLA_ERR_INVALID_ARG;
    if (!aligned16(X) || !aligned16(w_g) || (reinterpret_cast<uintptr_t>(gate) & 3u)) return ROLA_ERR_INVALID_ARG;
    ROLA_TRY(launch_gate(cfg->dtype, (long long)cfg->B * cfg->N, d_model, X, w_g, b_g, gate,
                         static_cast<cudaStream_t>(stream)));
    return ROLA_OK;
}

rola_status_t rola_out_proj(const rola_config_t* cfg, const void* O, const void* W_o, const float* b_o,
                            int32_t d_model, void* Y, void* ws, size_t ws_bytes, void* stream)
{
    return out_proj_impl(cfg, O, W_o, b_o, d_model, Y, ws, ws_bytes, static_cast<cudaStream_t>(stream), true);
}

rola_status_t rola_attention_block(const rola_config_t* cfg, const void* X, const void* w_g, float b_g,
                                   int32_t d_model, const void* q, const void* k, const void* v, const void* P_q,
                                   const void* P_k, const void* W_o, const float* b_o, float* gate, void* o, void* Y,
                                   int32_t* kv_idx_out, void* ws, size_t ws_bytes, void* stream)
{
    ROLA_CHECK(validate(cfg));
    if (!gate || !o) return ROLA_ERR_INVALID_ARG;
    ROLA_CHECK(check_ws(*cfg, ws, ws_bytes));
    ROLA_CHECK(rola_gate(cfg, X, w_g, b_g, d_model, gate, stream));
    ROLA_CHECK(rola_forward(cfg, q, k, v, P_q, P_k, gate, o, kv_idx_out, ws, ws_bytes, stream));
    // the projection records into the status word the forward cleared, without clearing it again
    return out_proj_impl(cfg, o, W_o, b_o, d_model, Y, ws, ws_bytes, static_cast<cudaStream_t>(stream), false);
}

rola_status_t rola_get_device_status(const void* ws, void* stream)
{
    if (!ws) return ROLA_ERR_WORKSPACE;
    DeviceStatus h;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (cudaStreamSynchronize(st) != cudaSuccess) return ROLA_ERR_CUDA;
    if (cudaMemcpy(&h, ws, sizeof(h), cudaMemcpyDeviceToHost) != cudaSuccess) return ROLA_ERR_CUDA;
    return h.code == 0 ? ROLA_OK : static_cast<rola_status_t>(h.code);
}

const char* rola_status_string(rola_status_t status)
{
    switch (status) {
        case ROLA_OK: return "ROLA_OK";
        case ROLA_ERR_INVALID_ARG: return "ROLA_ERR_INVALID_ARG: bad pointer, shape, alignment or value";
        case ROLA_ERR_UNSUPPORTED: return "ROLA_ERR_UNSUPPORTED: configuration not built (d_h, block, r)";
        case ROLA_ERR_WORKSPACE: return "ROLA_ERR_WORKSPACE: workspace NULL, misaligned or too small";
        case ROLA_ERR_CUDA: return "ROLA_ERR_CUDA: a CUDA launch or runtime call failed";
        case ROLA_ERR_TIMEOUT: return "ROLA_ERR_TIMEOUT: a device-side bounded wait expired";
        default: return "unknown rola_status_t";
    }
}

}  // extern "C"
