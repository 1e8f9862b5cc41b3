/*
 * rola.h -- C ABI of the RoLA hybrid-attention library for one GB300 (sm_103a).
 *
 * RoLA ("Rotary-Positioned Low-Rank Linear Attention") replaces dense 3D-RoPE
 * self-attention in a video DiT layer with
 *   - a block-sparse softmax branch over the kept 64-token key blocks of each
 *     64-token query block (Alg. 1, sparse-branch steps; Sec. 3 for the
 *     softmax form), and
 *   - a low-rank linear-attention branch whose features are rotated by the
 *     truncated 3D RoPE *after* the SiLU feature map (Eq. qklr), so one
 *     summary C = sum_q k~_q v_q^T per head (Eq. ctx) serves every query,
 * merged by the RMS-referenced token gate of Eq. (gate).
 *
 * Conventions shared by every entry point
 *   Memory     every tensor pointer is a DEVICE pointer owned by the caller,
 *              16-byte aligned and densely packed in the layout stated.  The
 *              library allocates nothing and keeps no global mutable state;
 *              scratch lives in the caller's workspace (see
 *              rola_workspace_bytes).
 *   Element    q, k, v, o, o_s, P_q, P_k are bf16 when cfg->dtype ==
 *   types      ROLA_BF16 and fp32 when cfg->dtype == ROLA_FP32 (validation
 *              mode: fp32 arithmetic everywhere, no bf16/tf32 rounding).
 *              C, z and gate are always fp32; kv_idx is int32.
 *   Layouts    q, k, v, o_s, o : [B][H][N][d_h]
 *              P_q, P_k        : [H][r][d_h]   (one r x d_h projection per head)
 *              C               : [B][H][r][d_h]
 *              z               : [B][H][r]
 *              gate            : [B][N]        (one scalar per token, shared by heads)
 *              kv_idx          : [B][H][nQB][n_keep], ascending block ids
 *   Tokens     token n of the flattened video sits at (t, x, y) with
 *              t = n / (Hh*Ww), x = (n / Ww) % Hh, y = n % Ww (t-major), plus
 *              cfg->pos_offset (Sec. 3 notation).
 *   Inputs     q and k are the backbone's normalised, PRE-RoPE vectors
 *              (q^n, k^n of Sec. 4.1 / Alg. 1); the library applies both the
 *              full RoPE (sparse branch) and the truncated RoPE (low-rank
 *              branch) itself.
 *   Streams    `stream` is a cudaStream_t (NULL = legacy default stream).  All
 *              calls are asynchronous on it.  Calls that share a workspace
 *              must be ordered on one stream.
 *   Errors     argument validation happens on the host before any launch
 *              and returns ROLA_ERR_INVALID_ARG / ROLA_ERR_UNSUPPORTED /
 *              ROLA_ERR_WORKSPACE with nothing launched (UNSUPPORTED also
 *              for shapes past the kernels' limits: B*H > 65535, more than
 *              7008 blocks, B*H*nB*n_keep >= 2^31); a launch failure
 *              returns ROLA_ERR_CUDA.  A device-side bounded wait that gives
 *              up records ROLA_ERR_TIMEOUT in the workspace status word,
 *              which rola_get_device_status reads.  No C++ exception
 *              crosses this ABI.
 */
#ifndef ROLA_H_
#define ROLA_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    ROLA_OK = 0,
    ROLA_ERR_INVALID_ARG = 1,  /* bad pointer, shape, alignment or value */
    ROLA_ERR_UNSUPPORTED = 2,  /* valid but not built here (e.g. d_h != 128) */
    ROLA_ERR_WORKSPACE = 3,    /* workspace NULL, misaligned or too small */
    ROLA_ERR_CUDA = 4,         /* a CUDA launch or runtime call failed */
    ROLA_ERR_TIMEOUT = 5       /* a device-side bounded wait expired */
} rola_status_t;

typedef enum {
    ROLA_BF16 = 0,             /* bf16 storage, tensor-core MMAs, fp32 accumulation */
    ROLA_FP32 = 1              /* fp32 storage and fp32 arithmetic (validation mode) */
} rola_dtype_t;

/*
 * Layer configuration (plain old data).  Fill with rola_config_init, then
 * set the shape.  Defaults follow the paper where it gives a value and the
 * stated reading where it does not.
 */
typedef struct {
    int32_t B, H, N, d_h;      /* batch, heads, tokens, head dim (d_h == 128) */
    int32_t T, Hh, Ww;         /* latent grid; N == T*Hh*Ww (Sec. 3) */
    int32_t pos_offset[3];     /* added to (t, x, y); 0 normally */
    int32_t rope_split[3];     /* d_t, d_x, d_y; each even, sum == d_h (Sec. 3); default 44,42,42 */
    double rope_theta;         /* RoPE base; default 10000 */
    int32_t block;             /* block size for queries and keys; 64 */
    float keep_ratio;          /* n_keep = clamp(floor(keep_ratio*nKB + 0.5), 1, nKB) */
    int32_t r;                 /* low-rank width (Sec. 4.2), 8 <= r <= d_h, r % 8 == 0; the bf16
                                  kernels run at r rounded up to 16 with zero rows of P */
    float eps_lr;              /* RMSNorm epsilon of the low-rank readout; default 1e-6 */
    float eps_fuse;            /* epsilon of the sparse-output RMS r_p, Eq. (gate); default 1e-6 */
    float gate_bias;           /* g = sigmoid(gate_bias) when gate == NULL; default -1.946 */
    rola_dtype_t dtype;        /* ROLA_BF16 (default) or ROLA_FP32 */
    int32_t wait_limit_ms;     /* bound of every device-side wait (0 = 2000 ms); at most 60000 */
    int32_t debug_flags;       /* 0 normally.  ROLA_DEBUG_SKIP_FIRST_K_COPY makes each CTA of the
                                  bf16 sparse kernel skip its first K copy (of the bf16 backward
                                  kernels: the first K pair, the first Q / dO pair; of the bf16
                                  pre-pass: its first k, v, q load), so a bounded wait runs out
                                  and the call reports ROLA_ERR_TIMEOUT (tests the timeout path) */
    int32_t lowrank_rope;      /* where the truncated RoPE sits in the low-rank features; one of
                                  rola_lowrank_rope_t, default ROLA_LOWRANK_ROPE_OUTSIDE */
    int32_t lowrank_act;       /* feature map phi of the low-rank features; one of
                                  rola_lowrank_act_t, default ROLA_LOWRANK_ACT_SILU */
    int32_t block_geometry;    /* which tokens form a block of the sparse branch; one of
                                  rola_block_geometry_t, default ROLA_BLOCK_FLAT */
    int32_t query_block;       /* tokens per query block of the mask, ROLA_BLOCK_FLAT only: 0 or 64
                                  (the key blocks' size, default) or 128 -- each 128-token query chunk
                                  is pooled, scored and given its n_keep key blocks as one unit (the
                                  b_q = 128 / b_kv = 64 tiling of the block-sparse video attentions
                                  the paper builds on); the forward entry points only */
} rola_config_t;

#define ROLA_DEBUG_SKIP_FIRST_K_COPY 1

/*
 * Placement of the truncated rotation R_r in the low-rank features (the three
 * orderings the paper compares in its RoPE-placement study, Tab. mechanism):
 *   OUTSIDE  k~_q = R_r(q) SiLU(P_k k^n_q)   Eq. (qklr), the RoLA branch
 *   INSIDE   k~_q = SiLU(R_r(q) P_k k^n_q)   Prop. inside (App. inside): no
 *            exact relative factorisation, the summary leaks absolute position
 *   NONE     k~_q = SiLU(P_k k^n_q)          position-blind low-rank branch
 * and the same for q~_p.  The sparse branch always uses the full RoPE.
 */
typedef enum {
    ROLA_LOWRANK_ROPE_OUTSIDE = 0,
    ROLA_LOWRANK_ROPE_INSIDE = 1,
    ROLA_LOWRANK_ROPE_NONE = 2
} rola_lowrank_rope_t;

/*
 * Feature map phi of the low-rank branch (SiLU in Eq. qklr; the others are
 * the activation ablation, Tab. abl_activation), applied coordinatewise to
 * P x wherever SiLU appears in the formulas of this header:
 *   SILU      x / (1 + exp(-x))              the RoLA default
 *   IDENTITY  x                              plain (rotary) linear features
 *   TANH      tanh(x)
 *   RELU      max(x, 0)
 *   GELU      x Phi(x) = x (1 + erf(x / sqrt 2)) / 2   (the exact form)
 */
typedef enum {
    ROLA_LOWRANK_ACT_SILU = 0,
    ROLA_LOWRANK_ACT_IDENTITY = 1,
    ROLA_LOWRANK_ACT_TANH = 2,
    ROLA_LOWRANK_ACT_RELU = 3,
    ROLA_LOWRANK_ACT_GELU = 4
} rola_lowrank_act_t;

/*
 * Block geometry of the sparse branch (the paper does not describe it):
 *   FLAT  block i = tokens 64 i .. 64 i + 63 of the t-major sequence (the
 *         last block ragged); nQB = nKB = ceil(N / 64)
 *   CUBE  block i = the 4 x 4 x 4 cube (ct, cx, cy) of the latent grid,
 *         i = (ct * ceil(Hh/4) + cx) * ceil(Ww/4) + cy, holding the tokens
 *         (t, x, y) with t / 4 = ct, x / 4 = cx, y / 4 = cy (edge cubes hold
 *         fewer); nQB = nKB = ceil(T/4) ceil(Hh/4) ceil(Ww/4)
 * Block means, scores, kv_idx and the sparse branch all use the blocks of
 * the configured geometry; the low-rank branch does not depend on it.
 */
typedef enum {
    ROLA_BLOCK_FLAT = 0,
    ROLA_BLOCK_CUBE = 1
} rola_block_geometry_t;

/* Fill *cfg with defaults (shape fields zero).  Returns ROLA_ERR_INVALID_ARG on NULL. */
rola_status_t rola_config_init(rola_config_t* cfg);

/* The number of key blocks nKB: ceil(N / block), or the cube count for ROLA_BLOCK_CUBE; 0 if cfg
 * is invalid.  It is also the number of query blocks unless cfg->query_block is 128. */
int32_t rola_num_blocks(const rola_config_t* cfg);

/* The number of query blocks nQB, the rows of kv_idx: ceil(N / 128) when cfg->query_block is 128,
 * else rola_num_blocks(cfg); 0 if cfg is invalid. */
int32_t rola_num_query_blocks(const rola_config_t* cfg);

/* Kept key blocks per query block, clamp(floor(keep_ratio*nKB + 0.5), 1, nKB); 0 if cfg is invalid. */
int32_t rola_num_keep(const rola_config_t* cfg);

/* Bytes of workspace every entry point below accepts for this cfg (the
 * largest any of them needs); 0 if cfg is invalid.  The workspace must be
 * 256-byte aligned.  Its first bytes hold the device status word. */
size_t rola_workspace_bytes(const rola_config_t* cfg);

/*
 * Kernel (1): block mask.  Rotates q and k by the full 3D RoPE R(p)
 * (Sec. 3, Eq. shiftinv), mean-pools each block (of cfg->block_geometry)
 * over its tokens, scores every
 * (query block, key block) pair as q_bar . k_bar / sqrt(d_h) and keeps the
 * n_keep highest-scoring key blocks of each query block (Alg. 1, "topk
 * ratio"; the pooling / scoring rule is this library's reading of the
 * unspecified selection of the sparse engine).  Ties go to the lower block
 * id.  The selection turns floating point into integers, so it is an fp32
 * decision with every rounding fixed: the fp32 (cos, sin) table,
 * y0 = fma(x0, c, -fl(x1 s)), y1 = fma(x0, s, fl(x1 c)); a block's slots
 * (64, or 128 query tokens) summed pairwise in slot order, empty slots +0,
 * one division by its token count; each score an ascending-d fma chain from
 * +0 times fl(1/sqrt(d_h)).  Every kernel of this library evaluates it so.
 *   q, k    : [B][H][N][d_h] pre-RoPE, dtype
 *   kv_idx  : out, int32 [B][H][nQB][n_keep], ascending within each row
 */
rola_status_t rola_block_mask(const rola_config_t* cfg, const void* q, const void* k,
                              int32_t* kv_idx, void* ws, size_t ws_bytes, void* stream);

/*
 * Kernel (2): block-sparse softmax attention (Alg. 1, sparse branch):
 *   O^s_p = sum_{q in kept(i)} softmax_q(<R(p) q_p, R(q) k_q> / sqrt(d_h)) v_q
 * for p in query block i, over the key blocks kv_idx lists for block i.
 * Softmax is evaluated online in fp32.
 *   q, k, v : [B][H][N][d_h] (q, k pre-RoPE), dtype
 *   kv_idx  : int32 [B][H][nQB][n_keep], each row ascending, ids < nKB
 *   o_s     : out, [B][H][N][d_h], dtype
 */
rola_status_t rola_sparse_attn(const rola_config_t* cfg, const void* q, const void* k, const void* v,
                               const int32_t* kv_idx, void* o_s, void* ws, size_t ws_bytes,
                               void* stream);

/*
 * Kernel (3): low-rank summary, Eq. (qklr) and Eq. (ctx):
 *   k~_q = R_r(q) SiLU(P_k k^n_q),   C = sum_q k~_q v_q^T,   z = sum_q k~_q
 * (k~ as cfg->lowrank_rope places the rotation, with cfg->lowrank_act's feature map).
 * R_r keeps the first r coordinates (r/2 complete pairs) of the native RoPE
 * ordering (Sec. 4.2).  The reduction over N is split across CTAs (one
 * contiguous token range each) and combined in a fixed order, so results are
 * bitwise reproducible on a given GPU model (the split follows its SM count).
 *   k, v    : [B][H][N][d_h] (k pre-RoPE), dtype;  P_k : [H][r][d_h], dtype
 *   C       : out, fp32 [B][H][r][d_h];   z : out, fp32 [B][H][r], or NULL
 */
rola_status_t rola_lowrank_summary(const rola_config_t* cfg, const void* k, const void* v,
                                   const void* P_k, float* C, float* z, void* ws, size_t ws_bytes,
                                   void* stream);

/*
 * Kernel (4): low-rank readout and gated fusion, Eq. (ctx) and Eq. (gate):
 *   q~_p   = R_r(p) SiLU(P_q q^n_p)            (as cfg->lowrank_rope places R_r; SiLU or
 *                                               cfg->lowrank_act's feature map)
 *   O^lr_p = y_p / sqrt(mean_i y_{p,i}^2 + eps_lr),   y_p = q~_p^T C
 *   r_p    = sqrt(mean_i (O^s_{p,i})^2 + eps_fuse)
 *   O_p    = (O^s_p / r_p + g_p O^lr_p) r_p
 * q~ never leaves the chip.
 *   q       : [B][H][N][d_h] pre-RoPE, dtype;  P_q : [H][r][d_h], dtype
 *   C       : fp32 [B][H][r][d_h];  gate : fp32 [B][N] or NULL (sigmoid(gate_bias))
 *   o_s     : [B][H][N][d_h], dtype;  o : out, same layout, may alias o_s
 */
rola_status_t rola_lowrank_apply(const rola_config_t* cfg, const void* q, const void* P_q,
                                 const float* C, const float* gate, const void* o_s, void* o,
                                 void* ws, size_t ws_bytes, void* stream);

/*
 * The whole module (Alg. 1, the per-head steps between the QKV projection
 * and W_o): block mask, sparse branch, low-rank summary, readout and fusion.
 * In bf16 the rotation, the block pooling and the summary share one pass
 * over q, k and v; the mask, C and O are those of the separate entry points
 * (same arithmetic, same bits).
 *   o          : out, [B][H][N][d_h] fused per-head output O^fused, dtype
 *   kv_idx_out : out, the mask used (int32 [B][H][nQB][n_keep]), or NULL
 */
rola_status_t rola_forward(const rola_config_t* cfg, const void* q, const void* k, const void* v,
                           const void* P_q, const void* P_k, const float* gate, void* o,
                           int32_t* kv_idx_out, void* ws, size_t ws_bytes, void* stream);

/*
 * rola_forward for training: the same computation, keeping what rola_backward
 * reads.  kv_idx_out is required here.
 *   o_s : out, [B][H][N][d_h] sparse-branch output O^s, dtype (must not alias o)
 *   lse : out, fp32 [B][H][N], log sum_j exp(<q^r_p, k^r_j> / sqrt(d_h)) over the
 *         kept keys of each query row (natural log)
 *   C   : out, fp32 [B][H][r][d_h], the low-rank summary
 */
rola_status_t rola_forward_train(const rola_config_t* cfg, const void* q, const void* k, const void* v,
                                 const void* P_q, const void* P_k, const float* gate, void* o,
                                 int32_t* kv_idx_out, void* o_s, float* lse, float* C, void* ws,
                                 size_t ws_bytes, void* stream);

/* Bytes of workspace rola_backward needs (256-byte aligned); 0 if cfg is invalid. */
size_t rola_backward_workspace_bytes(const rola_config_t* cfg);

/*
 * Backward pass: the gradients of L = sum_p dO_p . O_p through the forward
 * pass under the block mask kv_idx (the top-k selection is piecewise constant,
 * so no gradient flows through it), for the single-stage fine-tune that trains
 * q, k, v (the backbone's projections), P_q, P_k and the gate (Sec. impl).
 * Undoes the fusion (Eq. gate), the RMSNorm readout and the summary (Eq. ctx),
 * the low-rank features (Eq. qklr, with the configured placement and map), the
 * block-sparse softmax attention and the full RoPE (Sec. 3), in that order.
 *   q, k, v, P_q, P_k, gate : the forward inputs
 *   kv_idx, o_s, lse, C     : what rola_forward_train returned for them
 *   dO      : [B][H][N][d_h], dtype
 *   dq, dk, dv : out, [B][H][N][d_h], dtype
 *   dP_q, dP_k : out, fp32 [H][r][d_h], summed over the batch
 *   dgate   : out, fp32 [B][N], dL/dg_p summed over the heads (for gate == NULL:
 *             the gradient at the constant sigmoid(gate_bias)), or NULL
 * bf16: tensor cores (tcgen05 for the block-sparse gradients, mma.sync for the
 * low-rank ones) with fp32 accumulation; fp32: fp32 arithmetic throughout.
 * Results are bitwise reproducible (fixed-order reductions).  Both block
 * geometries.
 */
rola_status_t rola_backward(const rola_config_t* cfg, const void* q, const void* k, const void* v,
                            const void* P_q, const void* P_k, const float* gate, const int32_t* kv_idx,
                            const void* o_s, const float* lse, const float* C, const void* dO, void* dq,
                            void* dk, void* dv, float* dP_q, float* dP_k, float* dgate, void* ws,
                            size_t ws_bytes, void* stream);

/*
 * rola_forward with stage timing: identical computation and launches, plus
 * cudaEventRecord(stage_events[i], stream) at five stage boundaries --
 *   [0] start  [1] after the block mask (fp32) or the fused pass over
 *   q, k, v (bf16: rotation, pooling, summary partials)  [2] after the
 *   low-rank summary (fp32) or the block scores, top-k and summary combine
 *   (bf16)  [3] after the sparse branch  [4] after the readout + fusion.
 * stage_events: array of 5 cudaEvent_t created by the caller (owned by the
 * caller), or NULL (then this is rola_forward).
 */
rola_status_t rola_forward_timed(const rola_config_t* cfg, const void* q, const void* k, const void* v,
                                 const void* P_q, const void* P_k, const float* gate, void* o,
                                 int32_t* kv_idx_out, void* ws, size_t ws_bytes, void* stream,
                                 void* const* stage_events);

/*
 * Token gate of the gated fusion (Sec. fusion; Alg. 1, token-wise scalar gate):
 *   g_p = sigmoid(x_p . w_g + b_g)
 * one scalar per token from the attention block's input hidden states; the
 * result is the `gate` argument of rola_forward / rola_lowrank_apply.
 *   X       : [B][N][d_model], cfg->dtype (bf16 or fp32);  w_g : [d_model], cfg->dtype
 *   b_g     : the gate bias (the paper initialises it to -1.946, so g starts near 1/8)
 *   gate    : out, fp32 [B][N]
 * d_model must be a multiple of 8 and at least 8; X and w_g 16-byte aligned.
 * Uses cfg->B, cfg->N and cfg->dtype; needs no workspace.  Accumulates in fp32.
 */
rola_status_t rola_gate(const rola_config_t* cfg, const void* X, const void* w_g, float b_g,
                        int32_t d_model, float* gate, void* stream);

/*
 * Output projection of the attention block (Alg. 1, last step, "merge heads,
 * output projection"): per token the heads' fused outputs are concatenated,
 * head-major, and multiplied by W_o:
 *   Y[b][n][f] = sum_{h,d} O[b][h][n][d] * W_o[f][128 h + d]  (+ b_o[f])
 *   O    : [B][H][N][128], cfg->dtype -- the output of rola_forward, read in
 *          place (the concatenation is the GEMM's K index, no copy is made)
 *   W_o  : [d_model][H*128], cfg->dtype (row f = output feature f, the
 *          nn.Linear weight layout)
 *   b_o  : [d_model] fp32, or NULL for no bias
 *   Y    : out, [B][N][d_model], cfg->dtype, caller-allocated
 *   ws   : at least 256 bytes, 256-byte aligned (the module's workspace will
 *          do); only its status word is used: cleared, then set to
 *          ROLA_ERR_TIMEOUT if a bounded device wait expires
 * d_model must be a positive multiple of 64; O, W_o, Y (and b_o) 16-byte
 * aligned.  bf16: tcgen05 tensor-core GEMM with fp32 accumulation in TMEM, one
 * bf16 rounding of each output; fp32: plain fp32 arithmetic (validation).
 * Uses cfg->B, H, N, dtype and wait_limit_ms.
 */
rola_status_t rola_out_proj(const rola_config_t* cfg, const void* O, const void* W_o, const float* b_o,
                            int32_t d_model, void* Y, void* ws, size_t ws_bytes, void* stream);

/*
 * The attention block after the QKV projection and the pre-RoPE norms
 * (Alg. 1 from the gate on): the token gate from the block input X
 * (rola_gate), the RoLA module on q, k, v (rola_forward, with that gate), and
 * the output projection (rola_out_proj), in this order on `stream`.
 *   X, w_g, b_g, d_model : as rola_gate (d_model also the width of Y and W_o)
 *   q, k, v, P_q, P_k    : as rola_forward
 *   W_o, b_o             : as rola_out_proj
 *   gate : out, fp32 [B][N], the gate values (caller-owned scratch)
 *   o    : out, [B][H][N][128], the module's per-head output
 *   Y    : out, [B][N][d_model]
 *   kv_idx_out : nullable, as rola_forward
 *   ws   : rola_workspace_bytes(cfg) bytes; rola_get_device_status(ws)
 *          afterwards covers the module and the projection
 */
rola_status_t rola_attention_block(const rola_config_t* cfg, const void* X, const void* w_g, float b_g,
                                   int32_t d_model, const void* q, const void* k, const void* v, const void* P_q,
                                   const void* P_k, const void* W_o, const float* b_o, float* gate, void* o, void* Y,
                                   int32_t* kv_idx_out, void* ws, size_t ws_bytes, void* stream);

/*
 * rola_lowrank_summary_static: the low-rank summary (C and optionally z, as
 * rola_lowrank_summary computes them) for callers that cannot give the
 * library any device scratch -- e.g. a plugin whose host framework owns the
 * allocator and hands the op only its inputs and outputs, or a runtime that
 * forbids device allocation once it is serving.  The paper has no
 * counterpart; this is a deployment variant of the entry point above.
 *
 * It takes no workspace and allocates nothing: its scratch (RoPE table and
 * split-N partial sums) is one file-scope __device__ array of 16 MiB that
 * every GPU loading the library holds until the process exits.  The first
 * call on a device looks up that array's device address and caches it; make
 * that first call before any stream capture.  Every call reuses the same
 * array, so calls whose executions overlap on the GPU (other streams, other
 * host threads) race and must be serialised by the caller.
 *   k, v, P_k, C, z : as rola_lowrank_summary (device pointers, caller-owned)
 * Returns ROLA_ERR_UNSUPPORTED when the layer's least scratch exceeds the
 * 16 MiB array: a 256-byte status word, the RoPE table of
 * (T + Hh + Ww) * 64 * 8 bytes rounded up to 256, and one partial slot per
 * head, B*H*4*(rp*128 + rp) bytes with rp = r rounded up to a multiple of 16;
 * the usual validation codes otherwise.  When the array cannot hold the
 * regular number of splits it uses fewer, so C may differ from
 * rola_lowrank_summary's in the last bits (same fixed-order sum, coarser split).
 * There is no status word for the caller to read: if a bounded device wait
 * of the bf16 kernel gives up (cfg->wait_limit_ms), C and z come back filled
 * with NaN.  ROLA_DEBUG_SKIP_FIRST_K_COPY makes every CTA of that kernel skip
 * its first load, so its waits run out (tests this path).
 */
rola_status_t rola_lowrank_summary_static(const rola_config_t* cfg, const void* k, const void* v,
                                          const void* P_k, float* C, float* z, void* stream);

/*
 * Synchronises `stream`, then reads the device status word at the start of
 * ws: ROLA_OK, or ROLA_ERR_TIMEOUT if a bounded device wait expired since the
 * workspace was last cleared by an entry point.  ROLA_ERR_CUDA if the
 * synchronisation or copy fails.
 */
rola_status_t rola_get_device_status(const void* ws, void* stream);

/* Static, human-readable name of a status code. */
const char* rola_status_string(rola_status_t status);

#ifdef __cplusplus
}
#endif

#endif /* ROLA_H_ */
