/*
 * RoLA hybrid attention -- plain fp64 CPU oracle.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the slow, obviously-correct
 * reference the CUDA library is checked against.  Only the tests, the smoke
 * check and the bench's CPU-baseline leg may load it; the product path never
 * does.  It shares no code, header, table or constant with the CUDA library.
 *
 * Every input arrives as float32 (an exact copy of the bf16 / fp32 device
 * inputs) and is upcast to double on read.  All arithmetic is fp64, each
 * step written in the order the paper states it, with no blocking, fusion
 * or reordering:
 *
 *   positions        Sec. 3 (Preliminary, notation): p = (t, x, y), token n
 *                    of the flattened video is t-major.
 *   full 3D RoPE     Sec. 3, Eq. (shiftinv): block-diagonal rotation R(p),
 *                    d_h = d_t + d_x + d_y, pairs (2m, 2m+1) (Sec. 4.5,
 *                    even/odd split), frequency theta^(-2i/d_axis).
 *   truncated RoPE   Sec. 4.2: R_r(p) keeps the first r coordinates (r/2
 *                    complete pairs) of the native ordering.
 *   block mask       Alg. 1 "SparseAttn ... with topk ratio"; the selection
 *                    rule itself is not given by the paper -- this oracle
 *                    mean-pools the rotated q / k over each block, scores
 *                    q_bar . k_bar / sqrt(d_h) and keeps the n_keep largest
 *                    per query block (ties -> lower block index).
 *   block geometry   not described by the paper either: contiguous chunks of
 *                    `block` tokens of the t-major sequence (geometry 0), or
 *                    4 x 4 x 4 cubes of the (t, x, y) latent grid (geometry
 *                    1, the tiling of the sparse video attentions the paper
 *                    builds on), numbered t-major over the cube grid; edge
 *                    cubes hold the tokens that fall inside the grid.
 *                    Geometry 0 may also give the query side longer chunks
 *                    (qblock, e.g. 128 queries against 64-token key blocks,
 *                    the b_q / b_kv tiling of those attentions): each query
 *                    block is pooled, scored and given its n_keep key blocks
 *                    as one unit.
 *   sparse branch    Sec. 3 (softmax(QK^T / sqrt d_h) V) restricted to the
 *                    kept key blocks; Alg. 1 sparse-branch steps.
 *   low-rank branch  Eq. (qklr): q~ = R_r(p) SiLU(P_q q^n), k~ = R_r(q)
 *                    SiLU(P_k k^n); Eq. (ctx): C = sum_q k~_q v_q^T,
 *                    O^lr = RMSNorm(q~^T C) with no gain.
 *   fusion           Eq. (gate): r_p = sqrt(mean_i O^s_{p,i}^2 + eps),
 *                    O = (O^s / r_p + g_p O^lr) r_p.
 *   variants         Prop. (inside): SiLU(R_r(p) P x) ("inside"), and the
 *                    no-RoPE ablation (Sec. 5.2) SiLU(P x); the feature map
 *                    of the activation ablation (Tab. abl_activation):
 *                    SiLU (default), identity, tanh, ReLU, GELU (the exact
 *                    x Phi(x) form; the paper does not say which GELU).
 *
 * Layouts: q, k, v, o: [B][H][N][d_h]; P_q, P_k: [H][r][d_h];
 * C: [B][H][r][d_h]; z: [B][H][r]; gate: [B][N] (NULL -> sigmoid(gate_bias));
 * kv_idx: [B][H][nQB][n_keep] ascending, nQB the query blocks (the key
 * blocks unless qblock is set).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

typedef struct {
    int32_t B, H, N, dh;
    int32_t T, Hh, Ww;
    int32_t pos_offset[3];
    int32_t split[3];
    double theta;
    int32_t block;
    double keep;          /* keep ratio; n_keep = clamp(floor(keep*nKB+0.5), 1, nKB) */
    int32_t r;
    double eps_lr, eps_f;
    double gate_bias;     /* g = sigmoid(gate_bias) when gate == NULL */
    int32_t rope_mode;    /* 0: RoPE outside SiLU (RoLA), 1: inside, 2: none */
    int32_t act;          /* 0: SiLU, 1: identity, 2: tanh, 3: ReLU, 4: GELU */
    int32_t geometry;     /* 0: contiguous chunks of `block` tokens, 1: 4x4x4 cubes */
    int32_t qblock;       /* geometry 0: tokens per query block (0: `block`); the key
                             blocks keep `block` tokens.  Ignored by geometry 1. */
} orc_cfg;

enum { CUBE = 4 };        /* cube edge of geometry 1 (CUBE^3 == block == 64) */

/* ------------------------------------------------------------------ */
/* sizes                                                              */
/* ------------------------------------------------------------------ */

int orc_num_blocks(const orc_cfg* c)
{
    if (c->geometry == 1)
        return ((c->T + CUBE - 1) / CUBE) * ((c->Hh + CUBE - 1) / CUBE) * ((c->Ww + CUBE - 1) / CUBE);
    return (c->N + c->block - 1) / c->block;
}

/* The block token n belongs to: its chunk n / block, or its cube
 * (t / 4, x / 4, y / 4) numbered t-major over the cube grid. */
int orc_block_of(const orc_cfg* c, int n)
{
    if (c->geometry != 1) return n / c->block;
    int t = n / (c->Hh * c->Ww), x = (n / c->Ww) % c->Hh, y = n % c->Ww;
    int nx = (c->Hh + CUBE - 1) / CUBE, ny = (c->Ww + CUBE - 1) / CUBE;
    return ((t / CUBE) * nx + x / CUBE) * ny + y / CUBE;
}

/* Query blocks.  The block-sparse video attentions the paper builds on
 * tile the query side more coarsely than the key side (b_q = 128 queries
 * against b_kv = 64 keys); with qblock set, the query blocks of geometry 0
 * are contiguous chunks of qblock tokens: pooled, scored and given their
 * n_keep key blocks as one unit.  Otherwise they are the key blocks. */
static int qblock_size(const orc_cfg* c)
{
    return (c->geometry != 1 && c->qblock > 0) ? c->qblock : c->block;
}

int orc_num_qblocks(const orc_cfg* c)
{
    if (c->geometry == 1) return orc_num_blocks(c);
    int qb = qblock_size(c);
    return (c->N + qb - 1) / qb;
}

int orc_qblock_of(const orc_cfg* c, int n)
{
    if (c->geometry == 1) return orc_block_of(c, n);
    return n / qblock_size(c);
}

/* Members of every query block, ascending: list[b * qblock_size + i], i < cnt[b]. */
static void qblock_members(const orc_cfg* c, int* list, int* cnt)
{
    int nQ = orc_num_qblocks(c), qb = qblock_size(c);
    for (int b = 0; b < nQ; ++b) cnt[b] = 0;
    for (int n = 0; n < c->N; ++n) {
        int b = orc_qblock_of(c, n);
        list[(size_t)b * qb + cnt[b]++] = n;
    }
}

/* Members of every block in ascending token order: list[b * block + i] for
 * i < cnt[b] (a block never holds more than `block` tokens). */
static void block_members(const orc_cfg* c, int* list, int* cnt)
{
    int nB = orc_num_blocks(c);
    for (int b = 0; b < nB; ++b) cnt[b] = 0;
    for (int n = 0; n < c->N; ++n) {
        int b = orc_block_of(c, n);
        list[(size_t)b * c->block + cnt[b]++] = n;
    }
}

int orc_num_keep(const orc_cfg* c)
{
    int nkb = orc_num_blocks(c);
    double x = floor(c->keep * (double)nkb + 0.5);
    int n = (int)x;
    if (n < 1) n = 1;
    if (n > nkb) n = nkb;
    return n;
}

/* ------------------------------------------------------------------ */
/* positions and RoPE (Sec. 3, Sec. 4.2)                              */
/* ------------------------------------------------------------------ */

/* token n -> (t, x, y), t-major flattening, plus the configured offset. */
void orc_position(const orc_cfg* c, int n, double pos[3])
{
    int hw = c->Hh * c->Ww;
    int t = n / hw;
    int x = (n / c->Ww) % c->Hh;
    int y = n % c->Ww;
    pos[0] = (double)(t + c->pos_offset[0]);
    pos[1] = (double)(x + c->pos_offset[1]);
    pos[2] = (double)(y + c->pos_offset[2]);
}

/* Rotation angle of pair m (coordinates 2m, 2m+1) at position pos. */
double orc_pair_angle(const orc_cfg* c, int m, const double pos[3])
{
    int pt = c->split[0] / 2, px = c->split[1] / 2;
    int axis, i, d_axis;
    if (m < pt) { axis = 0; i = m; d_axis = c->split[0]; }
    else if (m < pt + px) { axis = 1; i = m - pt; d_axis = c->split[1]; }
    else { axis = 2; i = m - pt - px; d_axis = c->split[2]; }
    double freq = pow(c->theta, -2.0 * (double)i / (double)d_axis);
    return pos[axis] * freq;
}

/* Turn the first npairs coordinate pairs of in by the angles whose (cos, sin)
 * are cs[2m], cs[2m+1]; coordinates beyond 2*npairs are copied unchanged.
 * in / out of length len may alias. */
static void rotate_pairs(int npairs, const double* cs, const double* in, double* out, int len)
{
    for (int m = 0; m < npairs; ++m) {
        double ca = cs[2 * m], sa = cs[2 * m + 1];
        double x = in[2 * m], y = in[2 * m + 1];
        out[2 * m] = x * ca - y * sa;
        out[2 * m + 1] = x * sa + y * ca;
    }
    for (int i = 2 * npairs; i < len; ++i) out[i] = in[i];
}

/* (cos, sin) of every pair angle at position pos: cs[2m], cs[2m+1], m < dh/2. */
static void pair_cs(const orc_cfg* c, const double pos[3], double* cs)
{
    for (int m = 0; m < c->dh / 2; ++m) {
        double a = orc_pair_angle(c, m, pos);
        cs[2 * m] = cos(a);
        cs[2 * m + 1] = sin(a);
    }
}

/* out = R(pos) restricted to the first 2*npairs coordinates, applied to in. */
void orc_rotate(const orc_cfg* c, int npairs, const double pos[3], const double* in,
                double* out, int len)
{
    double* cs = (double*)malloc(sizeof(double) * (size_t)c->dh);
    pair_cs(c, pos, cs);
    rotate_pairs(npairs, cs, in, out, len);
    free(cs);
}

/* The same (cos, sin) for every token position, computed once per call:
 * tcs[n*dh + 2m + {0,1}]. */
static double* token_cs(const orc_cfg* c)
{
    double* tcs = (double*)malloc(sizeof(double) * (size_t)c->N * c->dh);
#pragma omp parallel for schedule(static)
    for (int n = 0; n < c->N; ++n) {
        double pos[3];
        orc_position(c, n, pos);
        pair_cs(c, pos, tcs + (size_t)n * c->dh);
    }
    return tcs;
}

static double silu(double x) { return x / (1.0 + exp(-x)); }

/* The feature map phi of Eq. (qklr): SiLU by default, or one of the
 * activations of the ablation (Tab. abl_activation).  GELU is x * Phi(x)
 * with Phi the standard normal CDF, Phi(x) = (1 + erf(x / sqrt 2)) / 2. */
double orc_activation(const orc_cfg* c, double x)
{
    switch (c->act) {
        case 1: return x;
        case 2: return tanh(x);
        case 3: return x > 0.0 ? x : 0.0;
        case 4: return 0.5 * x * (1.0 + erf(x / sqrt(2.0)));
        default: return silu(x);
    }
}

/* ------------------------------------------------------------------ */
/* low-rank features, Eq. (qklr) and its two ablations                */
/* ------------------------------------------------------------------ */

/* feat[r] for one token: cs its pair (cos, sin), x [dh] (float input), P [r][dh] (one head). */
static void lowrank_feature(const orc_cfg* c, const double* cs, const float* x, const float* P,
                            double* feat)
{
    int r = c->r, dh = c->dh;
    double* u = (double*)malloc(sizeof(double) * (size_t)r);
    for (int a = 0; a < r; ++a) {
        double s = 0.0;
        for (int d = 0; d < dh; ++d) s += (double)P[(size_t)a * dh + d] * (double)x[d];
        u[a] = s;
    }
    if (c->rope_mode == 0) {            /* R_r(p) phi(P x) */
        for (int a = 0; a < r; ++a) u[a] = orc_activation(c, u[a]);
        rotate_pairs(r / 2, cs, u, feat, r);
    } else if (c->rope_mode == 1) {     /* phi(R_r(p) P x) */
        rotate_pairs(r / 2, cs, u, feat, r);
        for (int a = 0; a < r; ++a) feat[a] = orc_activation(c, feat[a]);
    } else {                            /* phi(P x) */
        for (int a = 0; a < r; ++a) feat[a] = orc_activation(c, u[a]);
    }
    free(u);
}

/* Low-rank features of every token of every head: out [B][H][N][r]. */
void orc_lowrank_features(const orc_cfg* c, const float* x, const float* P, double* out)
{
    int BH = c->B * c->H;
    double* tcs = token_cs(c);
#pragma omp parallel for schedule(dynamic, 1)
    for (int bh = 0; bh < BH; ++bh) {
        int h = bh % c->H;
        for (int n = 0; n < c->N; ++n)
            lowrank_feature(c, tcs + (size_t)n * c->dh, x + ((size_t)bh * c->N + n) * c->dh,
                            P + (size_t)h * c->r * c->dh, out + ((size_t)bh * c->N + n) * c->r);
    }
    free(tcs);
}

/* ------------------------------------------------------------------ */
/* summary C = sum_q k~_q v_q^T and z = sum_q k~_q, Eq. (ctx)         */
/* ------------------------------------------------------------------ */

void orc_lowrank_summary(const orc_cfg* c, const float* k, const float* v, const float* Pk,
                         double* C, double* z)
{
    int BH = c->B * c->H, r = c->r, dh = c->dh;
    double* tcs = token_cs(c);
#pragma omp parallel for schedule(dynamic, 1)
    for (int bh = 0; bh < BH; ++bh) {
        int h = bh % c->H;
        double* Cb = C + (size_t)bh * r * dh;
        double* zb = z ? z + (size_t)bh * r : NULL;
        double* kt = (double*)malloc(sizeof(double) * (size_t)r);
        memset(Cb, 0, sizeof(double) * (size_t)r * dh);
        if (zb) memset(zb, 0, sizeof(double) * (size_t)r);
        for (int n = 0; n < c->N; ++n) {
            lowrank_feature(c, tcs + (size_t)n * dh, k + ((size_t)bh * c->N + n) * dh,
                            Pk + (size_t)h * r * dh, kt);
            const float* vn = v + ((size_t)bh * c->N + n) * dh;
            for (int a = 0; a < r; ++a) {
                for (int d = 0; d < dh; ++d) Cb[(size_t)a * dh + d] += kt[a] * (double)vn[d];
                if (zb) zb[a] += kt[a];
            }
        }
        free(kt);
    }
    free(tcs);
}

/* ------------------------------------------------------------------ */
/* readout, RMSNorm and fusion, Eq. (ctx) and Eq. (gate)             */
/* ------------------------------------------------------------------ */

static double gate_value(const orc_cfg* c, const float* gate, int b, int n)
{
    if (gate) return (double)gate[(size_t)b * c->N + n];
    return 1.0 / (1.0 + exp(-c->gate_bias));
}

/* O^lr for token n of head bh into olr[dh]; y (pre-RMSNorm) into y if non-NULL. */
static void lowrank_readout(const orc_cfg* c, const double* tcs, int bh, int n, const float* q,
                            const float* Pq, const double* C, double* olr, double* y)
{
    int r = c->r, dh = c->dh, h = bh % c->H;
    double* qt = (double*)malloc(sizeof(double) * (size_t)r);
    double* yy = (double*)malloc(sizeof(double) * (size_t)dh);
    lowrank_feature(c, tcs + (size_t)n * dh, q + ((size_t)bh * c->N + n) * dh, Pq + (size_t)h * r * dh, qt);
    const double* Cb = C + (size_t)bh * r * dh;
    double ss = 0.0;
    for (int d = 0; d < dh; ++d) {
        double s = 0.0;
        for (int a = 0; a < r; ++a) s += qt[a] * Cb[(size_t)a * dh + d];
        yy[d] = s;
        ss += s * s;
    }
    double inv = 1.0 / sqrt(ss / (double)dh + c->eps_lr);
    for (int d = 0; d < dh; ++d) {
        if (olr) olr[d] = yy[d] * inv;
        if (y) y[d] = yy[d];
    }
    free(qt);
    free(yy);
}

/* Fusion of one token: o_s [dh] (double), olr [dh], gate g -> out [dh]. */
static void fuse(const orc_cfg* c, const double* os, const double* olr, double g, double* out)
{
    int dh = c->dh;
    double ss = 0.0;
    for (int d = 0; d < dh; ++d) ss += os[d] * os[d];
    double rp = sqrt(ss / (double)dh + c->eps_f);
    for (int d = 0; d < dh; ++d) out[d] = (os[d] / rp + g * olr[d]) * rp;
}

/* Token list helper: the tokens of the selected query blocks (all if NULL). */
static int token_in_selection(const orc_cfg* c, int n, const uint8_t* qb_sel)
{
    return qb_sel == NULL || qb_sel[orc_qblock_of(c, n)];
}

/* O = fusion(O^s, RMSNorm(q~^T C)) for the tokens of the selected query
 * blocks (qb_sel[nQB] flags, NULL = all).  o_s is float [B][H][N][dh]. */
void orc_lowrank_apply(const orc_cfg* c, const float* q, const float* Pq, const double* C,
                       const float* gate, const float* o_s, const uint8_t* qb_sel, double* o)
{
    int BH = c->B * c->H, dh = c->dh;
    double* tcs = token_cs(c);
#pragma omp parallel for schedule(dynamic, 1)
    for (int bh = 0; bh < BH; ++bh) {
        int b = bh / c->H;
        double* olr = (double*)malloc(sizeof(double) * (size_t)dh);
        double* os = (double*)malloc(sizeof(double) * (size_t)dh);
        for (int n = 0; n < c->N; ++n) {
            if (!token_in_selection(c, n, qb_sel)) continue;
            size_t off = ((size_t)bh * c->N + n) * dh;
            lowrank_readout(c, tcs, bh, n, q, Pq, C, olr, NULL);
            for (int d = 0; d < dh; ++d) os[d] = (double)o_s[off + d];
            fuse(c, os, olr, gate_value(c, gate, b, n), o + off);
        }
        free(olr);
        free(os);
    }
    free(tcs);
}

/* Pre-RMSNorm readout y_p = q~_p^T C for every token: y [B][H][N][dh]. */
void orc_lowrank_readout(const orc_cfg* c, const float* q, const float* Pq, const double* C, double* y)
{
    int BH = c->B * c->H;
    double* tcs = token_cs(c);
#pragma omp parallel for schedule(dynamic, 1)
    for (int bh = 0; bh < BH; ++bh)
        for (int n = 0; n < c->N; ++n)
            lowrank_readout(c, tcs, bh, n, q, Pq, C, NULL, y + ((size_t)bh * c->N + n) * c->dh);
    free(tcs);
}

/* Explicit O(N^2) form of the pre-RMSNorm low-rank output,
 * y_p = sum_q (q~_p . k~_q) v_q  (Prop. exact, Step 2, read right to left). */
void orc_lowrank_explicit(const orc_cfg* c, const float* q, const float* k, const float* v,
                          const float* Pq, const float* Pk, double* y)
{
    int BH = c->B * c->H, r = c->r, dh = c->dh, N = c->N;
    double* tcs = token_cs(c);
#pragma omp parallel for schedule(dynamic, 1)
    for (int bh = 0; bh < BH; ++bh) {
        int h = bh % c->H;
        double* kt = (double*)malloc(sizeof(double) * (size_t)N * r);
        double* qt = (double*)malloc(sizeof(double) * (size_t)r);
        for (int n = 0; n < N; ++n)
            lowrank_feature(c, tcs + (size_t)n * dh, k + ((size_t)bh * N + n) * dh,
                            Pk + (size_t)h * r * dh, kt + (size_t)n * r);
        for (int p = 0; p < N; ++p) {
            lowrank_feature(c, tcs + (size_t)p * dh, q + ((size_t)bh * N + p) * dh,
                            Pq + (size_t)h * r * dh, qt);
            double* yp = y + ((size_t)bh * N + p) * dh;
            for (int d = 0; d < dh; ++d) yp[d] = 0.0;
            for (int n = 0; n < N; ++n) {
                double w = 0.0;
                for (int a = 0; a < r; ++a) w += qt[a] * kt[(size_t)n * r + a];
                const float* vn = v + ((size_t)bh * N + n) * dh;
                for (int d = 0; d < dh; ++d) yp[d] += w * (double)vn[d];
            }
        }
        free(kt);
        free(qt);
    }
    free(tcs);
}

/* ------------------------------------------------------------------ */
/* full RoPE of q / k for the sparse branch (Alg. 1, sparse steps)    */
/* ------------------------------------------------------------------ */

/* Rotated copy of x [B][H][N][dh] into xr (double). */
void orc_rope_full(const orc_cfg* c, const float* x, double* xr)
{
    int BH = c->B * c->H, dh = c->dh;
    double* tcs = token_cs(c);
#pragma omp parallel for schedule(dynamic, 1)
    for (int bh = 0; bh < BH; ++bh) {
        double* tmp = (double*)malloc(sizeof(double) * (size_t)dh);
        for (int n = 0; n < c->N; ++n) {
            size_t off = ((size_t)bh * c->N + n) * dh;
            for (int d = 0; d < dh; ++d) tmp[d] = (double)x[off + d];
            rotate_pairs(dh / 2, tcs + (size_t)n * dh, tmp, xr + off, dh);
        }
        free(tmp);
    }
    free(tcs);
}

/* ------------------------------------------------------------------ */
/* block mask: pooled scores + per-row top-n_keep                     */
/* ------------------------------------------------------------------ */

typedef struct { double s; int j; } scored;

static int cmp_scored(const void* a, const void* b)
{
    const scored* x = (const scored*)a;
    const scored* y = (const scored*)b;
    if (x->s > y->s) return -1;
    if (x->s < y->s) return 1;
    return (x->j < y->j) ? -1 : (x->j > y->j);   /* ties: lower block first */
}

static int cmp_int(const void* a, const void* b)
{
    int x = *(const int*)a, y = *(const int*)b;
    return (x > y) - (x < y);
}

/*
 * Block mask.  Outputs (any may be NULL except kv_idx):
 *   kv_idx [B][H][nQB][n_keep]   kept key blocks, ascending
 *   scores [B][H][nQB][nKB]      s_ij = q_bar_i . k_bar_j / sqrt(dh)
 *   gap    [B][H][nQB]           s_(n_keep) - s_(n_keep+1) in descending order
 *                                (+inf when n_keep == nKB)
 *   tau    [B][H][nQB]           twice the largest, over the row, of a
 *                                rigorous bound on |s32 - s| for the fp32
 *                                evaluation of orc_block_mask_f32 (u = 2^-24),
 *                                two scores entering every comparison.  A row
 *                                with gap > tau keeps the same set in fp32 and
 *                                in exact arithmetic; a row with gap <= tau is
 *                                a near-tie row, where the fp32 decision may
 *                                keep another valid set.
 *
 * The bound, per score, first order in u with a relative slack of 2^-12 for
 * the higher-order terms (Higham, Accuracy and Stability of Numerical
 * Algorithms, Sec. 3.1 and 4.2): a rotated coordinate y = x0 c - x1 s is off
 * by at most 3u (|x0| + |x1|) (c and s rounded once each, one product, one
 * fma); a pairwise sum over L levels adds gamma_L sum |y|; the division adds
 * u; so a pooled mean is off by at most (L + 4) u M_d, M_d the pooled
 * |x0| + |x1| of coordinate d's pair.  The d_h-term fma chain adds
 * gamma_dh sum |q_bar_d k_bar_d|, the scale (rounded once, one product) 2u of
 * |s|.  With a1 = sum |q_bar_d| |k_bar_d| and a2 = sum (M^q_d |k_bar_d| +
 * |q_bar_d| M^k_d):  |s32 - s| <= u ((d_h + 2) a1 + (L + 4) a2) / sqrt(d_h).
 */
void orc_block_mask(const orc_cfg* c, const float* q, const float* k, int32_t* kv_idx,
                    double* scores, double* gap, double* tau)
{
    int BH = c->B * c->H, dh = c->dh, N = c->N, bs = c->block;
    int nB = orc_num_blocks(c), nk = orc_num_keep(c);
    int nQ = orc_num_qblocks(c), qbs = qblock_size(c);
    int pool = qbs > bs ? qbs : bs;                         /* most slots a pooled mean sums */
    int levels = 0;                                         /* pairwise-summation depth, ceil(log2 pool) */
    while ((1 << levels) < pool) ++levels;
    double isd = 1.0 / sqrt((double)dh);
    const double u = ldexp(1.0, -24);
    double* tcs = token_cs(c);
    int* members = (int*)malloc(sizeof(int) * (size_t)nB * bs);
    int* count = (int*)malloc(sizeof(int) * (size_t)nB);
    int* qmembers = (int*)malloc(sizeof(int) * (size_t)nQ * qbs);
    int* qcount = (int*)malloc(sizeof(int) * (size_t)nQ);
    block_members(c, members, count);
    qblock_members(c, qmembers, qcount);
#pragma omp parallel for schedule(dynamic, 1)
    for (int bh = 0; bh < BH; ++bh) {
        size_t nbd = (size_t)nB * dh, nqd = (size_t)nQ * dh;
        double* qb = (double*)calloc(nqd, sizeof(double));   /* pooled means */
        double* kb = (double*)calloc(nbd, sizeof(double));
        double* qa = (double*)calloc(nqd, sizeof(double));   /* pooled |pair| magnitudes */
        double* ka = (double*)calloc(nbd, sizeof(double));
        double* xr = (double*)malloc(sizeof(double) * (size_t)dh);
        double* xi = (double*)malloc(sizeof(double) * (size_t)dh);
        scored* row = (scored*)malloc(sizeof(scored) * (size_t)nB);
        for (int which = 0; which < 2; ++which) {
            const float* x = which == 0 ? q : k;
            double* mean = which == 0 ? qb : kb;
            double* mag = which == 0 ? qa : ka;
            const int nblk = which == 0 ? nQ : nB;
            const int* cntv = which == 0 ? qcount : count;
            for (int n = 0; n < N; ++n) {
                size_t off = ((size_t)bh * N + n) * dh;
                for (int d = 0; d < dh; ++d) xi[d] = (double)x[off + d];
                rotate_pairs(dh / 2, tcs + (size_t)n * dh, xi, xr, dh);
                int blk = which == 0 ? orc_qblock_of(c, n) : orc_block_of(c, n);
                for (int d = 0; d < dh; ++d) {
                    mean[(size_t)blk * dh + d] += xr[d];
                    mag[(size_t)blk * dh + d] += fabs(xi[d & ~1]) + fabs(xi[d | 1]);
                }
            }
            for (int blk = 0; blk < nblk; ++blk) {
                int cnt = cntv[blk];
                for (int d = 0; d < dh; ++d) {
                    mean[(size_t)blk * dh + d] /= (double)cnt;
                    mag[(size_t)blk * dh + d] /= (double)cnt;
                }
            }
        }
        for (int i = 0; i < nQ; ++i) {
            const double* qi = qb + (size_t)i * dh;
            const double* qm = qa + (size_t)i * dh;
            double tmax = 0.0;
            for (int j = 0; j < nB; ++j) {
                const double* kj = kb + (size_t)j * dh;
                const double* km = ka + (size_t)j * dh;
                double s = 0.0, a1 = 0.0, a2 = 0.0;
                for (int d = 0; d < dh; ++d) {
                    s += qi[d] * kj[d];
                    a1 += fabs(qi[d]) * fabs(kj[d]);
                    a2 += qm[d] * fabs(kj[d]) + fabs(qi[d]) * km[d];
                }
                row[j].s = s * isd;
                row[j].j = j;
                if (scores) scores[((size_t)bh * nQ + i) * nB + j] = s * isd;
                /* per operand: rotation 3u, pairwise pooling over `levels`
                 * levels, one divide; dot product over dh terms; scale 2u. */
                double e = u * ((double)(dh + 2) * a1 + (double)(levels + 4) * a2) * isd * (1.0 + ldexp(1.0, -12));
                if (e > tmax) tmax = e;
            }
            qsort(row, (size_t)nB, sizeof(scored), cmp_scored);
            int32_t* out = kv_idx + ((size_t)bh * nQ + i) * nk;
            for (int t = 0; t < nk; ++t) out[t] = row[t].j;
            qsort(out, (size_t)nk, sizeof(int32_t), cmp_int);
            if (gap) gap[(size_t)bh * nQ + i] = nk < nB ? row[nk - 1].s - row[nk].s : INFINITY;
            if (tau) tau[(size_t)bh * nQ + i] = 2.0 * tmax;
        }
        free(qb); free(kb); free(qa); free(ka); free(xr); free(xi); free(row);
    }
    free(tcs);
    free(members);
    free(count);
    free(qmembers);
    free(qcount);
}

/*
 * The block mask as an fp32 decision.  Keeping the n_keep largest scores turns
 * floating-point values into integers, so the checker takes that decision in
 * the precision the CUDA path takes it in, fp32, with every rounding fixed by
 * the following evaluation (the definition above, step by step, in fp32):
 *   table    (c, s) of a pair: the fp64 cos / sin of the fp64 pair angle of
 *            orc_pair_angle, each rounded once to fp32;
 *   rotate   y0 = fma(x0, c, -(x1 s)), y1 = fma(x0, s, x1 c): each product
 *            and each fma rounded to fp32;
 *   pool     pairwise summation (Higham, Accuracy and Stability of Numerical
 *            Algorithms, Sec. 4.2) of the block's slots in slot order:
 *            sum(x[0..n)) = sum(x[0..h)) + sum(x[h..n)), h = floor(n/2), the
 *            slots being
 *            the `block` (query side: qblock) positions of a chunk, or the
 *            CUBE^3 positions 16 dt + 4 dx + dy of a cube; a slot outside the
 *            sequence or the grid holds +0.  Then one fp32 division by the
 *            number of tokens the block holds;
 *   score    an fp32 fma chain over d = 0, 1, ..., d_h - 1 starting from +0,
 *            then one fp32 product with the fp32 rounding of 1/sqrt(d_h);
 *   select   the n_keep largest of a row, ties to the lower block index
 *            (+0 and -0 are equal), listed ascending.
 * Outputs: kv_idx [B][H][nQB][n_keep]; scores32 [B][H][nQB][nKB] (may be
 * NULL), the fp32 scores widened to double.
 */
static float pairwise_f32(const float* x, int n)
{
    if (n == 1) return x[0];
    return pairwise_f32(x, n / 2) + pairwise_f32(x + n / 2, n - n / 2);
}

/* Token held by slot i of block b (-1: an empty slot); query side when qside. */
static int slot_token(const orc_cfg* c, int b, int i, int qside)
{
    if (c->geometry == 1) {
        int cubes_x = (c->Hh + CUBE - 1) / CUBE;          /* cube grid, t-major numbering */
        int cubes_y = (c->Ww + CUBE - 1) / CUBE;
        int ct = b / (cubes_x * cubes_y), cx = (b / cubes_y) % cubes_x, cy = b % cubes_y;
        int t = CUBE * ct + i / (CUBE * CUBE), x = CUBE * cx + (i / CUBE) % CUBE, y = CUBE * cy + i % CUBE;
        if (t >= c->T || x >= c->Hh || y >= c->Ww) return -1;
        return (t * c->Hh + x) * c->Ww + y;
    }
    int size = qside ? qblock_size(c) : c->block;
    int n = b * size + i;
    return n < c->N ? n : -1;
}

typedef struct { float s; int j; } scored32;

static int cmp_scored32(const void* a, const void* b)
{
    const scored32* x = (const scored32*)a;
    const scored32* y = (const scored32*)b;
    if (x->s > y->s) return -1;
    if (x->s < y->s) return 1;
    return (x->j > y->j) - (x->j < y->j);
}

void orc_block_mask_f32(const orc_cfg* c, const float* q, const float* k, int32_t* kv_idx, double* scores32)
{
    int BH = c->B * c->H, dh = c->dh, N = c->N;
    int nB = orc_num_blocks(c), nk = orc_num_keep(c), nQ = orc_num_qblocks(c);
    int kslots = c->geometry == 1 ? CUBE * CUBE * CUBE : c->block;
    int qslots = c->geometry == 1 ? kslots : qblock_size(c);
    const float scale = (float)(1.0 / sqrt((double)dh));
    /* the fp32 (cos, sin) of every pair at every token */
    float* tab = (float*)malloc(sizeof(float) * (size_t)N * dh);
#pragma omp parallel for schedule(static)
    for (int n = 0; n < N; ++n) {
        double pos[3];
        orc_position(c, n, pos);
        for (int m = 0; m < dh / 2; ++m) {
            double a = orc_pair_angle(c, m, pos);
            tab[(size_t)n * dh + 2 * m] = (float)cos(a);
            tab[(size_t)n * dh + 2 * m + 1] = (float)sin(a);
        }
    }
#pragma omp parallel for schedule(dynamic, 1)
    for (int bh = 0; bh < BH; ++bh) {
        float* qbar = (float*)malloc(sizeof(float) * (size_t)nQ * dh);
        float* kbar = (float*)malloc(sizeof(float) * (size_t)nB * dh);
        int maxslots = qslots > kslots ? qslots : kslots;
        float* col = (float*)malloc(sizeof(float) * (size_t)maxslots * dh);   /* [slot][d] rotated rows */
        scored32* row = (scored32*)malloc(sizeof(scored32) * (size_t)nB);
        for (int which = 0; which < 2; ++which) {
            const float* x = which == 0 ? q : k;
            float* mean = which == 0 ? qbar : kbar;
            int nblk = which == 0 ? nQ : nB, slots = which == 0 ? qslots : kslots;
            float* vals = (float*)malloc(sizeof(float) * (size_t)slots);
            for (int b = 0; b < nblk; ++b) {
                int cnt = 0;
                for (int i = 0; i < slots; ++i) {
                    int n = slot_token(c, b, i, which == 0);
                    float* yr = col + (size_t)i * dh;
                    if (n < 0) {
                        for (int d = 0; d < dh; ++d) yr[d] = 0.0f;
                        continue;
                    }
                    ++cnt;
                    const float* xn = x + ((size_t)bh * N + n) * dh;
                    const float* cs = tab + (size_t)n * dh;
                    for (int m = 0; m < dh / 2; ++m) {
                        float x0 = xn[2 * m], x1 = xn[2 * m + 1], cm = cs[2 * m], sm = cs[2 * m + 1];
                        float p1 = x1 * sm, p2 = x1 * cm;
                        yr[2 * m] = fmaf(x0, cm, -p1);
                        yr[2 * m + 1] = fmaf(x0, sm, p2);
                    }
                }
                for (int d = 0; d < dh; ++d) {
                    for (int i = 0; i < slots; ++i) vals[i] = col[(size_t)i * dh + d];
                    mean[(size_t)b * dh + d] = pairwise_f32(vals, slots) / (float)cnt;
                }
            }
            free(vals);
        }
        for (int i = 0; i < nQ; ++i) {
            const float* qi = qbar + (size_t)i * dh;
            for (int j = 0; j < nB; ++j) {
                const float* kj = kbar + (size_t)j * dh;
                float acc = 0.0f;
                for (int d = 0; d < dh; ++d) acc = fmaf(qi[d], kj[d], acc);
                row[j].s = acc * scale;
                row[j].j = j;
                if (scores32) scores32[((size_t)bh * nQ + i) * nB + j] = (double)row[j].s;
            }
            qsort(row, (size_t)nB, sizeof(scored32), cmp_scored32);
            int32_t* out = kv_idx + ((size_t)bh * nQ + i) * nk;
            for (int t = 0; t < nk; ++t) out[t] = row[t].j;
            qsort(out, (size_t)nk, sizeof(int32_t), cmp_int);
        }
        free(qbar); free(kbar); free(col); free(row);
    }
    free(tab);
}

/* ------------------------------------------------------------------ */
/* block-sparse softmax attention                                     */
/* ------------------------------------------------------------------ */

/* O^s for the tokens of the selected query blocks (qb_sel flags, NULL =
 * all).  qr, kr: rotated q / k (double) [B][H][N][dh]; v float; kv_idx
 * [B][H][nQB][n_keep]; o_s out double [B][H][N][dh] (rows outside the
 * selection untouched). */
void orc_sparse_attn(const orc_cfg* c, const double* qr, const double* kr, const float* v,
                     const int32_t* kv_idx, int n_keep, const uint8_t* qb_sel, double* o_s)
{
    int BH = c->B * c->H, dh = c->dh, N = c->N, bs = c->block;
    int nB = orc_num_blocks(c), nQ = orc_num_qblocks(c), qbs = qblock_size(c);
    double isd = 1.0 / sqrt((double)dh);
    int ntask = BH * nQ;
    int* members = (int*)malloc(sizeof(int) * (size_t)nB * bs);
    int* count = (int*)malloc(sizeof(int) * (size_t)nB);
    int* qmembers = (int*)malloc(sizeof(int) * (size_t)nQ * qbs);
    int* qcount = (int*)malloc(sizeof(int) * (size_t)nQ);
    block_members(c, members, count);
    qblock_members(c, qmembers, qcount);
#pragma omp parallel for schedule(dynamic, 1)
    for (int task = 0; task < ntask; ++task) {
        int bh = task / nQ, i = task % nQ;
        if (qb_sel && !qb_sel[i]) continue;
        const int32_t* kept = kv_idx + ((size_t)bh * nQ + i) * n_keep;
        int nkeys = 0;
        for (int t = 0; t < n_keep; ++t) nkeys += count[kept[t]];
        int* keys = (int*)malloc(sizeof(int) * (size_t)nkeys);
        double* s = (double*)malloc(sizeof(double) * (size_t)nkeys);
        int kk = 0;
        for (int t = 0; t < n_keep; ++t)
            for (int m = 0; m < count[kept[t]]; ++m) keys[kk++] = members[(size_t)kept[t] * bs + m];
        for (int mi = 0; mi < qcount[i]; ++mi) {
            int p = qmembers[(size_t)i * qbs + mi];
            const double* qp = qr + ((size_t)bh * N + p) * dh;
            double mx = -INFINITY;
            for (int t = 0; t < nkeys; ++t) {
                const double* kq = kr + ((size_t)bh * N + keys[t]) * dh;
                double acc = 0.0;
                for (int d = 0; d < dh; ++d) acc += qp[d] * kq[d];
                s[t] = acc * isd;
                if (s[t] > mx) mx = s[t];
            }
            double den = 0.0;
            for (int t = 0; t < nkeys; ++t) { s[t] = exp(s[t] - mx); den += s[t]; }
            double* op = o_s + ((size_t)bh * N + p) * dh;
            for (int d = 0; d < dh; ++d) op[d] = 0.0;
            for (int t = 0; t < nkeys; ++t) {
                const float* vq = v + ((size_t)bh * N + keys[t]) * dh;
                double w = s[t] / den;
                for (int d = 0; d < dh; ++d) op[d] += w * (double)vq[d];
            }
        }
        free(keys);
        free(s);
    }
    free(members);
    free(count);
    free(qmembers);
    free(qcount);
}

/* ------------------------------------------------------------------ */
/* full forward (Alg. 1, the per-head steps between QKV and W_o)      */
/* ------------------------------------------------------------------ */

/*
 * o [B][H][N][dh] for the tokens of the selected query blocks.  The mask is
 * computed here (kv_idx_out receives it if non-NULL), unless mask_override is
 * given.  Intermediates (o_s_out, C_out, z_out) are returned when non-NULL.
 */
void orc_forward(const orc_cfg* c, const float* q, const float* k, const float* v,
                 const float* Pq, const float* Pk, const float* gate,
                 const int32_t* mask_override, const uint8_t* qb_sel,
                 double* o, int32_t* kv_idx_out, double* o_s_out, double* C_out, double* z_out)
{
    size_t nel = (size_t)c->B * c->H * c->N * c->dh;
    int nQ = orc_num_qblocks(c), nk = orc_num_keep(c);
    size_t nmask = (size_t)c->B * c->H * nQ * nk;
    int32_t* mask = (int32_t*)malloc(sizeof(int32_t) * nmask);
    if (mask_override) memcpy(mask, mask_override, sizeof(int32_t) * nmask);
    else orc_block_mask(c, q, k, mask, NULL, NULL, NULL);
    if (kv_idx_out) memcpy(kv_idx_out, mask, sizeof(int32_t) * nmask);

    double* qr = (double*)malloc(sizeof(double) * nel);
    double* kr = (double*)malloc(sizeof(double) * nel);
    orc_rope_full(c, q, qr);
    orc_rope_full(c, k, kr);
    double* os = (double*)calloc(nel, sizeof(double));
    orc_sparse_attn(c, qr, kr, v, mask, nk, qb_sel, os);
    free(qr);
    free(kr);

    size_t nC = (size_t)c->B * c->H * c->r * c->dh;
    double* C = (double*)malloc(sizeof(double) * nC);
    double* z = (double*)malloc(sizeof(double) * (size_t)c->B * c->H * c->r);
    orc_lowrank_summary(c, k, v, Pk, C, z);

    int BH = c->B * c->H, dh = c->dh;
    double* tcs = token_cs(c);
#pragma omp parallel for schedule(dynamic, 1)
    for (int bh = 0; bh < BH; ++bh) {
        int b = bh / c->H;
        double* olr = (double*)malloc(sizeof(double) * (size_t)dh);
        for (int n = 0; n < c->N; ++n) {
            if (!token_in_selection(c, n, qb_sel)) continue;
            size_t off = ((size_t)bh * c->N + n) * dh;
            lowrank_readout(c, tcs, bh, n, q, Pq, C, olr, NULL);
            fuse(c, os + off, olr, gate_value(c, gate, b, n), o + off);
        }
        free(olr);
    }
    free(tcs);
    if (o_s_out) memcpy(o_s_out, os, sizeof(double) * nel);
    if (C_out) memcpy(C_out, C, sizeof(double) * nC);
    if (z_out) memcpy(z_out, z, sizeof(double) * (size_t)c->B * c->H * c->r);
    free(os);
    free(C);
    free(z);
    free(mask);
}

/* ------------------------------------------------------------------ */
/* backward pass: the gradients of the single-stage fine-tune         */
/* (Sec. impl, post-training: q, k, v, P_q, P_k and the gate train)   */
/* ------------------------------------------------------------------ */

/* phi'(x) of the configured feature map (the derivatives of the maps of
 * orc_activation; Phi' is the standard normal density). */
double orc_activation_grad(const orc_cfg* c, double x)
{
    switch (c->act) {
        case 1: return 1.0;
        case 2: { double t = tanh(x); return 1.0 - t * t; }
        case 3: return x > 0.0 ? 1.0 : 0.0;
        case 4: return 0.5 * (1.0 + erf(x / sqrt(2.0))) + x * exp(-0.5 * x * x) / sqrt(2.0 * acos(-1.0));
        default: { double sg = 1.0 / (1.0 + exp(-x)); return sg * (1.0 + x * (1.0 - sg)); }
    }
}

/* R^T on the first npairs pairs (the rotation by the opposite angles). */
static void rotate_pairs_t(int npairs, const double* cs, const double* in, double* out, int len)
{
    for (int m = 0; m < npairs; ++m) {
        double ca = cs[2 * m], sa = cs[2 * m + 1];
        double x = in[2 * m], y = in[2 * m + 1];
        out[2 * m] = x * ca + y * sa;
        out[2 * m + 1] = -x * sa + y * ca;
    }
    for (int i = 2 * npairs; i < len; ++i) out[i] = in[i];
}

/* Backward of one token's features: given df [r] = dL/d(feature), add
 * P^T du to dx [dh] and du x^T to dP [r][dh], du = dL/d(P x). */
static void lowrank_feature_bwd(const orc_cfg* c, const double* cs, const float* x, const float* P,
                                const double* df, double* dx, double* dP)
{
    int r = c->r, dh = c->dh;
    double* u = (double*)malloc(sizeof(double) * (size_t)r);
    double* w = (double*)malloc(sizeof(double) * (size_t)r);
    double* du = (double*)malloc(sizeof(double) * (size_t)r);
    for (int a = 0; a < r; ++a) {
        double sum = 0.0;
        for (int d = 0; d < dh; ++d) sum += (double)P[(size_t)a * dh + d] * (double)x[d];
        u[a] = sum;
    }
    if (c->rope_mode == 0) {            /* f = R_r phi(u):  du = phi'(u) (R_r^T df) */
        rotate_pairs_t(r / 2, cs, df, w, r);
        for (int a = 0; a < r; ++a) du[a] = orc_activation_grad(c, u[a]) * w[a];
    } else if (c->rope_mode == 1) {     /* f = phi(R_r u):  du = R_r^T (phi'(R_r u) df) */
        rotate_pairs(r / 2, cs, u, w, r);
        for (int a = 0; a < r; ++a) w[a] = orc_activation_grad(c, w[a]) * df[a];
        rotate_pairs_t(r / 2, cs, w, du, r);
    } else {                            /* f = phi(u) */
        for (int a = 0; a < r; ++a) du[a] = orc_activation_grad(c, u[a]) * df[a];
    }
    for (int a = 0; a < r; ++a)
        for (int d = 0; d < dh; ++d) {
            dx[d] += (double)P[(size_t)a * dh + d] * du[a];
            dP[(size_t)a * dh + d] += du[a] * (double)x[d];
        }
    free(u);
    free(w);
    free(du);
}

/*
 * Gradients of L = sum_p dO_p . O_p for the forward pass under the block mask
 * kv_idx (the top-k selection is piecewise constant in q and k, so nothing
 * flows through it): dq, dk, dv [B][H][N][dh]; dPq, dPk [H][r][dh] summed over
 * the batch; dgate [B][N] = dL/dg_p summed over the heads (also when gate is
 * NULL, for the constant g = sigmoid(gate_bias)).  The steps undo the forward
 * steps in reverse order: fusion, RMSNorm readout, features of q, summary,
 * features of k, block-sparse softmax attention, full RoPE.
 */
void orc_backward(const orc_cfg* c, const float* q, const float* k, const float* v, const float* Pq,
                  const float* Pk, const float* gate, const int32_t* kv_idx, const float* dO, double* dq,
                  double* dk, double* dv, double* dPq, double* dPk, double* dgate)
{
    int B = c->B, H = c->H, N = c->N, dh = c->dh, r = c->r, bs = c->block, BH = c->B * c->H;
    int nB = orc_num_blocks(c), nk = orc_num_keep(c);
    double isd = 1.0 / sqrt((double)dh);
    size_t nel = (size_t)BH * N * dh, nrd = (size_t)r * dh;
    /* forward quantities the chain rule needs */
    double* qr = (double*)malloc(sizeof(double) * nel);
    double* kr = (double*)malloc(sizeof(double) * nel);
    double* os = (double*)calloc(nel, sizeof(double));
    double* C = (double*)malloc(sizeof(double) * (size_t)BH * nrd);
    orc_rope_full(c, q, qr);
    orc_rope_full(c, k, kr);
    orc_sparse_attn(c, qr, kr, v, kv_idx, nk, NULL, os);
    orc_lowrank_summary(c, k, v, Pk, C, NULL);
    double* tcs = token_cs(c);
    int* members = (int*)malloc(sizeof(int) * (size_t)nB * bs);
    int* count = (int*)malloc(sizeof(int) * (size_t)nB);
    block_members(c, members, count);
    int nQ = orc_num_qblocks(c), qbs = qblock_size(c);
    int* qmembers = (int*)malloc(sizeof(int) * (size_t)nQ * qbs);
    int* qcount = (int*)malloc(sizeof(int) * (size_t)nQ);
    qblock_members(c, qmembers, qcount);
    double* dPq_bh = (double*)calloc((size_t)BH * nrd, sizeof(double));
    double* dPk_bh = (double*)calloc((size_t)BH * nrd, sizeof(double));
    double* dg_bh = (double*)calloc((size_t)BH * N, sizeof(double));
    memset(dq, 0, sizeof(double) * nel);
    memset(dk, 0, sizeof(double) * nel);
    memset(dv, 0, sizeof(double) * nel);
#pragma omp parallel for schedule(dynamic, 1)
    for (int bh = 0; bh < BH; ++bh) {
        int b = bh / H, h = bh % H;
        size_t head = (size_t)bh * N * dh;
        const double* Cb = C + (size_t)bh * nrd;
        double* dOs = (double*)calloc((size_t)N * dh, sizeof(double));
        double* dqr = (double*)calloc((size_t)N * dh, sizeof(double));
        double* dkr = (double*)calloc((size_t)N * dh, sizeof(double));
        double* dC = (double*)calloc(nrd, sizeof(double));
        double* olr = (double*)malloc(sizeof(double) * (size_t)dh);
        double* y = (double*)malloc(sizeof(double) * (size_t)dh);
        double* dy = (double*)malloc(sizeof(double) * (size_t)dh);
        double* ft = (double*)malloc(sizeof(double) * (size_t)r);
        double* dft = (double*)malloc(sizeof(double) * (size_t)r);
        /* fusion O = (O^s / r_p + g O^lr) r_p and readout O^lr = y / rho, y = q~^T C */
        for (int p = 0; p < N; ++p) {
            const double* osp = os + head + (size_t)p * dh;
            const float* dop = dO + head + (size_t)p * dh;
            double g = gate_value(c, gate, b, p);
            lowrank_readout(c, tcs, bh, p, q, Pq, C, olr, y);
            double ss = 0.0, yy = 0.0, a = 0.0;
            for (int d = 0; d < dh; ++d) {
                ss += osp[d] * osp[d];
                yy += y[d] * y[d];
                a += olr[d] * (double)dop[d];
            }
            double rp = sqrt(ss / (double)dh + c->eps_f);
            double rho = sqrt(yy / (double)dh + c->eps_lr);
            double dr = g * a;                          /* dL/dr_p */
            dg_bh[(size_t)bh * N + p] = rp * a;         /* dL/dg_p from this head */
            double od = 0.0;                            /* O^lr . dL/dO^lr */
            for (int d = 0; d < dh; ++d) {
                dOs[(size_t)p * dh + d] = (double)dop[d] + dr * osp[d] / ((double)dh * rp);
                od += olr[d] * g * rp * (double)dop[d];
            }
            for (int d = 0; d < dh; ++d) dy[d] = (g * rp * (double)dop[d] - olr[d] * od / (double)dh) / rho;
            lowrank_feature(c, tcs + (size_t)p * dh, q + head + (size_t)p * dh, Pq + (size_t)h * nrd, ft);
            for (int aa = 0; aa < r; ++aa) {
                double sum = 0.0;
                for (int d = 0; d < dh; ++d) {
                    sum += Cb[(size_t)aa * dh + d] * dy[d];
                    dC[(size_t)aa * dh + d] += ft[aa] * dy[d];
                }
                dft[aa] = sum;
            }
            lowrank_feature_bwd(c, tcs + (size_t)p * dh, q + head + (size_t)p * dh, Pq + (size_t)h * nrd, dft,
                                dq + head + (size_t)p * dh, dPq_bh + (size_t)bh * nrd);
        }
        /* summary C = sum_j k~_j v_j^T */
        for (int j = 0; j < N; ++j) {
            const float* vj = v + head + (size_t)j * dh;
            lowrank_feature(c, tcs + (size_t)j * dh, k + head + (size_t)j * dh, Pk + (size_t)h * nrd, ft);
            for (int aa = 0; aa < r; ++aa) {
                double sum = 0.0;
                for (int d = 0; d < dh; ++d) {
                    sum += dC[(size_t)aa * dh + d] * (double)vj[d];
                    dv[head + (size_t)j * dh + d] += ft[aa] * dC[(size_t)aa * dh + d];
                }
                dft[aa] = sum;
            }
            lowrank_feature_bwd(c, tcs + (size_t)j * dh, k + head + (size_t)j * dh, Pk + (size_t)h * nrd, dft,
                                dk + head + (size_t)j * dh, dPk_bh + (size_t)bh * nrd);
        }
        /* block-sparse softmax attention: s = q^r k^r / sqrt(d_h), P = softmax(s), O^s = P v */
        for (int i = 0; i < nQ; ++i) {
            const int32_t* kept = kv_idx + ((size_t)bh * nQ + i) * nk;
            int nkeys = 0;
            for (int t = 0; t < nk; ++t) nkeys += count[kept[t]];
            int* keys = (int*)malloc(sizeof(int) * (size_t)nkeys);
            double* pr = (double*)malloc(sizeof(double) * (size_t)nkeys);
            double* dpr = (double*)malloc(sizeof(double) * (size_t)nkeys);
            int kk = 0;
            for (int t = 0; t < nk; ++t)
                for (int m = 0; m < count[kept[t]]; ++m) keys[kk++] = members[(size_t)kept[t] * bs + m];
            for (int mi = 0; mi < qcount[i]; ++mi) {
                int p = qmembers[(size_t)i * qbs + mi];
                const double* qp = qr + head + (size_t)p * dh;
                const double* dop = dOs + (size_t)p * dh;
                double mx = -INFINITY;
                for (int t = 0; t < nkeys; ++t) {
                    const double* kq = kr + head + (size_t)keys[t] * dh;
                    double acc = 0.0;
                    for (int d = 0; d < dh; ++d) acc += qp[d] * kq[d];
                    pr[t] = acc * isd;
                    if (pr[t] > mx) mx = pr[t];
                }
                double den = 0.0;
                for (int t = 0; t < nkeys; ++t) { pr[t] = exp(pr[t] - mx); den += pr[t]; }
                double Dp = 0.0;                        /* sum_t P_t dP_t */
                for (int t = 0; t < nkeys; ++t) {
                    pr[t] /= den;
                    const float* vq = v + head + (size_t)keys[t] * dh;
                    double acc = 0.0;
                    for (int d = 0; d < dh; ++d) acc += dop[d] * (double)vq[d];
                    dpr[t] = acc;
                    Dp += pr[t] * acc;
                }
                for (int t = 0; t < nkeys; ++t) {
                    int j = keys[t];
                    double dsv = pr[t] * (dpr[t] - Dp) * isd;     /* dL/d(q^r . k^r) */
                    const double* kq = kr + head + (size_t)j * dh;
                    for (int d = 0; d < dh; ++d) {
                        dqr[(size_t)p * dh + d] += dsv * kq[d];
                        dkr[(size_t)j * dh + d] += dsv * qp[d];
                        dv[head + (size_t)j * dh + d] += pr[t] * dop[d];
                    }
                }
            }
            free(keys);
            free(pr);
            free(dpr);
        }
        /* full RoPE: dq += R(p)^T dq^r, dk += R(p)^T dk^r */
        for (int n = 0; n < N; ++n) {
            rotate_pairs_t(dh / 2, tcs + (size_t)n * dh, dqr + (size_t)n * dh, dy, dh);
            for (int d = 0; d < dh; ++d) dq[head + (size_t)n * dh + d] += dy[d];
            rotate_pairs_t(dh / 2, tcs + (size_t)n * dh, dkr + (size_t)n * dh, dy, dh);
            for (int d = 0; d < dh; ++d) dk[head + (size_t)n * dh + d] += dy[d];
        }
        free(dOs); free(dqr); free(dkr); free(dC); free(olr); free(y); free(dy); free(ft); free(dft);
    }
    memset(dPq, 0, sizeof(double) * (size_t)H * nrd);
    memset(dPk, 0, sizeof(double) * (size_t)H * nrd);
    for (int bh = 0; bh < BH; ++bh)
        for (size_t e = 0; e < nrd; ++e) {
            dPq[(size_t)(bh % H) * nrd + e] += dPq_bh[(size_t)bh * nrd + e];
            dPk[(size_t)(bh % H) * nrd + e] += dPk_bh[(size_t)bh * nrd + e];
        }
    for (int b = 0; b < B; ++b)
        for (int p = 0; p < N; ++p) {
            double sum = 0.0;
            for (int h = 0; h < H; ++h) sum += dg_bh[((size_t)b * H + h) * N + p];
            dgate[(size_t)b * N + p] = sum;
        }
    free(qr); free(kr); free(os); free(C); free(tcs); free(members); free(count);
    free(qmembers); free(qcount);
    free(dPq_bh); free(dPk_bh); free(dg_bh);
}

/* Token gate of the gated fusion (Sec. fusion, Alg. 1 "token-wise scalar
 * gate"): g_p = sigmoid(x_p . w_g + b_g), one scalar per token from the
 * attention block's input hidden state x_p (d_model wide).  X is [B][N][D],
 * w [D], g [B][N]. */
void orc_gate(int B, int N, int D, const float* X, const float* w, double b, double* g)
{
#pragma omp parallel for schedule(static)
    for (long p = 0; p < (long)B * N; ++p) {
        const float* x = X + (size_t)p * D;
        double logit = b;
        for (int d = 0; d < D; ++d) logit += (double)x[d] * (double)w[d];
        g[p] = 1.0 / (1.0 + exp(-logit));
    }
}

/* Output projection (Alg. 1, last step, "merge heads, output projection"):
 * the heads' fused outputs are concatenated per token, o_cat[n] =
 * (O^fused_1[n], ..., O^fused_H[n]) (length H * dh, head-major), and
 * Y[b][n][f] = sum_k o_cat[n][k] W[f][k] (+ bias[f]).  O is [B][H][N][dh]
 * (double), W [d_model][H * dh] (the row of output feature f), bias
 * [d_model] or NULL, Y [B][N][d_model].  Only the tokens with rows[n] != 0
 * are computed (rows NULL: all); the others are left untouched. */
void orc_out_proj(int B, int N, int H, int dh, int d_model, const double* O, const float* W, const float* bias,
                  const uint8_t* rows, double* Y)
{
    int K = H * dh;
#pragma omp parallel for schedule(dynamic, 16)
    for (long p = 0; p < (long)B * N; ++p) {
        int b = (int)(p / N), n = (int)(p % N);
        if (rows && !rows[n]) continue;
        double* cat = (double*)malloc(sizeof(double) * (size_t)K);
        for (int h = 0; h < H; ++h)
            for (int d = 0; d < dh; ++d) cat[h * dh + d] = O[(((size_t)b * H + h) * N + n) * dh + d];
        for (int f = 0; f < d_model; ++f) {
            double y = bias ? (double)bias[f] : 0.0;
            for (int k = 0; k < K; ++k) y += cat[k] * (double)W[(size_t)f * K + k];
            Y[(size_t)p * d_model + f] = y;
        }
        free(cat);
    }
}
