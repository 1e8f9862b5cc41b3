// Pre-pass of the bf16 path: one read of q, k and v feeds
//   (1) the full 3D RoPE of q and k (Sec. 3, Eq. shiftinv): q^r, k^r for the
//       sparse branch, and their 64-token block means for the block mask
//       (Alg. 1 "topk ratio");
//   (2) the low-rank summary (Eq. qklr, Eq. ctx; Sec. 4.5 kernel 1):
//       k~_n = R_r(n) SiLU(P_k k^n_n),  C = sum_n k~_n v_n^T,  z = sum_n k~_n.
// Without q the kernel computes (2) alone (the summary entry point).
//
// Work unit = (head, 64-token block).  G persistent CTAs take contiguous unit
// ranges [c U / G, (c + 1) U / G), so every CTA moves the same number of bytes
// to within one unit and no wave is left partly empty.  A range spans one or
// more heads; the CTA keeps C and z of the current head in registers and
// writes them to partial slot c + head when the head changes or the range
// ends.  The slots of one head belong to consecutive CTAs, and the combine
// kernel adds them in CTA order, so C is bitwise reproducible on a GPU model.
//
// A unit is processed as two 32-token halves, each a stage of the TMA ring
// (k, v and q boxes of 32 x 128, 8 KB each), which keeps a CTA small enough
// that two fit on an SM for r <= 48 (16 warps per SM hide the latency of the
// dependent MMA and rotation chains).  Per half, 8 warps:
//   rotate q, k (warp w = token rows 4w .. 4w + 3, lane = 4 coordinates),
//   store q^r, k^r, pool; U = K P_k^T (mma.sync; warp = 16 tokens x a quarter
//   or half of the r columns); k~ = R_r SiLU(U) to shared memory; the half's
//   barrier; C^T += V^T k~ (warp = 16 of the 128 d columns, all r rows).
// The block means are pairwise sums (the summation order the block mask is
// defined with, every rounding fixed, so the decision is the same on any
// kernel that evaluates it): a thread adds its four rows as a tree (levels 1
// and 2), writes those nodes to a double-buffered shared tile, and after the
// half's barrier thread c adds the 8 nodes of column c (levels 3-5); after the
// second half the two halves' nodes are added and divided by the block's
// token count -- the same bits as the stand-alone rotate + pool kernel.
//
// The loads of half-stage i + S - 1 are issued (by lane 0 of warps 0-2, one
// box each) right after half-stage i's barrier, when every thread is done
// with half-stage i - 1 and its stage is free.  Every wait on an mbarrier is
// bounded; a wait that gives up records ROLA_ERR_TIMEOUT, the threads agree on
// it at the half's barrier (a barrier reduction, so none is left waiting),
// and the copies still in flight are waited for before the CTA exits.
#include <cudaTypedefs.h>

#include "common.cuh"
#include "tcgen05.cuh"
#include "tensor_map.cuh"

namespace rola {
namespace {

using namespace tc;

constexpr int kWarps = 8;
constexpr int kThreads = 32 * kWarps;
constexpr int kHalfRows = 32;
constexpr uint32_t kHalf = kHalfRows * 128 * 2;      // one 32-token half of one tensor
constexpr int kMaxStages = 8;

// Byte offset of 16-byte chunk c (0..15) of row r (0..31) in a 32-row half
// tile as a [chunk][row][64] TMA box with 128-byte swizzle writes it.
__device__ __forceinline__ uint32_t hsw(int r, int c)
{
    return (c >> 3) * (kHalfRows * 128) + r * 128 + (((c & 7) ^ (r & 7)) << 4);
}

template <int R>
struct Cfg {
    static constexpr int NT = R / 8;                             // n-tiles of U
    static constexpr int NSPLIT = NT % 4 == 0 ? 4 : 2;           // column groups of U
    static constexpr int NTW = NT / NSPLIT;                      // n-tiles per warp
    static constexpr int KT = 2 * R + 16;                        // bytes per k~ row (padded)
    static constexpr int kCtasPerSm = R <= 48 ? 2 : 1;
};

struct Layout {
    int stages;
    uint32_t stage_bytes, P, kt, part, zsm, bars, total;
    __host__ __device__ Layout(int R, bool fuse)
    {
        const bool two = R <= 48;                                 // two CTAs per SM
        stages = two ? (fuse ? 3 : 4) : (fuse ? 6 : 8);
        stage_bytes = fuse ? 3 * kHalf : 2 * kHalf;
        P = stages * stage_bytes;                                 // P_k of the current head, r rows x 256 B
        kt = P + R * 256;                                         // k~, two buffers of 32 rows
        part = kt + 2 * kHalfRows * (2 * R + 16);                 // pooling nodes [2][8][q|k 256] fp32
        zsm = part + (fuse ? 2 * 8 * 256 * 4 : 0);
        bars = zsm + 2 * R * 4;                                   // full[kMaxStages], abort
        total = bars + kMaxStages * 8 + 16;
    }
};

struct Params {
    Shape s;
    const __nv_bfloat16* Pk;
    const float2* tab;
    __nv_bfloat16* qr;            // null: summary only
    __nv_bfloat16* kr;
    float* qbar;
    float* kbar;
    float* partials;
    DeviceStatus* status;
    int units;                    // B * H * nC
};

__device__ __forceinline__ void record_timeout(const Params& p, int where)
{
    if (atomicCAS(&p.status->code, 0, (int)ROLA_ERR_TIMEOUT) == 0) p.status->where = where;
}

// Rotates the 4 bf16 coordinates in w (2 pairs, (cos, sin) in cs) into y
// (fp32) and, for a token inside the sequence, stores them as bf16 at dst;
// a token past the end gives y = +0 (an empty slot of the pairwise sum).
__device__ __forceinline__ void rotate4(const uint2& w, const float2 (&cs)[2], __nv_bfloat16* dst, bool valid,
                                        float (&y)[4])
{
    const uint32_t wv[2] = {w.x, w.y};
    uint32_t out[2];
#pragma unroll
    for (int q = 0; q < 2; ++q) {
        const float2 x = unpack_bf16(wv[q]);
        const float2 r = rope_rotate(x.x, x.y, cs[q]);
        out[q] = pack_bf16(r.x, r.y);
        y[2 * q] = valid ? r.x : 0.0f;
        y[2 * q + 1] = valid ? r.y : 0.0f;
    }
    if (valid) *reinterpret_cast<uint2*>(dst) = make_uint2(out[0], out[1]);
}

__device__ __forceinline__ uint2 lds64(uint32_t a)
{
    uint2 w;
    asm volatile("ld.shared.v2.b32 {%0,%1}, [%2];\n" : "=r"(w.x), "=r"(w.y) : "r"(a));
    return w;
}


// SiLU with the approximate divide (the features enter the MMA in bf16).  The
// kernel is instantiated for it and for ActAblation (the other feature maps).
struct SiluFast {
    int kind;    // always ROLA_LOWRANK_ACT_SILU
    __device__ float operator()(float x) const { return __fdividef(x, 1.0f + __expf(-x)); }
};

template <int R, typename Act>
__global__ void __launch_bounds__(kThreads, Cfg<R>::kCtasPerSm) prepass_kernel(
    const __grid_constant__ CUtensorMap map_q, const __grid_constant__ CUtensorMap map_k,
    const __grid_constant__ CUtensorMap map_v, const Params p)
{
    using C = Cfg<R>;
    constexpr int NTW = C::NTW;
    extern __shared__ __align__(1024) uint8_t smem[];
    const bool fuse = p.qr != nullptr;
    const Layout lay(R, fuse);
    if (smem_u32(smem) & 1023u) {          // the 128-byte swizzle of the TMA boxes needs 1024-byte alignment
        if (threadIdx.x == 0) atomicCAS(&p.status->code, 0, (int)ROLA_ERR_UNSUPPORTED);
        return;
    }
    const Shape& s = p.s;
    const int S = lay.stages;
    const uint32_t sbase = smem_u32(smem);
    const uint32_t sP = sbase + lay.P, sKt = sbase + lay.kt;
    float* zsm = reinterpret_cast<float*>(smem + lay.zsm);
    const uint32_t full0 = sbase + lay.bars;
    volatile int* abort = reinterpret_cast<volatile int*>(smem + lay.bars + kMaxStages * 8);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int u0 = (int)((long long)blockIdx.x * p.units / gridDim.x);
    const int u1 = (int)((long long)(blockIdx.x + 1) * p.units / gridDim.x);
    const int count = 2 * (u1 - u0);                // half-stages of this CTA

    if (tid == 0) {
        *abort = 0;
        for (int i = 0; i < S; ++i) mbar_init(full0 + 8 * i, 1);
        fence_mbar_init();
        tma_prefetch_desc(&map_k);
        tma_prefetch_desc(&map_v);
        if (fuse) tma_prefetch_desc(&map_q);
    }
    __syncthreads();

    // loads of the j-th half-stage of the range into stage j % S: lane 0 of
    // warps 0, 1, 2 issue the k, v, q boxes; thread 0 also arms the barrier
    const uint32_t bytes = fuse ? 3 * kHalf : 2 * kHalf;
    auto issue = [&](int j) {
        // test hook: the CTA's first half-stage is never loaded (nor its bytes armed), so the waits on it run out
        if ((s.debug_flags & ROLA_DEBUG_SKIP_FIRST_K_COPY) && j == 0) return;
        const int u = u0 + (j >> 1), bh = u / s.nC, row = (u - bh * s.nC) * 64 + (j & 1) * kHalfRows;
        const uint32_t dst = sbase + (j % S) * lay.stage_bytes, bar = full0 + 8 * (j % S);
        if (tid == 0) {
            mbar_expect_tx(bar, bytes);
            tma_load_4d(dst, &map_k, bar, 0, row, 0, bh);
        } else if (tid == 32) {
            tma_load_4d(dst + kHalf, &map_v, bar, 0, row, 0, bh);
        } else if (tid == 64 && fuse) {
            tma_load_4d(dst + 2 * kHalf, &map_q, bar, 0, row, 0, bh);
        }
    };
    int issued = count < S ? count : S;
    for (int j = 0; j < issued; ++j) issue(j);

    const int g = lane >> 2, t4 = lane & 3, mi = lane >> 3;
    const int mt = warp & 1, cg = warp >> 1;        // U: tokens 16 mt .. +15 of the half, column group cg
    const bool u_warp = cg < C::NSPLIT;             // (with two column groups, warps 4-7 skip U)
    // rotation and pooling: rows 4 warp .. 4 warp + 3 of the half, coordinates
    // 4 lane .. 4 lane + 3 (pairs 2 lane, 2 lane + 1); a warp's 8-byte shared
    // loads cover one whole row
    const int cq = lane;
    const int hw = s.Hh * s.Ww;
    int axis[2];
#pragma unroll
    for (int q = 0; q < 2; ++q) {
        const int m = cq * 2 + q;
        axis[q] = m < s.pt ? 0 : (m < s.pt + s.px ? 1 : 2);
    }
    int kaxis[NTW];                                 // axis of pair nt * 4 + t4 of each of this warp's n-tiles
#pragma unroll
    for (int j = 0; j < NTW; ++j) {
        const int m = (cg * NTW + j) * 4 + t4;
        kaxis[j] = m < s.pt ? 0 : (m < s.pt + s.px ? 1 : 2);
    }
    // grid position (t, x, y) of flat token n, and of the token `step` further on
    auto position = [&](int n, int& t, int& x, int& y) {
        t = n / hw;
        const int rem = n - t * hw;
        x = rem / s.Ww;
        y = rem - x * s.Ww;
    };
    auto advance = [&](int step, int& t, int& x, int& y) {
        y += step;
        while (y >= s.Ww) {
            y -= s.Ww;
            if (++x == s.Hh) {
                x = 0;
                ++t;
            }
        }
    };
    auto table_row = [&](int axis, int t, int x, int y) {
        return axis == 0 ? min(t, s.T - 1) : (axis == 1 ? s.T + x : s.T + s.Hh + y);
    };

    float cacc[R / 16][2][4];
    float zacc[NTW][2];
    auto clear = [&]() {
#pragma unroll
        for (int a = 0; a < R / 16; ++a)
#pragma unroll
            for (int b = 0; b < 2; ++b) cacc[a][b][0] = cacc[a][b][1] = cacc[a][b][2] = cacc[a][b][3] = 0.0f;
#pragma unroll
        for (int j = 0; j < NTW; ++j) zacc[j][0] = zacc[j][1] = 0.0f;
    };
    // partial C [R][128] and z [R] of head hb -> slot blockIdx.x + hb
    auto flush = [&](int hb) {
        float* dst = p.partials + (size_t)(blockIdx.x + hb) * (size_t)(R * kDh + R);
#pragma unroll
        for (int a = 0; a < R / 16; ++a)
#pragma unroll
            for (int nt = 0; nt < 2; ++nt) {
                const int d = warp * 16 + nt * 8 + t4 * 2, row = a * 16 + g;
                *reinterpret_cast<float2*>(dst + (size_t)row * kDh + d) = make_float2(cacc[a][nt][0], cacc[a][nt][1]);
                *reinterpret_cast<float2*>(dst + (size_t)(row + 8) * kDh + d) =
                    make_float2(cacc[a][nt][2], cacc[a][nt][3]);
            }
#pragma unroll
        for (int j = 0; j < NTW; ++j)
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                float x = zacc[j][e];
                x += __shfl_xor_sync(0xffffffffu, x, 4);
                x += __shfl_xor_sync(0xffffffffu, x, 8);
                x += __shfl_xor_sync(0xffffffffu, x, 16);
                if (g == 0 && u_warp) zsm[mt * R + (cg * NTW + j) * 8 + t4 * 2 + e] = x;
            }
        bar_sync(1, kThreads);
        if (tid < R) dst[R * kDh + tid] = zsm[tid] + zsm[R + tid];
    };

    clear();
    int hb = -1;
    bool failed = false;
    // grid positions of this thread's first k~ token and first rotation row in
    // the current half; carried 32 tokens forward per half (a division only at
    // the start of the range, since consecutive units are consecutive blocks)
    int kt_t, kt_x, kt_y, rt_t, rt_x, rt_y;
    {
        const int blk0 = u0 - (u0 / s.nC) * s.nC;
        position(blk0 * kBlock + mt * 16 + g, kt_t, kt_x, kt_y);
        position(blk0 * kBlock + 4 * warp, rt_t, rt_x, rt_y);
    }
    float pool0 = 0.0f;                             // pairwise node of the block's first half, column tid
    float* nodes = reinterpret_cast<float*>(smem + lay.part);
    int i = 0;                                      // half-stage index
    for (; i < count; ++i) {
        const int u = u0 + (i >> 1), h = i & 1;
        const int bh = u / s.nC, blk = u - bh * s.nC;
        const int st = i % S, buf = i & 1;
        if (h == 0 && bh != hb) {
            if (hb >= 0) {
                flush(hb);
                clear();
            }
            // P_k of the new head (every reader of the old one has passed the last barrier)
            const __nv_bfloat16* src = p.Pk + (size_t)(bh % s.H) * s.r * kDh;
            for (int e = tid; e < R * 16; e += kThreads) {
                const uint4 w = (e >> 4) < s.r ? __ldg(reinterpret_cast<const uint4*>(src) + e) : make_uint4(0, 0, 0, 0);
                asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};\n" ::"r"(sP + sw128(e >> 4, e & 15)), "r"(w.x),
                             "r"(w.y), "r"(w.z), "r"(w.w)
                             : "memory");
            }
            bar_sync(1, kThreads);
            if (hb >= 0) {                         // a new head starts at its block 0
                position(mt * 16 + g, kt_t, kt_x, kt_y);
                position(4 * warp, rt_t, rt_x, rt_y);
            }
            hb = bh;
        }
        const uint32_t stage = sbase + st * lay.stage_bytes;
        const uint32_t kb = stage, vb = stage + kHalf, qb = stage + 2 * kHalf;
        const uint32_t ktb = sKt + buf * (kHalfRows * C::KT);
        const int n_half = blk * kBlock + h * kHalfRows;          // first token of this half
        // (cos, sin) of the k~ pairs of this thread's two tokens, needed after U
        float2 kcs[2][NTW];
        {
            int t = kt_t, x = kt_x, y = kt_y;
#pragma unroll
            for (int hr = 0; hr < 2; ++hr) {
#pragma unroll
                for (int j = 0; j < NTW; ++j)
                    kcs[hr][j] = __ldg(p.tab + table_row(kaxis[j], t, x, y) * kPairs + (cg * NTW + j) * 4 + t4);
                advance(8, t, x, y);
            }
        }
        // (cos, sin) of the rotation's pairs for this thread's four rows
        float2 cs[4][2];
        if (fuse) {
            int t = rt_t, x = rt_x, y = rt_y;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
#pragma unroll
                for (int q = 0; q < 2; ++q) cs[j][q] = __ldg(p.tab + table_row(axis[q], t, x, y) * kPairs + cq * 2 + q);
                advance(1, t, x, y);
            }
        }
        advance(kHalfRows, kt_t, kt_x, kt_y);          // the next half's positions
        advance(kHalfRows, rt_t, rt_x, rt_y);
        // warp-uniform, so that the warp-wide shuffles and MMAs below see every lane
        const bool ok = __all_sync(0xffffffffu, mbar_wait(full0 + 8 * st, (i / S) & 1, abort, s.wait_limit_ns));
        if (ok) {
            if (fuse) {
                // ---- rotate q and k, store q^r and k^r, pool levels 1-2 (pairwise, the stand-alone kernel's bits)
                uint2 wq[4], wk[4];
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const uint32_t a = hsw(4 * warp + j, cq >> 1) + (cq & 1) * 8;
                    wq[j] = lds64(qb + a);
                    wk[j] = lds64(kb + a);
                }
                float yq[4][4], yk[4][4];
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const int n = n_half + 4 * warp + j;
                    const bool valid = n < s.N;
                    const size_t go = ((size_t)bh * s.N + (valid ? n : 0)) * kDh + cq * 4;
                    rotate4(wq[j], cs[j], p.qr + go, valid, yq[j]);
                    rotate4(wk[j], cs[j], p.kr + go, valid, yk[j]);
                }
                float4 nq, nk;                           // (y0 + y1) + (y2 + y3) per coordinate
                nq.x = (yq[0][0] + yq[1][0]) + (yq[2][0] + yq[3][0]);
                nq.y = (yq[0][1] + yq[1][1]) + (yq[2][1] + yq[3][1]);
                nq.z = (yq[0][2] + yq[1][2]) + (yq[2][2] + yq[3][2]);
                nq.w = (yq[0][3] + yq[1][3]) + (yq[2][3] + yq[3][3]);
                nk.x = (yk[0][0] + yk[1][0]) + (yk[2][0] + yk[3][0]);
                nk.y = (yk[0][1] + yk[1][1]) + (yk[2][1] + yk[3][1]);
                nk.z = (yk[0][2] + yk[1][2]) + (yk[2][2] + yk[3][2]);
                nk.w = (yk[0][3] + yk[1][3]) + (yk[2][3] + yk[3][3]);
                float* nb = nodes + (buf * 8 + warp) * 256;
                reinterpret_cast<float4*>(nb)[cq] = nq;
                reinterpret_cast<float4*>(nb + 128)[cq] = nk;
            }
            if (u_warp) {
                // ---- U = K P_k^T for tokens 16 mt .. +15 of the half and this warp's n-tiles
                float uacc[NTW][4];
#pragma unroll
                for (int j = 0; j < NTW; ++j) uacc[j][0] = uacc[j][1] = uacc[j][2] = uacc[j][3] = 0.0f;
#pragma unroll
                for (int kc = 0; kc < 8; ++kc) {
                    uint32_t a0, a1, a2, a3;
                    ldsm_x4(kb + hsw(mt * 16 + (lane & 7) + (mi & 1) * 8, kc * 2 + (mi >> 1)), a0, a1, a2, a3);
#pragma unroll
                    for (int np = 0; np < NTW / 2; ++np) {
                        const int nt = cg * NTW + 2 * np;
                        uint32_t b0, b1, b2, b3;
                        ldsm_x4(sP + sw128(nt * 8 + (mi >> 1) * 8 + (lane & 7), kc * 2 + (mi & 1)), b0, b1, b2, b3);
                        mma_bf16(uacc[2 * np], a0, a1, a2, a3, b0, b1);
                        mma_bf16(uacc[2 * np + 1], a0, a1, a2, a3, b2, b3);
                    }
                    if (NTW & 1) {
                        const int nt = cg * NTW + NTW - 1;
                        uint32_t b0, b1;
                        ldsm_x2(sP + sw128(nt * 8 + (lane & 7), kc * 2 + (mi & 1)), b0, b1);
                        mma_bf16(uacc[NTW - 1], a0, a1, a2, a3, b0, b1);
                    }
                }
                // ---- k~ = R_r SiLU(U) (or the placement cfg selects); tokens past N contribute nothing
#pragma unroll
                for (int hr = 0; hr < 2; ++hr) {
                    const int tl = mt * 16 + g + hr * 8, n = n_half + tl;
                    const bool valid = n < s.N;
#pragma unroll
                    for (int j = 0; j < NTW; ++j) {
                        const int nt = cg * NTW + j;
                        const float2 cs2 = valid ? kcs[hr][j] : make_float2(0.0f, 0.0f);
                        const float2 y = lowrank_pair(uacc[j][2 * hr], uacc[j][2 * hr + 1], cs2, s.lr_rope, Act{s.lr_act});
                        zacc[j][0] += y.x;
                        zacc[j][1] += y.y;
                        asm volatile("st.shared.b32 [%0], %1;\n" ::"r"(ktb + tl * C::KT + (nt * 8 + t4 * 2) * 2),
                                     "r"(pack_bf16(y.x, y.y))
                                     : "memory");
                    }
                }
            }
        }
        // every thread reaches this barrier once per half; it also settles a timeout
        if (bar_red_or(1, kThreads, !ok)) {
            failed = true;
            break;
        }
        if (i >= 1 && issued < count) {       // half-stage i - 1 is done everywhere: refill its stage
            issue(issued);
            ++issued;
        }
        if (fuse) {
            // ---- pooling levels 3-5: column tid (q: 0..127, k: 128..255) over the 8 nodes of this half
            // (the buffer is written again two halves on, after every thread has passed the next barrier)
            const float* nb = nodes + buf * 8 * 256 + tid;
            const float half_sum = ((nb[0] + nb[256]) + (nb[512] + nb[768])) +
                                   ((nb[1024] + nb[1280]) + (nb[1536] + nb[1792]));
            if (h == 0) {
                pool0 = half_sum;
            } else {
                // the top node: first half + second half, then the mean over the block's tokens
                // (with 128-token query blocks the query side keeps the sum: one half of the 128-token tree)
                const int cnt = min(kBlock, s.N - blk * kBlock);
                const float sum = pool0 + half_sum;
                (tid < kDh ? p.qbar : p.kbar)[((size_t)bh * s.nC + blk) * kDh + (tid & (kDh - 1))] =
                    (tid < kDh && s.qb2) ? sum : sum / (float)cnt;
            }
        }
        // ---- C^T += V^T k~ : this warp's 16 d columns, all r rows, 32 tokens
#pragma unroll
        for (int kc = 0; kc < kHalfRows / 16; ++kc) {
            uint32_t b0, b1, b2, b3;
            ldsm_x4_t(vb + hsw(kc * 16 + (mi & 1) * 8 + (lane & 7), warp * 2 + (mi >> 1)), b0, b1, b2, b3);
#pragma unroll
            for (int a = 0; a < R / 16; ++a) {
                uint32_t a0, a1, a2, a3;
                ldsm_x4_t(ktb + (kc * 16 + (mi >> 1) * 8 + (lane & 7)) * C::KT + (a * 2 + (mi & 1)) * 16, a0, a1, a2,
                          a3);
                mma_bf16(cacc[a][0], a0, a1, a2, a3, b0, b1);
                mma_bf16(cacc[a][1], a0, a1, a2, a3, b2, b3);
            }
        }
    }
    if (failed) {
        // the copies issued and not yet waited for must land before the CTA exits
        if (tid == 0) {
            record_timeout(p, 7);
            int never = 0;
            for (int j = i; j < issued; ++j) mbar_wait(full0 + 8 * (j % S), (j / S) & 1, &never, s.wait_limit_ns);
        }
        return;
    }
    if (hb >= 0) flush(hb);
}

__global__ void prepass_combine_kernel(Shape s, int ctas, int units, const float* __restrict__ partials,
                                       float* __restrict__ C, float* __restrict__ z, __nv_bfloat16* __restrict__ Cbf)
{
    const int bh = blockIdx.y;
    const int per = s.rp * kDh + s.rp;                 // one partial slot (rp rows)
    const int e = blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= per) return;
    // CTAs whose unit ranges meet head bh: those holding its first and last unit, and all between
    const int c0 = (int)((((long long)bh * s.nC + 1) * ctas - 1) / units);
    const int c1 = (int)((((long long)(bh + 1) * s.nC) * ctas - 1) / units);
    float x = 0.0f;
    for (int c = c0; c <= c1; ++c) x += partials[(size_t)(c + bh) * per + e];
    // C and z have r rows; the bf16 copy keeps all rp (rows past r are exactly zero)
    if (e < s.rp * kDh) {
        if (e < s.r * kDh) C[(size_t)bh * s.r * kDh + e] = x;
        if (Cbf) Cbf[(size_t)bh * s.rp * kDh + e] = __float2bfloat16_rn(x);
    } else if (z && e - s.rp * kDh < s.r) {
        z[(size_t)bh * s.r + (e - s.rp * kDh)] = x;
    }
}

template <int R, typename Act>
cudaError_t launch_ra(const CUtensorMap& mq, const CUtensorMap& mk, const CUtensorMap& mv, const Params& p, int ctas,
                      bool fuse, cudaStream_t st)
{
    const Layout lay(R, fuse);
    cudaError_t e = cudaFuncSetAttribute(prepass_kernel<R, Act>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)lay.total);
    if (e != cudaSuccess) return e;
    prepass_kernel<R, Act><<<ctas, kThreads, lay.total, st>>>(mq, mk, mv, p);
    return cudaGetLastError();
}

template <int R>
cudaError_t launch_r(const CUtensorMap& mq, const CUtensorMap& mk, const CUtensorMap& mv, const Params& p, int ctas,
                     bool fuse, cudaStream_t st)
{
    return p.s.lr_act == ROLA_LOWRANK_ACT_SILU ? launch_ra<R, SiluFast>(mq, mk, mv, p, ctas, fuse, st)
                                               : launch_ra<R, ActAblation>(mq, mk, mv, p, ctas, fuse, st);
}

}  // namespace

int prepass_ctas(const Shape& s, int max_ctas)
{
    int dev = 0, nsm = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev) !=
                                                   cudaSuccess)
        return 0;
    const long long units = (long long)s.B * s.H * s.nC;
    long long g = (long long)nsm * (s.rp <= 48 ? 2 : 1);     // CTAs per SM as Cfg<R>::kCtasPerSm
    if (g > max_ctas) g = max_ctas;
    if (g > kMaxPrepassCtas) g = kMaxPrepassCtas;
    if (g > units) g = units;
    return (int)g;
}

cudaError_t launch_prepass(const Shape& s, int ctas, const void* q, const void* k, const void* v,
                           const void* P_k, const float2* tab, void* qr, void* kr, float* qbar, float* kbar,
                           float* partials, DeviceStatus* status, cudaStream_t st)
{
    if (ctas <= 0 || ctas > kMaxPrepassCtas || ctas > s.B * s.H * s.nC) return cudaErrorInvalidValue;
    const bool fuse = q != nullptr;
    CUtensorMap mq, mk, mv;
    if (!make_block_map(&mk, k, s, kHalfRows) || !make_block_map(&mv, v, s, kHalfRows)) return cudaErrorInvalidValue;
    if (fuse) {
        if (!make_block_map(&mq, q, s, kHalfRows)) return cudaErrorInvalidValue;
    } else {
        mq = mk;
    }
    Params p;
    p.s = s;
    p.Pk = static_cast<const __nv_bfloat16*>(P_k);
    p.tab = tab;
    p.qr = fuse ? static_cast<__nv_bfloat16*>(qr) : nullptr;
    p.kr = fuse ? static_cast<__nv_bfloat16*>(kr) : nullptr;
    p.qbar = qbar;
    p.kbar = kbar;
    p.partials = partials;
    p.status = status;
    p.units = s.B * s.H * s.nC;
    switch (s.rp) {
        case 16: return launch_r<16>(mq, mk, mv, p, ctas, fuse, st);
        case 32: return launch_r<32>(mq, mk, mv, p, ctas, fuse, st);
        case 48: return launch_r<48>(mq, mk, mv, p, ctas, fuse, st);
        case 64: return launch_r<64>(mq, mk, mv, p, ctas, fuse, st);
        case 80: return launch_r<80>(mq, mk, mv, p, ctas, fuse, st);
        case 96: return launch_r<96>(mq, mk, mv, p, ctas, fuse, st);
        case 112: return launch_r<112>(mq, mk, mv, p, ctas, fuse, st);
        case 128: return launch_r<128>(mq, mk, mv, p, ctas, fuse, st);
        default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_prepass_combine(const Shape& s, int ctas, const float* partials, float* C, float* z,
                                   __nv_bfloat16* Cbf, cudaStream_t st)
{
    const int per = s.rp * kDh + s.rp;
    const int units = s.B * s.H * s.nC;
    prepass_combine_kernel<<<dim3((per + 255) / 256, s.B * s.H), 256, 0, st>>>(s, ctas, units, partials, C, z, Cbf);
    return cudaGetLastError();
}

}  // namespace rola
