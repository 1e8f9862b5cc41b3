// Backward pass of the block-sparse softmax attention, query side, on the
// 5th-generation tensor cores (bf16, fp32 accumulation in TMEM):
//
//   P = exp(q^r k^r / sqrt d - lse),  dP = dO^s v^T,  dS = P (dP - D),  dq^r = dS k^r / sqrt d
//
// over the kept key blocks of each query block (Sec. 3 softmax form, its
// gradient).  As in the forward kernel the problem is transposed so that every
// MMA has M = 128: for a query block (N = 64 queries) and a pair of kept key
// blocks (M = 128 keys)
//   S^T  = K_pair  Q^T       A = K pair (K-major),   B = Q (K-major)       TMEM
//   dP^T = V_pair  dO^T      A = V pair (K-major),   B = dO (K-major)      TMEM
//   dS^T = P^T (dP^T - D)    by the dS warps (thread = key), bf16 into shared memory
//   dQ^T += K_pair^T dS^T    A = the same K pair read MN-major (M = d), B = dS^T (MN-major)
// The log-sum-exp of each query is known, so no running maximum is needed.
//
// Roles (384 threads, one persistent CTA per SM):
//   warps 0-7  dS and epilogue: two warpgroups of 32 query columns; thread
//              wtid owns TMEM lane wtid (a key of S^T / dP^T, a d of dQ^T)
//   warp  8    TMA: Q and dO (per query block) and the K pairs
//   warp  9    TMA: the V pairs
//   warp 10    S^T and dP^T issuer, TMEM owner
//   warp 11    dQ^T issuer
// Rings: K pairs 3 deep (held until the tile's dQ^T MMA), V pairs 2 deep,
// S^T / dP^T / dS^T double-buffered, dQ^T double-buffered across query blocks.
// Every mbarrier wait is bounded; a wait that gives up records ROLA_ERR_TIMEOUT
// and the CTA drains what it issued and frees TMEM.
#include <stddef.h>

#include "common.cuh"
#include "tcgen05.cuh"
#include "tensor_map.cuh"

namespace rola {
namespace {

using namespace tc;

constexpr int kDsWarps = 8;
constexpr int kCols = 32;                      // query columns per dS warpgroup
constexpr int kProdKWarp = 8, kProdVWarp = 9, kSWarp = 10, kQWarp = 11;
constexpr int kThreads = 32 * 12;
constexpr int kWGThreads = 128;
constexpr uint32_t kBlockBytes = 64 * 128 * 2;   // one query block (Q or dO), [chunk][row][64]
constexpr uint32_t kPairBytes = 128 * 128 * 2;   // a pair of key blocks, [chunk][block][row]
constexpr uint32_t kDsBytes = 128 * 64 * 2;      // dS^T tile [key][64 q]
constexpr int KS = 3, VS = 2;
constexpr uint32_t kSmemQ = 0, kSmemO = kBlockBytes, kSmemK = 2 * kBlockBytes;
constexpr uint32_t kSmemV = kSmemK + KS * kPairBytes;
constexpr uint32_t kSmemDs = kSmemV + VS * kPairBytes;
constexpr uint32_t kSmemTiles = kSmemDs + 2 * kDsBytes;   // 224 KB
constexpr uint32_t kTmemCols = 512;              // S^T x2, dP^T x2, dQ^T x2 (64 columns each)

namespace dq {

enum Bar { Q_FULL = 0, Q_EMPTY = 1, K_FULL = 2, K_EMPTY = K_FULL + KS, V_FULL = K_EMPTY + KS, V_EMPTY = V_FULL + VS,
           S_FULL = V_EMPTY + VS, S_EMPTY = S_FULL + 2, DS_FULL = S_EMPTY + 2, DS_EMPTY = DS_FULL + 2,
           O_FULL = DS_EMPTY + 2, O_EMPTY = O_FULL + 2, DRAIN = O_EMPTY + 2, NUM_BARS = DRAIN + 2 };

struct Smem {
    alignas(16) float lse2[64];     // lse of the block's queries, log2 units
    alignas(16) float D[64];        // dO^s . O^s of the block's queries
    uint64_t bar[NUM_BARS];
    uint32_t tmem_base;
    int abort;
};
static_assert(kSmemTiles % 1024 == 0, "the control block starts aligned");

struct Params {
    Shape s;
    const int32_t* kv_idx;
    const float* lse;
    const float* Dv;
    const float* dq_lr;                 // fp32 low-rank part of dq
    const float2* tab;
    __nv_bfloat16* dq;
    DeviceStatus* status;
    int total_items;
    int tiles;
};

__device__ __forceinline__ void record_timeout(const Params& p, int where)
{
    if (atomicCAS(&p.status->code, 0, (int)ROLA_ERR_TIMEOUT) == 0) p.status->where = 16 + where;
}

}  // namespace dq

template <int NC>
__device__ __forceinline__ void ld_cols(uint32_t taddr, float (&v)[NC])
{
#pragma unroll
    for (int c = 0; c < NC / 16; ++c) tmem_ld16(taddr + c * 16, *reinterpret_cast<float(*)[16]>(&v[c * 16]));
    tmem_ld_wait(*reinterpret_cast<float(*)[16]>(&v[0]));
#pragma unroll
    for (int c = 1; c < NC / 16; ++c) reg_fence(*reinterpret_cast<float(*)[16]>(&v[c * 16]));
}

template <bool kCube>
__global__ void __launch_bounds__(kThreads, 1) sparse_bwd_dq_tc_kernel(const __grid_constant__ CUtensorMap map_q,
                                                                       const __grid_constant__ CUtensorMap map_o,
                                                                       const __grid_constant__ CUtensorMap map_k,
                                                                       const __grid_constant__ CUtensorMap map_v,
                                                                       const dq::Params p)
{
    using namespace dq;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    if (smem_u32(smem_raw) & 1023u) {
        if (threadIdx.x == 0) atomicCAS(&p.status->code, 0, (int)ROLA_ERR_UNSUPPORTED);
        return;
    }
    Smem& sm = *reinterpret_cast<Smem*>(smem_raw + kSmemTiles);
    const uint32_t sbase = smem_u32(smem_raw);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    auto bar = [&](int i) { return smem_u32(&sm.bar[i]); };
    const Shape& s = p.s;
    const int T = p.tiles, nB = s.nB;

    if (tid == 0) {
        sm.abort = 0;
        mbar_init(bar(Q_FULL), 1);
        mbar_init(bar(Q_EMPTY), 1);
        for (int i = 0; i < KS; ++i) {
            mbar_init(bar(K_FULL + i), 1);
            mbar_init(bar(K_EMPTY + i), 1);
        }
        for (int i = 0; i < VS; ++i) {
            mbar_init(bar(V_FULL + i), 1);
            mbar_init(bar(V_EMPTY + i), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar(S_FULL + i), 1);
            mbar_init(bar(S_EMPTY + i), kDsWarps);
            mbar_init(bar(DS_FULL + i), kDsWarps);
            mbar_init(bar(DS_EMPTY + i), 1);
            mbar_init(bar(O_FULL + i), 1);
            mbar_init(bar(O_EMPTY + i), kDsWarps);
        }
        mbar_init(bar(DRAIN), 1);
        mbar_init(bar(DRAIN + 1), 1);
        fence_mbar_init();
    }
    if (warp == kSWarp) {
        tmem_alloc(smem_u32(&sm.tmem_base), kTmemCols);
        tmem_relinquish();
    }
    if ((warp == kProdKWarp || warp == kProdVWarp) && lane == 0) {
        tma_prefetch_desc(&map_q);
        tma_prefetch_desc(&map_o);
        tma_prefetch_desc(&map_k);
        tma_prefetch_desc(&map_v);
    }
    fence_before_sync();
    __syncthreads();
    fence_after_sync();
    const uint32_t tmem = sm.tmem_base;
    volatile int* abort = &sm.abort;

    if (warp == kProdKWarp || warp == kProdVWarp) {
        // ------------------------------------------------------------ TMA producers
        // lane 2h + c loads d-chunk c of block h of the pair (8 KB boxes) into
        // the [chunk][block][row] layout; the K warp also loads Q and dO.
        const bool is_v = warp == kProdVWarp;
        const int h = lane >> 1, kc = lane & 1;
        const int NS = is_v ? VS : KS;
        const uint32_t ring = is_v ? kSmemV : kSmemK;
        const int full0 = is_v ? V_FULL : K_FULL, empty0 = is_v ? V_EMPTY : K_EMPTY;
        const CUtensorMap* map = is_v ? &map_v : &map_k;
        int k = 0, issued_q = 0, issued = 0;
        bool ok = true;
        for (int item = blockIdx.x; item < p.total_items && ok; item += gridDim.x, ++k) {
            const int bh = item / nB, qb = item - bh * nB;
            const int32_t* kept = p.kv_idx + (size_t)item * s.n_keep;
            if (!is_v) {
                if (k >= 1) ok = mbar_wait(bar(Q_EMPTY), (k - 1) & 1, abort, s.wait_limit_ns);
                ok = __shfl_sync(0xffffffffu, ok, 0);
                if (!ok) break;
                if (lane == 0) {
                    mbar_expect_tx(bar(Q_FULL), 2 * kBlockBytes);
                    tma_load_4d(sbase + kSmemQ, &map_q, bar(Q_FULL), 0, qb * 64, 0, bh);
                    tma_load_4d(sbase + kSmemO, &map_o, bar(Q_FULL), 0, qb * 64, 0, bh);
                }
                ++issued_q;
            }
            for (int t = 0; t < T; ++t) {
                const int g = k * T + t, st = g % NS;
                const int ja = __ldg(kept + 2 * t);
                const int jb = 2 * t + 1 < s.n_keep ? __ldg(kept + 2 * t + 1) : -1;
                const int nblk = jb >= 0 ? 2 : 1;
                if (g >= NS) ok = mbar_wait(bar(empty0 + st), ((g / NS) - 1) & 1, abort, s.wait_limit_ns);
                ok = __shfl_sync(0xffffffffu, ok, 0);
                if (!ok) break;
                // test hook: the CTA's first K pair is never loaded, so the waits on it run out
                const bool skip = !is_v && (s.debug_flags & ROLA_DEBUG_SKIP_FIRST_K_COPY) && g == 0;
                if (lane == 0 && !skip) mbar_expect_tx(bar(full0 + st), nblk * 16384u);
                __syncwarp();
                if (lane < 4 && h < nblk && !skip)
                    tma_load_3d(sbase + ring + st * kPairBytes + kc * 16384 + h * 8192, map, bar(full0 + st), kc * 64,
                                (h ? jb : ja) * 64, bh);
                ++issued;
            }
        }
        if (!ok && lane == 0) record_timeout(p, is_v ? 4 : 1);
        if (lane == 0) {
            int never = 0;
            if (issued_q > 0) mbar_wait(bar(Q_FULL), (issued_q - 1) & 1, &never, s.wait_limit_ns);
            for (int u = issued > NS ? issued - NS : 0; u < issued; ++u)
                mbar_wait(bar(full0 + u % NS), (u / NS) & 1, &never, s.wait_limit_ns);
        }
    } else if (warp == kSWarp || warp == kQWarp) {
        // ------------------------------------------------------------ MMA issuers
        if (lane == 0) {
            const bool qw = warp == kQWarp;
            const uint32_t id_s = idesc_bf16(128, 64, false, false);
            const uint32_t id_q = idesc_bf16(128, 64, true, true);
            const uint64_t dq_ = smem_desc(sbase + kSmemQ, 16, 1024);      // Q: B of S^T (K-major)
            const uint64_t do_ = smem_desc(sbase + kSmemO, 16, 1024);      // dO: B of dP^T (K-major)
            const uint64_t dk = smem_desc(sbase + kSmemK, 16, 1024);       // K pairs: A of S^T (K-major)
            const uint64_t dv = smem_desc(sbase + kSmemV, 16, 1024);       // V pairs: A of dP^T (K-major)
            const uint64_t dkt = smem_desc(sbase + kSmemK, 16384, 1024);   // K pairs: A of dQ^T (MN-major, M = d)
            const uint64_t dds = smem_desc(sbase + kSmemDs, 8192, 1024);   // dS^T: B of dQ^T (MN-major)
            const uint32_t q_lo = (uint32_t)dq_, q_hi = (uint32_t)(dq_ >> 32);
            const uint32_t o_lo = (uint32_t)do_, o_hi = (uint32_t)(do_ >> 32);
            const uint32_t k_lo = (uint32_t)dk, k_hi = (uint32_t)(dk >> 32);
            const uint32_t v_lo = (uint32_t)dv, v_hi = (uint32_t)(dv >> 32);
            const uint32_t kt_lo = (uint32_t)dkt, kt_hi = (uint32_t)(dkt >> 32);
            const uint32_t ds_lo = (uint32_t)dds, ds_hi = (uint32_t)(dds >> 32);
            bool ok = true;
            int k = 0;
            for (int item = blockIdx.x; item < p.total_items && ok; item += gridDim.x, ++k) {
                const int ob = k & 1;
                if (!qw) {
                    if (!(ok = mbar_wait(bar(Q_FULL), k & 1, abort, s.wait_limit_ns))) break;
                    for (int t = 0; t < T; ++t) {
                        const int g = k * T + t, sb = g & 1, ks = g % KS, vs = g % VS;
                        if (!(ok = mbar_wait(bar(K_FULL + ks), (g / KS) & 1, abort, s.wait_limit_ns))) break;
                        if (!(ok = mbar_wait(bar(V_FULL + vs), (g / VS) & 1, abort, s.wait_limit_ns))) break;
                        if (g >= 2 && !(ok = mbar_wait(bar(S_EMPTY + sb), ((g >> 1) - 1) & 1, abort, s.wait_limit_ns)))
                            break;
                        fence_after_sync();
                        const uint32_t a = k_lo + ks * (kPairBytes >> 4), av = v_lo + vs * (kPairBytes >> 4);
#pragma unroll
                        for (int kk = 0; kk < 8; ++kk) {
                            const uint32_t ko = (kk >> 2) * 1024 + (kk & 3) * 2, qo = (kk >> 2) * 512 + (kk & 3) * 2;
                            mma_ss_split(tmem + sb * 64, a + ko, k_hi, q_lo + qo, q_hi, id_s, kk > 0 ? 1u : 0u);
                        }
#pragma unroll
                        for (int kk = 0; kk < 8; ++kk) {
                            const uint32_t ko = (kk >> 2) * 1024 + (kk & 3) * 2, qo = (kk >> 2) * 512 + (kk & 3) * 2;
                            mma_ss_split(tmem + 128 + sb * 64, av + ko, v_hi, o_lo + qo, o_hi, id_s, kk > 0 ? 1u : 0u);
                        }
                        mma_commit(bar(S_FULL + sb));
                        mma_commit(bar(V_EMPTY + vs));
                        if (t == T - 1) mma_commit(bar(Q_EMPTY));
                    }
                } else {
                    for (int t = 0; t < T; ++t) {
                        const int g = k * T + t, sb = g & 1, ks = g % KS;
                        const bool half = 2 * t + 1 >= s.n_keep;
                        if (!(ok = mbar_wait(bar(DS_FULL + sb), (g >> 1) & 1, abort, s.wait_limit_ns))) break;
                        if (t == 0 && k >= 2 &&
                            !(ok = mbar_wait(bar(O_EMPTY + ob), ((k >> 1) - 1) & 1, abort, s.wait_limit_ns)))
                            break;
                        fence_after_sync();
                        const uint32_t a = kt_lo + ks * (kPairBytes >> 4), b = ds_lo + sb * (kDsBytes >> 4);
                        const uint32_t d = tmem + 256 + ob * 64;
                        const int nk = half ? 4 : 8;          // K steps of 16 keys (a half tile has 64)
                        for (int kk = 0; kk < nk; ++kk)
                            mma_ss_split(d, a + kk * 128, kt_hi, b + kk * 128, ds_hi, id_q, (t > 0 || kk > 0) ? 1u : 0u);
                        mma_commit(bar(DS_EMPTY + sb));
                        mma_commit(bar(K_EMPTY + ks));
                    }
                    if (!ok) break;
                    mma_commit(bar(O_FULL + ob));
                }
            }
            if (!ok) record_timeout(p, qw ? 5 : 2);
            int never = 0;
            const uint32_t drain = bar(qw ? DRAIN + 1 : DRAIN);
            mma_commit(drain);
            mbar_wait(drain, 0, &never, s.wait_limit_ns);
        }
    } else {
        // ------------------------------------------------------------ dS + epilogue
        const int wg = warp >> 2, wtid = tid & 127;
        const int col0 = wg * kCols;
        const float c_log2 = s.sm_scale_log2;
        const uint32_t lane_off = (uint32_t)((warp & 3) * 32) << 16;
        bool ok = true;
        int k = 0;
        for (int item = blockIdx.x; item < p.total_items && ok; item += gridDim.x, ++k) {
            const int bh = item / nB, qb = item - bh * nB;
            const int32_t* kept = p.kv_idx + (size_t)item * s.n_keep;
            const int ob = k & 1;
            const uint32_t qmask = slot_mask32_g<kCube>(s, qb, col0);      // query columns of this warpgroup that are tokens
            const int rows = min(64, s.N - qb * 64) - col0;                // (contiguous blocks: the first `rows` are)
            auto colok = [&](int q) { if constexpr (kCube) return ((qmask >> q) & 1u) != 0; else return q < rows; };
            bar_sync(1 + wg, kWGThreads);                         // the previous block's columns are consumed
            if (wtid < kCols) {
                // lse and D in block order: row 64 qb + slot of the head's Np rows
                const size_t r = (size_t)bh * s.Np + (size_t)qb * 64 + col0 + wtid;
                const bool v = (qmask >> wtid) & 1u;
                sm.lse2[col0 + wtid] = v ? p.lse[r] * 1.4426950408889634f : 0.0f;
                sm.D[col0 + wtid] = v ? p.Dv[r] : 0.0f;
            }
            bar_sync(1 + wg, kWGThreads);
            int ja_n = __ldg(kept);
            int jb_n = s.n_keep > 1 ? __ldg(kept + 1) : -1;
            for (int t = 0; t < T; ++t) {
                const int g = k * T + t, sb = g & 1;
                const int ja = ja_n, jb = jb_n;
                if (t + 1 < T) {
                    ja_n = __ldg(kept + 2 * t + 2);
                    jb_n = 2 * t + 3 < s.n_keep ? __ldg(kept + 2 * t + 3) : -1;
                }
                const int blk = wtid < 64 ? ja : jb;
                const bool valid = blk >= 0 && slot_token_g<kCube>(s, blk, wtid & 63) >= 0;
                if (!(ok = mbar_wait(bar(S_FULL + sb), (g >> 1) & 1, abort, s.wait_limit_ns))) break;
                fence_after_sync();
                float x[kCols], y[kCols];
                ld_cols<kCols>(tmem + lane_off + sb * 64 + col0, x);
                ld_cols<kCols>(tmem + lane_off + 128 + sb * 64 + col0, y);
                fence_before_sync();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(S_EMPTY + sb));
                uint32_t pk[kCols / 2];
#pragma unroll
                for (int q = 0; q < kCols; q += 2) {
                    float d0 = 0.0f, d1 = 0.0f;
                    if (valid) {
                        const float2 l2 = *reinterpret_cast<const float2*>(&sm.lse2[col0 + q]);
                        const float2 dd = *reinterpret_cast<const float2*>(&sm.D[col0 + q]);
                        const float p0 = colok(q) ? fast_exp2(fmaf(x[q], c_log2, -l2.x)) : 0.0f;
                        const float p1 = colok(q + 1) ? fast_exp2(fmaf(x[q + 1], c_log2, -l2.y)) : 0.0f;
                        d0 = p0 * (y[q] - dd.x);
                        d1 = p1 * (y[q + 1] - dd.y);
                    }
                    pk[q >> 1] = pack_bf16(d0, d1);
                }
                if (g >= 2 && !(ok = mbar_wait(bar(DS_EMPTY + sb), ((g >> 1) - 1) & 1, abort, s.wait_limit_ns)))
                    break;
                const uint32_t prow = sbase + kSmemDs + sb * kDsBytes + (wtid >> 3) * 1024 + (wtid & 7) * 128;
#pragma unroll
                for (int c = 0; c < kCols / 8; ++c) {
                    const int chunk = wg * (kCols / 8) + c;
                    asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};\n" ::"r"(prow + ((chunk ^ (wtid & 7)) << 4)),
                                 "r"(pk[4 * c]), "r"(pk[4 * c + 1]), "r"(pk[4 * c + 2]), "r"(pk[4 * c + 3])
                                 : "memory");
                }
                fence_proxy_async_smem();
                fence_before_sync();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(DS_FULL + sb));
            }
            if (!ok) break;
            // ---- epilogue: dq = low-rank rows + R(p)^T (dQ^T / sqrt d); thread wtid holds
            // d = wtid of this warpgroup's 32 query rows; the pair partner d ^ 1 is lane ^ 1.
            // The low-rank rows are read before the wait for the block's last dQ^T MMA.
            const int d = wtid, m = d >> 1;
            const size_t head = (size_t)bh * s.N * kDh + d;
            // token of column q (the block's slot col0 + q); tokens are rows of the head's N
            auto tok = [&](int q) {
                if constexpr (kCube) return (qmask >> q) & 1u ? slot_token_g<true>(s, qb, col0 + q) : -1;
                else return q < rows ? qb * 64 + col0 + q : -1;
            };
            float lr[kCols];
            float2 cs[kCols];
            const size_t base = ((size_t)bh * s.N + (size_t)qb * 64 + col0) * kDh + d;   // contiguous blocks
#pragma unroll
            for (int q = 0; q < kCols; ++q) {
                const int n = tok(q);
                if constexpr (kCube) lr[q] = n >= 0 ? __ldg(p.dq_lr + head + (size_t)n * kDh) : 0.0f;
                else lr[q] = q < rows ? __ldg(p.dq_lr + base + (size_t)q * kDh) : 0.0f;
                cs[q] = rope_cs(p.tab, s, n >= 0 ? n : 0, m);
            }
            if (!(ok = mbar_wait(bar(O_FULL + ob), (k >> 1) & 1, abort, s.wait_limit_ns))) break;
            fence_after_sync();
            float ov[kCols];
            ld_cols<kCols>(tmem + lane_off + 256 + ob * 64 + col0, ov);
            fence_before_sync();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(O_EMPTY + ob));
#pragma unroll
            for (int q = 0; q < kCols; ++q) {
                const float xv = ov[q] * 0.08838834764831845f;
                const float other = __shfl_xor_sync(0xffffffffu, xv, 1);
                const int n = tok(q);
                if (n >= 0) {
                    const float x0 = (d & 1) ? other : xv, x1 = (d & 1) ? xv : other;
                    // R^T: (x0 c + x1 s, x1 c - x0 s)
                    const float r = (d & 1) ? __fmaf_rn(x1, cs[q].x, -__fmul_rn(x0, cs[q].y))
                                            : __fmaf_rn(x0, cs[q].x, __fmul_rn(x1, cs[q].y));
                    p.dq[kCube ? head + (size_t)n * kDh : base + (size_t)q * kDh] = __float2bfloat16_rn(lr[q] + r);
                }
            }
        }
        if (!ok) record_timeout(p, 3);
    }
    fence_before_sync();
    __syncthreads();
    fence_after_sync();
    if (warp == kSWarp) tmem_dealloc(tmem, kTmemCols);
}

// ===========================================================================
// Key side: dK and dV.  An item is a key block (N = 64 keys) of a head; the
// query blocks that kept it (the transposed mask, ascending) are taken in
// pairs (M = 128 queries):
//   S  = Q_pair K^T        A = Q pair (K-major),   B = K block (K-major)   TMEM
//   dP = dO_pair V^T       A = dO pair (K-major),  B = V block (K-major)   TMEM
//   P, dS = P (dP - D)     by the dS warps (thread = query row), bf16 into shared memory
//   dV^T += dO_pair^T P    A = the dO pair read MN-major (M = d), B = P (MN-major)
//   dK^T += Q_pair^T dS    A = the Q pair read MN-major,          B = dS (MN-major)
// Roles as in the query-side kernel (warp 9 idles): warp 8 loads K, V (per
// item) and the Q / dO pairs (2-deep ring), warp 10 issues S and dP, warp 11
// issues dV^T and dK^T.  A key block no query block kept gets its low-rank
// rows only.

namespace kv {

constexpr int QS = 2;
constexpr uint32_t kQOBytes = 2 * kPairBytes;                     // Q pair + dO pair
constexpr uint32_t kSmK = 0, kSmV = kBlockBytes, kSmQO = 2 * kBlockBytes;
constexpr uint32_t kSmP = kSmQO + QS * kQOBytes, kSmDs = kSmP + 2 * kDsBytes;
constexpr uint32_t kTiles = kSmDs + 2 * kDsBytes;                 // 224 KB

enum Bar { KV_FULL = 0, KV_EMPTY = 1, QO_FULL = 2, QO_EMPTY = QO_FULL + QS, S_FULL = QO_EMPTY + QS,
           S_EMPTY = S_FULL + 2, DS_FULL = S_EMPTY + 2, DS_EMPTY = DS_FULL + 2, O_FULL = DS_EMPTY + 2,
           O_EMPTY = O_FULL + 2, DRAIN = O_EMPTY + 2, NUM_BARS = DRAIN + 2 };

struct Smem {
    uint64_t bar[NUM_BARS];
    uint32_t tmem_base;
    int abort;
};
static_assert(kTiles % 1024 == 0, "the control block starts aligned");

struct Params {
    Shape s;
    const int32_t* off;                 // [BH][nB + 1]
    const int32_t* list;                // [BH][nB * n_keep]
    const float* lse;
    const float* Dv;
    const float* dk_lr;
    const float* dv_lr;
    const float2* tab;
    __nv_bfloat16* dk;
    __nv_bfloat16* dv;
    DeviceStatus* status;
    int total_items;
};

__device__ __forceinline__ void timeout(const Params& p, int where)
{
    if (atomicCAS(&p.status->code, 0, (int)ROLA_ERR_TIMEOUT) == 0) p.status->where = 32 + where;
}

}  // namespace kv

template <bool kCube>
__global__ void __launch_bounds__(kThreads, 1) sparse_bwd_dkdv_tc_kernel(const __grid_constant__ CUtensorMap map_k,
                                                                         const __grid_constant__ CUtensorMap map_v,
                                                                         const __grid_constant__ CUtensorMap map_q,
                                                                         const __grid_constant__ CUtensorMap map_o,
                                                                         const kv::Params p)
{
    using namespace kv;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    if (smem_u32(smem_raw) & 1023u) {
        if (threadIdx.x == 0) atomicCAS(&p.status->code, 0, (int)ROLA_ERR_UNSUPPORTED);
        return;
    }
    kv::Smem& sm = *reinterpret_cast<kv::Smem*>(smem_raw + kTiles);
    const uint32_t sbase = smem_u32(smem_raw);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    auto bar = [&](int i) { return smem_u32(&sm.bar[i]); };
    const Shape& s = p.s;
    const int nB = s.nB;
    // the query blocks that kept key block kb of head bh: l[e0 .. e1)
    auto range = [&](int item, int& bh, int& kb, int& e0, int& len) {
        bh = item / nB;
        kb = item - bh * nB;
        const int32_t* o = p.off + (size_t)bh * (nB + 1);
        e0 = __ldg(o + kb);
        len = __ldg(o + kb + 1) - e0;
    };

    if (tid == 0) {
        sm.abort = 0;
        mbar_init(bar(KV_FULL), 1);
        mbar_init(bar(KV_EMPTY), 1);
        for (int i = 0; i < QS; ++i) {
            mbar_init(bar(QO_FULL + i), 1);
            mbar_init(bar(QO_EMPTY + i), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar(S_FULL + i), 1);
            mbar_init(bar(S_EMPTY + i), kDsWarps);
            mbar_init(bar(DS_FULL + i), kDsWarps);
            mbar_init(bar(DS_EMPTY + i), 1);
            mbar_init(bar(O_FULL + i), 1);
            mbar_init(bar(O_EMPTY + i), kDsWarps);
        }
        mbar_init(bar(DRAIN), 1);
        mbar_init(bar(DRAIN + 1), 1);
        fence_mbar_init();
    }
    if (warp == kSWarp) {
        tmem_alloc(smem_u32(&sm.tmem_base), kTmemCols);
        tmem_relinquish();
    }
    if (warp == kProdKWarp && lane == 0) {
        tma_prefetch_desc(&map_k);
        tma_prefetch_desc(&map_v);
        tma_prefetch_desc(&map_q);
        tma_prefetch_desc(&map_o);
    }
    fence_before_sync();
    __syncthreads();
    fence_after_sync();
    const uint32_t tmem = sm.tmem_base;
    volatile int* abort = &sm.abort;

    if (warp == kProdKWarp) {
        // ------------------------------------------------------------ TMA producer
        // lanes 0-3: d-chunk (lane & 1) of Q block (lane >> 1) of the pair,
        // lanes 4-7: the same of dO; the [chunk][block][row] layout.
        const int h = (lane >> 1) & 1, kc = lane & 1;
        const bool is_o = lane >= 4;
        int ko = 0, g = 0, issued_kv = 0;
        bool ok = true;
        for (int item = blockIdx.x; item < p.total_items && ok; item += gridDim.x) {
            int bh, kb, e0, len;
            range(item, bh, kb, e0, len);
            if (len == 0) continue;
            if (ko >= 1) ok = mbar_wait(bar(KV_EMPTY), (ko - 1) & 1, abort, s.wait_limit_ns);
            ok = __shfl_sync(0xffffffffu, ok, 0);
            if (!ok) break;
            if (lane == 0) {
                mbar_expect_tx(bar(KV_FULL), 2 * kBlockBytes);
                tma_load_4d(sbase + kSmK, &map_k, bar(KV_FULL), 0, kb * 64, 0, bh);
                tma_load_4d(sbase + kSmV, &map_v, bar(KV_FULL), 0, kb * 64, 0, bh);
            }
            ++issued_kv;
            const int32_t* l = p.list + (size_t)bh * nB * s.n_keep + e0;
            const int T = (len + 1) / 2;
            for (int t = 0; t < T && ok; ++t, ++g) {
                const int slot = g % QS;
                const int qa = __ldg(l + 2 * t), qb2 = 2 * t + 1 < len ? __ldg(l + 2 * t + 1) : -1;
                const int nblk = qb2 >= 0 ? 2 : 1;
                if (g >= QS) ok = mbar_wait(bar(QO_EMPTY + slot), ((g / QS) - 1) & 1, abort, s.wait_limit_ns);
                ok = __shfl_sync(0xffffffffu, ok, 0);
                if (!ok) break;
                // test hook: the CTA's first Q / dO pair is never loaded, so the waits on it run out
                const bool skip = (s.debug_flags & ROLA_DEBUG_SKIP_FIRST_K_COPY) && g == 0;
                if (lane == 0 && !skip) mbar_expect_tx(bar(QO_FULL + slot), nblk * 2 * 16384u);
                __syncwarp();
                if (lane < 8 && h < nblk && !skip)
                    tma_load_3d(sbase + kSmQO + slot * kQOBytes + (is_o ? kPairBytes : 0) + kc * 16384 + h * 8192,
                                is_o ? &map_o : &map_q, bar(QO_FULL + slot), kc * 64, (h ? qb2 : qa) * 64, bh);
            }
            ++ko;
        }
        if (!ok && lane == 0) timeout(p, 1);
        if (lane == 0) {
            int never = 0;
            if (issued_kv > 0) mbar_wait(bar(KV_FULL), (issued_kv - 1) & 1, &never, s.wait_limit_ns);
            for (int u = g > QS ? g - QS : 0; u < g; ++u)
                mbar_wait(bar(QO_FULL + u % QS), (u / QS) & 1, &never, s.wait_limit_ns);
        }
    } else if (warp == kSWarp || warp == kQWarp) {
        // ------------------------------------------------------------ MMA issuers
        if (lane == 0) {
            const bool gw = warp == kQWarp;
            const uint32_t id_s = idesc_bf16(128, 64, false, false);
            const uint32_t id_g = idesc_bf16(128, 64, true, true);
            const uint64_t dk = smem_desc(sbase + kSmK, 16, 1024);             // K: B of S (K-major)
            const uint64_t dvb = smem_desc(sbase + kSmV, 16, 1024);            // V: B of dP (K-major)
            const uint64_t dqa = smem_desc(sbase + kSmQO, 16, 1024);           // Q pair: A of S (K-major)
            const uint64_t dqm = smem_desc(sbase + kSmQO, 16384, 1024);        // Q pair: A of dK^T (MN-major)
            const uint64_t dpb = smem_desc(sbase + kSmP, 8192, 1024);          // P: B of dV^T (MN-major)
            const uint64_t dsb = smem_desc(sbase + kSmDs, 8192, 1024);         // dS: B of dK^T (MN-major)
            const uint32_t k_lo = (uint32_t)dk, k_hi = (uint32_t)(dk >> 32);
            const uint32_t v_lo = (uint32_t)dvb, v_hi = (uint32_t)(dvb >> 32);
            const uint32_t qa_lo = (uint32_t)dqa, qa_hi = (uint32_t)(dqa >> 32);
            const uint32_t qm_lo = (uint32_t)dqm, qm_hi = (uint32_t)(dqm >> 32);
            const uint32_t p_lo = (uint32_t)dpb, p_hi = (uint32_t)(dpb >> 32);
            const uint32_t ds_lo = (uint32_t)dsb, ds_hi = (uint32_t)(dsb >> 32);
            constexpr uint32_t kO = kPairBytes >> 4;                          // dO pair after the Q pair
            bool ok = true;
            int ko = 0, g = 0;
            for (int item = blockIdx.x; item < p.total_items && ok; item += gridDim.x) {
                int bh, kb, e0, len;
                range(item, bh, kb, e0, len);
                if (len == 0) continue;
                const int T = (len + 1) / 2, ob = ko & 1;
                if (!gw) {
                    if (!(ok = mbar_wait(bar(KV_FULL), ko & 1, abort, s.wait_limit_ns))) break;
                    for (int t = 0; t < T; ++t, ++g) {
                        const int sb = g & 1, slot = g % QS;
                        if (!(ok = mbar_wait(bar(QO_FULL + slot), (g / QS) & 1, abort, s.wait_limit_ns))) break;
                        if (g >= 2 && !(ok = mbar_wait(bar(S_EMPTY + sb), ((g >> 1) - 1) & 1, abort, s.wait_limit_ns)))
                            break;
                        fence_after_sync();
                        const uint32_t a = qa_lo + slot * (kQOBytes >> 4);
#pragma unroll
                        for (int kk = 0; kk < 8; ++kk) {
                            const uint32_t ao = (kk >> 2) * 1024 + (kk & 3) * 2, bo = (kk >> 2) * 512 + (kk & 3) * 2;
                            mma_ss_split(tmem + sb * 64, a + ao, qa_hi, k_lo + bo, k_hi, id_s, kk > 0 ? 1u : 0u);
                        }
#pragma unroll
                        for (int kk = 0; kk < 8; ++kk) {
                            const uint32_t ao = (kk >> 2) * 1024 + (kk & 3) * 2, bo = (kk >> 2) * 512 + (kk & 3) * 2;
                            mma_ss_split(tmem + 128 + sb * 64, a + kO + ao, qa_hi, v_lo + bo, v_hi, id_s,
                                         kk > 0 ? 1u : 0u);
                        }
                        mma_commit(bar(S_FULL + sb));
                        if (t == T - 1) mma_commit(bar(KV_EMPTY));
                    }
                } else {
                    for (int t = 0; t < T; ++t, ++g) {
                        const int sb = g & 1, slot = g % QS;
                        const bool half = 2 * t + 1 >= len;
                        if (!(ok = mbar_wait(bar(DS_FULL + sb), (g >> 1) & 1, abort, s.wait_limit_ns))) break;
                        if (t == 0 && ko >= 2 &&
                            !(ok = mbar_wait(bar(O_EMPTY + ob), ((ko >> 1) - 1) & 1, abort, s.wait_limit_ns)))
                            break;
                        fence_after_sync();
                        const uint32_t aq = qm_lo + slot * (kQOBytes >> 4);
                        const uint32_t bp = p_lo + sb * (kDsBytes >> 4), bs = ds_lo + sb * (kDsBytes >> 4);
                        const int nk = half ? 4 : 8;          // K steps of 16 queries
                        for (int kk = 0; kk < nk; ++kk)
                            mma_ss_split(tmem + 256 + ob * 64, aq + kO + kk * 128, qm_hi, bp + kk * 128, p_hi, id_g,
                                         (t > 0 || kk > 0) ? 1u : 0u);
                        for (int kk = 0; kk < nk; ++kk)
                            mma_ss_split(tmem + 384 + ob * 64, aq + kk * 128, qm_hi, bs + kk * 128, ds_hi, id_g,
                                         (t > 0 || kk > 0) ? 1u : 0u);
                        mma_commit(bar(DS_EMPTY + sb));
                        mma_commit(bar(QO_EMPTY + slot));
                    }
                    if (!ok) break;
                    mma_commit(bar(O_FULL + ob));
                }
                ++ko;
            }
            if (!ok) timeout(p, gw ? 5 : 2);
            int never = 0;
            const uint32_t drain = bar(gw ? DRAIN + 1 : DRAIN);
            mma_commit(drain);
            mbar_wait(drain, 0, &never, s.wait_limit_ns);
        }
    } else if (warp < kDsWarps) {
        // ------------------------------------------------------------ dS + epilogue
        // thread wtid: TMEM lane wtid = query row wtid of the pair (block wtid / 64)
        // for S and dP, d = wtid for dV^T and dK^T; warpgroup wg: key columns
        // [32 wg, 32 wg + 32)
        const int wg = warp >> 2, wtid = tid & 127;
        const int col0 = wg * kCols;
        const float c_log2 = s.sm_scale_log2;
        const uint32_t lane_off = (uint32_t)((warp & 3) * 32) << 16;
        bool ok = true;
        int ko = 0, g = 0;
        for (int item = blockIdx.x; item < p.total_items && ok; item += gridDim.x) {
            int bh, kb, e0, len;
            range(item, bh, kb, e0, len);
            const uint32_t kmask = slot_mask32_g<kCube>(s, kb, col0);      // key columns of this warpgroup that are tokens
            const int keys = min(64, s.N - kb * 64) - col0;                // (contiguous blocks: the first `keys` are)
            auto keyok = [&](int j) { if constexpr (kCube) return ((kmask >> j) & 1u) != 0; else return j < keys; };
            const int d = wtid;
            const size_t head = (size_t)bh * s.N * kDh + d;
            auto ktok = [&](int j) {
                if constexpr (kCube) return (kmask >> j) & 1u ? slot_token_g<true>(s, kb, col0 + j) : -1;
                else return j < keys ? kb * 64 + col0 + j : -1;
            };
            if (len == 0) {
                // no query block kept this key block: the low-rank part alone
                for (int j = 0; j < kCols; ++j) {
                    const int n = ktok(j);
                    if (n >= 0) {
                        p.dk[head + (size_t)n * kDh] = __float2bfloat16_rn(p.dk_lr[head + (size_t)n * kDh]);
                        p.dv[head + (size_t)n * kDh] = __float2bfloat16_rn(p.dv_lr[head + (size_t)n * kDh]);
                    }
                }
                continue;
            }
            const int32_t* l = p.list + (size_t)bh * nB * s.n_keep + e0;
            const int T = (len + 1) / 2, ob = ko & 1;
            // this thread's query row of tile t is in block l[2t + wtid / 64]; the block ids are
            // fetched two tiles ahead, the row's lse and D one tile ahead
            auto block_of = [&](int t) {
                const int e = 2 * t + (wtid >> 6);
                return t < T && e < len ? __ldg(l + e) : -1;
            };
            // (lse and D in block order: row 64 qblk + slot of the head's Np rows; nq < N marks a token)
            auto row_of = [&](int qblk, int& nq, float& l2q, float& Dqq) {
                if constexpr (kCube) {
                    const bool v = qblk >= 0 && slot_token_g<true>(s, qblk, wtid & 63) >= 0;
                    nq = v ? 0 : s.N;
                    const size_t r = (size_t)bh * s.Np + (size_t)(v ? qblk : 0) * 64 + (wtid & 63);
                    l2q = v ? __ldg(p.lse + r) * 1.4426950408889634f : 0.0f;
                    Dqq = v ? __ldg(p.Dv + r) : 0.0f;
                } else {
                    nq = qblk >= 0 ? qblk * 64 + (wtid & 63) : s.N;
                    const bool v = nq < s.N;
                    l2q = v ? __ldg(p.lse + (size_t)bh * s.N + nq) * 1.4426950408889634f : 0.0f;
                    Dqq = v ? __ldg(p.Dv + (size_t)bh * s.N + nq) : 0.0f;
                }
            };
            int n_nx, blk_nx2 = block_of(1);
            float l2_nx, D_nx;
            row_of(block_of(0), n_nx, l2_nx, D_nx);
            for (int t = 0; t < T; ++t, ++g) {
                const int sb = g & 1;
                const int n = n_nx;
                const float l2 = l2_nx, Dq = D_nx;
                if (t + 1 < T) {
                    row_of(blk_nx2, n_nx, l2_nx, D_nx);
                    blk_nx2 = block_of(t + 2);
                }
                const bool vq = n < s.N;
                if (!(ok = mbar_wait(bar(S_FULL + sb), (g >> 1) & 1, abort, s.wait_limit_ns))) break;
                fence_after_sync();
                float x[kCols], y[kCols];
                ld_cols<kCols>(tmem + lane_off + sb * 64 + col0, x);
                ld_cols<kCols>(tmem + lane_off + 128 + sb * 64 + col0, y);
                fence_before_sync();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(S_EMPTY + sb));
                uint32_t pp[kCols / 2], pd[kCols / 2];
#pragma unroll
                for (int j = 0; j < kCols; j += 2) {
                    const float p0 = vq && keyok(j) ? fast_exp2(fmaf(x[j], c_log2, -l2)) : 0.0f;
                    const float p1 = vq && keyok(j + 1) ? fast_exp2(fmaf(x[j + 1], c_log2, -l2)) : 0.0f;
                    pp[j >> 1] = pack_bf16(p0, p1);
                    pd[j >> 1] = pack_bf16(p0 * (y[j] - Dq), p1 * (y[j + 1] - Dq));
                }
                if (g >= 2 && !(ok = mbar_wait(bar(DS_EMPTY + sb), ((g >> 1) - 1) & 1, abort, s.wait_limit_ns)))
                    break;
                const uint32_t roff = (wtid >> 3) * 1024 + (wtid & 7) * 128;
                const uint32_t prow = sbase + kSmP + sb * kDsBytes + roff, drow = sbase + kSmDs + sb * kDsBytes + roff;
#pragma unroll
                for (int c = 0; c < kCols / 8; ++c) {
                    const uint32_t sw = ((wg * (kCols / 8) + c) ^ (wtid & 7)) << 4;
                    asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};\n" ::"r"(prow + sw), "r"(pp[4 * c]),
                                 "r"(pp[4 * c + 1]), "r"(pp[4 * c + 2]), "r"(pp[4 * c + 3])
                                 : "memory");
                    asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};\n" ::"r"(drow + sw), "r"(pd[4 * c]),
                                 "r"(pd[4 * c + 1]), "r"(pd[4 * c + 2]), "r"(pd[4 * c + 3])
                                 : "memory");
                }
                fence_proxy_async_smem();
                fence_before_sync();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(DS_FULL + sb));
            }
            if (!ok) break;
            // ---- epilogue: dv = low-rank + dV, dk = low-rank + R^T (dK / sqrt d); thread wtid
            // holds d = wtid of this warpgroup's 32 keys; the pair partner d ^ 1 is lane ^ 1.
            // The low-rank rows are read before the wait for the block's last MMAs.
            float lk[kCols], lv[kCols];
            const size_t base = ((size_t)bh * s.N + (size_t)kb * 64 + col0) * kDh + d;   // contiguous blocks
#pragma unroll
            for (int j = 0; j < kCols; ++j) {
                if constexpr (kCube) {
                    const int n = ktok(j);
                    lk[j] = n >= 0 ? __ldg(p.dk_lr + head + (size_t)n * kDh) : 0.0f;
                    lv[j] = n >= 0 ? __ldg(p.dv_lr + head + (size_t)n * kDh) : 0.0f;
                } else {
                    lk[j] = j < keys ? __ldg(p.dk_lr + base + (size_t)j * kDh) : 0.0f;
                    lv[j] = j < keys ? __ldg(p.dv_lr + base + (size_t)j * kDh) : 0.0f;
                }
            }
            if (!(ok = mbar_wait(bar(O_FULL + ob), (ko >> 1) & 1, abort, s.wait_limit_ns))) break;
            fence_after_sync();
            float av[kCols], ak[kCols];
            ld_cols<kCols>(tmem + lane_off + 256 + ob * 64 + col0, av);
            ld_cols<kCols>(tmem + lane_off + 384 + ob * 64 + col0, ak);
            fence_before_sync();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(O_EMPTY + ob));
            const int m = d >> 1;
#pragma unroll
            for (int j = 0; j < kCols; ++j) {
                const float xk = ak[j] * 0.08838834764831845f;
                const float other = __shfl_xor_sync(0xffffffffu, xk, 1);
                const int nk = ktok(j);
                if (nk >= 0) {
                    const float2 cs = rope_cs(p.tab, s, nk, m);
                    const float x0 = (d & 1) ? other : xk, x1 = (d & 1) ? xk : other;
                    const float r = (d & 1) ? __fmaf_rn(x1, cs.x, -__fmul_rn(x0, cs.y))
                                            : __fmaf_rn(x0, cs.x, __fmul_rn(x1, cs.y));
                    const size_t e = kCube ? head + (size_t)nk * kDh : base + (size_t)j * kDh;
                    p.dk[e] = __float2bfloat16_rn(lk[j] + r);
                    p.dv[e] = __float2bfloat16_rn(lv[j] + av[j]);
                }
            }
            ++ko;
        }
        if (!ok) timeout(p, 3);
    }
    fence_before_sync();
    __syncthreads();
    fence_after_sync();
    if (warp == kSWarp) tmem_dealloc(tmem, kTmemCols);
}

}  // namespace

cudaError_t launch_sparse_bwd_dq_tc(const Shape& s, const void* qr, const void* kr, const void* v, const void* dOs,
                                    const int32_t* kv_idx, const float* lse, const float* Dv, const float2* tab,
                                    const float* dq_lr, void* dq, DeviceStatus* status, cudaStream_t st)
{
    // the maps span the block-ordered rows (the token order itself for contiguous chunks)
    Shape rows = s;
    rows.N = s.Np;
    CUtensorMap mq, mo, mk, mv;
    if (!make_block_map(&mq, qr, rows) || !make_block_map(&mo, dOs, rows) || !make_chunk_map(&mk, kr, rows) ||
        !make_chunk_map(&mv, v, rows))
        return cudaErrorInvalidValue;
    int dev = 0, nsm = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    dq::Params p;
    p.s = s;
    p.kv_idx = kv_idx;
    p.lse = lse;
    p.Dv = Dv;
    p.dq_lr = dq_lr;
    p.tab = tab;
    p.dq = static_cast<__nv_bfloat16*>(dq);
    p.status = status;
    p.total_items = s.B * s.H * s.nB;
    p.tiles = (s.n_keep + 1) / 2;
    const size_t smem = kSmemTiles + sizeof(dq::Smem);
    auto kernel = s.cube ? sparse_bwd_dq_tc_kernel<true> : sparse_bwd_dq_tc_kernel<false>;
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int grid = p.total_items < nsm ? p.total_items : nsm;
    kernel<<<grid, kThreads, smem, st>>>(mq, mo, mk, mv, p);
    return cudaGetLastError();
}

cudaError_t launch_sparse_bwd_dkdv_tc(const Shape& s, const void* qr, const void* kr, const void* v, const void* dOs,
                                      const int32_t* off, const int32_t* list, const float* lse, const float* Dv,
                                      const float2* tab, const float* dk_lr, const float* dv_lr, void* dk, void* dv,
                                      DeviceStatus* status, cudaStream_t st)
{
    Shape rows = s;
    rows.N = s.Np;
    CUtensorMap mk, mv, mq, mo;
    if (!make_block_map(&mk, kr, rows) || !make_block_map(&mv, v, rows) || !make_chunk_map(&mq, qr, rows) ||
        !make_chunk_map(&mo, dOs, rows))
        return cudaErrorInvalidValue;
    int dev = 0, nsm = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    kv::Params p;
    p.s = s;
    p.off = off;
    p.list = list;
    p.lse = lse;
    p.Dv = Dv;
    p.dk_lr = dk_lr;
    p.dv_lr = dv_lr;
    p.tab = tab;
    p.dk = static_cast<__nv_bfloat16*>(dk);
    p.dv = static_cast<__nv_bfloat16*>(dv);
    p.status = status;
    p.total_items = s.B * s.H * s.nB;
    const size_t smem = kv::kTiles + sizeof(kv::Smem);
    auto kernel = s.cube ? sparse_bwd_dkdv_tc_kernel<true> : sparse_bwd_dkdv_tc_kernel<false>;
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int grid = p.total_items < nsm ? p.total_items : nsm;
    kernel<<<grid, kThreads, smem, st>>>(mk, mv, mq, mo, p);
    return cudaGetLastError();
}

}  // namespace rola
