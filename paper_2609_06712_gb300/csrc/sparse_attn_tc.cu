// Block-sparse softmax attention on the 5th-generation tensor cores (kernel 2, bf16).
//
//   O^s_p = sum_{q in kept(i)} softmax_q(q^r_p . k^r_q / sqrt(d_h)) v_q,   p in query block i
//
// (Sec. 3 softmax form restricted to the kept key blocks, Alg. 1 sparse branch.)
//
// Mapping to tcgen05.  A query block has only 64 rows, but every MMA here
// has M = 128: the kernel works on the TRANSPOSED problem, with a pair of
// kept 64-key blocks as the 128-row operand.
//   S^T[key][q]  = K_pair (128 x 128, smem, K-major)  x  Q^T (N = 64, smem, K-major)
//   O^T[d][q]   += V_pair^T (128 x 128 keys, smem, MN-major) x P^T (128 keys x 64 q, smem, MN-major)
// S^T and O^T live in TMEM (fp32); TMEM lane = key (for S^T) or d (for O^T).
//
// Softmax.  A softmax thread owns one key (one TMEM lane) and sees that
// key's 64 scores.  Per-query statistics therefore cross threads, so the
// running maximum m_q is kept lazily: scores are exponentiated against the
// current m_q; only when some score exceeds m_q by more than 2^8 (in base 2)
// does the warpgroup compute the tile's exact column maxima, raise m_q and
// rescale O^T (in TMEM) and its row sums.  The first tile of a query block
// always takes that path.  Row sums are accumulated per thread and reduced
// across the 128 threads once per query block.  Weights are rounded to bf16
// for the P V product and the row sums add the same rounded values.
//
// Warp roles (192 threads, one persistent CTA per SM):
//   warps 0-3  softmax + epilogue (TMEM lanes 32w .. 32w+31)
//   warp  4    TMA producer: Q (per query block), K and V pairs (per tile)
//   warp  5    MMA issuer and TMEM owner
// Double buffers: Q, K, V, S^T, P^T and O^T, so the next tile's Q K^T runs
// while the current tile's softmax does, and the next query block's first
// tiles run while the current one's epilogue does.  Every wait on an
// mbarrier is bounded (2 s); a wait that gives up records ROLA_ERR_TIMEOUT
// in the workspace status word, and the CTA stops issuing, drains what it
// issued and releases its TMEM.
#include <cudaTypedefs.h>

#include "common.cuh"
#include "tcgen05.cuh"

namespace rola {
namespace {

using namespace tc;

constexpr int kThreads = 192;
constexpr int kSoftmaxThreads = 128;
constexpr uint32_t kQBytes = 64 * 128 * 2;          // one query block
constexpr uint32_t kKVBytes = 128 * 128 * 2;        // a pair of key blocks
constexpr uint32_t kPBytes = 128 * 64 * 2;          // P^T tile
constexpr uint32_t kOBytes = 64 * 128 * 2;          // output staging
constexpr uint32_t kSmemQ = 0;
constexpr uint32_t kSmemK = kSmemQ + 2 * kQBytes;
constexpr uint32_t kSmemV = kSmemK + 2 * kKVBytes;
constexpr uint32_t kSmemP = kSmemV + 2 * kKVBytes;
constexpr uint32_t kSmemO = kSmemP + 2 * kPBytes;
constexpr uint32_t kSmemTiles = kSmemO + kOBytes;   // 208 KB, 1024-aligned pieces
constexpr uint32_t kTmemCols = 256;                 // S^T x2 (64 cols each), O^T x2
constexpr uint64_t kWaitLimitNs = 2000000000ull;
constexpr float kRescaleThreshold = 8.0f;           // log2 units

enum Bar { Q_FULL = 0, Q_EMPTY = 2, K_FULL = 4, K_EMPTY = 6, V_FULL = 8, V_EMPTY = 10, S_FULL = 12,
           S_EMPTY = 14, P_FULL = 16, PV_DONE = 18, O_FULL = 20, O_EMPTY = 22, DRAIN = 24, NUM_BARS = 25 };

struct Smem {
    uint64_t bar[NUM_BARS];
    uint32_t tmem_base;
    int abort;
    float m[64];          // running maximum per query (log2 units)
    float alpha[64];      // rescale factors of the current tile
    float red[4][64];     // cross-warp reduction scratch
    float inv_l[64];
};

struct Params {
    Shape s;
    const int32_t* kv_idx;
    __nv_bfloat16* o;
    DeviceStatus* status;
    int total_items;      // B*H*nB
    int tiles;            // ceil(n_keep / 2)
};

__device__ __forceinline__ void record_timeout(const Params& p, int where)
{
    if (atomicCAS(&p.status->code, 0, (int)ROLA_ERR_TIMEOUT) == 0) p.status->where = where;
}

// Column reduction of v[64] over the 128 softmax threads; result for
// column q in out[q] (q < 64).  MAX selects max, else sum.  Uses named barrier 1.
template <bool MAX>
__device__ __forceinline__ void column_reduce(float (&v)[64], Smem& sm, int tid, float* out)
{
    const int lane = tid & 31, warp = tid >> 5;
#pragma unroll
    for (int step = 0; step < 5; ++step) {
        const int off = 16 >> step;
        const int half = 32 >> step;              // values kept after this step
        const bool upper = (lane & off) != 0;
#pragma unroll
        for (int i = 0; i < 32; ++i) {
            if (i < half) {
                float keep = upper ? v[i + half] : v[i];
                float send = upper ? v[i] : v[i + half];
                float recv = __shfl_xor_sync(0xffffffffu, send, off);
                v[i] = MAX ? fmaxf(keep, recv) : keep + recv;
            }
        }
    }
    // lane holds columns 2*lane, 2*lane+1
    sm.red[warp][2 * lane] = v[0];
    sm.red[warp][2 * lane + 1] = v[1];
    bar_sync(1, kSoftmaxThreads);
    if (tid < 64) {
        float a = sm.red[0][tid], b = sm.red[1][tid], c = sm.red[2][tid], d = sm.red[3][tid];
        out[tid] = MAX ? fmaxf(fmaxf(a, b), fmaxf(c, d)) : (a + b) + (c + d);
    }
    bar_sync(1, kSoftmaxThreads);
}

__device__ __forceinline__ void tmem_ld64(uint32_t taddr, float (&v)[64])
{
    float (&a)[16] = *reinterpret_cast<float(*)[16]>(&v[0]);
    float (&b)[16] = *reinterpret_cast<float(*)[16]>(&v[16]);
    float (&c)[16] = *reinterpret_cast<float(*)[16]>(&v[32]);
    float (&d)[16] = *reinterpret_cast<float(*)[16]>(&v[48]);
    tmem_ld16(taddr, a);
    tmem_ld16(taddr + 16, b);
    tmem_ld16(taddr + 32, c);
    tmem_ld16(taddr + 48, d);
    tmem_ld_wait(a);
    reg_fence(b);
    reg_fence(c);
    reg_fence(d);
}

__global__ void __launch_bounds__(kThreads, 1) sparse_attn_tc_kernel(const __grid_constant__ CUtensorMap map_q,
                                                                     const __grid_constant__ CUtensorMap map_k,
                                                                     const __grid_constant__ CUtensorMap map_v,
                                                                     const Params p)
{
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* tiles = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    Smem& sm = *reinterpret_cast<Smem*>(tiles + kSmemTiles);
    const uint32_t sbase = smem_u32(tiles);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    auto bar = [&](int i) { return smem_u32(&sm.bar[i]); };

    const Shape& s = p.s;
    const int T = p.tiles;
    const int nB = s.nB;

    if (tid == 0) {
        sm.abort = 0;
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar(Q_FULL + i), 1);
            mbar_init(bar(Q_EMPTY + i), 1);
            mbar_init(bar(K_FULL + i), 1);
            mbar_init(bar(K_EMPTY + i), 1);
            mbar_init(bar(V_FULL + i), 1);
            mbar_init(bar(V_EMPTY + i), 1);
            mbar_init(bar(S_FULL + i), 1);
            mbar_init(bar(S_EMPTY + i), 4);
            mbar_init(bar(P_FULL + i), 4);
            mbar_init(bar(PV_DONE + i), 1);
            mbar_init(bar(O_FULL + i), 1);
            mbar_init(bar(O_EMPTY + i), 4);
        }
        mbar_init(bar(DRAIN), 1);
        fence_mbar_init();
    }
    if (warp == 5) {
        tmem_alloc(smem_u32(&sm.tmem_base), kTmemCols);
        tmem_relinquish();
    }
    if (warp == 4 && lane == 0) {
        tma_prefetch_desc(&map_q);
        tma_prefetch_desc(&map_k);
        tma_prefetch_desc(&map_v);
    }
    fence_before_sync();
    __syncthreads();
    fence_after_sync();
    const uint32_t tmem = sm.tmem_base;
    volatile int* abort = &sm.abort;

    if (warp == 4) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            int k = 0, issued_q = 0, issued_k = 0, issued_v = 0;
            bool ok = true;
            for (int item = blockIdx.x; item < p.total_items && ok; item += gridDim.x, ++k) {
                const int bh = item / nB, qb = item - bh * nB;
                const int32_t* kept = p.kv_idx + (size_t)item * s.n_keep;
                const int qs = k & 1;
                if (k >= 2 && !(ok = mbar_wait(bar(Q_EMPTY + qs), ((k >> 1) - 1) & 1, abort, kWaitLimitNs))) break;
                mbar_expect_tx(bar(Q_FULL + qs), kQBytes);
                for (int c = 0; c < 2; ++c)
                    tma_load_3d(sbase + kSmemQ + qs * kQBytes + c * 8192, &map_q, bar(Q_FULL + qs), c * 64, qb * 64, bh);
                ++issued_q;
                for (int t = 0; t < T; ++t) {
                    const int g = k * T + t, st = g & 1;
                    const int ja = __ldg(kept + 2 * t);
                    const int jb = 2 * t + 1 < s.n_keep ? __ldg(kept + 2 * t + 1) : -1;
                    const uint32_t bytes = (jb >= 0 ? 2u : 1u) * 16384u;
                    if (g >= 2 && !(ok = mbar_wait(bar(K_EMPTY + st), ((g >> 1) - 1) & 1, abort, kWaitLimitNs))) break;
                    mbar_expect_tx(bar(K_FULL + st), bytes);
                    for (int c = 0; c < 2; ++c) {
                        tma_load_3d(sbase + kSmemK + st * kKVBytes + c * 16384, &map_k, bar(K_FULL + st), c * 64,
                                    ja * 64, bh);
                        if (jb >= 0)
                            tma_load_3d(sbase + kSmemK + st * kKVBytes + c * 16384 + 8192, &map_k, bar(K_FULL + st),
                                        c * 64, jb * 64, bh);
                    }
                    ++issued_k;
                    if (g >= 2 && !(ok = mbar_wait(bar(V_EMPTY + st), ((g >> 1) - 1) & 1, abort, kWaitLimitNs))) break;
                    mbar_expect_tx(bar(V_FULL + st), bytes);
                    for (int c = 0; c < 2; ++c) {
                        tma_load_3d(sbase + kSmemV + st * kKVBytes + c * 16384, &map_v, bar(V_FULL + st), c * 64,
                                    ja * 64, bh);
                        if (jb >= 0)
                            tma_load_3d(sbase + kSmemV + st * kKVBytes + c * 16384 + 8192, &map_v, bar(V_FULL + st),
                                        c * 64, jb * 64, bh);
                    }
                    ++issued_v;
                }
            }
            if (!ok) record_timeout(p, 1);
            // every TMA this thread issued must land before the CTA exits: wait
            // for the latest issued phase of each buffer, bounded by time only
            int never = 0;
            for (int b = 0; b < 2; ++b) {
                if (issued_q > b) {
                    const int last = issued_q - 1 - ((issued_q - 1 - b) & 1);
                    mbar_wait(bar(Q_FULL + b), (last >> 1) & 1, &never, kWaitLimitNs);
                }
                if (issued_k > b) {
                    const int last = issued_k - 1 - ((issued_k - 1 - b) & 1);
                    mbar_wait(bar(K_FULL + b), (last >> 1) & 1, &never, kWaitLimitNs);
                }
                if (issued_v > b) {
                    const int last = issued_v - 1 - ((issued_v - 1 - b) & 1);
                    mbar_wait(bar(V_FULL + b), (last >> 1) & 1, &never, kWaitLimitNs);
                }
            }
        }
    } else if (warp == 5) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t id_qk = idesc_bf16(128, 64, false, false);
            const uint32_t id_pv = idesc_bf16(128, 64, true, true);
            bool ok = true;
            int k = 0;
            // PV of global tile gp (item-local tile tp) into O buffer ob
            auto issue_pv = [&](int gp, int tp, int ob, int kitem) -> bool {
                const int pb = gp & 1;
                if (!mbar_wait(bar(P_FULL + pb), (gp >> 1) & 1, abort, kWaitLimitNs)) return false;
                if (!mbar_wait(bar(V_FULL + pb), (gp >> 1) & 1, abort, kWaitLimitNs)) return false;
                if (tp == 0 && kitem >= 2 &&
                    !mbar_wait(bar(O_EMPTY + ob), ((kitem >> 1) - 1) & 1, abort, kWaitLimitNs))
                    return false;
                fence_after_sync();
                const bool half = 2 * tp + 1 >= s.n_keep;
                const uint32_t vaddr = sbase + kSmemV + pb * kKVBytes;
                const uint32_t paddr = sbase + kSmemP + pb * kPBytes;
                const uint32_t d = tmem + 128 + ob * 64;
#pragma unroll
                for (int kk = 0; kk < 8; ++kk) {
                    if (half && kk >= 4) break;
                    mma_ss(d, smem_desc(vaddr + kk * 2048, 16384, 1024), smem_desc(paddr + kk * 2048, 8192, 1024),
                           id_pv, (tp > 0 || kk > 0) ? 1u : 0u);
                }
                mma_commit(bar(PV_DONE + pb));
                mma_commit(bar(V_EMPTY + pb));
                return true;
            };
            for (int item = blockIdx.x; item < p.total_items && ok; item += gridDim.x, ++k) {
                const int qs = k & 1, ob = k & 1;
                if (!(ok = mbar_wait(bar(Q_FULL + qs), (k >> 1) & 1, abort, kWaitLimitNs))) break;
                const uint32_t qaddr = sbase + kSmemQ + qs * kQBytes;
                for (int t = 0; t < T; ++t) {
                    const int g = k * T + t, st = g & 1;
                    if (!(ok = mbar_wait(bar(K_FULL + st), (g >> 1) & 1, abort, kWaitLimitNs))) break;
                    if (g >= 2 && !(ok = mbar_wait(bar(S_EMPTY + st), ((g >> 1) - 1) & 1, abort, kWaitLimitNs))) break;
                    fence_after_sync();
                    const uint32_t kaddr = sbase + kSmemK + st * kKVBytes;
                    const uint32_t d = tmem + st * 64;
#pragma unroll
                    for (int kk = 0; kk < 8; ++kk)
                        mma_ss(d, smem_desc(kaddr + (kk >> 2) * 16384 + (kk & 3) * 32, 16, 1024),
                               smem_desc(qaddr + (kk >> 2) * 8192 + (kk & 3) * 32, 16, 1024), id_qk, kk > 0 ? 1u : 0u);
                    mma_commit(bar(S_FULL + st));
                    mma_commit(bar(K_EMPTY + st));
                    if (t == T - 1) mma_commit(bar(Q_EMPTY + qs));
                    if (t >= 1 && !(ok = issue_pv(g - 1, t - 1, ob, k))) break;
                }
                if (!ok) break;
                if (!(ok = issue_pv(k * T + T - 1, T - 1, ob, k))) break;
                mma_commit(bar(O_FULL + ob));
            }
            if (!ok) record_timeout(p, 2);
            // drain: every MMA issued by this thread completes before TMEM is released
            int never = 0;
            mma_commit(bar(DRAIN));
            mbar_wait(bar(DRAIN), 0, &never, kWaitLimitNs);
        }
    } else {
        // ------------------------------------------------------------ softmax + epilogue
        const float c_log2 = s.sm_scale_log2;
        const uint32_t lane_off = (uint32_t)(warp * 32) << 16;
        bool ok = true;
        int k = 0;
        for (int item = blockIdx.x; item < p.total_items && ok; item += gridDim.x, ++k) {
            const int bh = item / nB, qb = item - bh * nB;
            const int32_t* kept = p.kv_idx + (size_t)item * s.n_keep;
            const int ob = k & 1;
            if (tid < 64) sm.m[tid] = -INFINITY;
            float l[64];
#pragma unroll
            for (int q = 0; q < 64; ++q) l[q] = 0.0f;
            bar_sync(1, kSoftmaxThreads);
            for (int t = 0; t < T; ++t) {
                const int g = k * T + t, sb = g & 1;
                const int ja = __ldg(kept + 2 * t);
                const int jb = 2 * t + 1 < s.n_keep ? __ldg(kept + 2 * t + 1) : -1;
                const int blk = tid < 64 ? ja : jb;
                const int key = blk * 64 + (tid & 63);
                const bool valid = blk >= 0 && key < s.N;
                if (!(ok = mbar_wait(bar(S_FULL + sb), (g >> 1) & 1, abort, kWaitLimitNs))) break;
                fence_after_sync();
                const uint32_t saddr = tmem + lane_off + sb * 64;
                float x[64];
                tmem_ld64(saddr, x);
                bool need = false;
#pragma unroll
                for (int q = 0; q < 64; q += 4) {
                    float4 m4 = *reinterpret_cast<const float4*>(&sm.m[q]);
                    float mm[4] = {m4.x, m4.y, m4.z, m4.w};
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        float xv = valid ? x[q + e] * c_log2 : -INFINITY;
                        x[q + e] = xv;
                        need |= xv > mm[e] + kRescaleThreshold;
                    }
                }
                if (bar_red_or(1, kSoftmaxThreads, need)) {
                    column_reduce<true>(x, sm, tid, sm.alpha);        // alpha <- tile maxima (x consumed)
                    if (tid < 64) {
                        const float mo = sm.m[tid];
                        const float mn = fmaxf(mo, sm.alpha[tid]);
                        sm.alpha[tid] = fast_exp2(mo - mn);            // 0 when mo = -inf
                        sm.m[tid] = mn;
                    }
                    bar_sync(1, kSoftmaxThreads);
                    tmem_ld64(saddr, x);                               // S^T is still ours: reload
#pragma unroll
                    for (int q = 0; q < 64; ++q) x[q] = valid ? x[q] * c_log2 : -INFINITY;
                    if (t > 0) {
                        // O^T must hold PV(t-1) before it is rescaled
                        if (!(ok = mbar_wait(bar(PV_DONE + ((g - 1) & 1)), ((g - 1) >> 1) & 1, abort, kWaitLimitNs)))
                            break;
                        fence_after_sync();
                        const uint32_t oaddr = tmem + lane_off + 128 + ob * 64;
#pragma unroll
                        for (int c = 0; c < 4; ++c) {
                            float ov[16];
                            tmem_ld16(oaddr + c * 16, ov);
                            tmem_ld_wait(ov);
#pragma unroll
                            for (int e = 0; e < 16; ++e) ov[e] *= sm.alpha[c * 16 + e];
                            tmem_st16(oaddr + c * 16, ov);
                        }
                        tmem_st_wait();
#pragma unroll
                        for (int q = 0; q < 64; ++q) l[q] *= sm.alpha[q];
                    }
                }
                fence_before_sync();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(S_EMPTY + sb));
                // P^T row of this key, bf16, 128-byte-swizzled
                uint32_t pk[32];
#pragma unroll
                for (int q = 0; q < 64; q += 4) {
                    float4 m4 = *reinterpret_cast<const float4*>(&sm.m[q]);
                    float mm[4] = {m4.x, m4.y, m4.z, m4.w};
#pragma unroll
                    for (int e = 0; e < 4; e += 2) {
                        float p0 = fast_exp2(x[q + e] - mm[e]);
                        float p1 = fast_exp2(x[q + e + 1] - mm[e + 1]);
                        uint32_t u = pack_bf16(p0, p1);
                        float2 r = unpack_bf16(u);
                        l[q + e] += r.x;
                        l[q + e + 1] += r.y;
                        pk[(q + e) >> 1] = u;
                    }
                }
                if (g >= 2 && !(ok = mbar_wait(bar(PV_DONE + sb), ((g >> 1) - 1) & 1, abort, kWaitLimitNs))) break;
                const uint32_t prow = sbase + kSmemP + sb * kPBytes + (tid >> 3) * 1024 + (tid & 7) * 128;
#pragma unroll
                for (int c = 0; c < 8; ++c)
                    asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};\n" ::"r"(prow + ((c ^ (tid & 7)) << 4)),
                                 "r"(pk[4 * c]), "r"(pk[4 * c + 1]), "r"(pk[4 * c + 2]), "r"(pk[4 * c + 3])
                                 : "memory");
                fence_proxy_async_smem();
                fence_before_sync();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(P_FULL + sb));
            }
            if (!ok) break;
            // ---- epilogue: O^s = O^T / l, transposed through shared memory
            if (!(ok = mbar_wait(bar(O_FULL + ob), (k >> 1) & 1, abort, kWaitLimitNs))) break;
            fence_after_sync();
            column_reduce<false>(l, sm, tid, sm.inv_l);
            if (tid < 64) sm.inv_l[tid] = 1.0f / sm.inv_l[tid];
            bar_sync(1, kSoftmaxThreads);
            {
                float ov[64];
                tmem_ld64(tmem + lane_off + 128 + ob * 64, ov);
                fence_before_sync();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(O_EMPTY + ob));
                __nv_bfloat16* ostage = reinterpret_cast<__nv_bfloat16*>(tiles + kSmemO);
#pragma unroll
                for (int q = 0; q < 64; ++q) ostage[q * 128 + tid] = __float2bfloat16_rn(ov[q] * sm.inv_l[q]);
            }
            bar_sync(1, kSoftmaxThreads);
            {
                const uint4* src = reinterpret_cast<const uint4*>(tiles + kSmemO);
                __nv_bfloat16* dst = p.o + ((size_t)bh * s.N + (size_t)qb * 64) * kDh;
#pragma unroll
                for (int it = 0; it < 8; ++it) {
                    const int e = it * kSoftmaxThreads + tid;
                    const int row = e >> 4, c = e & 15;
                    if (qb * 64 + row < s.N)
                        *reinterpret_cast<uint4*>(dst + (size_t)row * kDh + c * 8) = src[e];
                }
            }
            bar_sync(1, kSoftmaxThreads);
        }
        if (!ok) record_timeout(p, 3);
    }
    fence_before_sync();
    __syncthreads();
    fence_after_sync();
    if (warp == 5) tmem_dealloc(tmem, kTmemCols);
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn()
{
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        void* f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
    }
    return fn;
}

// [BH][N][128] bf16 viewed as a 3-D tensor (d, token, head); 64 x 64 boxes,
// 128-byte swizzle; rows past N read as zero.
bool make_map(CUtensorMap* m, const void* ptr, const Shape& s)
{
    auto enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[3] = {(cuuint64_t)kDh, (cuuint64_t)s.N, (cuuint64_t)s.B * s.H};
    cuuint64_t strides[2] = {(cuuint64_t)kDh * 2, (cuuint64_t)s.N * kDh * 2};
    cuuint32_t box[3] = {64, 64, 1};
    cuuint32_t es[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(ptr), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

cudaError_t launch_sparse_attn_tc(const Shape& s, const void* qr, const void* kr, const void* v,
                                  const int32_t* kv_idx, void* o_s, DeviceStatus* status, cudaStream_t st)
{
    CUtensorMap mq, mk, mv;
    if (!make_map(&mq, qr, s) || !make_map(&mk, kr, s) || !make_map(&mv, v, s)) return cudaErrorInvalidValue;
    int dev = 0, nsm = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    Params p;
    p.s = s;
    p.kv_idx = kv_idx;
    p.o = static_cast<__nv_bfloat16*>(o_s);
    p.status = status;
    p.total_items = s.B * s.H * s.nB;
    p.tiles = (s.n_keep + 1) / 2;
    const size_t smem = 1024 + kSmemTiles + sizeof(Smem);
    e = cudaFuncSetAttribute(sparse_attn_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int grid = p.total_items < nsm ? p.total_items : nsm;
    sparse_attn_tc_kernel<<<grid, kThreads, smem, st>>>(mq, mk, mv, p);
    return cudaGetLastError();
}

}  // namespace rola
