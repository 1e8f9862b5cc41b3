// Block-sparse softmax attention on the 5th-generation tensor cores (kernel 2, bf16).
//
//   O^s_p = sum_{q in kept(i)} softmax_q(q^r_p . k^r_q / sqrt(d_h)) v_q,   p in query block i
//
// (Sec. 3 softmax form restricted to the kept key blocks, Alg. 1 sparse branch.)
//
// This transposed form serves the 4 x 4 x 4 cube geometry, where a thread per
// key keeps the slot-validity test and the scatter of O^s rows local;
// contiguous key blocks run the row-wise kernel of sparse_attn_rows.cu.
//
// Mapping to tcgen05.  A query block has only 64 rows, but every MMA here
// has M = 128: the kernel works on the TRANSPOSED problem, with a pair of
// kept 64-key blocks as the 128-row operand.
//   S^T[key][q]  = K_pair (128 x 128, smem, K-major)  x  Q^T (N = 64, smem, K-major)
//   O^T[d][q]   += V_pair^T (128 x 128 keys, smem, MN-major) x P^T (128 keys x 64 q, smem, MN-major)
// Shared-memory tiles: Q [chunk][64 rows], K pair [chunk][block][64 rows],
// V pair [block][chunk][64 rows], rows of 128 B in 128-byte swizzle atoms.
// S^T and O^T live in TMEM (fp32); TMEM lane = key (for S^T) or d (for O^T).
//
// Softmax.  A softmax thread owns one key (one TMEM lane) and sees that
// key's 64 scores.  Per-query statistics therefore cross threads, so the
// running maximum m_q is kept lazily: scores are exponentiated against the
// current m_q; only when some score exceeds m_q by more than 2^8 (in base 2)
// does the warpgroup compute the tile's exact column maxima, raise m_q and
// rescale O^T (in TMEM) and its row sums.  The first tile of a query block
// always takes that path.  Row sums are accumulated per thread in fp32 and
// reduced across the 128 threads once per query block; the weights enter the
// P V product rounded to bf16.
//
// Warp roles (384 threads, one persistent CTA per SM):
//   warps 0-7  softmax + epilogue: two warpgroups, each owning 32 of the 64
//              query columns of every tile (warp w reads TMEM lanes
//              32 (w mod 4) .. +31, so every warpgroup sees all 128 keys;
//              the warpgroup count is a compile-time parameter)
//   warp  8    TMA producer: Q (per query block) and the K pairs
//   warp  9    TMA producer: the V blocks
//   warp 10    Q K^T issuer and TMEM owner
//   warp 11    P V issuer
// Buffers: K pairs in a 2-deep ring and V blocks in a 7-deep ring of single
// blocks (a V block is needed a softmax later than its K pair, so V gets the
// deeper ring; 224 KB of the 227 KB go to tiles); S^T, P^T and O^T double-buffered, so the next tile's Q K^T
// runs while the current tile's softmax does and the next query block's
// first tiles run while the current one's epilogue does; Q single-buffered.  Every wait on an
// mbarrier is bounded (2 s); a wait that gives up records ROLA_ERR_TIMEOUT
// in the workspace status word, and the CTA stops issuing, drains what it
// issued and releases its TMEM.
#include <cudaTypedefs.h>
#include <stddef.h>

#include "common.cuh"
#include "tcgen05.cuh"
#include "tensor_map.cuh"

namespace rola {
namespace {

using namespace tc;

constexpr int kSoftmaxWG = 2;                        // softmax warpgroups, each owns 64/kSoftmaxWG query columns
constexpr int kCols = 64 / kSoftmaxWG;               // query columns per softmax warpgroup
constexpr int kSoftmaxWarps = 4 * kSoftmaxWG;
constexpr int kProducerKWarp = kSoftmaxWarps;      // Q and the K pairs
constexpr int kProducerVWarp = kSoftmaxWarps + 1;  // V blocks
constexpr int kMmaWarp = kSoftmaxWarps + 2;        // Q K^T issuer, TMEM owner
constexpr int kPvWarp = kSoftmaxWarps + 3;         // P V issuer
constexpr int kThreads = 32 * (kSoftmaxWarps + 4);
constexpr int kWGThreads = 128;
constexpr uint32_t kQBytes = 64 * 128 * 2;          // one query block
constexpr uint32_t kKVBytes = 128 * 128 * 2;        // a pair of key blocks
constexpr uint32_t kPBytes = 128 * 64 * 2;          // P^T tile
constexpr int KS = 2;                               // K ring: pairs of key blocks ([chunk][block][row])
constexpr int VB = 7;                               // V ring: single key blocks (16 KB, [chunk][row])
constexpr uint32_t kVBlockBytes = 64 * 128 * 2;
constexpr uint32_t kSmemQ = 0;
constexpr uint32_t kSmemK = kSmemQ + kQBytes;
constexpr uint32_t kSmemV = kSmemK + KS * kKVBytes;
constexpr uint32_t kSmemP = kSmemV + VB * kVBlockBytes;
constexpr uint32_t kSmemTiles = kSmemP + 2 * kPBytes;   // 224 KB, 1024-aligned pieces
constexpr uint32_t kTmemCols = 256;                 // S^T x2 (64 cols each), O^T x2
constexpr float kRescaleThreshold = 8.0f;           // log2 units

enum Bar { Q_FULL = 0, Q_EMPTY = 1, K_FULL = 2, K_EMPTY = K_FULL + KS, V_FULL = K_EMPTY + KS,
           V_EMPTY = V_FULL + VB, S_FULL = V_EMPTY + VB, S_EMPTY = S_FULL + 2, P_FULL = S_EMPTY + 2,
           PV_DONE = P_FULL + 2, O_FULL = PV_DONE + 2, O_EMPTY = O_FULL + 2, DRAIN = O_EMPTY + 2, NUM_BARS = DRAIN + 2 };

// Per-CTA control block after the tiles.  The float arrays are read with
// 16-byte vector loads, so they come first and are 16-byte aligned.
struct Smem {
    alignas(16) float m[64];          // minus the running maximum per query (log2 units)
    alignas(16) float alpha[64];      // rescale factors of the current tile
    alignas(16) float delta[64];      // the raise of m_q of the current tile (log2 units)
    alignas(16) float red[kSoftmaxWG][4][kCols];   // cross-warp reduction scratch, per warpgroup
    alignas(16) float inv_l[64];
    uint64_t bar[NUM_BARS];
    uint32_t tmem_base;
    int abort;
};
static_assert(offsetof(Smem, m) % 16 == 0 && offsetof(Smem, alpha) % 16 == 0 && offsetof(Smem, inv_l) % 16 == 0,
              "vector-loaded arrays are 16-byte aligned");
static_assert(kSmemTiles % 1024 == 0, "the control block starts 16-byte aligned");

struct Params {
    Shape s;
    const int32_t* kv_idx;
    __nv_bfloat16* o;
    float* lse;           // nullable: log-sum-exp per query row (natural log)
    DeviceStatus* status;
    int total_items;      // B*H*nB
    int tiles;            // ceil(n_keep / 2)
};

__device__ __forceinline__ void record_timeout(const Params& p, int where)
{
    if (atomicCAS(&p.status->code, 0, (int)ROLA_ERR_TIMEOUT) == 0) p.status->where = where;
}

// Column reduction of v[kCols] over the 128 threads of softmax warpgroup wg;
// result for column c in out[c] (c < kCols).  MAX selects max, else sum.
// A butterfly halves the columns a lane holds at each step; with kCols = 16
// a last exchange leaves column lane / 2 on lanes 2c and 2c + 1.  Uses named
// barrier 1 + wg.
template <bool MAX>
__device__ __forceinline__ void column_reduce(float (&v)[kCols], Smem& sm, int wg, int wtid, float* out)
{
    const int lane = wtid & 31, warp = wtid >> 5;
    constexpr int kSteps = kCols == 32 ? 5 : 4;
#pragma unroll
    for (int step = 0; step < kSteps; ++step) {
        const int off = 16 >> step;
        const int half = (kCols / 2) >> step;     // values kept after this step
        const bool upper = (lane & off) != 0;
#pragma unroll
        for (int i = 0; i < kCols / 2; ++i) {
            if (i < half) {
                float keep = upper ? v[i + half] : v[i];
                float send = upper ? v[i] : v[i + half];
                float recv = __shfl_xor_sync(0xffffffffu, send, off);
                v[i] = MAX ? fmaxf(keep, recv) : keep + recv;
            }
        }
    }
    int col = lane;
    if (kCols == 16) {
        const float recv = __shfl_xor_sync(0xffffffffu, v[0], 1);
        v[0] = MAX ? fmaxf(v[0], recv) : v[0] + recv;
        col = lane >> 1;
    }
    if (kCols == 32 || (lane & 1) == 0) sm.red[wg][warp][col] = v[0];
    bar_sync(1 + wg, kWGThreads);
    if (wtid < kCols) {
        float a = sm.red[wg][0][wtid], b = sm.red[wg][1][wtid], c = sm.red[wg][2][wtid], d = sm.red[wg][3][wtid];
        out[wtid] = MAX ? fmaxf(fmaxf(a, b), fmaxf(c, d)) : (a + b) + (c + d);
    }
    bar_sync(1 + wg, kWGThreads);
}

// Two neighbouring query columns in one packed f32x2 instruction (each element
// an IEEE fma / add, so the results are those of the scalar forms):
// (a, b) = (a * m0 + c0, b * m1 + c1) and (a, b) += (p, q)
__device__ __forceinline__ void ffma2(float& a, float& b, float m0, float m1, float c0, float c1)
{
    asm("{\n.reg .b64 ra, rm, rc;\nmov.b64 ra, {%0, %1};\nmov.b64 rm, {%2, %3};\nmov.b64 rc, {%4, %5};\n"
        "fma.rn.f32x2 ra, ra, rm, rc;\nmov.b64 {%0, %1}, ra;\n}\n"
        : "+f"(a), "+f"(b) : "f"(m0), "f"(m1), "f"(c0), "f"(c1));
}
__device__ __forceinline__ void fadd2(float& a, float& b, float p, float q)
{
    asm("{\n.reg .b64 ra, rp;\nmov.b64 ra, {%0, %1};\nmov.b64 rp, {%2, %3};\n"
        "add.rn.f32x2 ra, ra, rp;\nmov.b64 {%0, %1}, ra;\n}\n"
        : "+f"(a), "+f"(b) : "f"(p), "f"(q));
}

template <int NC>
__device__ __forceinline__ void tmem_ld_cols(uint32_t taddr, float (&v)[NC])
{
    static_assert(NC % 16 == 0, "loads of 16 columns");
#pragma unroll
    for (int c = 0; c < NC / 16; ++c) tmem_ld16(taddr + c * 16, *reinterpret_cast<float(*)[16]>(&v[c * 16]));
    tmem_ld_wait(*reinterpret_cast<float(*)[16]>(&v[0]));
#pragma unroll
    for (int c = 1; c < NC / 16; ++c) reg_fence(*reinterpret_cast<float(*)[16]>(&v[c * 16]));
}

// kCube: blocks are 4x4x4 cubes.  q^r, k^r, v are then read in block order
// (the maps span the padded Np rows), a key is valid when its cube slot lies
// inside the grid, and each O^s row goes to the token of its slot.
template <bool kCube>
__global__ void __launch_bounds__(kThreads, 1) sparse_attn_tc_kernel(const __grid_constant__ CUtensorMap map_q,
                                                                     const __grid_constant__ CUtensorMap map_k,
                                                                     const __grid_constant__ CUtensorMap map_v,
                                                                     const Params p)
{
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    // the 128-byte-swizzle atoms need a 1024-byte aligned base; the kernel has
    // no static shared memory, so the dynamic block starts on the window base
    if (smem_u32(smem_raw) & 1023u) {
        if (threadIdx.x == 0) atomicCAS(&p.status->code, 0, (int)ROLA_ERR_UNSUPPORTED);
        return;
    }
    uint8_t* tiles = smem_raw;
    Smem& sm = *reinterpret_cast<Smem*>(tiles + kSmemTiles);
    const uint32_t sbase = smem_u32(tiles);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    auto bar = [&](int i) { return smem_u32(&sm.bar[i]); };

    const Shape& s = p.s;
    const int T = p.tiles;
    const int nB = s.nB;

    if (tid == 0) {
        sm.abort = 0;
        mbar_init(bar(Q_FULL), 1);
        mbar_init(bar(Q_EMPTY), 1);
        for (int i = 0; i < KS; ++i) {
            mbar_init(bar(K_FULL + i), 1);
            mbar_init(bar(K_EMPTY + i), 1);
        }
        for (int i = 0; i < VB; ++i) {
            mbar_init(bar(V_FULL + i), 1);
            mbar_init(bar(V_EMPTY + i), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar(S_FULL + i), 1);
            mbar_init(bar(S_EMPTY + i), kSoftmaxWarps);
            mbar_init(bar(P_FULL + i), kSoftmaxWarps);
            mbar_init(bar(PV_DONE + i), 1);
            mbar_init(bar(O_FULL + i), 1);
            mbar_init(bar(O_EMPTY + i), kSoftmaxWarps);
        }
        mbar_init(bar(DRAIN), 1);
        mbar_init(bar(DRAIN + 1), 1);
        fence_mbar_init();
    }
    if (warp == kMmaWarp) {
        tmem_alloc(smem_u32(&sm.tmem_base), kTmemCols);
        tmem_relinquish();
    }
    if ((warp == kProducerKWarp || warp == kProducerVWarp) && lane == 0) {
        tma_prefetch_desc(&map_q);
        tma_prefetch_desc(&map_k);
        tma_prefetch_desc(&map_v);
    }
    fence_before_sync();
    __syncthreads();
    fence_after_sync();
    const uint32_t tmem = sm.tmem_base;
    volatile int* abort = &sm.abort;

    if (warp == kProducerKWarp || warp == kProducerVWarp) {
        // ------------------------------------------------------------ TMA producers
        // The loads of a tile are issued from several lanes: the K warp's lanes
        // 2h + c load d-chunk c of block h of the K pair (8 KB boxes; K keeps
        // the [chunk][block][row] layout its M = 128 operand needs); the V
        // warp's lane h loads block h (one 16 KB box, [chunk][row], into a ring
        // of single-block slots so that V needs no pair alignment).  The K warp
        // also loads Q (16 KB).
        const bool is_v = warp == kProducerVWarp;
        const int h = is_v ? lane : (lane >> 1);        // block of the pair
        const int kc = lane & 1;                        // K d-chunk (K warp)
        int k = 0, issued_q = 0, issued_k = 0, issued_vb = 0;
        bool ok = true;
        for (int item = blockIdx.x; item < p.total_items && ok; item += gridDim.x, ++k) {
            const int bh = item / nB, qb = item - bh * nB;
            const int32_t* kept = p.kv_idx + ((size_t)bh * s.nQ + (qb >> s.qb2)) * s.n_keep;
            if (warp == kProducerKWarp) {
                if (k >= 1) ok = mbar_wait(bar(Q_EMPTY), (k - 1) & 1, abort, s.wait_limit_ns);
                ok = __shfl_sync(0xffffffffu, ok, 0);
                if (!ok) break;
                if (lane == 0) {
                    mbar_expect_tx(bar(Q_FULL), kQBytes);
                    tma_load_4d(sbase + kSmemQ, &map_q, bar(Q_FULL), 0, qb * 64, 0, bh);
                }
                ++issued_q;
            }
            for (int t = 0; t < T; ++t) {
                const int g = k * T + t;
                const int ja = __ldg(kept + 2 * t);
                const int jb = 2 * t + 1 < s.n_keep ? __ldg(kept + 2 * t + 1) : -1;
                const int nblk = jb >= 0 ? 2 : 1;
                if (is_v) {
                    // cumulative block index of block h of this tile; both lanes
                    // wait for their slots, then issue together (or neither does)
                    const int c = k * s.n_keep + 2 * t + h;
                    const int slot = c % VB;
                    bool okl = true;
                    if (lane < 2 && h < nblk && c >= VB)
                        okl = mbar_wait(bar(V_EMPTY + slot), ((c / VB) - 1) & 1, abort, s.wait_limit_ns);
                    ok = __shfl_sync(0xffffffffu, okl, 0) && __shfl_sync(0xffffffffu, okl, 1);
                    if (!ok) break;
                    if (lane < 2 && h < nblk) {
                        mbar_expect_tx(bar(V_FULL + slot), kVBlockBytes);
                        tma_load_4d(sbase + kSmemV + slot * kVBlockBytes, &map_v, bar(V_FULL + slot), 0,
                                    (h ? jb : ja) * 64, 0, bh);
                    }
                    issued_vb += nblk;
                } else {
                    const int st = g % KS;
                    if (g >= KS) ok = mbar_wait(bar(K_EMPTY + st), ((g / KS) - 1) & 1, abort, s.wait_limit_ns);
                    ok = __shfl_sync(0xffffffffu, ok, 0);
                    if (!ok) break;
                    // test hook: the first K copy of the CTA is never issued, so the waits on it run out
                    const bool skip = (s.debug_flags & ROLA_DEBUG_SKIP_FIRST_K_COPY) && g == 0;
                    if (lane == 0 && !skip) mbar_expect_tx(bar(K_FULL + st), nblk * 16384u);
                    __syncwarp();
                    if (lane < 4 && h < nblk && !skip)
                        tma_load_3d(sbase + kSmemK + st * kKVBytes + kc * 16384 + h * 8192, &map_k, bar(K_FULL + st),
                                    kc * 64, (h ? jb : ja) * 64, bh);
                    ++issued_k;
                }
            }
        }
        if (!ok && lane == 0) record_timeout(p, is_v ? 4 : 1);
        // every copy this warp issued must land before the CTA exits: wait for
        // the latest issued phase of each buffer, bounded by time only
        if (lane == 0) {
            int never = 0;
            if (issued_q > 0) mbar_wait(bar(Q_FULL), (issued_q - 1) & 1, &never, s.wait_limit_ns);
            const int NS = is_v ? VB : KS, issued = is_v ? issued_vb : issued_k;
            const int full0 = is_v ? V_FULL : K_FULL;
            // the last NS uses (tiles of K, blocks of V), one per slot
            for (int u = issued > NS ? issued - NS : 0; u < issued; ++u)
                mbar_wait(bar(full0 + u % NS), (u / NS) & 1, &never, s.wait_limit_ns);
        }
    } else if (warp == kMmaWarp || warp == kPvWarp) {
        // ------------------------------------------------------------ MMA issuers
        // Two issuing warps, so that a P V waiting for the softmax never holds
        // back the next Q K^T (and vice versa); each commits only its own MMAs.
        // Descriptors are built once; a K step adds its offset (in 16-byte
        // units) to the low word.
        if (lane == 0) {
            const bool pv = warp == kPvWarp;
            const uint32_t id_qk = idesc_bf16(128, 64, false, false);
            const uint32_t id_pv = idesc_bf16(128, 64, true, true);
            const uint64_t dq = smem_desc(sbase + kSmemQ, 16, 1024);            // Q: B of Q K^T (K-major)
            const uint64_t dk = smem_desc(sbase + kSmemK, 16, 1024);            // K pair ring: A of Q K^T
            const uint64_t dv = smem_desc(sbase + kSmemV, 8192, 1024);          // V block ring: A of P V (MN-major)
            const uint64_t dp = smem_desc(sbase + kSmemP, 8192, 1024);          // P^T: B of P V (MN-major)
            const uint32_t q_lo = (uint32_t)dq, q_hi = (uint32_t)(dq >> 32);
            const uint32_t k_lo = (uint32_t)dk, k_hi = (uint32_t)(dk >> 32);
            const uint32_t v_lo = (uint32_t)dv, v_hi = (uint32_t)(dv >> 32);
            const uint32_t p_lo = (uint32_t)dp, p_hi = (uint32_t)(dp >> 32);
            bool ok = true;
            int k = 0;
            for (int item = blockIdx.x; item < p.total_items && ok; item += gridDim.x, ++k) {
                const int ob = k & 1;
                if (!pv) {
                    if (!(ok = mbar_wait(bar(Q_FULL), k & 1, abort, s.wait_limit_ns))) break;
                    for (int t = 0; t < T; ++t) {
                        const int g = k * T + t, sb = g & 1, ks = g % KS;
                        if (!(ok = mbar_wait(bar(K_FULL + ks), (g / KS) & 1, abort, s.wait_limit_ns))) break;
                        if (g >= 2 && !(ok = mbar_wait(bar(S_EMPTY + sb), ((g >> 1) - 1) & 1, abort, s.wait_limit_ns)))
                            break;
                        fence_after_sync();
                        const uint32_t a = k_lo + ks * (kKVBytes >> 4);
                        const uint32_t d = tmem + sb * 64;
#pragma unroll
                        for (int kk = 0; kk < 8; ++kk)
                            mma_ss_split(d, a + (kk >> 2) * 1024 + (kk & 3) * 2, k_hi,
                                         q_lo + (kk >> 2) * 512 + (kk & 3) * 2, q_hi, id_qk, kk > 0 ? 1u : 0u);
                        mma_commit(bar(S_FULL + sb));
                        mma_commit(bar(K_EMPTY + ks));
                        if (t == T - 1) mma_commit(bar(Q_EMPTY));
                    }
                } else {
                    for (int t = 0; t < T; ++t) {
                        const int g = k * T + t, pb = g & 1;
                        const bool half = 2 * t + 1 >= s.n_keep;
                        const int c0 = k * s.n_keep + 2 * t;             // cumulative index of block a
                        const int va = c0 % VB, vb = (c0 + 1) % VB;
                        if (!(ok = mbar_wait(bar(P_FULL + pb), (g >> 1) & 1, abort, s.wait_limit_ns))) break;
                        if (!(ok = mbar_wait(bar(V_FULL + va), (c0 / VB) & 1, abort, s.wait_limit_ns))) break;
                        if (!half && !(ok = mbar_wait(bar(V_FULL + vb), ((c0 + 1) / VB) & 1, abort, s.wait_limit_ns)))
                            break;
                        if (t == 0 && k >= 2 &&
                            !(ok = mbar_wait(bar(O_EMPTY + ob), ((k >> 1) - 1) & 1, abort, s.wait_limit_ns)))
                            break;
                        fence_after_sync();
                        const uint32_t a0 = v_lo + va * (kVBlockBytes >> 4), a1 = v_lo + vb * (kVBlockBytes >> 4);
                        const uint32_t b0 = p_lo + pb * (kPBytes >> 4);
                        const uint32_t d = tmem + 128 + ob * 64;
                        mma_ss_split(d, a0, v_hi, b0, p_hi, id_pv, t > 0 ? 1u : 0u);
#pragma unroll
                        for (int kk = 1; kk < 4; ++kk)
                            mma_ss_split(d, a0 + kk * 128, v_hi, b0 + kk * 128, p_hi, id_pv, 1u);
                        if (!half) {
#pragma unroll
                            for (int kk = 0; kk < 4; ++kk)
                                mma_ss_split(d, a1 + kk * 128, v_hi, b0 + (4 + kk) * 128, p_hi, id_pv, 1u);
                        }
                        mma_commit(bar(PV_DONE + pb));
                        mma_commit(bar(V_EMPTY + va));
                        if (!half) mma_commit(bar(V_EMPTY + vb));
                    }
                    if (!ok) break;
                    mma_commit(bar(O_FULL + ob));
                }
            }
            if (!ok) record_timeout(p, pv ? 5 : 2);
            // drain: every MMA this thread issued completes before TMEM is released
            int never = 0;
            const uint32_t drain = bar(pv ? DRAIN + 1 : DRAIN);
            mma_commit(drain);
            mbar_wait(drain, 0, &never, s.wait_limit_ns);
        }
    } else {
        // ------------------------------------------------------------ softmax + epilogue
        // Softmax warpgroup wg owns query columns [32 wg, 32 wg + 32) of every
        // tile; thread wtid owns key wtid of the tile (TMEM lane wtid).  Per key
        // and query: t = s * log2(e)/sqrt(d) - m_q (one FFMA against the stored
        // -m_q), p = 2^t.  A tile whose t exceeds the threshold anywhere in the
        // warpgroup's columns takes the rescale path: exact column maxima of t,
        // m_q += max(tmax_q, 0), O^T columns and row sums scaled by 2^-delta.
        // The first tile of a query block starts from m_q = 0 and always takes
        // that path with delta = tmax (m_q becomes the tile's exact maximum).
        const int wg = warp >> 2, wtid = tid & 127;
        const int col0 = wg * kCols;
        const float c_log2 = s.sm_scale_log2;
        const uint32_t lane_off = (uint32_t)((warp & 3) * 32) << 16;
        bool ok = true;
        int k = 0;
        for (int item = blockIdx.x; item < p.total_items && ok; item += gridDim.x, ++k) {
            const int bh = item / nB, qb = item - bh * nB;
            const int32_t* kept = p.kv_idx + ((size_t)bh * s.nQ + (qb >> s.qb2)) * s.n_keep;
            const int ob = k & 1;
            if (wtid < kCols) sm.m[col0 + wtid] = 0.0f;       // holds -m_q
            float l[kCols];
#pragma unroll
            for (int q = 0; q < kCols; ++q) l[q] = 0.0f;
            int ja_n = __ldg(kept);
            int jb_n = s.n_keep > 1 ? __ldg(kept + 1) : -1;
            bar_sync(1 + wg, kWGThreads);
            for (int t = 0; t < T; ++t) {
                const int g = k * T + t, sb = g & 1;
                const int ja = ja_n, jb = jb_n;
                if (t + 1 < T) {                               // kept ids of the next tile, one tile ahead
                    ja_n = __ldg(kept + 2 * t + 2);
                    jb_n = 2 * t + 3 < s.n_keep ? __ldg(kept + 2 * t + 3) : -1;
                }
                const int blk = wtid < 64 ? ja : jb;
                bool valid;
                if constexpr (kCube) {
                    valid = blk >= 0 && cube_token(s, cube_origin_rcp(s, blk), wtid & 63) >= 0;
                } else {
                    const int key = blk * 64 + (wtid & 63);
                    valid = blk >= 0 && key < s.N;
                }
                if (!(ok = mbar_wait(bar(S_FULL + sb), (g >> 1) & 1, abort, s.wait_limit_ns))) break;
                fence_after_sync();
                const uint32_t saddr = tmem + lane_off + sb * 64 + col0;
                float x[kCols];
                tmem_ld_cols<kCols>(saddr, x);
                fence_before_sync();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(S_EMPTY + sb));  // S^T buffer free for Q K^T(g + 2)
                bool need = t == 0;
                if (valid) {
#pragma unroll
                    for (int q = 0; q < kCols; q += 4) {
                        const float4 nm = *reinterpret_cast<const float4*>(&sm.m[col0 + q]);
                        ffma2(x[q], x[q + 1], c_log2, c_log2, nm.x, nm.y);
                        ffma2(x[q + 2], x[q + 3], c_log2, c_log2, nm.z, nm.w);
                        need |= (x[q] > kRescaleThreshold) | (x[q + 1] > kRescaleThreshold) |
                                (x[q + 2] > kRescaleThreshold) | (x[q + 3] > kRescaleThreshold);
                    }
                } else {
#pragma unroll
                    for (int q = 0; q < kCols; ++q) x[q] = -INFINITY;
                }
                if (bar_red_or(1 + wg, kWGThreads, need)) {
                    float xr[kCols];                                                // the reduction consumes its input
#pragma unroll
                    for (int q = 0; q < kCols; ++q) xr[q] = x[q];
                    column_reduce<true>(xr, sm, wg, wtid, sm.alpha + col0);   // alpha <- column maxima of t
                    if (wtid < kCols) {
                        const float tmax = sm.alpha[col0 + wtid];
                        const float delta = t == 0 ? tmax : fmaxf(tmax, 0.0f);
                        sm.m[col0 + wtid] -= delta;
                        sm.alpha[col0 + wtid] = fast_exp2(-delta);
                        sm.delta[col0 + wtid] = delta;
                    }
                    bar_sync(1 + wg, kWGThreads);
                    if (valid) {                                   // t against the new m: t - (m_new - m_old)
#pragma unroll
                        for (int q = 0; q < kCols; ++q) x[q] -= sm.delta[col0 + q];
                    } else {
#pragma unroll
                        for (int q = 0; q < kCols; ++q) x[q] = -INFINITY;
                    }
                    if (t > 0) {
                        // O^T must hold PV(t-1) before it is rescaled
                        if (!(ok = mbar_wait(bar(PV_DONE + ((g - 1) & 1)), ((g - 1) >> 1) & 1, abort, s.wait_limit_ns)))
                            break;
                        fence_after_sync();
                        const uint32_t oaddr = tmem + lane_off + 128 + ob * 64 + col0;
#pragma unroll
                        for (int c = 0; c < kCols / 16; ++c) {
                            float ov[16];
                            tmem_ld16(oaddr + c * 16, ov);
                            tmem_ld_wait(ov);
#pragma unroll
                            for (int e = 0; e < 16; ++e) ov[e] *= sm.alpha[col0 + c * 16 + e];
                            tmem_st16(oaddr + c * 16, ov);
                        }
                        tmem_st_wait();
#pragma unroll
                        for (int q = 0; q < kCols; ++q) l[q] *= sm.alpha[col0 + q];
                    }
                }
                // p = 2^t; this warpgroup's columns of the key's P^T row, bf16, 128-byte-swizzled
                uint32_t pk[kCols / 2];
#pragma unroll
                for (int q = 0; q < kCols; q += 2) {
                    const float p0 = fast_exp2(x[q]);
                    const float p1 = fast_exp2(x[q + 1]);
                    fadd2(l[q], l[q + 1], p0, p1);
                    pk[q >> 1] = pack_bf16(p0, p1);
                }
                if (g >= 2 && !(ok = mbar_wait(bar(PV_DONE + sb), ((g >> 1) - 1) & 1, abort, s.wait_limit_ns))) break;
                const uint32_t prow = sbase + kSmemP + sb * kPBytes + (wtid >> 3) * 1024 + (wtid & 7) * 128;
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
                if (lane == 0) mbar_arrive(bar(P_FULL + sb));
            }
            if (!ok) break;
            // ---- epilogue: O^s = O^T / l.  l is final after the last tile, so its
            // reduction overlaps the last P V; then thread wtid writes d = wtid of
            // this warpgroup's 32 query rows, so each warp store is one 64-byte segment
            column_reduce<false>(l, sm, wg, wtid, sm.inv_l + col0);
            if (wtid < kCols) {
                const float lsum = sm.inv_l[col0 + wtid];
                if (p.lse) {
                    // sum_j exp(s_j / sqrt d) = 2^(m_q) l_q, with -m_q stored in sm.m (log2 units)
                    int n;
                    if constexpr (kCube) n = cube_token(s, cube_origin_rcp(s, qb), col0 + wtid);
                    else n = qb * 64 + col0 + wtid < s.N ? qb * 64 + col0 + wtid : -1;
                    if (n >= 0) p.lse[(size_t)bh * s.N + n] = (log2f(lsum) - sm.m[col0 + wtid]) * 0.6931471805599453f;
                }
                sm.inv_l[col0 + wtid] = 1.0f / lsum;
            }
            bar_sync(1 + wg, kWGThreads);
            if (!(ok = mbar_wait(bar(O_FULL + ob), (k >> 1) & 1, abort, s.wait_limit_ns))) break;
            fence_after_sync();
            {
                float ov[kCols];
                tmem_ld_cols<kCols>(tmem + lane_off + 128 + ob * 64 + col0, ov);
                fence_before_sync();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(O_EMPTY + ob));
                if constexpr (kCube) {
                    // this warpgroup's 32 slots are (dt, dx, dy) = (2 wg + q / 16, q / 4 % 4, q % 4):
                    // offsets and bounds per row are compile-time against three runtime limits
                    static_assert(kCols == 32, "a warpgroup owns two 16-slot layers of the cube");
                    const CubeOrigin co = cube_origin_rcp(s, qb);
                    const int t0 = co.t + 2 * wg;
                    const int lt = s.T - t0, lx = s.Hh - co.x, ly = s.Ww - co.y;
                    const size_t plane = (size_t)s.Hh * s.Ww * kDh, line = (size_t)s.Ww * kDh;
                    const size_t row0 = ((size_t)bh * s.N + ((size_t)t0 * s.Hh + co.x) * s.Ww + co.y) * kDh + wtid;
#pragma unroll
                    for (int q = 0; q < kCols; ++q) {
                        const int dt = q >> 4, dx = (q >> 2) & 3, dy = q & 3;
                        if (dt < lt && dx < lx && dy < ly)
                            p.o[row0 + dt * plane + dx * line + dy * kDh] =
                                __float2bfloat16_rn(ov[q] * sm.inv_l[col0 + q]);
                    }
                } else {
                    __nv_bfloat16* dst = p.o + ((size_t)bh * s.N + (size_t)qb * 64 + col0) * kDh + wtid;
                    const int rows = min(64, s.N - qb * 64) - col0;     // rows of this warpgroup inside the sequence
#pragma unroll
                    for (int q = 0; q < kCols; ++q)
                        if (q < rows) dst[(size_t)q * kDh] = __float2bfloat16_rn(ov[q] * sm.inv_l[col0 + q]);
                }
            }
        }
        if (!ok) record_timeout(p, 3);
    }
    fence_before_sync();
    __syncthreads();
    fence_after_sync();
    if (warp == kMmaWarp) tmem_dealloc(tmem, kTmemCols);
}

}  // namespace

// The driver's cuTensorMapEncodeTiled, looked up once (thread-safe static initialisation).
static PFN_cuTensorMapEncodeTiled_v12000 encode_fn()
{
    static const PFN_cuTensorMapEncodeTiled_v12000 fn = []() -> PFN_cuTensorMapEncodeTiled_v12000 {
        void* f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
        return nullptr;
    }();
    return fn;
}

// [BH][N][128] bf16 viewed as a 3-D tensor (d, token, head); 64 x 64 boxes
// (one d-chunk of a key block), 128-byte swizzle; rows past N read as zero.
bool make_chunk_map(CUtensorMap* m, const void* ptr, const Shape& s)
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

// The same tensor viewed as 4-D (d within chunk, token, d-chunk, head) so that
// one 64 x 64 x 2 box brings a whole key block in as [chunk][row][64]: 16 KB,
// 128-byte swizzle, rows past N read as zero.
bool make_block_map(CUtensorMap* m, const void* ptr, const Shape& s, int rows)
{
    auto enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[4] = {64, (cuuint64_t)s.N, 2, (cuuint64_t)s.B * s.H};
    cuuint64_t strides[3] = {(cuuint64_t)kDh * 2, 128, (cuuint64_t)s.N * kDh * 2};
    cuuint32_t box[4] = {64, (cuuint32_t)rows, 2, 1};
    cuuint32_t es[4] = {1, 1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(ptr), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

cudaError_t launch_sparse_attn_tc(const Shape& s, const void* qr, const void* kr, const void* v,
                                  const int32_t* kv_idx, void* o_s, float* lse, DeviceStatus* status,
                                  cudaStream_t st)
{
    // the maps span the block-ordered rows (the token order itself for contiguous chunks)
    Shape rows = s;
    rows.N = s.Np;
    CUtensorMap mq, mk, mv;
    if (!make_block_map(&mq, qr, rows) || !make_chunk_map(&mk, kr, rows) || !make_block_map(&mv, v, rows))
        return cudaErrorInvalidValue;
    int dev = 0, nsm = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    Params p;
    p.s = s;
    p.kv_idx = kv_idx;
    p.o = static_cast<__nv_bfloat16*>(o_s);
    p.lse = lse;
    p.status = status;
    p.total_items = s.B * s.H * s.nB;
    p.tiles = (s.n_keep + 1) / 2;
    const size_t smem = kSmemTiles + sizeof(Smem);
    const int grid = p.total_items < nsm ? p.total_items : nsm;
    // contiguous key blocks run the row-wise kernel (sparse_attn_rows.cu); this one serves cubes
    if (!s.cube) return cudaErrorInvalidValue;
    auto kernel = sparse_attn_tc_kernel<true>;
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    kernel<<<grid, kThreads, smem, st>>>(mq, mk, mv, p);
    return cudaGetLastError();
}

}  // namespace rola
