// Block-sparse softmax attention, one softmax thread (pair) per query row
// (kernel 2, bf16).
//
//   O^s_p = sum_{q in kept(i)} softmax_q(q^r_p . k^r_q / sqrt(d_h)) v_q,   p in query block i
//
// (Sec. 3 softmax form restricted to the kept key blocks, Alg. 1 sparse
// branch.)  Query blocks of QN = 64 tokens (the mask of Alg. 1) or QN = 128
// tokens (a mask chosen per 128-token chunk); key blocks are 64 tokens.
//
// An item (one query block of one head) is the M = QN rows of tcgen05 MMAs:
//   S    = Q (QN q x 128 d, smem, K-major)  x  K_pair^T (N = 128 keys, smem, K-major)
//   O   += P (QN q x 128 keys, TMEM, bf16)  x  V_pair (N = 128 d, smem, MN-major)
// S, P and O live in TMEM with one query row per TMEM lane (M = 128: lanes
// 0-127; M = 64: lanes 0-15 of each 32-lane quarter, row r at lane
// 32 (r / 16) + r mod 16).  The softmax reads its row of S, keeps the row
// maximum and the row sum in registers and writes P back to TMEM as packed
// bf16 (the lower key in the low half), the A operand of the P V product, so
// no P tile passes through shared memory.  For QN = 128 a thread owns a row
// (128 keys); for QN = 64 the two half-warps share the 16 rows of their
// quarter, threads 0-15 taking keys 0-63 and threads 16-31 keys 64-127 of
// the same rows (the 16x32bx2 TMEM access shape), and combine the row maximum
// and the row sum with one shuffle.
//
// Softmax (lazy rescaling, base 2): each row keeps -m and its row sum l.  A
// tile's scores are t = s log2(e)/sqrt(d) - m; when the row's largest t of
// the tile exceeds 2^3 (or on the first tile of the item) m is raised to the
// tile maximum and the O row and l are scaled by 2^(m_old - m_new) (a warp
// takes that path when any of its rows needs it; the O row is rescaled after
// the previous P V has finished and before this tile's P is handed over).
// p = 2^t enters the row sum in fp32 and the product rounded to bf16.
//
// Warp roles (256 threads, one persistent CTA per SM):
//   warps 0-3  softmax + epilogue: warp w owns TMEM lane quarter w
//   warp  4    TMA producer: Q (per item) and the K pairs
//   warp  5    TMA producer: the V blocks
//   warp  6    S = Q K^T issuer and TMEM owner
//   warp  7    O += P V issuer
// Buffers (shared memory): Q (QN = 64: two 16 KB buffers, so the next item's
// Q arrives during this one; QN = 128: one of 32 KB), K pairs in a 3-deep
// ring (32 KB each), V blocks in a ring of single 16 KB blocks (6 for QN = 64,
// 5 for 128): 224 / 208 KB.  TMEM (512 columns): S double-buffered (2 x 128),
// O (128), P double-buffered (2 x 64 columns of bf16 pairs), so Q K^T of the
// next tile runs while the softmax of this one does.  Every mbarrier wait is
// bounded; a wait that gives up records ROLA_ERR_TIMEOUT in the status word
// and the CTA stops issuing, drains what it issued and releases its TMEM.
//
// Per 64-query block and 128-key tile the shared memory sees 64 KB of TMA
// writes (K, V) and 80 KB of operand reads (Q 16, K 32, V 32) for 4.2 MFLOP,
// against 176 KB in the transposed form of sparse_attn_tc.cu (which is kept
// for the cube geometry); an M = 64 MMA runs at half the M = 128 rate.
#include <cudaTypedefs.h>
#include <stddef.h>

#include "common.cuh"
#include "tcgen05.cuh"
#include "tensor_map.cuh"

namespace rola {
namespace {

using namespace tc;

constexpr int kSoftmaxWarps = 4;
constexpr int kProducerKWarp = 4, kProducerVWarp = 5, kMmaWarp = 6, kPvWarp = 7;
constexpr int kThreads = 256;
constexpr uint32_t kKPairBytes = 128 * 128 * 2;      // a pair of key blocks [d-chunk][block][64 rows][64]
constexpr uint32_t kVBlockBytes = 64 * 128 * 2;      // one key block of v [d-chunk][64 rows][64]
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kTmemS = 0;                       // S buffers at 0, 128
constexpr uint32_t kTmemO = 256;
constexpr uint32_t kTmemP = 384;                     // P buffers at 384, 448 (64 columns: 128 bf16 keys)
constexpr float kRescaleThreshold = 8.0f;            // log2 units

template <int QN>
struct Cfg {
    static_assert(QN == 64 || QN == 128, "query blocks of 64 or 128 rows");
    static constexpr int QB = QN == 64 ? 2 : 1;                  // Q buffers
    static constexpr int KS = 3;                                 // K ring (pairs)
    static constexpr int VB = QN == 64 ? 6 : 5;                  // V ring (single blocks)
    static constexpr int kCols = QN == 64 ? 64 : 128;            // keys of a tile per softmax thread
    static constexpr uint32_t kQBytes = QN * 128 * 2;            // [d-chunk][QN rows][64]
    static constexpr uint32_t kSmemQ = 0;
    static constexpr uint32_t kSmemK = kSmemQ + QB * kQBytes;
    static constexpr uint32_t kSmemV = kSmemK + KS * kKPairBytes;
    static constexpr uint32_t kSmemTiles = kSmemV + VB * kVBlockBytes;
    static constexpr int Q_FULL = 0, Q_EMPTY = Q_FULL + QB, K_FULL = Q_EMPTY + QB, K_EMPTY = K_FULL + KS,
                         V_FULL = K_EMPTY + KS, V_EMPTY = V_FULL + VB, S_FULL = V_EMPTY + VB, S_EMPTY = S_FULL + 2,
                         P_FULL = S_EMPTY + 2, PV_DONE = P_FULL + 2, O_FULL = PV_DONE + 2, O_EMPTY = O_FULL + 1,
                         DRAIN = O_EMPTY + 1, NUM_BARS = DRAIN + 2;
    static_assert(kSmemTiles % 1024 == 0, "the control block follows the 1024-aligned tiles");
};

template <int QN>
struct Ctrl {
    uint64_t bar[Cfg<QN>::NUM_BARS];
    uint32_t tmem_base;
    int abort;
};
static_assert(Cfg<64>::kSmemTiles + sizeof(Ctrl<64>) <= 232448 && Cfg<128>::kSmemTiles + sizeof(Ctrl<128>) <= 232448,
              "tiles and control block fit the 227 KB a CTA may have");

struct Params {
    Shape s;
    const int32_t* kv_idx;   // [B*H][nQ][n_keep]
    __nv_bfloat16* o;        // O^s [B*H][N][128]
    float* lse;              // nullable: log-sum-exp per query row (natural log)
    DeviceStatus* status;
    int items_per_head;      // query blocks per (batch, head) = rows of the mask
    int total_items;         // B*H*items_per_head
    int tiles;               // ceil(n_keep / 2)
};

__device__ __forceinline__ void record_timeout(const Params& p, int where)
{
    if (atomicCAS(&p.status->code, 0, (int)ROLA_ERR_TIMEOUT) == 0) p.status->where = where;
}

// D[tmem] (+)= A[tmem] * B[smem]: A is M rows of K 16-bit values in TMEM,
// two per 32-bit column (the lower K index in the low half).
__device__ __forceinline__ void mma_ts_split(uint32_t d_tmem, uint32_t a_tmem, uint32_t b_lo, uint32_t b_hi,
                                             uint32_t idesc, uint32_t accum)
{
    asm volatile(
        "{\n.reg .pred p;\n.reg .b64 db;\n"
        "setp.ne.b32 p, %5, 0;\n"
        "mov.b64 db, {%2, %3};\n"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], db, %4, p;\n}\n" ::"r"(d_tmem),
        "r"(a_tmem), "r"(b_lo), "r"(b_hi), "r"(idesc), "r"(accum)
        : "memory");
}

// 16x32bx2 accesses: over the 16 lanes from taddr's lane, threads 0-15 take
// lane `lane` at columns [c, c + 16), threads 16-31 lane `lane - 16` at
// columns [c + OFF, c + OFF + 16).
template <int OFF>
__device__ __forceinline__ void tmem_ld16_half(uint32_t taddr, float (&v)[16])
{
    asm volatile(
        "tcgen05.ld.sync.aligned.16x32bx2.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16], %17;\n"
        : "=f"(v[0]), "=f"(v[1]), "=f"(v[2]), "=f"(v[3]), "=f"(v[4]), "=f"(v[5]), "=f"(v[6]), "=f"(v[7]),
          "=f"(v[8]), "=f"(v[9]), "=f"(v[10]), "=f"(v[11]), "=f"(v[12]), "=f"(v[13]), "=f"(v[14]), "=f"(v[15])
        : "r"(taddr), "n"(OFF));
}
template <int OFF>
__device__ __forceinline__ void tmem_st16_half(uint32_t taddr, const float (&v)[16])
{
    asm volatile(
        "tcgen05.st.sync.aligned.16x32bx2.x16.b32 [%0], %17, {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};\n" ::"r"(
            taddr),
        "f"(v[0]), "f"(v[1]), "f"(v[2]), "f"(v[3]), "f"(v[4]), "f"(v[5]), "f"(v[6]), "f"(v[7]), "f"(v[8]), "f"(v[9]),
        "f"(v[10]), "f"(v[11]), "f"(v[12]), "f"(v[13]), "f"(v[14]), "f"(v[15]), "n"(OFF)
        : "memory");
}

// A softmax thread's NC consecutive columns of its row starting at column c0:
// 32x32b for QN = 128 (the thread's own lane), 16x32bx2 with the half-warp
// split at column c0 + NC for QN = 64.
template <int QN, int NC>
__device__ __forceinline__ void row_load(uint32_t taddr, float (&v)[NC])
{
    static_assert(NC % 16 == 0, "loads of 16 columns");
#pragma unroll
    for (int c = 0; c < NC / 16; ++c) {
        float(&part)[16] = *reinterpret_cast<float(*)[16]>(&v[c * 16]);
        if constexpr (QN == 128) tmem_ld16(taddr + c * 16, part);
        else tmem_ld16_half<NC>(taddr + c * 16, part);
    }
    tmem_ld_wait(*reinterpret_cast<float(*)[16]>(&v[0]));
#pragma unroll
    for (int c = 1; c < NC / 16; ++c) reg_fence(*reinterpret_cast<float(*)[16]>(&v[c * 16]));
}
template <int QN, int NC>
__device__ __forceinline__ void row_store(uint32_t taddr, const float (&v)[NC])
{
#pragma unroll
    for (int c = 0; c < NC / 16; ++c) {
        const float(&part)[16] = *reinterpret_cast<const float(*)[16]>(&v[c * 16]);
        if constexpr (QN == 128) tmem_st16(taddr + c * 16, part);
        else tmem_st16_half<NC>(taddr + c * 16, part);
    }
}

// (a, b) = (a * m + c, b * m + c), one packed f32x2 instruction (each element an IEEE fma)
__device__ __forceinline__ void ffma2(float& a, float& b, float m, float c)
{
    asm("{\n.reg .b64 ra, rm, rc;\nmov.b64 ra, {%0, %1};\nmov.b64 rm, {%2, %2};\nmov.b64 rc, {%3, %3};\n"
        "fma.rn.f32x2 ra, ra, rm, rc;\nmov.b64 {%0, %1}, ra;\n}\n"
        : "+f"(a), "+f"(b) : "f"(m), "f"(c));
}
__device__ __forceinline__ void fadd2(float& a, float& b, float p, float q)
{
    asm("{\n.reg .b64 ra, rp;\nmov.b64 ra, {%0, %1};\nmov.b64 rp, {%2, %3};\n"
        "add.rn.f32x2 ra, ra, rp;\nmov.b64 {%0, %1}, ra;\n}\n"
        : "+f"(a), "+f"(b) : "f"(p), "f"(q));
}

template <int QN>
__global__ void __launch_bounds__(kThreads, 1) sparse_attn_rows_kernel(const __grid_constant__ CUtensorMap map_q,
                                                                       const __grid_constant__ CUtensorMap map_k,
                                                                       const __grid_constant__ CUtensorMap map_v,
                                                                       const Params p)
{
    using C = Cfg<QN>;
    constexpr int QB = C::QB, KS = C::KS, VB = C::VB, NC = C::kCols;
    constexpr uint32_t kQBytes = C::kQBytes, kSmemQ = C::kSmemQ, kSmemK = C::kSmemK, kSmemV = C::kSmemV;
    constexpr int Q_FULL = C::Q_FULL, Q_EMPTY = C::Q_EMPTY, K_FULL = C::K_FULL, K_EMPTY = C::K_EMPTY,
                  V_FULL = C::V_FULL, V_EMPTY = C::V_EMPTY, S_FULL = C::S_FULL, S_EMPTY = C::S_EMPTY,
                  P_FULL = C::P_FULL, PV_DONE = C::PV_DONE, O_FULL = C::O_FULL, O_EMPTY = C::O_EMPTY,
                  DRAIN = C::DRAIN;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    // the 128-byte-swizzle atoms need a 1024-byte aligned base; the kernel has
    // no static shared memory, so the dynamic block starts on the window base
    if (smem_u32(smem_raw) & 1023u) {
        if (threadIdx.x == 0) atomicCAS(&p.status->code, 0, (int)ROLA_ERR_UNSUPPORTED);
        return;
    }
    Ctrl<QN>& sm = *reinterpret_cast<Ctrl<QN>*>(smem_raw + C::kSmemTiles);
    const uint32_t sbase = smem_u32(smem_raw);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    auto bar = [&](int i) { return smem_u32(&sm.bar[i]); };

    const Shape& s = p.s;
    const int T = p.tiles;
    const int nI = p.items_per_head;

    if (tid == 0) {
        sm.abort = 0;
        for (int i = 0; i < QB; ++i) {
            mbar_init(bar(Q_FULL + i), 1);
            mbar_init(bar(Q_EMPTY + i), 1);
        }
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
            mbar_init(bar(DRAIN + i), 1);
        }
        mbar_init(bar(O_FULL), 1);
        mbar_init(bar(O_EMPTY), kSoftmaxWarps);
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
        // K warp: lane 0 loads Q (one box); lanes 2h + c load d-chunk c of
        // block h of the K pair (8 KB boxes, [chunk][block][row] so that the
        // pair is one N = 128 operand).  V warp: lanes 2h + c load d-chunk c of
        // block h into its slot of the ring of single blocks ([chunk][row]).
        // A lane's copies are processed one after another, so every copy of a
        // tile gets a lane of its own.
        const bool is_v = warp == kProducerVWarp;
        const int h = lane >> 1;                        // block of the pair
        const int kc = lane & 1;                        // d-chunk
        int k = 0, issued_q = 0, issued_k = 0, issued_vb = 0;
        bool ok = true;
        for (int item = blockIdx.x; item < p.total_items && ok; item += gridDim.x, ++k) {
            const int bh = item / nI, qb = item - bh * nI;
            const int32_t* kept = p.kv_idx + (size_t)item * s.n_keep;
            if (!is_v) {
                const int qs = k % QB;
                if (k >= QB) ok = mbar_wait(bar(Q_EMPTY + qs), ((k / QB) - 1) & 1, abort, s.wait_limit_ns);
                ok = __shfl_sync(0xffffffffu, ok, 0);
                if (!ok) break;
                if (lane == 0) {
                    mbar_expect_tx(bar(Q_FULL + qs), kQBytes);
                    tma_load_4d(sbase + kSmemQ + qs * kQBytes, &map_q, bar(Q_FULL + qs), 0, qb * QN, 0, bh);
                }
                ++issued_q;
            }
            for (int t = 0; t < T; ++t) {
                const int g = k * T + t;
                const int ja = __ldg(kept + 2 * t);
                const int jb = 2 * t + 1 < s.n_keep ? __ldg(kept + 2 * t + 1) : -1;
                const int nblk = jb >= 0 ? 2 : 1;
                if (is_v) {
                    const int c = k * s.n_keep + 2 * t + h;       // cumulative block index of block h
                    const int slot = c % VB;
                    bool okl = true;
                    if (lane < 4 && kc == 0 && h < nblk && c >= VB)
                        okl = mbar_wait(bar(V_EMPTY + slot), ((c / VB) - 1) & 1, abort, s.wait_limit_ns);
                    ok = __shfl_sync(0xffffffffu, okl, 0) && __shfl_sync(0xffffffffu, okl, 2);
                    if (!ok) break;
                    if (lane < 4 && kc == 0 && h < nblk) mbar_expect_tx(bar(V_FULL + slot), kVBlockBytes);
                    __syncwarp();
                    if (lane < 4 && h < nblk)
                        tma_load_3d(sbase + kSmemV + slot * kVBlockBytes + kc * 8192, &map_v, bar(V_FULL + slot),
                                    kc * 64, (h ? jb : ja) * 64, bh);
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
                        tma_load_3d(sbase + kSmemK + st * kKPairBytes + kc * 16384 + h * 8192, &map_k,
                                    bar(K_FULL + st), kc * 64, (h ? jb : ja) * 64, bh);
                    ++issued_k;
                }
            }
        }
        if (!ok && lane == 0) record_timeout(p, is_v ? 4 : 1);
        // every copy this warp issued lands before the CTA exits (bounded by time only)
        if (lane == 0) {
            int never = 0;
            for (int u = issued_q > QB ? issued_q - QB : 0; u < issued_q; ++u)
                mbar_wait(bar(Q_FULL + u % QB), (u / QB) & 1, &never, s.wait_limit_ns);
            const int NS = is_v ? VB : KS, issued = is_v ? issued_vb : issued_k;
            const int full0 = is_v ? V_FULL : K_FULL;
            for (int u = issued > NS ? issued - NS : 0; u < issued; ++u)
                mbar_wait(bar(full0 + u % NS), (u / NS) & 1, &never, s.wait_limit_ns);
        }
    } else if (warp == kMmaWarp || warp == kPvWarp) {
        // ------------------------------------------------------------ MMA issuers
        if (lane == 0) {
            const bool pv = warp == kPvWarp;
            const uint32_t id_qk = idesc_bf16(QN, 128, false, false);
            const uint32_t id_pv = idesc_bf16(QN, 128, false, true);
            const uint64_t dq = smem_desc(sbase + kSmemQ, 16, 1024);     // Q: A of Q K^T (K-major)
            const uint64_t dk = smem_desc(sbase + kSmemK, 16, 1024);     // K pair ring: B of Q K^T (K-major)
            const uint64_t dv = smem_desc(sbase + kSmemV, 8192, 1024);   // V block ring: B of P V (MN-major, d chunks 8 KB apart)
            const uint32_t q_lo = (uint32_t)dq, q_hi = (uint32_t)(dq >> 32);
            const uint32_t k_lo = (uint32_t)dk, k_hi = (uint32_t)(dk >> 32);
            const uint32_t v_lo = (uint32_t)dv, v_hi = (uint32_t)(dv >> 32);
            bool ok = true;
            int k = 0;
            for (int item = blockIdx.x; item < p.total_items && ok; item += gridDim.x, ++k) {
                if (!pv) {
                    const int qs = k % QB;
                    if (!(ok = mbar_wait(bar(Q_FULL + qs), (k / QB) & 1, abort, s.wait_limit_ns))) break;
                    const uint32_t a = q_lo + qs * (kQBytes >> 4);
                    for (int t = 0; t < T; ++t) {
                        const int g = k * T + t, sb = g & 1, ks = g % KS;
                        if (!(ok = mbar_wait(bar(K_FULL + ks), (g / KS) & 1, abort, s.wait_limit_ns))) break;
                        if (g >= 2 && !(ok = mbar_wait(bar(S_EMPTY + sb), ((g >> 1) - 1) & 1, abort, s.wait_limit_ns)))
                            break;
                        fence_after_sync();
                        const uint32_t b = k_lo + ks * (kKPairBytes >> 4);
                        // K step kk: d-chunk kk / 4 (Q: QN rows of 128 B on, K pair: 16 KB on), 32 bytes per 16 d
#pragma unroll
                        for (int kk = 0; kk < 8; ++kk)
                            mma_ss_split(tmem + kTmemS + sb * 128, a + (kk >> 2) * (QN * 8) + (kk & 3) * 2, q_hi,
                                         b + (kk >> 2) * 1024 + (kk & 3) * 2, k_hi, id_qk, kk > 0 ? 1u : 0u);
                        mma_commit(bar(S_FULL + sb));
                        mma_commit(bar(K_EMPTY + ks));
                        if (t == T - 1) mma_commit(bar(Q_EMPTY + qs));
                    }
                } else {
                    for (int t = 0; t < T; ++t) {
                        const int g = k * T + t, pb = g & 1;
                        const bool half = 2 * t + 1 >= s.n_keep;
                        const int c0 = k * s.n_keep + 2 * t;
                        const int va = c0 % VB, vb = (c0 + 1) % VB;
                        if (!(ok = mbar_wait(bar(P_FULL + pb), (g >> 1) & 1, abort, s.wait_limit_ns))) break;
                        if (!(ok = mbar_wait(bar(V_FULL + va), (c0 / VB) & 1, abort, s.wait_limit_ns))) break;
                        if (!half && !(ok = mbar_wait(bar(V_FULL + vb), ((c0 + 1) / VB) & 1, abort, s.wait_limit_ns)))
                            break;
                        if (t == 0 && k >= 1 && !(ok = mbar_wait(bar(O_EMPTY), (k - 1) & 1, abort, s.wait_limit_ns)))
                            break;
                        fence_after_sync();
                        // K step kk (16 keys): 8 TMEM columns of P, 2 KB of the V block
                        const uint32_t a = tmem + kTmemP + pb * 64;
                        const uint32_t b0 = v_lo + va * (kVBlockBytes >> 4), b1 = v_lo + vb * (kVBlockBytes >> 4);
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk)
                            mma_ts_split(tmem + kTmemO, a + kk * 8, b0 + kk * 128, v_hi, id_pv,
                                         (t > 0 || kk > 0) ? 1u : 0u);
                        if (!half) {
#pragma unroll
                            for (int kk = 0; kk < 4; ++kk)
                                mma_ts_split(tmem + kTmemO, a + 32 + kk * 8, b1 + kk * 128, v_hi, id_pv, 1u);
                        }
                        mma_commit(bar(PV_DONE + pb));
                        mma_commit(bar(V_EMPTY + va));
                        if (!half) mma_commit(bar(V_EMPTY + vb));
                    }
                    if (!ok) break;
                    mma_commit(bar(O_FULL));
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
        // QN = 128: thread tid owns row tid, keys 0-127 of a tile, d 0-127 of O.
        // QN = 64: thread (w, lane) owns row 16 w + lane mod 16, keys and d
        // [64 hf, 64 hf + 64) with hf = lane / 16 (its partner is lane ^ 16).
        const int hf = QN == 64 ? lane >> 4 : 0;
        const int row = QN == 64 ? 16 * warp + (lane & 15) : tid;
        const float c_log2 = s.sm_scale_log2;
        const uint32_t lane_off = (uint32_t)(warp * 32) << 16;
        bool ok = true;
        int k = 0;
        for (int item = blockIdx.x; item < p.total_items && ok; item += gridDim.x, ++k) {
            const int bh = item / nI, qb = item - bh * nI;
            const int32_t* kept = p.kv_idx + (size_t)item * s.n_keep;
            float neg_m = 0.0f;                      // -m (log2 units)
            float l0 = 0.0f, l1 = 0.0f, l2 = 0.0f, l3 = 0.0f;
            int ja_n = __ldg(kept);
            int jb_n = s.n_keep > 1 ? __ldg(kept + 1) : -1;
            for (int t = 0; t < T; ++t) {
                const int g = k * T + t, sb = g & 1;
                const int ja = ja_n, jb = jb_n;
                if (t + 1 < T) {                     // kept ids of the next tile, one tile ahead
                    ja_n = __ldg(kept + 2 * t + 2);
                    jb_n = 2 * t + 3 < s.n_keep ? __ldg(kept + 2 * t + 3) : -1;
                }
                // keys of the pair inside the sequence: block a's first na, block b's first nb
                const int na = min(64, s.N - ja * 64);
                const int nb = jb >= 0 ? min(64, s.N - jb * 64) : 0;
                if (!(ok = mbar_wait(bar(S_FULL + sb), (g >> 1) & 1, abort, s.wait_limit_ns))) break;
                fence_after_sync();
                float x[NC];
                row_load<QN, NC>(tmem + lane_off + kTmemS + sb * 128, x);
                fence_before_sync();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(S_EMPTY + sb));    // S buffer free for Q K^T(g + 2)
                if constexpr (QN == 128) {
                    if (na < 64 || nb < 64) {
#pragma unroll
                        for (int j = 0; j < 64; ++j) {
                            if (j >= na) x[j] = -INFINITY;
                            if (j >= nb) x[64 + j] = -INFINITY;
                        }
                    }
                } else {
                    const int nv = hf ? nb : na;
                    if (nv < 64) {
#pragma unroll
                        for (int j = 0; j < 64; ++j)
                            if (j >= nv) x[j] = -INFINITY;
                    }
                }
                // the tile's row maximum (eight independent chains; the two halves of a row meet by shuffle)
                float mx[8];
#pragma unroll
                for (int i = 0; i < 8; ++i) mx[i] = x[i];
#pragma unroll
                for (int j = 8; j < NC; ++j) mx[j & 7] = fmaxf(mx[j & 7], x[j]);
                float tile_max = fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])),
                                       fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7])));
                if constexpr (QN == 64) tile_max = fmaxf(tile_max, __shfl_xor_sync(0xffffffffu, tile_max, 16));
                const bool need = t == 0 || fmaf(tile_max, c_log2, neg_m) > kRescaleThreshold;
                if (__any_sync(0xffffffffu, need)) {
                    const float neg_m_new = need ? -tile_max * c_log2 : neg_m;
                    if (t > 0) {
                        // the O row must hold P V(g - 1) before it is scaled by 2^(m_old - m_new)
                        const float alpha = fast_exp2(neg_m_new - neg_m);
                        if (!(ok = mbar_wait(bar(PV_DONE + ((g - 1) & 1)), ((g - 1) >> 1) & 1, abort,
                                             s.wait_limit_ns)))
                            break;
                        fence_after_sync();
                        const uint32_t oaddr = tmem + lane_off + kTmemO;
                        // a thread holds as many d columns of its O row as it has keys of a tile
#pragma unroll
                        for (int c = 0; c < NC / 16; ++c) {
                            float ov[16];
                            if constexpr (QN == 128) tmem_ld16(oaddr + c * 16, ov);
                            else tmem_ld16_half<64>(oaddr + c * 16, ov);
                            tmem_ld_wait(ov);
#pragma unroll
                            for (int e = 0; e < 16; ++e) ov[e] *= alpha;
                            if constexpr (QN == 128) tmem_st16(oaddr + c * 16, ov);
                            else tmem_st16_half<64>(oaddr + c * 16, ov);
                        }
                        tmem_st_wait();
                        l0 *= alpha;
                        l1 *= alpha;
                        l2 *= alpha;
                        l3 *= alpha;
                    }
                    neg_m = neg_m_new;
                }
                // p = 2^t, row sum in fp32, P packed to bf16 pairs (lower key in the low half)
                uint32_t pk[NC / 2];
#pragma unroll
                for (int j = 0; j < NC; j += 4) {
                    ffma2(x[j], x[j + 1], c_log2, neg_m);
                    ffma2(x[j + 2], x[j + 3], c_log2, neg_m);
                    const float p0 = fast_exp2(x[j]), p1 = fast_exp2(x[j + 1]);
                    const float p2 = fast_exp2(x[j + 2]), p3 = fast_exp2(x[j + 3]);
                    if ((j & 4) == 0) {
                        fadd2(l0, l1, p0, p1);
                        fadd2(l2, l3, p2, p3);
                    } else {
                        fadd2(l2, l3, p0, p1);
                        fadd2(l0, l1, p2, p3);
                    }
                    pk[j >> 1] = pack_bf16(p0, p1);
                    pk[(j >> 1) + 1] = pack_bf16(p2, p3);
                }
                // P buffer g & 1 is free once P V(g - 2) is done
                if (g >= 2 && !(ok = mbar_wait(bar(PV_DONE + sb), ((g >> 1) - 1) & 1, abort, s.wait_limit_ns)))
                    break;
                row_store<QN, NC / 2>(tmem + lane_off + kTmemP + sb * 64, *reinterpret_cast<const float(*)[NC / 2]>(pk));
                tmem_st_wait();
                fence_before_sync();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(P_FULL + sb));
            }
            if (!ok) break;
            // ---- epilogue: O^s row = O / l
            float lsum = (l0 + l1) + (l2 + l3);
            if constexpr (QN == 64) lsum += __shfl_xor_sync(0xffffffffu, lsum, 16);
            const int n = qb * QN + row;
            if (p.lse && hf == 0 && n < s.N) p.lse[(size_t)bh * s.N + n] = (log2f(lsum) - neg_m) * 0.6931471805599453f;
            const float inv_l = 1.0f / lsum;
            if (!(ok = mbar_wait(bar(O_FULL), k & 1, abort, s.wait_limit_ns))) break;
            fence_after_sync();
            float ov[NC];                                     // this thread's d columns of the O row
            row_load<QN, NC>(tmem + lane_off + kTmemO, ov);
            fence_before_sync();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(O_EMPTY));             // O free for the next item's P V
            if (n < s.N) {
                uint4* dst = reinterpret_cast<uint4*>(p.o + ((size_t)bh * s.N + n) * kDh + hf * 64);
#pragma unroll
                for (int c = 0; c < NC / 8; ++c) {
                    uint4 u;
                    u.x = pack_bf16(ov[8 * c] * inv_l, ov[8 * c + 1] * inv_l);
                    u.y = pack_bf16(ov[8 * c + 2] * inv_l, ov[8 * c + 3] * inv_l);
                    u.z = pack_bf16(ov[8 * c + 4] * inv_l, ov[8 * c + 5] * inv_l);
                    u.w = pack_bf16(ov[8 * c + 6] * inv_l, ov[8 * c + 7] * inv_l);
                    dst[c] = u;
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

template <int QN>
cudaError_t launch_rows(const Shape& s, const void* qr, const void* kr, const void* v, const int32_t* kv_idx,
                        void* o_s, float* lse, DeviceStatus* status, cudaStream_t st)
{
    CUtensorMap mq, mk, mv;
    if (!make_block_map(&mq, qr, s, QN) || !make_chunk_map(&mk, kr, s) || !make_chunk_map(&mv, v, s))
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
    p.items_per_head = s.nQ;
    p.total_items = s.B * s.H * s.nQ;
    p.tiles = (s.n_keep + 1) / 2;
    const size_t smem = Cfg<QN>::kSmemTiles + sizeof(Ctrl<QN>);
    const int grid = p.total_items < nsm ? p.total_items : nsm;
    e = cudaFuncSetAttribute(sparse_attn_rows_kernel<QN>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    sparse_attn_rows_kernel<QN><<<grid, kThreads, smem, st>>>(mq, mk, mv, p);
    return cudaGetLastError();
}

}  // namespace

// Contiguous 64-token key blocks; 64-token query blocks (s.qb2 == 0, the mask
// has nQ = nB rows) or 128-token query chunks (s.qb2 == 1).
cudaError_t launch_sparse_attn_rows(const Shape& s, const void* qr, const void* kr, const void* v,
                                    const int32_t* kv_idx, void* o_s, float* lse, DeviceStatus* status,
                                    cudaStream_t st)
{
    if (s.cube) return cudaErrorInvalidValue;
    return s.qb2 ? launch_rows<128>(s, qr, kr, v, kv_idx, o_s, lse, status, st)
                 : launch_rows<64>(s, qr, kr, v, kv_idx, o_s, lse, status, st);
}

}  // namespace rola
