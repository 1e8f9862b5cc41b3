// Low-rank readout and gated fusion of the bf16 path (kernel 4):
//   q~_p   = R_r(p) SiLU(P_q q^n_p)                     Eq. (qklr) (or the placement cfg selects)
//   O^lr_p = y_p / sqrt(mean_i y_{p,i}^2 + eps_lr),     y_p = q~_p^T C      Eq. (ctx)
//   r_p    = sqrt(mean_i (O^s_{p,i})^2 + eps_fuse)
//   O_p    = O^s_p + g_p r_p O^lr_p                     Eq. (gate), (O^s/r_p + g O^lr) r_p
//
// Work unit = (head, 64-token block); G persistent CTAs (two per SM for
// r <= 48, else one) take
// contiguous unit ranges, so P_q and C (bf16) are loaded once per head a CTA
// meets instead of once per block.  Each unit's q and O^s blocks arrive by TMA
// (one 16 KB [chunk][row][64] box each) in a ring of stages; the fused O is
// written over O^s in the stage and leaves by a TMA store, which also clips
// the rows past N of the last block.  The loads of unit i + S - 1 go out after
// unit i's first barrier, once the store that last read that stage is done
// reading it.
//
// Eight warps per unit: warp w takes tokens 16 (w & 3) .. +15 and half h = w >> 2
// of the work: U = Q P_q^T for half of the r columns (then q~ to shared
// memory), y = q~ C for d in [64 h, 64 h + 64); the row sums of y^2 and of
// (O^s)^2 are combined over the two halves through shared memory.
#include <cudaTypedefs.h>

#include "common.cuh"
#include "tcgen05.cuh"
#include "tensor_map.cuh"

namespace rola {
namespace {

using namespace tc;

constexpr int kWarps = 8;
constexpr int kThreads = 32 * kWarps;
constexpr uint32_t kBox = 64 * 128 * 2;
constexpr int kMaxStages = 4;

// r <= 48: two CTAs per SM (16 warps) with a 2-deep ring; wider r: one CTA
// with a 4-deep ring (P_q and C take more shared memory and registers)
template <int R>
struct Occupancy {
    static constexpr int ctas = R <= 48 ? 2 : 1;
    static constexpr int stages = R <= 48 ? 2 : 4;
};

template <int R>
struct Layout {
    static constexpr int NT = R / 8;
    static constexpr int NTW = NT / 2;               // n-tiles of U per warp
    static constexpr int QT = 2 * R + 16;            // bytes per q~ row (padded against bank conflicts)
    static constexpr uint32_t stage_bytes = 2 * kBox;   // q | O^s
    static constexpr uint32_t P = Occupancy<R>::stages * stage_bytes;
    static constexpr uint32_t C = P + R * 256;
    static constexpr uint32_t qt = C + R * 256;
    static constexpr uint32_t red = qt + 64 * QT;    // [y^2 | O^s^2][half][64 rows] fp32
    static constexpr uint32_t bars = red + 2 * 2 * 64 * 4;
    static constexpr uint32_t total = bars + kMaxStages * 8 + 16;
};

struct Params {
    Shape s;
    const __nv_bfloat16* Pq;
    const __nv_bfloat16* Cbf;
    const float* gate;
    const float2* tab;
    DeviceStatus* status;
    int units;
};

// SiLU with the MUFU exponential; the kernel is instantiated for it and for
// ActAblation (the other feature maps of the activation ablation).
struct SiluMufu {
    int kind;    // always ROLA_LOWRANK_ACT_SILU
    __device__ float operator()(float x) const { return silu(x); }
};

template <int R, typename Act>
__global__ void __launch_bounds__(kThreads, Occupancy<R>::ctas) readout_kernel(const __grid_constant__ CUtensorMap map_q,
                                                              const __grid_constant__ CUtensorMap map_os,
                                                              const __grid_constant__ CUtensorMap map_o,
                                                              const Params p)
{
    using L = Layout<R>;
    constexpr int NTW = L::NTW;
    constexpr int kStages = Occupancy<R>::stages;
    extern __shared__ __align__(1024) uint8_t smem[];
    if (smem_u32(smem) & 1023u) {
        if (threadIdx.x == 0) atomicCAS(&p.status->code, 0, (int)ROLA_ERR_UNSUPPORTED);
        return;
    }
    const Shape& s = p.s;
    const uint32_t sbase = smem_u32(smem), sP = sbase + L::P, sC = sbase + L::C, sQt = sbase + L::qt;
    float* red = reinterpret_cast<float*>(smem + L::red);
    const uint32_t full0 = sbase + L::bars;
    volatile int* abort = reinterpret_cast<volatile int*>(smem + L::bars + kMaxStages * 8);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int g = lane >> 2, t4 = lane & 3, mi = lane >> 3;
    const int mt = warp & 3, half = warp >> 2;
    const int u0 = (int)((long long)blockIdx.x * p.units / gridDim.x);
    const int u1 = (int)((long long)(blockIdx.x + 1) * p.units / gridDim.x);
    const int count = u1 - u0;

    if (tid == 0) {
        *abort = 0;
        for (int i = 0; i < kStages; ++i) mbar_init(full0 + 8 * i, 1);
        fence_mbar_init();
        tma_prefetch_desc(&map_q);
        tma_prefetch_desc(&map_os);
        tma_prefetch_desc(&map_o);
    }
    __syncthreads();

    // loads of the j-th unit into stage j % S, by thread 0 (the thread that
    // stores, so that its bulk-group waits order a refill after the store)
    auto issue = [&](int j) {
        const int u = u0 + j, bh = u / s.nC, blk = u - bh * s.nC, st = j % kStages;
        const uint32_t dst = sbase + st * L::stage_bytes, bar = full0 + 8 * st;
        if (tid == 0) {
            mbar_expect_tx(bar, 2 * kBox);
            tma_load_4d(dst, &map_q, bar, 0, blk * 64, 0, bh);
            tma_load_4d(dst + kBox, &map_os, bar, 0, blk * 64, 0, bh);
        }
    };
    int issued = count < kStages ? count : kStages;
    for (int j = 0; j < issued; ++j) issue(j);

    int kaxis[NTW];
#pragma unroll
    for (int j = 0; j < NTW; ++j) {
        const int m = (half * NTW + j) * 4 + t4;
        kaxis[j] = m < s.pt ? 0 : (m < s.pt + s.px ? 1 : 2);
    }
    const int hw = s.Hh * s.Ww;

    int hb = -1;
    bool failed = false;
    int i = 0;
    for (int u = u0; u < u1; ++u, ++i) {
        const int bh = u / s.nC, blk = u - bh * s.nC, b = bh / s.H;
        const int st = i % kStages;
        if (bh != hb) {
            // P_q of the head and C of (batch, head); every reader of the old ones has passed the last barrier
            const uint4* srcP = reinterpret_cast<const uint4*>(p.Pq + (size_t)(bh % s.H) * s.r * kDh);
            const uint4* srcC = reinterpret_cast<const uint4*>(p.Cbf + (size_t)bh * R * kDh);   // rp rows
            for (int e = tid; e < R * 16; e += kThreads) {
                const uint4 a = (e >> 4) < s.r ? __ldg(srcP + e) : make_uint4(0, 0, 0, 0), c = __ldg(srcC + e);
                const uint32_t off = sw128(e >> 4, e & 15);
                asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};\n" ::"r"(sP + off), "r"(a.x), "r"(a.y), "r"(a.z),
                             "r"(a.w)
                             : "memory");
                asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};\n" ::"r"(sC + off), "r"(c.x), "r"(c.y), "r"(c.z),
                             "r"(c.w)
                             : "memory");
            }
            bar_sync(1, kThreads);
            hb = bh;
        }
        const uint32_t qb = sbase + st * L::stage_bytes, ob = qb + kBox;
        const int n_base = blk * kBlock;
        // (cos, sin) of this thread's q~ pairs for its two tokens
        float2 kcs[2][NTW];
        {
            const int n = n_base + mt * 16 + g;
            int t = n / hw;
            const int rem = n - t * hw;
            int x = rem / s.Ww, y = rem - x * s.Ww;
#pragma unroll
            for (int hr = 0; hr < 2; ++hr) {
#pragma unroll
                for (int j = 0; j < NTW; ++j) {
                    const int row = kaxis[j] == 0 ? min(t, s.T - 1) : (kaxis[j] == 1 ? s.T + x : s.T + s.Hh + y);
                    kcs[hr][j] = __ldg(p.tab + row * kPairs + (half * NTW + j) * 4 + t4);
                }
                y += 8;
                while (y >= s.Ww) {
                    y -= s.Ww;
                    if (++x == s.Hh) {
                        x = 0;
                        ++t;
                    }
                }
            }
        }
        // the gate of this thread's two rows, loaded ahead of use
        const int r_lo = mt * 16 + g, r_hi = r_lo + 8;
        float gp[2];
#pragma unroll
        for (int hr = 0; hr < 2; ++hr) {
            const int n = min(n_base + (hr ? r_hi : r_lo), s.N - 1);
            gp[hr] = p.gate ? __ldg(p.gate + (size_t)b * s.N + n) : s.default_gate;
        }
        const bool ok = mbar_wait(full0 + 8 * st, (i / kStages) & 1, abort, s.wait_limit_ns);
        if (ok) {
            // ---- U = Q P_q^T: tokens 16 mt .. +15, this warp's half of the r columns
            float uacc[NTW][4];
#pragma unroll
            for (int j = 0; j < NTW; ++j) uacc[j][0] = uacc[j][1] = uacc[j][2] = uacc[j][3] = 0.0f;
#pragma unroll
            for (int kc = 0; kc < 8; ++kc) {
                uint32_t a0, a1, a2, a3;
                ldsm_x4(qb + tsw(mt * 16 + (lane & 7) + (mi & 1) * 8, kc * 2 + (mi >> 1)), a0, a1, a2, a3);
#pragma unroll
                for (int np = 0; np < NTW / 2; ++np) {
                    const int nt = half * NTW + 2 * np;
                    uint32_t b0, b1, b2, b3;
                    ldsm_x4(sP + sw128(nt * 8 + (mi >> 1) * 8 + (lane & 7), kc * 2 + (mi & 1)), b0, b1, b2, b3);
                    mma_bf16(uacc[2 * np], a0, a1, a2, a3, b0, b1);
                    mma_bf16(uacc[2 * np + 1], a0, a1, a2, a3, b2, b3);
                }
                if (NTW & 1) {
                    const int nt = half * NTW + NTW - 1;
                    uint32_t b0, b1;
                    ldsm_x2(sP + sw128(nt * 8 + (lane & 7), kc * 2 + (mi & 1)), b0, b1);
                    mma_bf16(uacc[NTW - 1], a0, a1, a2, a3, b0, b1);
                }
            }
            // ---- q~ (bf16) into shared memory; tokens past N give zero features
#pragma unroll
            for (int hr = 0; hr < 2; ++hr) {
                const int tl = mt * 16 + g + hr * 8;
#pragma unroll
                for (int j = 0; j < NTW; ++j) {
                    const int nt = half * NTW + j;
                    const float2 f = lowrank_pair(uacc[j][2 * hr], uacc[j][2 * hr + 1], kcs[hr][j], s.lr_rope,
                                                  Act{s.lr_act});
                    asm volatile("st.shared.b32 [%0], %1;\n" ::"r"(sQt + tl * L::QT + (nt * 8 + t4 * 2) * 2),
                                 "r"(pack_bf16(f.x, f.y))
                                 : "memory");
                }
            }
        }
        // every thread reaches this barrier once per unit; it also settles a timeout
        if (bar_red_or(1, kThreads, !ok)) {
            failed = true;
            break;
        }
        if (i >= 1 && issued < count) {
            // refill the stage of unit i - 1 once its store has finished reading it
            if (tid == 0) bulk_wait_read_all();
            issue(issued);
            ++issued;
        }
        // ---- y = q~ C for d in [64 half, 64 half + 64)
        float yacc[8][4];
#pragma unroll
        for (int j = 0; j < 8; ++j) yacc[j][0] = yacc[j][1] = yacc[j][2] = yacc[j][3] = 0.0f;
#pragma unroll
        for (int kc = 0; kc < R / 16; ++kc) {
            uint32_t a0, a1, a2, a3;
            ldsm_x4(sQt + (mt * 16 + (lane & 7) + (mi & 1) * 8) * L::QT + (kc * 2 + (mi >> 1)) * 16, a0, a1, a2, a3);
#pragma unroll
            for (int dp = 0; dp < 4; ++dp) {
                uint32_t b0, b1, b2, b3;
                ldsm_x4_t(sC + sw128(kc * 16 + (mi & 1) * 8 + (lane & 7), half * 8 + dp * 2 + (mi >> 1)), b0, b1, b2,
                          b3);
                mma_bf16(yacc[2 * dp], a0, a1, a2, a3, b0, b1);
                mma_bf16(yacc[2 * dp + 1], a0, a1, a2, a3, b2, b3);
            }
        }
        // ---- row sums of y^2 and (O^s)^2 over this half's 64 d, then over both halves
        float ssy[2] = {0.0f, 0.0f}, sso[2] = {0.0f, 0.0f};
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const int c = half * 8 + j;
            uint32_t wlo, whi;
            asm volatile("ld.shared.b32 %0, [%1];\n" : "=r"(wlo) : "r"(ob + tsw(r_lo, c) + t4 * 4));
            asm volatile("ld.shared.b32 %0, [%1];\n" : "=r"(whi) : "r"(ob + tsw(r_hi, c) + t4 * 4));
            const float2 lo = unpack_bf16(wlo), hi = unpack_bf16(whi);
            ssy[0] += yacc[j][0] * yacc[j][0] + yacc[j][1] * yacc[j][1];
            ssy[1] += yacc[j][2] * yacc[j][2] + yacc[j][3] * yacc[j][3];
            sso[0] += lo.x * lo.x + lo.y * lo.y;
            sso[1] += hi.x * hi.x + hi.y * hi.y;
        }
#pragma unroll
        for (int hr = 0; hr < 2; ++hr) {
            ssy[hr] += __shfl_xor_sync(0xffffffffu, ssy[hr], 1);
            ssy[hr] += __shfl_xor_sync(0xffffffffu, ssy[hr], 2);
            sso[hr] += __shfl_xor_sync(0xffffffffu, sso[hr], 1);
            sso[hr] += __shfl_xor_sync(0xffffffffu, sso[hr], 2);
        }
        if (t4 == 0) {
            red[(0 * 2 + half) * 64 + r_lo] = ssy[0];
            red[(0 * 2 + half) * 64 + r_hi] = ssy[1];
            red[(1 * 2 + half) * 64 + r_lo] = sso[0];
            red[(1 * 2 + half) * 64 + r_hi] = sso[1];
        }
        bar_sync(1, kThreads);
        // ---- O = O^s + g r_p O^lr, written over O^s in the stage
        float coef[2];
#pragma unroll
        for (int hr = 0; hr < 2; ++hr) {
            const int row = hr ? r_hi : r_lo;
            const float sy = red[0 * 64 + row] + red[1 * 64 + row];
            const float so = red[2 * 64 + row] + red[3 * 64 + row];
            coef[hr] = gp[hr] * sqrtf(so * (1.0f / kDh) + s.eps_fuse) * rsqrtf(sy * (1.0f / kDh) + s.eps_lr);
        }
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const int c = half * 8 + j;
            const uint32_t alo = ob + tsw(r_lo, c) + t4 * 4, ahi = ob + tsw(r_hi, c) + t4 * 4;
            uint32_t wlo, whi;
            asm volatile("ld.shared.b32 %0, [%1];\n" : "=r"(wlo) : "r"(alo));
            asm volatile("ld.shared.b32 %0, [%1];\n" : "=r"(whi) : "r"(ahi));
            const float2 lo = unpack_bf16(wlo), hi = unpack_bf16(whi);
            const uint32_t olo = pack_bf16(lo.x + coef[0] * yacc[j][0], lo.y + coef[0] * yacc[j][1]);
            const uint32_t ohi = pack_bf16(hi.x + coef[1] * yacc[j][2], hi.y + coef[1] * yacc[j][3]);
            asm volatile("st.shared.b32 [%0], %1;\n" ::"r"(alo), "r"(olo) : "memory");
            asm volatile("st.shared.b32 [%0], %1;\n" ::"r"(ahi), "r"(ohi) : "memory");
        }
        fence_proxy_async_smem();
        bar_sync(1, kThreads);
        if (tid == 0) {
            tma_store_4d(&map_o, ob, 0, n_base, 0, bh);
            bulk_commit();
        }
    }
    if (tid == 0) {
        if (failed) {
            if (atomicCAS(&p.status->code, 0, (int)ROLA_ERR_TIMEOUT) == 0) p.status->where = 8;
            // loads issued and not yet waited for must land before the CTA exits
            int never = 0;
            for (int j = i; j < issued; ++j)
                mbar_wait(full0 + 8 * (j % kStages), (j / kStages) & 1, &never, s.wait_limit_ns);
        }
        bulk_wait_all();
    }
}

template <int R, typename Act>
cudaError_t launch_ra(const CUtensorMap& mq, const CUtensorMap& mos, const CUtensorMap& mo, const Params& p, int ctas,
                      cudaStream_t st)
{
    using L = Layout<R>;
    static_assert(L::total <= 232448, "fits the shared memory of one SM");
    cudaError_t e =
        cudaFuncSetAttribute(readout_kernel<R, Act>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)L::total);
    if (e != cudaSuccess) return e;
    readout_kernel<R, Act><<<ctas, kThreads, L::total, st>>>(mq, mos, mo, p);
    return cudaGetLastError();
}

template <int R>
cudaError_t launch_r(const CUtensorMap& mq, const CUtensorMap& mos, const CUtensorMap& mo, const Params& p, int ctas,
                     cudaStream_t st)
{
    return p.s.lr_act == ROLA_LOWRANK_ACT_SILU ? launch_ra<R, SiluMufu>(mq, mos, mo, p, ctas, st)
                                               : launch_ra<R, ActAblation>(mq, mos, mo, p, ctas, st);
}

}  // namespace

cudaError_t launch_readout(const Shape& s, const void* q, const void* P_q, const __nv_bfloat16* Cbf,
                           const float* gate, const void* o_s, void* o, const float2* tab, DeviceStatus* status,
                           cudaStream_t st)
{
    const int units = s.B * s.H * s.nC;
    int dev = 0, nsm = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    const int per_sm = s.rp <= 48 ? 2 : 1;                   // Occupancy<R>::ctas
    const int ctas = units < nsm * per_sm ? units : nsm * per_sm;
    CUtensorMap mq, mos, mo;
    if (!make_block_map(&mq, q, s) || !make_block_map(&mos, o_s, s) || !make_block_map(&mo, o, s))
        return cudaErrorInvalidValue;
    Params p;
    p.s = s;
    p.Pq = static_cast<const __nv_bfloat16*>(P_q);
    p.Cbf = Cbf;
    p.gate = gate;
    p.tab = tab;
    p.status = status;
    p.units = units;
    switch (s.rp) {
        case 16: return launch_r<16>(mq, mos, mo, p, ctas, st);
        case 32: return launch_r<32>(mq, mos, mo, p, ctas, st);
        case 48: return launch_r<48>(mq, mos, mo, p, ctas, st);
        case 64: return launch_r<64>(mq, mos, mo, p, ctas, st);
        case 80: return launch_r<80>(mq, mos, mo, p, ctas, st);
        case 96: return launch_r<96>(mq, mos, mo, p, ctas, st);
        case 112: return launch_r<112>(mq, mos, mo, p, ctas, st);
        case 128: return launch_r<128>(mq, mos, mo, p, ctas, st);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace rola
