// Output projection of the attention block (Alg. 1, last step: merge heads,
// output projection):
//
//   Y[b][n][f] = sum_{h,d} O[b][h][n][d] W_o[f][h * d_h + d]  (+ b_o[f])
//
// O is the per-head fused output the module writes ([B][H][N][128], bf16);
// "concat_h" needs no copy: the K index k = 128 h + d of the GEMM selects head
// h, so every K step of 64 reads a 128 x 64 box of one head's rows.  W_o is in
// the nn.Linear layout [d_model][H * 128] (row = output feature), Y is
// [B][N][d_model] bf16 (token-major, as the residual stream expects).
//
// A persistent warp-specialised tcgen05 GEMM, one CTA per SM.  Output tiles of
// 128 tokens x 256 features, one batch element each, taken in token-major
// order so that the CTAs in flight share their A rows and all of W_o in L2.
// Per K step of 64: A 128 x 64 (16 KB) and B 256 x 64 (32 KB), both K-major in
// 128-byte swizzle atoms, in a 4-deep TMA ring; four tcgen05.mma M = 128,
// N = 256, K = 16 accumulate fp32 in TMEM.  The accumulator is double-buffered
// (2 x 256 TMEM columns), so one tile's epilogue runs under the next tile's
// MMAs.
//
// Warp roles (192 threads):
//   warp 0     TMA producer
//   warp 1     MMA issuer, TMEM owner
//   warps 2-5  epilogue: warp w reads TMEM lanes 32 (w mod 4) .. +31 (its 32
//              tokens), adds the bias, rounds to bf16, writes 32 x 64 chunks
//              into a double-buffered 128-byte-swizzled staging tile and
//              stores each with one TMA store (rows past N are clipped).
// Every mbarrier wait is bounded; a wait that gives up records
// ROLA_ERR_TIMEOUT in the status word, and the CTA stops issuing, lets what it
// issued complete and frees its TMEM.
#include <cudaTypedefs.h>

#include "common.cuh"
#include "tcgen05.cuh"
#include "tensor_map.cuh"

namespace rola {
namespace {

using namespace tc;

constexpr int kTileM = 128, kTileN = 256, kStepK = 64;
constexpr int kStages = 4;
constexpr uint32_t kABytes = kTileM * kStepK * 2;            // 16 KB
constexpr uint32_t kBBytes = kTileN * kStepK * 2;            // 32 KB
constexpr uint32_t kStageBytes = kABytes + kBBytes;
constexpr uint32_t kStoreBytes = 32 * 64 * 2;                // one epilogue warp's 32 x 64 bf16 chunk
constexpr uint32_t kSmemStages = kStages * kStageBytes;      // 192 KB
constexpr uint32_t kSmemStore = kSmemStages;                 // 4 warps x 2 buffers x 4 KB
constexpr uint32_t kSmemTiles = kSmemStore + 8 * kStoreBytes;
constexpr int kThreads = 192;
constexpr int kEpiWarps = 4;
constexpr uint32_t kTmemCols = 2 * kTileN;

enum Bar { FULL = 0, EMPTY = FULL + kStages, ACC_FULL = EMPTY + kStages, ACC_EMPTY = ACC_FULL + 2,
           DRAIN = ACC_EMPTY + 2, NUM_BARS = DRAIN + 1 };

struct Ctrl {
    uint64_t bar[NUM_BARS];
    uint32_t tmem_base;
    int abort;
};

struct Params {
    int B, N, H, d_model;
    int m_tiles;          // ceil(N / 128) per batch element
    int n_tiles;          // ceil(d_model / 256)
    int tiles;            // B * m_tiles * n_tiles
    int k_steps;          // H * 128 / 64
    const float* bias;    // nullable, fp32 [d_model]
    DeviceStatus* status;
    uint64_t wait_limit_ns;
};

__device__ __forceinline__ void record_timeout(const Params& p, int where)
{
    if (atomicCAS(&p.status->code, 0, (int)ROLA_ERR_TIMEOUT) == 0) p.status->where = where;
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const void* map, uint32_t bar, int x, int y)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], [%2];\n" ::"r"(
            dst),
        "l"(map), "r"(bar), "r"(x), "r"(y)
        : "memory");
}

__device__ __forceinline__ void tma_store_3d(const void* map, uint32_t src, int x, int y, int z)
{
    asm volatile("cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%2, %3, %4}], [%1];\n" ::"l"(map),
                 "r"(src), "r"(x), "r"(y), "r"(z)
                 : "memory");
}

// Waits until at most one of this thread's committed bulk stores still reads shared memory.
__device__ __forceinline__ void bulk_wait_read_1() { asm volatile("cp.async.bulk.wait_group.read 1;\n" ::: "memory"); }

// Tile t -> (batch, token tile, feature tile); feature tiles vary fastest.
__device__ __forceinline__ void tile_coords(const Params& p, int t, int& b, int& mt, int& nt)
{
    nt = t % p.n_tiles;
    const int rest = t / p.n_tiles;
    mt = rest % p.m_tiles;
    b = rest / p.m_tiles;
}

__global__ void __launch_bounds__(kThreads, 1) out_proj_kernel(const __grid_constant__ CUtensorMap map_o,
                                                               const __grid_constant__ CUtensorMap map_w,
                                                               const __grid_constant__ CUtensorMap map_y,
                                                               const Params p)
{
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    if (smem_u32(smem_raw) & 1023u) {     // the 128-byte swizzle atoms need a 1024-byte aligned base
        if (threadIdx.x == 0) atomicCAS(&p.status->code, 0, (int)ROLA_ERR_UNSUPPORTED);
        return;
    }
    Ctrl& cb = *reinterpret_cast<Ctrl*>(smem_raw + kSmemTiles);
    const uint32_t sbase = smem_u32(smem_raw);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    auto bar = [&](int i) { return smem_u32(&cb.bar[i]); };

    if (tid == 0) {
        cb.abort = 0;
        for (int i = 0; i < kStages; ++i) {
            mbar_init(bar(FULL + i), 1);
            mbar_init(bar(EMPTY + i), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar(ACC_FULL + i), 1);
            mbar_init(bar(ACC_EMPTY + i), kEpiWarps);
        }
        mbar_init(bar(DRAIN), 1);
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(&cb.tmem_base), kTmemCols);
        tmem_relinquish();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&map_o);
        tma_prefetch_desc(&map_w);
        tma_prefetch_desc(&map_y);
    }
    fence_before_sync();
    __syncthreads();
    fence_after_sync();
    const uint32_t tmem = cb.tmem_base;
    volatile int* abort = &cb.abort;
    const uint64_t limit = p.wait_limit_ns;

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            bool ok = true;
            int g = 0;                                  // K steps issued by this CTA
            for (int t = blockIdx.x; t < p.tiles && ok; t += gridDim.x) {
                int b, mt, nt;
                tile_coords(p, t, b, mt, nt);
                for (int ks = 0; ks < p.k_steps; ++ks, ++g) {
                    const int s = g % kStages;
                    if (g >= kStages && !(ok = mbar_wait(bar(EMPTY + s), ((g / kStages) - 1) & 1, abort, limit)))
                        break;
                    const uint32_t dst = sbase + s * kStageBytes;
                    mbar_expect_tx(bar(FULL + s), kStageBytes);
                    // A: head ks / 2, d-chunk ks % 2, tokens 128 mt .. +127 of batch element b
                    tma_load_4d(dst, &map_o, bar(FULL + s), (ks & 1) * kStepK, mt * kTileM, ks >> 1, b);
                    // B: features 256 nt .. +255, K columns 64 ks .. +63
                    tma_load_2d(dst + kABytes, &map_w, bar(FULL + s), ks * kStepK, nt * kTileN);
                }
            }
            if (!ok) record_timeout(p, 1);
            // the copies still in flight land before the CTA exits: wait for the last use of each stage
            int never = 0;
            for (int u = g > kStages ? g - kStages : 0; u < g; ++u)
                mbar_wait(bar(FULL + u % kStages), (u / kStages) & 1, &never, limit);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16(kTileM, kTileN, false, false);
            const uint64_t da = smem_desc(sbase, 16, 1024), db = smem_desc(sbase + kABytes, 16, 1024);
            const uint32_t a_lo = (uint32_t)da, a_hi = (uint32_t)(da >> 32);
            const uint32_t b_lo = (uint32_t)db, b_hi = (uint32_t)(db >> 32);
            bool ok = true;
            int g = 0, it = 0;
            for (int t = blockIdx.x; t < p.tiles && ok; t += gridDim.x, ++it) {
                const int ab = it & 1;
                if (it >= 2 && !(ok = mbar_wait(bar(ACC_EMPTY + ab), ((it >> 1) - 1) & 1, abort, limit))) break;
                fence_after_sync();
                const uint32_t d = tmem + ab * kTileN;
                for (int ks = 0; ks < p.k_steps; ++ks, ++g) {
                    const int s = g % kStages;
                    if (!(ok = mbar_wait(bar(FULL + s), (g / kStages) & 1, abort, limit))) break;
                    fence_after_sync();
                    const uint32_t off = s * (kStageBytes >> 4);
#pragma unroll
                    for (int kk = 0; kk < kStepK / 16; ++kk)
                        mma_ss_split(d, a_lo + off + kk * 2, a_hi, b_lo + off + kk * 2, b_hi, idesc,
                                     (ks > 0 || kk > 0) ? 1u : 0u);
                    mma_commit(bar(EMPTY + s));
                }
                if (!ok) break;
                mma_commit(bar(ACC_FULL + ab));
            }
            if (!ok) record_timeout(p, 2);
            // every MMA issued completes before TMEM is released
            int never = 0;
            mma_commit(bar(DRAIN));
            mbar_wait(bar(DRAIN), 0, &never, limit);
        }
    } else {
        // ------------------------------------------------------------ epilogue
        const int q = warp & 3;                          // TMEM lane quarter: tokens 32 q .. +31 of the tile
        const uint32_t lane_off = (uint32_t)(q * 32) << 16;
        const int ew = warp - 2;                         // this warp's staging buffers
        bool ok = true;
        int it = 0, chunk = 0;
        for (int t = blockIdx.x; t < p.tiles && ok; t += gridDim.x, ++it) {
            int b, mt, nt;
            tile_coords(p, t, b, mt, nt);
            const int ab = it & 1;
            if (!(ok = mbar_wait(bar(ACC_FULL + ab), (it >> 1) & 1, abort, limit))) break;
            fence_after_sync();
            const int row0 = mt * kTileM + q * 32;       // first token of this warp's rows
            for (int c = 0; c < kTileN / 64; ++c, ++chunk) {
                const int f0 = nt * kTileN + c * 64;
                float v[64];
#pragma unroll
                for (int j = 0; j < 4; ++j)
                    tmem_ld16(tmem + lane_off + ab * kTileN + c * 64 + j * 16, *reinterpret_cast<float(*)[16]>(&v[j * 16]));
                tmem_ld_wait(*reinterpret_cast<float(*)[16]>(&v[0]));
#pragma unroll
                for (int j = 1; j < 4; ++j) reg_fence(*reinterpret_cast<float(*)[16]>(&v[j * 16]));
                if (c == kTileN / 64 - 1) {
                    // the accumulator buffer is free for the tile after next
                    fence_before_sync();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(bar(ACC_EMPTY + ab));
                }
                if (p.bias) {
#pragma unroll
                    for (int j = 0; j < 64; j += 4) {
                        const float4 bb = f0 + j < p.d_model ? __ldg(reinterpret_cast<const float4*>(p.bias + f0 + j))
                                                             : make_float4(0.f, 0.f, 0.f, 0.f);
                        v[j] += bb.x; v[j + 1] += bb.y; v[j + 2] += bb.z; v[j + 3] += bb.w;
                    }
                }
                // staging buffer of this chunk: free once the store issued two chunks ago has read it
                const uint32_t buf = sbase + kSmemStore + (ew * 2 + (chunk & 1)) * kStoreBytes;
                if (lane == 0 && chunk >= 2) bulk_wait_read_1();
                __syncwarp();
#pragma unroll
                for (int cc = 0; cc < 8; ++cc) {
                    const uint32_t w0 = pack_bf16(v[8 * cc], v[8 * cc + 1]), w1 = pack_bf16(v[8 * cc + 2], v[8 * cc + 3]);
                    const uint32_t w2 = pack_bf16(v[8 * cc + 4], v[8 * cc + 5]), w3 = pack_bf16(v[8 * cc + 6], v[8 * cc + 7]);
                    asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};\n" ::"r"(buf + lane * 128 + ((cc ^ (lane & 7)) << 4)),
                                 "r"(w0), "r"(w1), "r"(w2), "r"(w3)
                                 : "memory");
                }
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0 && row0 < p.N && f0 < p.d_model) {
                    tma_store_3d(&map_y, buf, f0, row0, b);
                    bulk_commit();
                }
            }
        }
        if (!ok) record_timeout(p, 3);
        if (lane == 0) bulk_wait_all();                  // the stores have left shared memory
    }
    fence_before_sync();
    __syncthreads();
    fence_after_sync();
    if (warp == 1) tmem_dealloc(tmem, kTmemCols);
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn()
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

bool encode(CUtensorMap* m, int rank, const void* ptr, const cuuint64_t* dims, const cuuint64_t* strides,
            const cuuint32_t* box)
{
    auto enc = encode_fn();
    if (!enc) return false;
    const cuuint32_t es[4] = {1, 1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, const_cast<void*>(ptr), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// ---------------------------------------------------------------------------
// fp32 validation mode: the same product in plain fp32 SIMT arithmetic (no
// bf16, no tensor cores).  64 tokens x 64 features per CTA, 256 threads with
// 4 x 4 outputs each, K staged through shared memory 16 at a time.
constexpr int kF32Tile = 64, kF32Chunk = 16;

__global__ void __launch_bounds__(256) out_proj_f32_kernel(int N, int H, int d_model, const float* __restrict__ O,
                                                           const float* __restrict__ W, const float* __restrict__ bias,
                                                           float* __restrict__ Y)
{
    __shared__ float as[kF32Chunk][kF32Tile + 1];
    __shared__ float bs[kF32Chunk][kF32Tile + 1];
    const int b = blockIdx.z, n0 = blockIdx.y * kF32Tile, f0 = blockIdx.x * kF32Tile;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    const int K = H * kDh;
    float acc[4][4] = {};
    for (int k0 = 0; k0 < K; k0 += kF32Chunk) {
        const int h = k0 / kDh, d0 = k0 - h * kDh;
        for (int e = threadIdx.x; e < kF32Tile * kF32Chunk; e += 256) {
            const int r = e / kF32Chunk, kk = e % kF32Chunk;
            const int n = n0 + r, f = f0 + r;
            as[kk][r] = n < N ? O[(((size_t)b * H + h) * N + n) * kDh + d0 + kk] : 0.0f;
            bs[kk][r] = f < d_model ? W[(size_t)f * K + k0 + kk] : 0.0f;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < kF32Chunk; ++kk)
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(as[kk][ty + 16 * i], bs[kk][tx + 16 * j], acc[i][j]);
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int n = n0 + ty + 16 * i;
        if (n >= N) continue;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int f = f0 + tx + 16 * j;
            if (f < d_model) Y[((size_t)b * N + n) * d_model + f] = acc[i][j] + (bias ? bias[f] : 0.0f);
        }
    }
}

}  // namespace

cudaError_t launch_out_proj_f32(int B, int N, int H, int d_model, const float* O, const float* W, const float* bias,
                                float* Y, cudaStream_t st)
{
    dim3 grid((d_model + kF32Tile - 1) / kF32Tile, (N + kF32Tile - 1) / kF32Tile, B);
    out_proj_f32_kernel<<<grid, 256, 0, st>>>(N, H, d_model, O, W, bias, Y);
    return cudaGetLastError();
}

cudaError_t launch_out_proj(int B, int N, int H, int d_model, const void* O, const void* W, const float* bias,
                            void* Y, DeviceStatus* status, uint64_t wait_limit_ns, cudaStream_t st)
{
    CUtensorMap mo, mw, my;
    {   // O as (d, token, head, batch), 64 x 128 boxes
        const cuuint64_t dims[4] = {(cuuint64_t)kDh, (cuuint64_t)N, (cuuint64_t)H, (cuuint64_t)B};
        const cuuint64_t strides[3] = {(cuuint64_t)kDh * 2, (cuuint64_t)N * kDh * 2, (cuuint64_t)H * N * kDh * 2};
        const cuuint32_t box[4] = {kStepK, kTileM, 1, 1};
        if (!encode(&mo, 4, O, dims, strides, box)) return cudaErrorInvalidValue;
    }
    {   // W_o as (K, feature), 64 x 256 boxes
        const cuuint64_t dims[2] = {(cuuint64_t)H * kDh, (cuuint64_t)d_model};
        const cuuint64_t strides[1] = {(cuuint64_t)H * kDh * 2};
        const cuuint32_t box[2] = {kStepK, kTileN};
        if (!encode(&mw, 2, W, dims, strides, box)) return cudaErrorInvalidValue;
    }
    {   // Y as (feature, token, batch), 64 x 32 boxes
        const cuuint64_t dims[3] = {(cuuint64_t)d_model, (cuuint64_t)N, (cuuint64_t)B};
        const cuuint64_t strides[2] = {(cuuint64_t)d_model * 2, (cuuint64_t)N * d_model * 2};
        const cuuint32_t box[3] = {64, 32, 1};
        if (!encode(&my, 3, Y, dims, strides, box)) return cudaErrorInvalidValue;
    }
    int dev = 0, nsm = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    Params p;
    p.B = B;
    p.N = N;
    p.H = H;
    p.d_model = d_model;
    p.m_tiles = (N + kTileM - 1) / kTileM;
    p.n_tiles = (d_model + kTileN - 1) / kTileN;
    p.tiles = B * p.m_tiles * p.n_tiles;
    p.k_steps = H * kDh / kStepK;
    p.bias = bias;
    p.status = status;
    p.wait_limit_ns = wait_limit_ns;
    const size_t smem = kSmemTiles + sizeof(Ctrl);
    e = cudaFuncSetAttribute(out_proj_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int grid = p.tiles < nsm ? p.tiles : nsm;
    out_proj_kernel<<<grid, kThreads, smem, st>>>(mo, mw, my, p);
    return cudaGetLastError();
}

}  // namespace rola
