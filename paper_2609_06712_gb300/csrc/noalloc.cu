// rola_lowrank_summary_static: the low-rank summary with no caller workspace.
//
// Some callers cannot hand this library any device scratch: a plugin whose
// host framework owns the allocator and passes the op only its input and
// output tensors, or a runtime that forbids device allocation once it has
// started (fixed memory budget, no cudaMalloc on the serving path).  For
// them this entry point keeps its scratch -- a status word, the RoPE table and
// the partial sums of the summary -- in one file-scope __device__ array of
// kStaticScratchBytes, which every GPU that loads the library holds until
// the process exits.  It allocates nothing itself.
//
// The array's name is usable only in device code; host code needs its
// device address, which cudaGetSymbolAddress returns.  That lookup is done
// once per device, on the first call made while that device is current, and
// cached.  Make that first call before any stream capture.
//
// Every call shares the one array and it keeps the last call's contents.
// Everything a call reads from it, the call has written first (the status
// word is cleared, the table and every partial are overwritten in full) --
// except when a bounded device wait of the bf16 kernel gives up: that kernel
// then stops without writing its partials, so the call's last kernel, seeing
// the status word set, overwrites C and z with NaN (the caller has no
// workspace whose status it could read).  Calls whose executions overlap on
// the GPU -- on different streams, or from different host threads -- race on
// the array and must be serialised by the caller.
#include <mutex>

#include "common.cuh"

namespace rola {
namespace {

constexpr size_t kStaticScratchBytes = size_t(16) << 20;   // 16 MiB per device
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

std::mutex g_lock;
void* g_scratch_ptr[kMaxDevices] = {};

// Device address of g_static_scratch on the current device (looked up once).
cudaError_t scratch_address(void** out)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> guard(g_lock);
    if (!g_scratch_ptr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_static_scratch);
        if (e != cudaSuccess) return e;
        g_scratch_ptr[dev] = p;
    }
    *out = g_scratch_ptr[dev];
    return cudaSuccess;
}

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

// After the combine: if a wait of the pre-pass gave up, C and z hold sums of stale
// partials, so they become NaN.  Nothing is written when the status word is clear.
__global__ void poison_on_timeout_kernel(const DeviceStatus* status, float* C, int nC, float* z, int nz)
{
    if (status->code == 0) return;
    const float nan = __int_as_float(0x7fc00000);
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < nC + nz; i += gridDim.x * blockDim.x) {
        if (i < nC) C[i] = nan;
        else if (z) z[i - nC] = nan;
    }
}

}  // namespace
}  // namespace rola

using namespace rola;

extern "C" rola_status_t rola_lowrank_summary_static(const rola_config_t* cfg, const void* k, const void* v,
                                                     const void* P_k, float* C, float* z, void* stream)
{
    rola_status_t st = validate(cfg);
    if (st != ROLA_OK) return st;
    auto a16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; };
    if (!k || !v || !P_k || !C || !a16(k) || !a16(v) || !a16(P_k) || !a16(C) || (z && !a16(z)))
        return ROLA_ERR_INVALID_ARG;
    const Shape s = make_shape(*cfg);
    // scratch = status word | RoPE table | summary partials (slots of r*128 + r floats);
    // fewer CTAs (bf16) or splits (fp32) if needed to fit, but at least one slot per head
    const size_t head = align256(sizeof(DeviceStatus));
    const size_t table = align256(sizeof(float2) * (size_t)(cfg->T + cfg->Hh + cfg->Ww) * kPairs);
    const size_t slot = sizeof(float) * ((size_t)s.rp * kDh + s.rp);
    const size_t bh = (size_t)s.B * s.H;
    if (head + table + bh * slot > kStaticScratchBytes) return ROLA_ERR_UNSUPPORTED;   // layer too large
    const size_t fit = (kStaticScratchBytes - head - table) / slot;                   // slots available
    void* base = nullptr;
    if (scratch_address(&base) != cudaSuccess) return ROLA_ERR_CUDA;
    unsigned char* b = static_cast<unsigned char*>(base);
    DeviceStatus* status = reinterpret_cast<DeviceStatus*>(b);
    float2* tab = reinterpret_cast<float2*>(b + head);
    float* partials = reinterpret_cast<float*>(b + head + table);
    cudaStream_t cs = static_cast<cudaStream_t>(stream);
    if (cudaMemsetAsync(status, 0, sizeof(DeviceStatus), cs) != cudaSuccess) return ROLA_ERR_CUDA;
    if (launch_rope_table(*cfg, tab, cs) != cudaSuccess) return ROLA_ERR_CUDA;
    if (cfg->dtype == ROLA_BF16) {
        const size_t cap = fit - bh + 1;                                    // CTAs whose slots fit
        const int ctas = prepass_ctas(s, cap < (size_t)kMaxPrepassCtas ? (int)cap : kMaxPrepassCtas);
        if (ctas <= 0) return ROLA_ERR_CUDA;
        if (launch_prepass(s, ctas, nullptr, k, v, P_k, tab, nullptr, nullptr, nullptr, nullptr, partials, status,
                           cs) != cudaSuccess ||
            launch_prepass_combine(s, ctas, partials, C, z, nullptr, cs) != cudaSuccess)
            return ROLA_ERR_CUDA;
        const int nC = (int)(bh * (size_t)s.r * kDh), nz = z ? (int)(bh * (size_t)s.r) : 0;
        poison_on_timeout_kernel<<<(nC + nz + 255) / 256 < 1024 ? (nC + nz + 255) / 256 : 1024, 256, 0, cs>>>(
            status, C, nC, z, nz);
        if (cudaGetLastError() != cudaSuccess) return ROLA_ERR_CUDA;
    } else {
        int nsplit = summary_splits(s);
        if ((size_t)nsplit > fit / bh) nsplit = (int)(fit / bh);
        if (launch_lowrank_summary(cfg->dtype, s, nsplit, k, v, P_k, tab, partials, C, z, nullptr, cs) !=
            cudaSuccess)
            return ROLA_ERR_CUDA;
    }
    return ROLA_OK;
}
