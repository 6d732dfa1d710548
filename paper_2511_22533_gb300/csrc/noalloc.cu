// noalloc.cu -- f3dc_gemm_noalloc: the transformer's tcgen05 GEMM for
// callers that must not allocate device memory.
//
// Some callers cannot call cudaMalloc: code that runs while a CUDA graph is
// being captured in global mode (allocation calls are illegal there), code
// inside a framework that owns all device memory through its own pool and
// forbids side allocations, and latency-critical loops that must never hit
// the driver's allocator.  f3dc_gemm needs a split-K workspace when a problem
// has few row tiles and gets it from a per-device allocation; this variant
// computes exactly the same thing but takes that workspace from a
// fixed-size array in the library's own device image, so a call allocates
// nothing.
#include <mutex>
#include <string>
#include <vector>

#include "../../include/f3dc.h"
#include "kernels.h"

using namespace f3dc;

namespace {

// Largest split-K partial tile (128 rows x 256 fp32 columns) and the number
// of them the array holds: a split never uses more partial tiles than the
// GEMM's grid has CTAs, i.e. than the device has SMs, so 160 tiles cover
// every GB300 (152 SMs).  Behind them, one arrival counter per output tile.
constexpr size_t kPartialTileBytes = 128 * 256 * sizeof(float);
constexpr size_t kPartialTiles = 160;
constexpr size_t kPartialBytes = kPartialTiles * kPartialTileBytes;  // 20 MiB
constexpr size_t kCounterBytes = kGemmMaxCounterTiles * sizeof(int32_t);

// Every GPU that loads libf3dc holds this array until the process exits.
static __device__ __align__(256) unsigned char g_gemm_scratch[kPartialBytes + kCounterBytes];

// Device address of g_gemm_scratch for each device, resolved once with that
// device current.  In host code the array's name is only a host-side stand-in.
std::mutex g_scratch_lock;
std::vector<std::pair<int, unsigned char *>> g_scratch_addr;
// failures are reported through f3dc_last_error(NULL)
f3dc_status fail(f3dc_status st, const std::string &msg)
{
    set_host_error(msg);
    return st;
}

}  // namespace

extern "C" f3dc_status f3dc_gemm_noalloc(const void *A, const void *B, const void *bias, const float *gate, void *out,
                                         int32_t M, int32_t N, int32_t K, int32_t epilogue, void *stream)
{
    if (!A || !B || !out) return fail(F3DC_ERR_INVALID_ARG, "null pointer");
    if (M < 1 || N < 64 || N % 64 != 0 || K < 64 || K % 64 != 0)
        return fail(F3DC_ERR_INVALID_ARG, "need M >= 1, N and K positive multiples of 64");
    if (epilogue < F3DC_EPI_BIAS || epilogue > F3DC_EPI_RESID) return fail(F3DC_ERR_INVALID_ARG, "bad epilogue");
    if (((uintptr_t)out & 15) || (bias && ((uintptr_t)bias & 15)) || (gate && ((uintptr_t)gate & 15)))
        return fail(F3DC_ERR_INVALID_ARG, "pointers must be 16-byte aligned");
    int dev = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return fail(F3DC_ERR_CUDA, std::string("device query: ") + cudaGetErrorString(e));

    // the same tiling and split rule as f3dc_gemm, so the result is the same
    const int bn = N % 256 == 0 ? 256 : (N % 128 == 0 ? 128 : 64);
    const int tiles = ((M + kTileRows - 1) / kTileRows) * (N / bn);
    const int grid = gemm_grid(tiles, sms);
    const int splits = gemm_split_count(tiles, grid, K / 64, sms, true);
    const size_t need = splits > 1 ? gemm_ws_bytes(bn, tiles * splits) : 0;
    if (need > kPartialBytes)
        return fail(F3DC_ERR_INVALID_ARG, "this problem needs " + std::to_string(need) +
                                              " bytes of split-K scratch; the static scratch holds " +
                                              std::to_string(kPartialBytes) + " (use f3dc_gemm)");

    unsigned char *scratch = nullptr;
    {
        std::lock_guard<std::mutex> g(g_scratch_lock);
        for (auto &a : g_scratch_addr)
            if (a.first == dev) scratch = a.second;
        if (!scratch) {  // first call on this device: resolve the array's address
            e = cudaGetSymbolAddress(reinterpret_cast<void **>(&scratch), g_gemm_scratch);
            if (e != cudaSuccess || !scratch)
                return fail(F3DC_ERR_CUDA, std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e));
            g_scratch_addr.push_back({dev, scratch});
        }
    }

    CUtensorMap ta, tb;
    if (!make_tmap_bf16(&ta, A, M, K, K, 128, 64) || !make_tmap_bf16(&tb, B, N, K, K, gemm_b_box_rows(bn), 64))
        return fail(F3DC_ERR_INVALID_ARG, "cuTensorMapEncodeTiled rejected A or B (alignment?)");
    GemmParams p;
    memset(&p, 0, sizeof(p));
    p.M = M;
    p.N = N;
    p.K = K;
    p.m_tiles = (M + kTileRows - 1) / kTileRows;
    p.out = out;
    p.ldo = N;
    p.bias = reinterpret_cast<const bf16 *>(bias);
    p.gate = gate;
    p.ws = reinterpret_cast<float *>(scratch);
    p.counters = reinterpret_cast<int32_t *>(scratch + kPartialBytes);
    p.ws_units = sms;
    cudaStream_t s = (cudaStream_t)stream;
    // the array keeps whatever the previous call left: the arrival counters
    // must start at zero (the partial tiles are always written before read)
    e = cudaMemsetAsync(p.counters, 0, kCounterBytes, s);
    if (e != cudaSuccess) return fail(F3DC_ERR_CUDA, std::string("clearing counters: ") + cudaGetErrorString(e));
    const int epi = epilogue == F3DC_EPI_BIAS ? kEpiBias : (epilogue == F3DC_EPI_GELU ? kEpiGelu : kEpiResid);
    e = launch_gemm(&ta, &tb, p, epi, bn, grid, s);
    if (e != cudaSuccess) return fail(F3DC_ERR_CUDA, std::string("launch: ") + cudaGetErrorString(e));
    return F3DC_OK;
}
