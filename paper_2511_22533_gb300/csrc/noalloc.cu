// noalloc.cu -- f3dc_gemm_noalloc: the transformer's tcgen05 GEMM for
// callers that must not allocate device memory, and the device status word
// of the standalone kernel calls (f3dc_gemm, f3dc_gemm_noalloc,
// f3dc_attention; read by f3dc_gemm_status).
//
// Some callers cannot call cudaMalloc: code that runs while a CUDA graph is
// being captured in global mode (allocation calls are illegal there), code
// inside a framework that owns all device memory through its own pool and
// forbids side allocations, and latency-critical loops that must never hit
// the driver's allocator.  f3dc_gemm needs a split-K workspace when a problem
// has few row tiles and gets it from a per-device allocation; this variant
// makes the same launch decisions (CTA-pair kernel, or the single-CTA kernel
// with the same split rule) and so computes bit for bit the same result, but
// takes that workspace from a fixed-size array in the library's own device
// image, so a call allocates nothing.
#include <cstring>
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

// Status word (F3DC_DEV_* bits) that the standalone GEMM and attention
// kernels record into (a bounded wait that ran out), sticky until
// f3dc_gemm_status reads it.
// __device__ variables start at zero.
static __device__ __align__(256) uint32_t g_gemm_status;

// Device addresses of the two symbols for each device, resolved once with
// that device current.  In host code a symbol's name is only a host-side
// stand-in, never a device address.
struct DeviceSyms {
    int dev;
    unsigned char *scratch;
    uint32_t *status;
};
std::mutex g_syms_lock;
std::vector<DeviceSyms> g_syms;

// failures are reported through f3dc_last_error(NULL)
f3dc_status fail(f3dc_status st, const std::string &msg)
{
    set_host_error(msg);
    return st;
}

// The current device's symbol addresses (first use on a device resolves them).
cudaError_t device_syms(DeviceSyms *out)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> g(g_syms_lock);
    for (const DeviceSyms &s : g_syms)
        if (s.dev == dev) {
            *out = s;
            return cudaSuccess;
        }
    DeviceSyms s{dev, nullptr, nullptr};
    e = cudaGetSymbolAddress(reinterpret_cast<void **>(&s.scratch), g_gemm_scratch);
    if (e == cudaSuccess) e = cudaGetSymbolAddress(reinterpret_cast<void **>(&s.status), g_gemm_status);
    if (e != cudaSuccess) return e;
    if (!s.scratch || !s.status) return cudaErrorInvalidSymbol;
    g_syms.push_back(s);
    *out = s;
    return cudaSuccess;
}

}  // namespace

uint32_t *f3dc::gemm_status_word()
{
    DeviceSyms s;
    return device_syms(&s) == cudaSuccess ? s.status : nullptr;
}

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

    // the launch decisions of f3dc_gemm, so the result is the same bit for bit
    const int bn = N % 256 == 0 ? 256 : (N % 128 == 0 ? 128 : 64);
    const int m_tiles = (M + kTileRows - 1) / kTileRows;
    const int tiles = m_tiles * (N / bn);
    const int grid = gemm_grid(tiles, sms);
    const int splits = gemm_split_count(tiles, grid, K / 64, sms, true);
    const bool pair = bn == 256 && K % 128 == 0 && splits == 1;
    const size_t need = splits > 1 ? gemm_ws_bytes(bn, tiles * splits) : 0;
    if (need > kPartialBytes)
        return fail(F3DC_ERR_INVALID_ARG, "this problem needs " + std::to_string(need) +
                                              " bytes of split-K scratch; the static scratch holds " +
                                              std::to_string(kPartialBytes) + " (use f3dc_gemm)");

    DeviceSyms syms;
    e = device_syms(&syms);
    if (e != cudaSuccess) return fail(F3DC_ERR_CUDA, std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e));

    CUtensorMap ta, tb;
    if (!make_tmap_bf16(&ta, A, M, K, K, 128, 64) ||
        !make_tmap_bf16(&tb, B, N, K, K, pair ? kGemmPairBBox : gemm_b_box_rows(bn), 64))
        return fail(F3DC_ERR_INVALID_ARG, "cuTensorMapEncodeTiled rejected A or B (alignment?)");
    GemmParams p;
    memset(&p, 0, sizeof(p));
    p.M = M;
    p.N = N;
    p.K = K;
    p.m_tiles = m_tiles;
    p.out = out;
    p.ldo = N;
    p.bias = reinterpret_cast<const bf16 *>(bias);
    p.gate = gate;
    p.err = syms.status;
    const int epi = epilogue == F3DC_EPI_BIAS ? kEpiBias : (epilogue == F3DC_EPI_GELU ? kEpiGelu : kEpiResid);
    cudaStream_t s = (cudaStream_t)stream;
    if (pair) {
        p.narrow_below = sms / 2;
        e = launch_gemm_pair(&ta, &tb, p, epi, (m_tiles + 1) / 2 * (N / 128), s);
        if (e != cudaSuccess) return fail(F3DC_ERR_CUDA, std::string("launch: ") + cudaGetErrorString(e));
        return F3DC_OK;
    }
    p.ws = reinterpret_cast<float *>(syms.scratch);
    p.counters = reinterpret_cast<int32_t *>(syms.scratch + kPartialBytes);
    p.ws_units = sms;
    // the array keeps whatever the previous call left (a call whose split
    // wait ran out leaves its counters raised): the arrival counters must
    // start at zero; the partial tiles are always written before they are read
    e = cudaMemsetAsync(p.counters, 0, kCounterBytes, s);
    if (e != cudaSuccess) return fail(F3DC_ERR_CUDA, std::string("clearing counters: ") + cudaGetErrorString(e));
    e = launch_gemm(&ta, &tb, p, epi, bn, grid, s);
    if (e != cudaSuccess) return fail(F3DC_ERR_CUDA, std::string("launch: ") + cudaGetErrorString(e));
    return F3DC_OK;
}

extern "C" f3dc_status f3dc_gemm_status(uint32_t *status_out)
{
    if (!status_out) return fail(F3DC_ERR_INVALID_ARG, "null status_out");
    DeviceSyms syms;
    cudaError_t e = device_syms(&syms);
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    uint32_t v = 0;
    if (e == cudaSuccess) e = cudaMemcpy(&v, syms.status, sizeof(v), cudaMemcpyDeviceToHost);
    if (e == cudaSuccess) e = cudaMemset(syms.status, 0, sizeof(v));
    if (e != cudaSuccess) return fail(F3DC_ERR_CUDA, std::string("reading the GEMM status: ") + cudaGetErrorString(e));
    *status_out = v;
    return F3DC_OK;
}
