// k_rows.cu -- bandwidth-bound row kernels of the cached step:
//   K2 gather + input embedding of the active tokens (Sec. 4.2 compaction)
//   K7 LayerNorm with adaLN modulation or affine parameters (Supp. Sec. F)
//   final layer (LN + adaLN + Linear W -> C)
//   K3 cache merge + Euler update + history write (Algorithm 1 step 3) with
//      the optional dynamic-voxel count of the stand-in decoder (Eq. 1)
//   K9 timestep embedding and the modulation GEMV of every block
// All row kernels are persistent grid-stride loops over rows of the packed
// active matrix whose row count is read from the device plan, so a step can
// be launched without the host knowing the active counts.
#include "common.cuh"
#include "kernels.h"

namespace f3dc {

namespace {

constexpr int kRowThreads = 256;  // 8 warps, one row per warp

F3DC_DEV float4 ld_f4(const float *p) { return *reinterpret_cast<const float4 *>(p); }
F3DC_DEV void st_f4(float *p, float4 v) { *reinterpret_cast<float4 *>(p) = v; }

F3DC_DEV void bf16x8_to_f32(uint4 u, float (&f)[8])
{
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        f[2 * j] = bf16_bits_to_f32(w[j] & 0xFFFFu);
        f[2 * j + 1] = bf16_bits_to_f32(w[j] >> 16);
    }
}

F3DC_DEV float bf16_at(const bf16 *p, size_t i)
{
    return bf16_bits_to_f32(reinterpret_cast<const uint16_t *>(p)[i]);
}

// ------------------------------------------------------------------ K2
// Work unit: 32 consecutive packed rows (a quarter of a 128-row tile, so one
// sample).  Threads 0..31 resolve the unit's rows to tokens (tile -> sample
// -> active index -> latent) once and stage index and latent in shared
// memory; then every thread owns one float4 of columns (its 4 x 8 input
// weights and 4 biases held in registers for the whole kernel) and streams
// the rows, issuing the position-embedding loads of 8 rows before using any.
// Per column: acc = b_n, acc = fma(S_c, W_nc, acc) for c = 0..7, x = pos + acc.
constexpr int kGatherUnit = 32;
template <int NV>
struct GatherCfg {
    static constexpr int kT = 32 * NV;                        // threads per row
    static constexpr int kThreads = kT < 256 ? 256 : kT;
    static constexpr int kRPI = kThreads / kT;                 // rows per pass
    static constexpr int kU = kRPI >= 8 ? 1 : (NV == 16 ? 4 : 8 / kRPI);  // passes unrolled
};

template <int NV>
__global__ void __launch_bounds__(GatherCfg<NV>::kThreads, GatherCfg<NV>::kThreads >= 512 ? 1 : 2)
    k_gather_embed(const float *S, int N, const int32_t *active_idx, const Plan *plan, const int32_t *tile_sample,
                   const bf16 *in_w, const bf16 *in_b, const float *pos, float *x, int cfg_B, uint32_t *err)
{
    using Cfg = GatherCfg<NV>;
    constexpr int W = 128 * NV;
    __shared__ int s_idx[kGatherUnit];
    __shared__ float4 s_lat[kGatherUnit][2];
    const int t = threadIdx.x, q = t % Cfg::kT, rsub = t / Cfg::kT;
    // this thread's columns 4q .. 4q+3: weights and biases
    float wv[4][8], bv[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        bf16x8_to_f32(__ldg(reinterpret_cast<const uint4 *>(in_w) + 4 * q + u), wv[u]);
        bv[u] = bf16_at(in_b, 4 * q + u);
    }
    griddep_launch();
    griddep_wait();
    const int units = plan->m_rows / kGatherUnit;
    for (int unit = blockIdx.x; unit < units; unit += gridDim.x) {
        const int r0 = unit * kGatherUnit;
        if (t < kGatherUnit) {
            const int b = tile_sample[r0 / kTileRows];
            const int sb = cfg_B > 0 && b >= cfg_B ? b - cfg_B : b;  // guided step: unguided copy of sb
            const int j = r0 + t - plan->row_off[b];
            int i = -1;
            if (j < plan->n_active[b]) {
                i = active_idx[(size_t)sb * N + j];
                if ((unsigned)i >= (unsigned)N) {
                    raise_error(err, kDevBadIndex);
                    i = -1;
                }
            }
            s_idx[t] = i;
            if (i >= 0) {
                const float *Si = S + ((size_t)sb * N + i) * kChannels;
                s_lat[t][0] = ld_f4(Si);
                s_lat[t][1] = ld_f4(Si + 4);
            }
        }
        __syncthreads();
#pragma unroll 1
        for (int p0 = 0; p0 < kGatherUnit; p0 += Cfg::kRPI * Cfg::kU) {
            float4 pe[Cfg::kU];
#pragma unroll
            for (int u = 0; u < Cfg::kU; ++u) {
                const int i = s_idx[p0 + u * Cfg::kRPI + rsub];
                pe[u] = i >= 0 ? __ldg(reinterpret_cast<const float4 *>(pos + (size_t)i * W) + q)
                               : make_float4(0.f, 0.f, 0.f, 0.f);
            }
#pragma unroll
            for (int u = 0; u < Cfg::kU; ++u) {
                const int rr = p0 + u * Cfg::kRPI + rsub;
                float4 o = make_float4(0.f, 0.f, 0.f, 0.f);
                if (s_idx[rr] >= 0) {  // padding rows stay zero: every downstream value finite
                    const float4 l0 = s_lat[rr][0], l1 = s_lat[rr][1];
                    const float sl[8] = {l0.x, l0.y, l0.z, l0.w, l1.x, l1.y, l1.z, l1.w};
                    float acc[4];
#pragma unroll
                    for (int c4 = 0; c4 < 4; ++c4) {
                        acc[c4] = bv[c4];
#pragma unroll
                        for (int c = 0; c < 8; ++c) acc[c4] = fmaf(sl[c], wv[c4][c], acc[c4]);
                    }
                    o = make_float4(pe[u].x + acc[0], pe[u].y + acc[1], pe[u].z + acc[2], pe[u].w + acc[3]);
                }
                st_f4(x + (size_t)(r0 + rr) * W + 4 * q, o);
            }
        }
        __syncthreads();
    }
}

// ------------------------------------------------------------------ K7
// One warp per row, lane l owning float4 columns q * 32 + l.  The per-column
// modulation (adaLN scale / shift, or LN gain / bias) is staged in shared
// memory once per CTA while the first row is in flight, and each warp loads
// its next row while it normalises the current one, so the kernel streams
// rows at a persistent grid of two CTAs per SM instead of paying two
// dependent memory round trips per row.
template <int NV>
__global__ void __launch_bounds__(kRowThreads, 2) k_layernorm(const float *x, int W, const Plan *plan, int mode,
                                                              const float *shift, const float *scale,
                                                              const bf16 *g, const bf16 *bb, bf16 *out)
{
    griddep_launch();
    griddep_wait();
    __shared__ float4 s_mul[NV * 32], s_add[NV * 32];  // y = xhat * mul + add per column
    const int m_rows = plan->m_rows;
    const int lane = threadIdx.x & 31, wpb = blockDim.x >> 5;
    const int stride = gridDim.x * wpb;
    int r = blockIdx.x * wpb + (threadIdx.x >> 5);
    if (blockIdx.x * wpb >= m_rows) return;  // the whole CTA is idle
    // the first row's loads are issued before the modulation is staged, so
    // the two memory round trips overlap
    float4 v[NV];
    if (r < m_rows) {
#pragma unroll
        for (int q = 0; q < NV; ++q) v[q] = ld_f4(x + (size_t)r * W + 4 * (q * 32 + lane));
    }
    for (int c4 = threadIdx.x; c4 < NV * 32; c4 += blockDim.x) {
        const int n0 = 4 * c4;
        if (mode == 0) {
            const float4 sc = ld_f4(scale + n0);
            s_mul[c4] = make_float4(1.f + sc.x, 1.f + sc.y, 1.f + sc.z, 1.f + sc.w);
            s_add[c4] = ld_f4(shift + n0);
        } else {
            const uint2 gw = __ldg(reinterpret_cast<const uint2 *>(reinterpret_cast<const uint16_t *>(g) + n0));
            const uint2 bw = __ldg(reinterpret_cast<const uint2 *>(reinterpret_cast<const uint16_t *>(bb) + n0));
            s_mul[c4] = make_float4(bf16_bits_to_f32(gw.x & 0xFFFFu), bf16_bits_to_f32(gw.x >> 16),
                                    bf16_bits_to_f32(gw.y & 0xFFFFu), bf16_bits_to_f32(gw.y >> 16));
            s_add[c4] = make_float4(bf16_bits_to_f32(bw.x & 0xFFFFu), bf16_bits_to_f32(bw.x >> 16),
                                    bf16_bits_to_f32(bw.y & 0xFFFFu), bf16_bits_to_f32(bw.y >> 16));
        }
    }
    __syncthreads();
    if (r >= m_rows) return;
    for (;;) {
        const int rn = r + stride;
        float4 vn[NV];
        if (rn < m_rows) {
#pragma unroll
            for (int q = 0; q < NV; ++q) vn[q] = ld_f4(x + (size_t)rn * W + 4 * (q * 32 + lane));
        }
        float mean, rstd;
        ln_row_stats<NV>(v, W, mean, rstd);
        uint16_t *orow = reinterpret_cast<uint16_t *>(out) + (size_t)r * W;
#pragma unroll
        for (int q = 0; q < NV; ++q) {
            const int n0 = 4 * (q * 32 + lane);
            *reinterpret_cast<uint2 *>(orow + n0) = ln_out4(v[q], mean, rstd, s_mul[q * 32 + lane], s_add[q * 32 + lane]);
        }
        if (rn >= m_rows) break;
        r = rn;
#pragma unroll
        for (int q = 0; q < NV; ++q) v[q] = vn[q];
    }
}

template <int NV>
__global__ void __launch_bounds__(kRowThreads) k_final_layer(const float *x, int W, const Plan *plan,
                                                             const float *shift, const float *scale,
                                                             const bf16 *out_w, const bf16 *out_b, float *v_active)
{
    griddep_launch();
    griddep_wait();
    const int m_rows = plan->m_rows;
    const int lane = threadIdx.x & 31, wpb = blockDim.x >> 5;
    for (int r = blockIdx.x * wpb + (threadIdx.x >> 5); r < m_rows; r += gridDim.x * wpb) {
        const float *xr = x + (size_t)r * W;
        float4 v[NV];
#pragma unroll
        for (int q = 0; q < NV; ++q) v[q] = ld_f4(xr + 4 * (q * 32 + lane));
        float mean, rstd;
        ln_row_stats<NV>(v, W, mean, rstd);
        float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int q = 0; q < NV; ++q) {
            const int n0 = 4 * (q * 32 + lane);
            const float4 sc = ld_f4(scale + n0), sh = ld_f4(shift + n0);
            const float y[4] = {(v[q].x - mean) * rstd * (1.f + sc.x) + sh.x,
                                (v[q].y - mean) * rstd * (1.f + sc.y) + sh.y,
                                (v[q].z - mean) * rstd * (1.f + sc.z) + sh.z,
                                (v[q].w - mean) * rstd * (1.f + sc.w) + sh.w};
#pragma unroll
            for (int c = 0; c < 8; ++c) {
                const uint2 wp = __ldg(reinterpret_cast<const uint2 *>(
                    reinterpret_cast<const uint16_t *>(out_w) + (size_t)c * W + n0));
                acc[c] += y[0] * bf16_bits_to_f32(wp.x & 0xFFFFu) + y[1] * bf16_bits_to_f32(wp.x >> 16) +
                          y[2] * bf16_bits_to_f32(wp.y & 0xFFFFu) + y[3] * bf16_bits_to_f32(wp.y >> 16);
            }
        }
#pragma unroll
        for (int c = 0; c < 8; ++c) acc[c] = warp_sum(acc[c]);
        if (lane == 0) {
            float o[8];
#pragma unroll
            for (int c = 0; c < 8; ++c) o[c] = acc[c] + bf16_at(out_b, c);
            st_f4(v_active + (size_t)r * 8, make_float4(o[0], o[1], o[2], o[3]));
            st_f4(v_active + (size_t)r * 8 + 4, make_float4(o[4], o[5], o[6], o[7]));
        }
    }
}

// ------------------------------------------------------------------ K3
// Two tokens per thread (256 apart, so a warp's 32 consecutive tokens stay
// in one sample): the latent, the token's packed row and its cached
// velocity are loaded for both tokens at once, and only an active token's
// fresh velocity waits for its row index -- one dependent round trip
// instead of two.
constexpr int kMergeThreads = 256;
constexpr int kMergeTok = 2;
constexpr int kMaxG = 512;

__global__ void __launch_bounds__(kMergeThreads) k_merge_euler(const MergeArgs a)
{
    griddep_launch();
    griddep_wait();
    __shared__ float dec[8 * kMaxG];
    const bool count = a.dyn != nullptr;
    if (count) {
        for (int q = threadIdx.x; q < 8 * a.G; q += blockDim.x)
            dec[q] = bf16_bits_to_f32(a.dec_w[q]);
        __syncthreads();
    }
    const size_t total = (size_t)a.B * a.N;
    const size_t tok0 = (size_t)blockIdx.x * (kMergeThreads * kMergeTok) + threadIdx.x;
    float so[kMergeTok][8];
    int row[kMergeTok];
    uint4 pv[kMergeTok];
#pragma unroll
    for (int u = 0; u < kMergeTok; ++u) {
        const size_t tok = tok0 + (size_t)u * kMergeThreads;
        row[u] = -1;
        if (tok < total) {
            const float4 s0 = ld_f4(a.S + tok * 8), s1 = ld_f4(a.S + tok * 8 + 4);
            so[u][0] = s0.x; so[u][1] = s0.y; so[u][2] = s0.z; so[u][3] = s0.w;
            so[u][4] = s1.x; so[u][5] = s1.y; so[u][6] = s1.z; so[u][7] = s1.w;
            row[u] = a.row_of_token[tok];
            pv[u] = *reinterpret_cast<const uint4 *>(a.v_prev1 + tok * 8);
        }
    }
    const size_t half = a.cfg_s != 0.0f ? (size_t)(a.plan->m_rows / 2) : 0;
    float va[kMergeTok][8], vu[kMergeTok][8];
    bool bad[kMergeTok];
#pragma unroll
    for (int u = 0; u < kMergeTok; ++u) {
        const size_t tok = tok0 + (size_t)u * kMergeThreads;
        bad[u] = false;
        if (tok < total && row[u] >= 0) {
            const size_t ru = a.cfg_s != 0.0f ? (size_t)row[u] + half : 0;
            if (row[u] >= a.max_rows || ru >= (size_t)a.max_rows) {
                bad[u] = true;
            } else {
                const float4 v0 = ld_f4(a.v_active + (size_t)row[u] * 8), v1 = ld_f4(a.v_active + (size_t)row[u] * 8 + 4);
                va[u][0] = v0.x; va[u][1] = v0.y; va[u][2] = v0.z; va[u][3] = v0.w;
                va[u][4] = v1.x; va[u][5] = v1.y; va[u][6] = v1.z; va[u][7] = v1.w;
                if (a.cfg_s != 0.0f) {
                    const float4 u0 = ld_f4(a.v_active + ru * 8), u1 = ld_f4(a.v_active + ru * 8 + 4);
                    vu[u][0] = u0.x; vu[u][1] = u0.y; vu[u][2] = u0.z; vu[u][3] = u0.w;
                    vu[u][4] = u1.x; vu[u][5] = u1.y; vu[u][6] = u1.z; vu[u][7] = u1.w;
                }
            }
        }
    }
#pragma unroll
    for (int u = 0; u < kMergeTok; ++u) {
        const size_t tok = tok0 + (size_t)u * kMergeThreads;
        const bool valid = tok < total;
        int flips = 0;
        int b = 0;
        if (valid) {
            b = (int)(tok / a.N);
            uint32_t vb[8];
            if (row[u] >= 0) {
                if (bad[u]) {
                    raise_error(a.err, kDevBadIndex);
#pragma unroll
                    for (int c = 0; c < 8; ++c) vb[c] = 0;
                } else {
                    float v[8];
#pragma unroll
                    for (int c = 0; c < 8; ++c) v[c] = va[u][c];
                    if (a.cfg_s != 0.0f) {
                        // guided step: v_u + s (v_c - v_u), the unguided copy's row
                        // half the plan further (subtract, multiply, add)
#pragma unroll
                        for (int c = 0; c < 8; ++c)
                            v[c] = __fadd_rn(vu[u][c], __fmul_rn(a.cfg_s, __fsub_rn(v[c], vu[u][c])));
                    }
#pragma unroll
                    for (int c = 0; c < 8; ++c) vb[c] = f32_to_bf16_bits(v[c]);
                }
            } else {  // cached token: reuse the stored velocity bit for bit
                const uint32_t pw[4] = {pv[u].x, pv[u].y, pv[u].z, pv[u].w};
#pragma unroll
                for (int c = 0; c < 8; ++c) vb[c] = (pw[c >> 1] >> ((c & 1) * 16)) & 0xFFFFu;
            }
            float sn[8];
#pragma unroll
            for (int c = 0; c < 8; ++c) sn[c] = __fsub_rn(so[u][c], __fmul_rn(a.dt, bf16_bits_to_f32(vb[c])));
            st_f4(a.S + tok * 8, make_float4(sn[0], sn[1], sn[2], sn[3]));
            st_f4(a.S + tok * 8 + 4, make_float4(sn[4], sn[5], sn[6], sn[7]));
            uint4 vo;
            vo.x = vb[0] | (vb[1] << 16);
            vo.y = vb[2] | (vb[3] << 16);
            vo.z = vb[4] | (vb[5] << 16);
            vo.w = vb[6] | (vb[7] << 16);
            *reinterpret_cast<uint4 *>(a.v_out + tok * 8) = vo;
            if (count) {
                for (int j = 0; j < a.G; ++j) {
                    float lo = 0.0f, ln = 0.0f;
#pragma unroll
                    for (int c = 0; c < 8; ++c) {
                        lo = __fadd_rn(lo, __fmul_rn(so[u][c], dec[c * a.G + j]));
                        ln = __fadd_rn(ln, __fmul_rn(sn[c], dec[c * a.G + j]));
                    }
                    flips += (lo > 0.0f) != (ln > 0.0f);
                }
            }
        }
        if (count) {
            // N % 32 == 0 is enforced at create, so a warp's 32 consecutive
            // tokens never span two samples
            int f = flips;
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) f += __shfl_xor_sync(0xffffffffu, f, o);
            if ((threadIdx.x & 31) == 0 && valid && f)
                atomicAdd(reinterpret_cast<unsigned long long *>(a.dyn + b), (unsigned long long)f);
        }
    }
}

__global__ void k_scatter_rows(const float *v_active, const Plan *plan, int N, float *v_out)
{
    griddep_launch();
    griddep_wait();
    const int b = blockIdx.y;
    const int na = plan->n_active[b], off = plan->row_off[b];
    for (int j = blockIdx.x * blockDim.x + threadIdx.x; j < na; j += gridDim.x * blockDim.x) {
        const float *src = v_active + (size_t)(off + j) * 8;
        float *dst = v_out + ((size_t)b * N + j) * 8;
        st_f4(dst, ld_f4(src));
        st_f4(dst + 4, ld_f4(src + 4));
    }
}

// ------------------------------------------------------------------ K9
F3DC_DEV void time_freq(float t, float *freq)
{
    const int f = threadIdx.x;  // 128 threads
    const float w = expf(-9.210340371976184f * (float)f / 128.0f);  // ln(10000)
    const float arg = 1000.0f * t * w;
    freq[f] = cosf(arg);
    freq[128 + f] = sinf(arg);
}

__global__ void k_time_freq(float t, float *freq)
{
    griddep_launch();
    griddep_wait();
    time_freq(t, freq);
}

// one block per time: freq[v] = sinusoid of t[v]
__global__ void k_time_freq_many(const float *t, float *freq)
{
    griddep_launch();
    griddep_wait();
    time_freq(t[blockIdx.x], freq + (size_t)blockIdx.x * 256);
}

F3DC_DEV float silu(float v) { return v / (1.0f + expf(-v)); }

constexpr int kGemvThreads = 512;
constexpr int kGemvMaxK = 4096;
constexpr int kGemvXs = 8192;  // staged input floats: NV * K <= 8192

// One warp per pair of weight rows.  Lane l owns the 4-wide column groups
// g = l, l + 32, ... (k = 4g .. 4g + 3): it loads them as 8-byte pieces of
// both rows -- eight pieces per row in flight for one or two vectors, fewer
// for more -- and reads the matching inputs as one float4 each, so a
// warp's shared-memory reads are consecutive (conflict-free).  NV vectors (x [NV, K] -> y [NV, rows], row
// strides K and rows) share each weight load; every output is summed in the
// same order for any NV.  Two CTAs of 16 warps per SM.
template <int NV>
__global__ void __launch_bounds__(kGemvThreads, 2) k_gemv(const float *x, int K, const bf16 *w, const bf16 *bias,
                                                          float *y, int rows, int silu_in, int silu_out)
{
    griddep_launch();
    griddep_wait();
    __shared__ float4 xs4[kGemvXs / 4];  // NV * K floats
    float *xs = reinterpret_cast<float *>(xs4);
    for (int k = threadIdx.x; k < NV * K; k += blockDim.x) xs[k] = silu_in ? silu(x[k]) : x[k];
    __syncthreads();
    const int lane = threadIdx.x & 31, wpb = blockDim.x >> 5;
    const int groups = K / 4;  // 4 bf16 (one uint2) per lane per step
    const uint2 *W2 = reinterpret_cast<const uint2 *>(w);
    for (int r = (blockIdx.x * wpb + (threadIdx.x >> 5)) * 2; r < rows; r += gridDim.x * wpb * 2) {
        const bool two = r + 1 < rows;
        float acc0[NV], acc1[NV];
#pragma unroll
        for (int v = 0; v < NV; ++v) acc0[v] = acc1[v] = 0.f;
        constexpr int kDepth = NV >= 8 ? 2 : (NV >= 4 ? 4 : 8);  // pieces per row in flight
        for (int g0 = lane; g0 < groups; g0 += kDepth * 32) {
            uint2 u0[kDepth], u1[kDepth];
#pragma unroll
            for (int c = 0; c < kDepth; ++c) {
                const int g = g0 + c * 32;
                u0[c] = g < groups ? __ldg(W2 + (size_t)r * (K / 4) + g) : make_uint2(0, 0);
                u1[c] = two && g < groups ? __ldg(W2 + (size_t)(r + 1) * (K / 4) + g) : make_uint2(0, 0);
            }
#pragma unroll
            for (int c = 0; c < kDepth; ++c) {
                const int g = g0 + c * 32;
                if (g >= groups) break;
                const float f0[4] = {bf16_bits_to_f32(u0[c].x & 0xFFFFu), bf16_bits_to_f32(u0[c].x >> 16),
                                     bf16_bits_to_f32(u0[c].y & 0xFFFFu), bf16_bits_to_f32(u0[c].y >> 16)};
                const float f1[4] = {bf16_bits_to_f32(u1[c].x & 0xFFFFu), bf16_bits_to_f32(u1[c].x >> 16),
                                     bf16_bits_to_f32(u1[c].y & 0xFFFFu), bf16_bits_to_f32(u1[c].y >> 16)};
#pragma unroll
                for (int v = 0; v < NV; ++v) {
                    const float4 xv = xs4[(v * K) / 4 + g];
                    const float xa[4] = {xv.x, xv.y, xv.z, xv.w};
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        acc0[v] = fmaf(f0[j], xa[j], acc0[v]);
                        acc1[v] = fmaf(f1[j], xa[j], acc1[v]);
                    }
                }
            }
        }
#pragma unroll
        for (int v = 0; v < NV; ++v) {
            const float s0 = warp_sum(acc0[v]), s1 = warp_sum(acc1[v]);
            if (lane == 0) {
                float v0 = s0 + (bias ? bf16_at(bias, r) : 0.f);
                y[(size_t)v * rows + r] = silu_out ? silu(v0) : v0;
                if (two) {
                    float v1 = s1 + (bias ? bf16_at(bias, r + 1) : 0.f);
                    y[(size_t)v * rows + r + 1] = silu_out ? silu(v1) : v1;
                }
            }
        }
    }
}

int row_grid(int num_sms, int max_rows)
{
    const int wpb = kRowThreads / 32;
    int g = num_sms * 4;
    const int need = (max_rows + wpb - 1) / wpb;
    return need < g ? (need > 0 ? need : 1) : g;
}

}  // namespace

template <int NV>
void launch_gather_nv(const float *S, int N, const int32_t *active_idx, const Plan *plan, const int32_t *tile_sample,
                      const bf16 *in_w, const bf16 *in_b, const float *pos, float *x, int max_rows, int num_sms,
                      int cfg_B, uint32_t *err, cudaStream_t s)
{
    const int units = max_rows / kGatherUnit;
    const int grid = units < 2 * num_sms ? (units > 0 ? units : 1) : 2 * num_sms;
    launch_k(k_gather_embed<NV>, dim3(grid), dim3(GatherCfg<NV>::kThreads), 0, s, S, N, active_idx, plan, tile_sample,
             in_w, in_b, pos, x, cfg_B, err);
}

cudaError_t launch_gather_embed(const float *S, int N, int W, const int32_t *active_idx, const Plan *plan,
                                const int32_t *tile_sample, const bf16 *in_w, const bf16 *in_b,
                                const float *pos, float *x, int max_rows, int num_sms, int cfg_B,
                                uint32_t *err, cudaStream_t s)
{
#define F3DC_GATHER(NV)                                                                                        \
    launch_gather_nv<NV>(S, N, active_idx, plan, tile_sample, in_w, in_b, pos, x, max_rows, num_sms, cfg_B, err, s)
    switch (W / 128) {
    case 1: F3DC_GATHER(1); break;
    case 2: F3DC_GATHER(2); break;
    case 4: F3DC_GATHER(4); break;
    case 8: F3DC_GATHER(8); break;
    case 16: F3DC_GATHER(16); break;
    default: return cudaErrorInvalidValue;
    }
#undef F3DC_GATHER
    return cudaGetLastError();
}

__global__ void k_broadcast_row(bf16 *dst, size_t ld, const bf16 *src, int rows, int cols)
{
    griddep_launch();
    griddep_wait();
    const int c8 = cols / 8;
    for (size_t q = (size_t)blockIdx.x * blockDim.x + threadIdx.x; q < (size_t)rows * c8;
         q += (size_t)gridDim.x * blockDim.x) {
        const size_t r = q / c8, c = q - r * c8;
        reinterpret_cast<uint4 *>(dst + r * ld)[c] = reinterpret_cast<const uint4 *>(src)[c];
    }
}

cudaError_t launch_broadcast_row(bf16 *dst, size_t ld, const bf16 *src, int rows, int cols, cudaStream_t s)
{
    if (cols % 8 != 0 || ld % 8 != 0 || rows < 0) return cudaErrorInvalidValue;
    if (rows == 0) return cudaSuccess;
    const size_t total = (size_t)rows * (cols / 8);
    const int grid = (int)((total + 255) / 256 < 1024 ? (total + 255) / 256 : 1024);
    launch_k(k_broadcast_row, dim3(grid), dim3(256), 0, s, dst, ld, src, rows, cols);
    return cudaGetLastError();
}

cudaError_t launch_layernorm(const float *x, int W, const Plan *plan, int mode, const float *shift,
                             const float *scale, const bf16 *g, const bf16 *b, bf16 *out, int max_rows,
                             int num_sms, cudaStream_t s)
{
    const int need = (max_rows + kRowThreads / 32 - 1) / (kRowThreads / 32);
    const int grid = need < 2 * num_sms ? (need > 0 ? need : 1) : 2 * num_sms;
    switch (W / 128) {
    case 1: launch_k(k_layernorm<1>, dim3(grid), dim3(kRowThreads), 0, s, x, W, plan, mode, shift, scale, g, b, out); break;
    case 2: launch_k(k_layernorm<2>, dim3(grid), dim3(kRowThreads), 0, s, x, W, plan, mode, shift, scale, g, b, out); break;
    case 4: launch_k(k_layernorm<4>, dim3(grid), dim3(kRowThreads), 0, s, x, W, plan, mode, shift, scale, g, b, out); break;
    case 8: launch_k(k_layernorm<8>, dim3(grid), dim3(kRowThreads), 0, s, x, W, plan, mode, shift, scale, g, b, out); break;
    case 16: launch_k(k_layernorm<16>, dim3(grid), dim3(kRowThreads), 0, s, x, W, plan, mode, shift, scale, g, b, out); break;
    default: return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

cudaError_t launch_final_layer(const float *x, int W, const Plan *plan, const float *shift,
                               const float *scale, const bf16 *out_w, const bf16 *out_b, float *v_active,
                               int max_rows, int num_sms, cudaStream_t s)
{
    const int grid = row_grid(num_sms, max_rows);
    switch (W / 128) {
    case 1: launch_k(k_final_layer<1>, dim3(grid), dim3(kRowThreads), 0, s, x, W, plan, shift, scale, out_w, out_b, v_active); break;
    case 2: launch_k(k_final_layer<2>, dim3(grid), dim3(kRowThreads), 0, s, x, W, plan, shift, scale, out_w, out_b, v_active); break;
    case 4: launch_k(k_final_layer<4>, dim3(grid), dim3(kRowThreads), 0, s, x, W, plan, shift, scale, out_w, out_b, v_active); break;
    case 8: launch_k(k_final_layer<8>, dim3(grid), dim3(kRowThreads), 0, s, x, W, plan, shift, scale, out_w, out_b, v_active); break;
    case 16: launch_k(k_final_layer<16>, dim3(grid), dim3(kRowThreads), 0, s, x, W, plan, shift, scale, out_w, out_b, v_active); break;
    default: return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

cudaError_t launch_merge_euler(const MergeArgs &a, cudaStream_t s)
{
    if (a.dyn && (a.G > kMaxG || a.N % 32 != 0)) return cudaErrorInvalidValue;
    const size_t total = (size_t)a.B * a.N;
    const int grid = (int)((total + kMergeThreads * kMergeTok - 1) / (kMergeThreads * kMergeTok));
    launch_k(k_merge_euler, dim3(grid), dim3(kMergeThreads), 0, s, a);
    return cudaGetLastError();
}

cudaError_t launch_scatter_rows(const float *v_active, const Plan *plan, int B, int N, float *v_out,
                                cudaStream_t s)
{
    dim3 grid((N + 255) / 256, B);
    launch_k(k_scatter_rows, dim3(grid), dim3(256), 0, s, v_active, plan, N, v_out);
    return cudaGetLastError();
}

cudaError_t launch_time_freq(float t, float *freq, cudaStream_t s)
{
    launch_k(k_time_freq, dim3(1), dim3(128), 0, s, t, freq);
    return cudaGetLastError();
}

cudaError_t launch_time_freq_many(const float *t, int n, float *freq, cudaStream_t s)
{
    if (n < 1) return cudaErrorInvalidValue;
    launch_k(k_time_freq_many, dim3(n), dim3(128), 0, s, t, freq);
    return cudaGetLastError();
}

cudaError_t launch_gemv(const float *x, int K, const bf16 *w, const bf16 *b, float *y, int rows, int silu_in,
                        int silu_out, int num_sms, cudaStream_t s)
{
    return launch_gemv_many(x, 1, K, w, b, y, rows, silu_in, silu_out, num_sms, s);
}

// vectors per launch: 8, 4, 2 or 1, as many as the shared staging holds
static int gemv_group(int left, int K)
{
    return left >= 8 && 8 * K <= kGemvXs ? 8 : (left >= 4 && 4 * K <= kGemvXs ? 4 : (left >= 2 && 2 * K <= kGemvXs ? 2 : 1));
}

int gemv_many_kernels(int nv, int K)
{
    int n = 0;
    for (int v0 = 0; v0 < nv; v0 += gemv_group(nv - v0, K)) ++n;
    return n;
}

cudaError_t launch_gemv_many(const float *x, int nv, int K, const bf16 *w, const bf16 *b, float *y, int rows,
                             int silu_in, int silu_out, int num_sms, cudaStream_t s)
{
    if (K % 8 != 0 || K > kGemvMaxK || nv < 1) return cudaErrorInvalidValue;
    const int wpb = kGemvThreads / 32;
    int grid = (rows + 2 * wpb - 1) / (2 * wpb);
    if (grid > num_sms * 2) grid = num_sms * 2;
    // vectors in groups whose inputs fit the shared staging (8, 4, 2 or 1)
    for (int v0 = 0; v0 < nv;) {
        const int g = gemv_group(nv - v0, K);
        const float *xg = x + (size_t)v0 * K;
        float *yg = y + (size_t)v0 * rows;
        switch (g) {
        case 8: launch_k(k_gemv<8>, dim3(grid), dim3(kGemvThreads), 0, s, xg, K, w, b, yg, rows, silu_in, silu_out); break;
        case 4: launch_k(k_gemv<4>, dim3(grid), dim3(kGemvThreads), 0, s, xg, K, w, b, yg, rows, silu_in, silu_out); break;
        case 2: launch_k(k_gemv<2>, dim3(grid), dim3(kGemvThreads), 0, s, xg, K, w, b, yg, rows, silu_in, silu_out); break;
        default: launch_k(k_gemv<1>, dim3(grid), dim3(kGemvThreads), 0, s, xg, K, w, b, yg, rows, silu_in, silu_out); break;
        }
        v0 += g;
    }
    return cudaGetLastError();
}

}  // namespace f3dc
