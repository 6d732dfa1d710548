// k_gemm.cu -- K4: the dense projections of the flow transformer (QKV,
// attention output, cross-attention Q / output, MLP fc1 / fc2, condition
// K / V; Supp. Sec. F) on 5th-generation tensor cores.
//
// out[m, n] = epilogue( sum_k A[m, k] B[n, k] ),  A = activations [M, K]
// bf16, B = weights [N, K] bf16 (nn.Linear layout), fp32 accumulation.
//
// Two kernels.  The transformer's step GEMMs (N a multiple of 256) run on
// k_gemm_pair, a CTA-pair (cta_group::2) version described with it below.
// k_gemm, the single-CTA kernel, serves the other widths and split K: a
// persistent warp-specialised kernel, one CTA per SM (192 threads):
//   warp 0     TMA producer: 128x64 A and BNx64 B tiles, 128B-swizzled, into
//              a STAGES-deep shared-memory ring (mbarrier full / empty)
//   warp 1     TMEM allocator + single-thread tcgen05.mma issuer
//              (M=128, N=BN, K=16 per instruction), accumulating in TMEM;
//              two accumulator buffers so the epilogue of tile i overlaps
//              the MMAs of tile i+1
//   warps 2-5  epilogue: tcgen05.ld (thread = row), fused bias / GELU /
//              per-head RMSNorm / gated fp32 residual; each 128-row chunk
//              of 32 bf16 (or 16 fp32) columns is staged in 64B-swizzled
//              shared memory (three buffers) and written by one TMA tensor
//              store (residual: TMA fp32 reduce-add into x), so the output
//              leaves in whole rows instead of one 16-byte piece per thread
// Tiles are walked m-fastest so the CTAs in flight share weight tiles in L2.
// The tile count can come from device memory (the step's row plan), so the
// same launch serves any number of active tokens.
#include <stdio.h>

#include <atomic>

#include <cudaTypedefs.h>

#include "common.cuh"
#include "kernels.h"

namespace f3dc {

namespace {

constexpr int kGemmThreads = 192;
constexpr int kBK = 64;
constexpr int kAStage = 128 * kBK * 2;

// output staging: 128 rows x 64 bytes (32 bf16 or 16 fp32 columns)
constexpr int kOutChunkBytes = 128 * 64;
constexpr int kOutBufs = 3;

template <int BN>
struct GemmCfg {
    static constexpr int kBStage = BN * kBK * 2;
    static constexpr int kStages = BN == 256 ? 4 : (BN == 128 ? 6 : 8);
    static constexpr uint32_t kTmemCols = 2 * BN;
    static constexpr size_t kBarBytes = 256;
    static constexpr size_t kSmem =
        1024 + (size_t)kStages * (kAStage + kBStage) + (size_t)kOutBufs * kOutChunkBytes + kBarBytes;
};

F3DC_DEV bool mbar_wait_bounded(uint64_t *bar, uint32_t parity, uint64_t ns)
{
    const uint64_t t0 = globaltimer();
    while (!mbar_try_wait(bar, parity))
        if (globaltimer() - t0 > ns) return false;
    return true;
}

F3DC_DEV void load_bias32(const bf16 *bias, int col, float (&b)[32])
{
    if (!bias) {
#pragma unroll
        for (int j = 0; j < 32; ++j) b[j] = 0.f;
        return;
    }
    const uint4 *p = reinterpret_cast<const uint4 *>(bias + col);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const uint4 u = __ldg(p + q);
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            b[q * 8 + 2 * j] = bf16_bits_to_f32(w[j] & 0xFFFFu);
            b[q * 8 + 2 * j + 1] = bf16_bits_to_f32(w[j] >> 16);
        }
    }
}

// RMSNorm over groups of `dh` columns of a 32-column chunk pair.
F3DC_DEV void rms_scale(float *v, int n, const bf16 *g, int gcol)
{
    float ss = 0.f;
    for (int j = 0; j < n; ++j) ss += v[j] * v[j];
    const float rs = rsqrtf(ss / (float)n + 1e-6f);
    for (int j = 0; j < n; ++j)
        v[j] = v[j] * rs * bf16_bits_to_f32(reinterpret_cast<const uint16_t *>(g)[gcol + j]);
}

// Accumulator sources for the epilogue: 32 fp32 values of this thread's row
// at columns c0..c0+31 of the tile, from TMEM (the MMA's accumulator) or as
// the split-order sum of the split-K partial tiles in the workspace.
struct TmemSrc {
    uint32_t tbase;
    F3DC_DEV void operator()(int c0, float *v) const
    {
        uint32_t r[32];
        tmem_ld32(tbase + c0, r);
        tmem_wait_ld();
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
    }
};

template <int BN>
struct WsSrc {
    const float *ws;  // partials of split s of this tile: unit (s * tiles + tile), chunk-major
    int tile, tiles, splits, row;
    // A chunk's 32 columns of two splits are loaded at once (16 float4 loads
    // in flight per thread), then summed in split order from 0, so the
    // reduction costs one L2 latency per chunk and two splits
    F3DC_DEV void operator()(int c0, float *v) const
    {
        // chunk-major workspace (see the partial store): unit u = s * tiles + tile
        const size_t split_stride4 = (size_t)tiles * 128 * BN / 4;
        const float4 *base =
            reinterpret_cast<const float4 *>(ws + (((size_t)tile * (BN / 32) + c0 / 32) * 128 + row) * 32);
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] = 0.f;
#pragma unroll 1
        for (int s0 = 0; s0 < splits; s0 += 2) {
            float4 part[2][8];
#pragma unroll
            for (int u = 0; u < 2; ++u)
#pragma unroll
                for (int c4 = 0; c4 < 8; ++c4)
                    if (s0 + u < splits) part[u][c4] = __ldcg(base + (s0 + u) * split_stride4 + c4);
#pragma unroll
            for (int u = 0; u < 2; ++u)
                if (s0 + u < splits) {
#pragma unroll
                    for (int c4 = 0; c4 < 8; ++c4) {
                        v[4 * c4 + 0] += part[u][c4].x;
                        v[4 * c4 + 1] += part[u][c4].y;
                        v[4 * c4 + 2] += part[u][c4].z;
                        v[4 * c4 + 3] += part[u][c4].w;
                    }
                }
        }
    }
};

// Output staging shared by a group of four epilogue warps: a chunk is one
// 128-row box of 64-byte rows, 16-byte piece c of row r at 64 r + 16 (c ^
// ((r / 2) % 4)) (the TMA 64B swizzle), which spreads a warp's row-per-lane
// stores over all banks.  The box is written out by the group's issuer thread
// with a TMA store; before a buffer is reused nbufs chunks later its store
// has finished reading it.
struct OutStage {
    uint8_t *buf;             // nbufs x kOutChunkBytes
    const CUtensorMap *map;   // output tensor: bf16 [M, N] or fp32 [M, N] (RESID, reduce-add)
    int row;                  // this thread's row of the tile
    int ck;                   // chunks emitted so far by this group of four warps
    int nbufs = kOutBufs;     // staging buffers (>= 2)
    int bar = 3;              // named barrier of the four warps
    int issuer = 64;          // thread that issues the group's TMA stores
    F3DC_DEV uint8_t *slot() const { return buf + (ck % nbufs) * kOutChunkBytes; }
    F3DC_DEV void put16(int c, uint4 u) const
    {
        *reinterpret_cast<uint4 *>(slot() + row * 64 + ((c ^ ((row >> 1) & 3)) << 4)) = u;
    }
    // publish the chunk just written and send it to (x, y) of the output
    // (or of the tensor `to`, e.g. the split-K workspace).  After the
    // barrier the warps write the next chunk into the buffer of chunk
    // ck + 1 - nbufs, so the issuer first waits until that chunk's store has
    // read it (at most nbufs - 2 stores still reading).
    template <bool kReduce>
    F3DC_DEV void emit(int x, int y, const CUtensorMap *to = nullptr)
    {
        fence_proxy_async_smem();
        if ((int)threadIdx.x == issuer) {
            if (nbufs == 2)
                bulk_wait_read<0>();
            else
                bulk_wait_read<1>();
        }
        asm volatile("bar.sync %0, 128;" ::"r"(bar) : "memory");
        if ((int)threadIdx.x == issuer) {
            const CUtensorMap *m = to ? to : map;
            if (kReduce)
                tma_reduce_add_2d(m, slot(), x, y);
            else
                tma_store_2d(m, slot(), x, y);
            bulk_commit();
        }
        ++ck;
    }
};

F3DC_DEV void put_bf16x32(OutStage &o, const float *v)
{
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        uint4 u;
        u.x = pack_bf16x2(v[q * 8 + 0], v[q * 8 + 1]);
        u.y = pack_bf16x2(v[q * 8 + 2], v[q * 8 + 3]);
        u.z = pack_bf16x2(v[q * 8 + 4], v[q * 8 + 5]);
        u.w = pack_bf16x2(v[q * 8 + 6], v[q * 8 + 7]);
        o.put16(q, u);
    }
}

// Per-column operands of one 32-column chunk (BIAS, GELU, RESID epilogues),
// loaded ahead of the chunk's accumulator so their L2 latency is hidden.
struct ColOps {
    uint4 b[4];   // 32 bf16 biases (zeros without a bias)
    float4 g[8];  // 32 fp32 gates (RESID; ones without a gate)
};

template <int EPI>
F3DC_DEV void load_colops(const GemmParams &p, int col, ColOps &c)
{
    if (p.bias) {
        const uint4 *pb = reinterpret_cast<const uint4 *>(p.bias + col);
#pragma unroll
        for (int q = 0; q < 4; ++q) c.b[q] = __ldg(pb + q);
    } else {
#pragma unroll
        for (int q = 0; q < 4; ++q) c.b[q] = make_uint4(0u, 0u, 0u, 0u);
    }
    if constexpr (EPI == kEpiResid) {
        if (p.gate) {
            const float4 *pg = reinterpret_cast<const float4 *>(p.gate + col);
#pragma unroll
            for (int q = 0; q < 8; ++q) c.g[q] = __ldg(pg + q);
        } else {
#pragma unroll
            for (int q = 0; q < 8; ++q) c.g[q] = make_float4(1.f, 1.f, 1.f, 1.f);
        }
    }
}

// Applies the epilogue to the column chunks k0, k0 + kstep, ... of a tile
// bn columns wide (chunks of 64 columns for QKNORM, whose RMSNorm groups
// span 64, else 32).  Outside QKNORM the next chunk's biases and gates are
// loaded while the current chunk is processed; `first`, when given, holds the
// first chunk's (loaded by the caller before it waited for the accumulator).
template <int EPI, typename Src>
F3DC_DEV void epilogue_tile(const GemmParams &p, const Src &src, OutStage &o, int m0, int n0, int bn, int k0 = 0,
                            int kstep = 1, const ColOps *first = nullptr)
{
    if constexpr (EPI == kEpiQKNorm) {
#pragma unroll 1
        for (int c0 = 64 * k0; c0 < bn; c0 += 64 * kstep) {
            float v[64];
            src(c0, v);
            src(c0 + 32, v + 32);
            const int col = n0 + c0;
            {
                float b[32];
                load_bias32(p.bias, col, b);
#pragma unroll
                for (int j = 0; j < 32; ++j) v[j] += b[j];
                load_bias32(p.bias, col + 32, b);
#pragma unroll
                for (int j = 0; j < 32; ++j) v[32 + j] += b[j];
            }
            if (col < 2 * p.width) {
                const bf16 *g = col < p.width ? p.qn_g : p.kn_g;
                const int gc = col < p.width ? col : col - p.width;
                if (p.dh == 64) {
                    rms_scale(v, 64, g, gc);
                } else {
                    rms_scale(v, 32, g, gc);
                    rms_scale(v + 32, 32, g, gc + 32);
                }
            }
            put_bf16x32(o, v);
            o.template emit<false>(col, m0);
            put_bf16x32(o, v + 32);
            o.template emit<false>(col + 32, m0);
        }
    } else {
        ColOps nxt;
        if (first)
            nxt = *first;
        else if (32 * k0 < bn)
            load_colops<EPI>(p, n0 + 32 * k0, nxt);
#pragma unroll 1
        for (int c0 = 32 * k0; c0 < bn; c0 += 32 * kstep) {
            const int col = n0 + c0;
            const ColOps cur = nxt;
            if (c0 + 32 * kstep < bn) load_colops<EPI>(p, col + 32 * kstep, nxt);
            float v[32];
            src(c0, v);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const uint32_t w[4] = {cur.b[q].x, cur.b[q].y, cur.b[q].z, cur.b[q].w};
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    v[q * 8 + 2 * j] += bf16_bits_to_f32(w[j] & 0xFFFFu);
                    v[q * 8 + 2 * j + 1] += bf16_bits_to_f32(w[j] >> 16);
                }
            }
            if constexpr (EPI == kEpiGelu) {
#pragma unroll
                for (int j = 0; j < 32; ++j) v[j] = gelu_tanh(v[j]);
            }
            if constexpr (EPI == kEpiResid) {
                // x += gate * y as an fp32 reduce-add of gate * y, 16 columns per chunk
#pragma unroll
                for (int h = 0; h < 2; ++h) {
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        const float4 g = cur.g[4 * h + q];
                        const float *w = v + 16 * h + 4 * q;
                        o.put16(q, make_uint4(__float_as_uint(g.x * w[0]), __float_as_uint(g.y * w[1]),
                                              __float_as_uint(g.z * w[2]), __float_as_uint(g.w * w[3])));
                    }
                    o.template emit<true>(col + 16 * h, m0);
                }
            } else {
                put_bf16x32(o, v);
                o.template emit<false>(col, m0);
            }
        }
    }
}

// Work decomposition shared by the three roles: unit u covers tile u % tiles
// (m fastest) and K blocks [split * kb_per, ...) with split = u / tiles.
struct Units {
    int m_tiles, tiles, splits, kb_per, kb_n, total;
    F3DC_DEV void decode(int u, int &m0, int &n0, int &kb0, int &kb1, int BN) const
    {
        const int t = u % tiles, s = u / tiles;
        m0 = (t % m_tiles) * 128;
        n0 = (t / m_tiles) * BN;
        kb0 = s * kb_per;
        kb1 = min(kb_n, kb0 + kb_per);
    }
};

template <int BN, int EPI>
__global__ void __launch_bounds__(kGemmThreads, 1)
    k_gemm(const __grid_constant__ CUtensorMap tma, const __grid_constant__ CUtensorMap tmb,
           const __grid_constant__ CUtensorMap tmo, const __grid_constant__ CUtensorMap tmw, const GemmParams p)
{
    using Cfg = GemmCfg<BN>;
    constexpr int S = Cfg::kStages;
    constexpr int kBBox = BN < 128 ? BN : 128;  // rows of one B box (gemm_b_box_rows)
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sa = smem;
    uint8_t *sb = smem + S * kAStage;
    uint8_t *so = sb + S * Cfg::kBStage;  // output staging (1024-aligned)
    uint64_t *bars = reinterpret_cast<uint64_t *>(so + kOutBufs * kOutChunkBytes);
    uint64_t *full = bars, *empty = bars + S, *accf = bars + 2 * S, *acce = accf + 2, *drain = acce + 2;
    uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(drain + 1);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_holder + 1);
    volatile int *split_flag = reinterpret_cast<volatile int *>(tmem_holder + 2);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    griddep_launch();

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(&accf[0], 1);
        mbar_init(&accf[1], 1);
        mbar_init(&acce[0], 4);  // one arrival per epilogue warp
        mbar_init(&acce[1], 4);
        mbar_init(drain, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(tmem_holder, Cfg::kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_holder;
    // the previous kernel's outputs (A, the row plan, x) are complete
    griddep_wait();
    Units U;
    U.m_tiles = p.m_tiles_dev ? *p.m_tiles_dev : p.m_tiles;
    // narrow mode: a 256-wide kernel whose tile count would leave too many SMs
    // idle (the row count is only known here) runs 128-wide tiles instead,
    // with the same stages (half of each B stage used) and TMEM buffers
    const bool narrow = BN == 256 && p.ws == nullptr && U.m_tiles * (p.N / BN) < p.narrow_below;
    const int bn = narrow ? BN / 2 : BN;
    U.tiles = U.m_tiles * (p.N / bn);
    U.kb_n = p.K / kBK;
    U.splits = gemm_split_count(U.tiles, (int)gridDim.x, U.kb_n, p.ws_units, p.ws != nullptr);
    U.kb_per = (U.kb_n + U.splits - 1) / U.splits;
    U.total = U.tiles * U.splits;
    const int total = U.total;

    if (warp == 0) {
        if (lane == 0) {
            tma_prefetch(&tma);
            tma_prefetch(&tmb);
            int s = 0;
            uint32_t ph = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < total && ok; t += gridDim.x) {
                int m0, n0, kb0, kb1;
                U.decode(t, m0, n0, kb0, kb1, bn);
                for (int kb = kb0; kb < kb1; ++kb) {
                    if (!mbar_wait(&empty[s], ph ^ 1, abort_flag, p.err)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(&full[s], kAStage + bn * kBK * 2);
                    tma_load_2d(sa + s * kAStage, &tma, kb * kBK, m0, &full[s]);
                    // B in boxes of kBBox rows, stacked in the stage (the
                    // 8-row swizzle atoms continue across boxes)
                    for (int hb = 0; hb < bn; hb += kBBox)
                        tma_load_2d(sb + s * Cfg::kBStage + hb * (kBK * 2), &tmb, kb * kBK, n0 + hb, &full[s]);
                    if (++s == S) {
                        s = 0;
                        ph ^= 1;
                    }
                }
            }
        }
    } else if (warp == 1) {
        // Barrier reads take long even when the phase is complete: the
        // issuer tests the next stage's `full` barrier before issuing the
        // current stage's MMAs, so the read overlaps them, and takes the
        // bounded wait only when the test found the stage not yet loaded.
        // The whole warp runs the loop (barrier outcomes as warp votes) and
        // elect.sync issues.
        {
            constexpr uint32_t idesc_w = make_idesc_bf16(128, BN, 0, 0);
            constexpr uint32_t idesc_n = make_idesc_bf16(128, BN / 2 < 16 ? 16 : BN / 2, 0, 0);
            const uint32_t idesc = narrow ? idesc_n : idesc_w;
            // stage-0 descriptors; stage s adds s * stage bytes / 16, a K
            // step of 16 elements inside the 128B swizzle atom adds 2
            const uint64_t a_desc0 = make_sdesc(smem_u32(sa), 16, 1024, kSwizzle128);
            const uint64_t b_desc0 = make_sdesc(smem_u32(sb), 16, 1024, kSwizzle128);
            int s = 0, it = 0;
            uint32_t ph = 0;
            bool ok = true;
            bool ready = warp_all(mbar_test(&full[0], 0));
            for (int t = blockIdx.x; t < total && ok; t += gridDim.x, ++it) {
                const int buf = it & 1;
                const uint32_t aph = (it >> 1) & 1;
                if (!warp_all(mbar_test(&acce[buf], aph ^ 1)) &&
                    !warp_all(mbar_wait(&acce[buf], aph ^ 1, abort_flag, p.err)))
                    break;
                const uint32_t d = tmem + buf * BN;
                int m0, n0, kb0, kb1;
                U.decode(t, m0, n0, kb0, kb1, bn);
                for (int kb = kb0; kb < kb1; ++kb) {
                    if (!ready && !warp_all(mbar_wait(&full[s], ph, abort_flag, p.err))) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const int s_next = s + 1 == S ? 0 : s + 1;
                    const uint32_t ph_next = s_next == 0 ? ph ^ 1 : ph;
                    ready = warp_all(mbar_test(&full[s_next], ph_next));  // read overlaps the MMAs below
                    const uint64_t ad = a_desc0 + (uint64_t)s * (kAStage >> 4);
                    const uint64_t bd = b_desc0 + (uint64_t)s * (Cfg::kBStage >> 4);
#pragma unroll
                    for (int k = 0; k < kBK / 16; ++k)
                        mma_bf16_elect(d, ad + 2 * k, bd + 2 * k, idesc, (kb != kb0) || (k != 0));
                    mma_commit_elect(&empty[s]);
                    s = s_next;
                    ph = ph_next;
                }
                if (ok) mma_commit_elect(&accf[buf]);
            }
        }
    } else {
        const int q = warp & 3;
        const int row = q * 32 + lane;
        OutStage o{so, &tmo, row, 0};
        int it = 0;
        for (int t = blockIdx.x; t < total; t += gridDim.x, ++it) {
            const int buf = it & 1;
            const uint32_t aph = (it >> 1) & 1;
            // the four epilogue warps meet at named barriers inside the tile,
            // so they take the wait's outcome together (a timeout seen by one
            // warp ends the loop for all)
            const uint32_t got = mbar_wait(&accf[buf], aph, abort_flag, p.err) ? 1u : 0u;
            uint32_t all;
            asm volatile("{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n bar.red.and.pred q, 3, 128, p;\n"
                         " selp.u32 %0, 1, 0, q;\n}\n"
                         : "=r"(all)
                         : "r"(got)
                         : "memory");
            if (!all) break;
            tc_fence_after();
            int m0, n0, kb0, kb1;
            U.decode(t, m0, n0, kb0, kb1, bn);
            const TmemSrc tsrc{tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(buf * BN)};
            if (U.splits == 1) {
                epilogue_tile<EPI>(p, tsrc, o, m0, n0, bn);
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&acce[buf]);
                continue;
            }
            // split K.  Each split stores its fp32 partial tile in the
            // workspace, chunk-major (unit u's 32-column chunk k: 128 rows of
            // 32 floats at row (u * BN / 32 + k) * 128 of the workspace
            // tensor), through the staged TMA stores; frees TMEM; and arrives
            // on the tile's counter.  Once every split has arrived, split s
            // reduces chunks s, s + S, ... of the tile -- all partials summed
            // in split order, so results do not depend on timing -- and
            // applies the epilogue to them.  When splitting, a CTA holds at
            // most one unit (tiles * splits <= grid <= SMs, one CTA per SM),
            // so the wait below never waits on work queued behind itself.
            const int tile = t % U.tiles, split = t / U.tiles;
#pragma unroll 1
            for (int c0 = 0; c0 < BN; c0 += 32) {
                float v[32];
                tsrc(c0, v);
                const int y = (t * (BN / 32) + c0 / 32) * 128;
#pragma unroll
                for (int h = 0; h < 2; ++h) {
#pragma unroll
                    for (int q4 = 0; q4 < 4; ++q4) {
                        const float *w = v + 16 * h + 4 * q4;
                        o.put16(q4, make_uint4(__float_as_uint(w[0]), __float_as_uint(w[1]), __float_as_uint(w[2]),
                                               __float_as_uint(w[3])));
                    }
                    o.template emit<false>(16 * h, y, &tmw);
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&acce[buf]);
            asm volatile("bar.sync 2, 128;" ::: "memory");
            if (threadIdx.x == 64) {
                // the partial's TMA stores are complete and visible before
                // the arrival
                bulk_wait_all();
                asm volatile("fence.proxy.async.global;" ::: "memory");
                __threadfence();
                atomicAdd(p.counters + tile, 1);
                int ok = 1;
                const uint64_t t0 = globaltimer();
                const uint64_t limit = p.split_wait_ns ? p.split_wait_ns : kWaitLimitNs;
                while (*reinterpret_cast<volatile int32_t *>(p.counters + tile) < U.splits + p.split_extra) {
                    if (*abort_flag || globaltimer() - t0 > limit) {
                        *abort_flag = 1;
                        raise_error(p.err, kDevTimeout);
                        ok = 0;
                        break;
                    }
                }
                __threadfence();
                *split_flag = ok;
            }
            asm volatile("bar.sync 2, 128;" ::: "memory");
            if (!*split_flag) break;
            __threadfence();
            const WsSrc<BN> wsrc{p.ws, tile, U.tiles, U.splits, row};
            epilogue_tile<EPI>(p, wsrc, o, m0, n0, BN, split, U.splits);
            asm volatile("bar.sync 2, 128;" ::: "memory");
            if (threadIdx.x == 64) {
                // every split has read what it needs: the last one to get here
                // returns the counter to 0 for the next launch
                if (atomicAdd(p.counters + tile, 1) == 2 * U.splits - 1) p.counters[tile] = 0;
            }
        }
        // this CTA's output stores complete before it ends
        if (threadIdx.x == 64) bulk_wait_all();
    }
    __syncthreads();
    if (*abort_flag) {
        // drain: wait (bounded) for this CTA's outstanding MMAs and copies
        if (warp == 1) {
            mma_commit_elect(drain);  // the MMAs' issuing lane
            if (lane == 0) mbar_wait_bounded(drain, 0, 100000000ull);
        }
        if (threadIdx.x == 0) spin_ns(200000);
        __syncthreads();
    }
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, Cfg::kTmemCols);
    }
}

// ------------------------------------------------------------ CTA pair
// cta_group::2 GEMM for 256-wide tiles.  A cluster of two CTAs computes a
// 256 x 256 tile (256 x 128 in narrow mode): each CTA loads its 128 rows of A
// and its half of the tile's B rows into its own shared memory (128 K per stage), the even CTA
// issues the 256-row MMAs for both, and each CTA's TMEM receives its own 128
// rows of the accumulator, which its epilogue warps write out.  Per SM that
// is 32 KB of operands per 512 MMA clocks instead of the 48 KB a 128 x 256
// tile of one CTA needs, so the operand stream from L2 keeps up with the
// tensor core.
//   full[s]  (even CTA): both CTAs' TMA bytes of stage s (the even CTA's
//            producer posts the expected count)
//   empty[s] (both):     stage s consumed (multicast MMA commit)
//   accf[b]  (both):     accumulator buffer b complete (multicast commit)
//   acce[b]  (even CTA): buffer b read by the epilogue warps of both CTAs
// A stage holds 128 K: two 64-column boxes per operand row block, each a
// 128B-swizzled K-major region of its own ([half][rows][128 B]).
constexpr int kPairBK = 128;
constexpr int kPairHalf = 128 * 128;                // one 64-K box of 128 rows (16 KB)
constexpr int kPairAStage = 2 * kPairHalf;          // this CTA's 128 A rows x 128 K
constexpr int kPairBStage = 2 * kPairHalf;          // this CTA's (up to) 128 B rows x 128 K
constexpr int kPairStages = 3;
constexpr uint32_t kPairTmemCols = 512;             // two buffers of 256 columns
// eight epilogue warps in two groups of four (one warp per TMEM lane quarter
// in each), group g writing the tile's column chunks g, g + 2, ..., each
// group through two staging buffers of its own
constexpr int kPairThreads = 320;
constexpr int kPairOutBufs = 2;
constexpr size_t kPairSmem = 1024 + (size_t)kPairStages * (kPairAStage + kPairBStage) +
                             2 * (size_t)kPairOutBufs * kOutChunkBytes + 256;

template <int EPI>
__global__ void __launch_bounds__(kPairThreads, 1)
    k_gemm_pair(const __grid_constant__ CUtensorMap tma, const __grid_constant__ CUtensorMap tmb,
                const __grid_constant__ CUtensorMap tmo, const GemmParams p)
{
    constexpr int S = kPairStages;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sa = smem;
    uint8_t *sb = smem + S * kPairAStage;
    uint8_t *so = sb + S * kPairBStage;
    uint64_t *bars = reinterpret_cast<uint64_t *>(so + 2 * kPairOutBufs * kOutChunkBytes);
    uint64_t *full = bars, *empty = bars + S, *accf = bars + 2 * S, *acce = accf + 2, *drain = acce + 2;
    uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(drain + 1);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_holder + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = cluster_rank();
    griddep_launch();

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(&accf[0], 1);
        mbar_init(&accf[1], 1);
        mbar_init(&acce[0], 16);  // eight epilogue warps in each CTA
        mbar_init(&acce[1], 16);
        mbar_init(drain, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc_pair(tmem_holder, kPairTmemCols);
        tmem_relinquish_pair();
    }
    if (warp == 0 && lane == 0) {
        // the weights are constant: pull this CTA's share of B into L2 while
        // the previous kernel finishes, so the first stages' loads hit L2
        const int kbx = p.K / 64, boxes = (p.N / (int)kGemmPairBBox) * kbx;
        for (int i = blockIdx.x; i < boxes; i += gridDim.x)
            tma_prefetch_l2_2d(&tmb, (i % kbx) * 64, (i / kbx) * (int)kGemmPairBBox);
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync();  // both CTAs' barriers are initialised before any remote signal
    tc_fence_after();
    const uint32_t tmem = *tmem_holder;
    griddep_wait();
    const int m_tiles = p.m_tiles_dev ? *p.m_tiles_dev : p.m_tiles;
    const bool narrow = m_tiles * (p.N / 256) < p.narrow_below;
    const int bn = narrow ? 128 : 256;  // tile width; this CTA holds bn / 2 B rows
    const int pm_tiles = (m_tiles + 1) / 2;
    const int tiles = pm_tiles * (p.N / bn);
    const int kb_n = p.K / kPairBK;
    const int cl = blockIdx.x >> 1, ncl = gridDim.x >> 1;
    const uint32_t full_c = mapa_shared(smem_u32(full), 0);  // the even CTA's full[0]
    const uint32_t acce_c = mapa_shared(smem_u32(acce), 0);

    if (warp == 0) {
        if (lane == 0) {
            tma_prefetch(&tma);
            tma_prefetch(&tmb);
            const uint32_t stage_bytes = 2u * (kPairAStage + (uint32_t)(bn / 2) * kPairBK * 2);  // both CTAs
            int s = 0;
            uint32_t ph = 0;
            bool ok = true;
            for (int t = cl; t < tiles && ok; t += ncl) {
                const int arow = (t % pm_tiles) * 256 + (int)rank * 128;
                const int brow = (t / pm_tiles) * bn + (int)rank * (bn / 2);
                for (int kb = 0; kb < kb_n; ++kb) {
                    if (!mbar_wait(&empty[s], ph ^ 1, abort_flag, p.err)) {
                        ok = false;
                        break;
                    }
                    if (rank == 0) mbar_arrive_expect_tx(&full[s], stage_bytes);
                    const uint32_t fb = full_c + 8u * (uint32_t)s;
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        const int x = kb * kPairBK + h * 64;
                        tma_load_2d_pair(sa + s * kPairAStage + h * kPairHalf, &tma, x, arow, fb);
                        for (int hb = 0; hb < bn / 2; hb += (int)kGemmPairBBox)
                            tma_load_2d_pair(sb + s * kPairBStage + h * kPairHalf + hb * 128, &tmb, x, brow + hb, fb);
                    }
                    if (++s == S) {
                        s = 0;
                        ph ^= 1;
                    }
                }
            }
        }
    } else if (warp == 1) {
        // the even CTA's warp issues for the pair: the whole warp runs the
        // loop (barrier outcomes as warp votes) and elect.sync issues
        if (rank == 0) {
            constexpr uint32_t idesc_w = make_idesc_bf16(256, 256, 0, 0);
            constexpr uint32_t idesc_n = make_idesc_bf16(256, 128, 0, 0);
            const uint32_t idesc = narrow ? idesc_n : idesc_w;
            const uint64_t a_desc0 = make_sdesc(smem_u32(sa), 16, 1024, kSwizzle128);
            const uint64_t b_desc0 = make_sdesc(smem_u32(sb), 16, 1024, kSwizzle128);
            int s = 0, it = 0;
            uint32_t ph = 0;
            bool ok = true;
            bool ready = warp_all(mbar_test(&full[0], 0));
            for (int t = cl; t < tiles && ok; t += ncl, ++it) {
                const int buf = it & 1;
                const uint32_t aph = (it >> 1) & 1;
                if (!warp_all(mbar_test(&acce[buf], aph ^ 1)) &&
                    !warp_all(mbar_wait(&acce[buf], aph ^ 1, abort_flag, p.err)))
                    break;
                const uint32_t d = tmem + buf * 256;
                for (int kb = 0; kb < kb_n; ++kb) {
                    if (!ready && !warp_all(mbar_wait(&full[s], ph, abort_flag, p.err))) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const int s_next = s + 1 == S ? 0 : s + 1;
                    const uint32_t ph_next = s_next == 0 ? ph ^ 1 : ph;
                    ready = warp_all(mbar_test(&full[s_next], ph_next));
                    const uint64_t ad = a_desc0 + (uint64_t)s * (kPairAStage >> 4);
                    const uint64_t bd = b_desc0 + (uint64_t)s * (kPairBStage >> 4);
#pragma unroll
                    for (int k = 0; k < kPairBK / 16; ++k) {
                        const uint64_t off = (uint64_t)(k >> 2) * (kPairHalf >> 4) + 2 * (k & 3);
                        mma_bf16_pair_elect(d, ad + off, bd + off, idesc, (kb != 0) || (k != 0));
                    }
                    mma_commit_pair_mc_elect(&empty[s], 3);
                    s = s_next;
                    ph = ph_next;
                }
                if (ok) mma_commit_pair_mc_elect(&accf[buf], 3);
            }
        }
    } else {
        const int q = warp & 3;
        const int row = q * 32 + lane;
        const int grp = (warp - 2) >> 2;
        OutStage o{so + grp * kPairOutBufs * kOutChunkBytes, &tmo, row, 0, kPairOutBufs, 3 + grp, 64 + 128 * grp};
        int it = 0;
        for (int t = cl; t < tiles; t += ncl, ++it) {
            const int buf = it & 1;
            const uint32_t aph = (it >> 1) & 1;
            const int n0 = (t / pm_tiles) * bn;
            ColOps first;
            if constexpr (EPI != kEpiQKNorm) load_colops<EPI>(p, n0 + 32 * grp, first);
            const uint32_t got = mbar_wait(&accf[buf], aph, abort_flag, p.err) ? 1u : 0u;
            uint32_t all;
            asm volatile("{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n bar.red.and.pred q, %2, 128, p;\n"
                         " selp.u32 %0, 1, 0, q;\n}\n"
                         : "=r"(all)
                         : "r"(got), "r"(o.bar)
                         : "memory");
            if (!all) break;
            tc_fence_after();
            const int m0 = (t % pm_tiles) * 256 + (int)rank * 128;
            // the odd CTA's rows of the last pair lie beyond the plan when
            // the tile count is odd: computed, not stored
            if (m0 < m_tiles * 128) {
                const TmemSrc tsrc{tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(buf * 256)};
                epilogue_tile<EPI>(p, tsrc, o, m0, n0, bn, grp, 2, &first);
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_cluster(acce_c + 8u * (uint32_t)buf);
        }
        if ((int)threadIdx.x == o.issuer) bulk_wait_all();
    }
    __syncthreads();
    if (*abort_flag) {
        if (warp == 1 && rank == 0) {
            mma_commit_pair_elect(drain);  // the MMAs' issuing lane
            if (lane == 0) mbar_wait_bounded(drain, 0, 100000000ull);
        }
        if (threadIdx.x == 0) spin_ns(200000);
        __syncthreads();
    }
    // neither CTA leaves while the other may still signal its barriers or
    // (the even CTA's MMAs) write its TMEM
    cluster_sync();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc_pair(tmem, kPairTmemCols);
    }
}

template <int EPI>
cudaError_t launch_pair_one(const CUtensorMap *ta, const CUtensorMap *tb, const CUtensorMap *to, const GemmParams &p,
                            int max_pair_tiles, cudaStream_t s)
{
    // per device: the shared-memory attribute and the resident-cluster count
    // are taken on each device's first launch (0 = not yet known)
    static std::atomic<int> max_clusters_of[64];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    int max_clusters = max_clusters_of[dev & 63].load(std::memory_order_acquire);
    if (!max_clusters) {
        e = cudaFuncSetAttribute(k_gemm_pair<EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kPairSmem);
        if (e != cudaSuccess) return e;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(2);
        cfg.blockDim = dim3(kPairThreads);
        cfg.dynamicSmemBytes = kPairSmem;
        cudaLaunchAttribute at[1];
        at[0].id = cudaLaunchAttributeClusterDimension;
        at[0].val.clusterDim.x = 2;
        at[0].val.clusterDim.y = 1;
        at[0].val.clusterDim.z = 1;
        cfg.attrs = at;
        cfg.numAttrs = 1;
        int n = 0;
        e = cudaOccupancyMaxActiveClusters(&n, k_gemm_pair<EPI>, &cfg);
        if (e != cudaSuccess) return e;
        if (n < 1) return cudaErrorInvalidConfiguration;
        max_clusters = n;
        max_clusters_of[dev & 63].store(n, std::memory_order_release);
    }
    const int clusters = max_pair_tiles < max_clusters ? (max_pair_tiles > 0 ? max_pair_tiles : 1) : max_clusters;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(2 * clusters);
    cfg.blockDim = dim3(kPairThreads);
    cfg.dynamicSmemBytes = kPairSmem;
    cfg.stream = s;
    cudaLaunchAttribute at[2];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = 2;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    at[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = at;
    cfg.numAttrs = 2;
    e = cudaLaunchKernelEx(&cfg, k_gemm_pair<EPI>, *ta, *tb, *to, p);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

template <int BN, int EPI>
cudaError_t launch_one(const CUtensorMap *ta, const CUtensorMap *tb, const CUtensorMap *to, const CUtensorMap *tw,
                       const GemmParams &p, int grid, cudaStream_t s)
{
    // the shared-memory attribute is per device: set it on each device's first launch
    static std::atomic<uint64_t> attr_devices{0};
    const size_t smem = GemmCfg<BN>::kSmem;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const uint64_t bit = 1ull << (dev & 63);
    if (!(attr_devices.load(std::memory_order_acquire) & bit)) {
        e = cudaFuncSetAttribute(k_gemm<BN, EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        attr_devices.fetch_or(bit, std::memory_order_acq_rel);
    }
    launch_k(k_gemm<BN, EPI>, dim3(grid), dim3(kGemmThreads), smem, s, *ta, *tb, *to, *tw, p);
    return cudaGetLastError();
}

template <int BN>
cudaError_t launch_bn(const CUtensorMap *ta, const CUtensorMap *tb, const CUtensorMap *to, const CUtensorMap *tw,
                      const GemmParams &p, int epi, int grid, cudaStream_t s)
{
    switch (epi) {
    case kEpiBias: return launch_one<BN, kEpiBias>(ta, tb, to, tw, p, grid, s);
    case kEpiGelu: return launch_one<BN, kEpiGelu>(ta, tb, to, tw, p, grid, s);
    case kEpiResid: return launch_one<BN, kEpiResid>(ta, tb, to, tw, p, grid, s);
    case kEpiQKNorm: return launch_one<BN, kEpiQKNorm>(ta, tb, to, tw, p, grid, s);
    default: return cudaErrorInvalidValue;
    }
}

PFN_cuTensorMapEncodeTiled_v12000 tmap_encoder()
{
    static PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
    if (!encode) {
        cudaDriverEntryPointQueryResult q;
        void *fn = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
                cudaSuccess ||
            q != cudaDriverEntryPointSuccess || !fn)
            return nullptr;
        encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    return encode;
}

// The epilogue's output tensor: rows [0, M), columns [0, N), row stride ldo
// elements; boxes of 128 rows x 64 bytes (32 bf16 or 16 fp32 columns), 64B
// swizzle, matching OutStage.
bool make_tmap_out(CUtensorMap *map, void *base, uint64_t rows, uint64_t cols, uint64_t ld, bool f32)
{
    PFN_cuTensorMapEncodeTiled_v12000 encode = tmap_encoder();
    const uint64_t esz = f32 ? 4 : 2;
    if (!encode || ((uintptr_t)base & 15) != 0 || (ld * esz) % 16 != 0) return false;
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {ld * esz};
    cuuint32_t box[2] = {(cuuint32_t)(64 / esz), 128};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = encode(map, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, dims,
                        strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

}  // namespace

size_t gemm_smem_bytes(int bn)
{
    switch (bn) {
    case 64: return GemmCfg<64>::kSmem;
    case 128: return GemmCfg<128>::kSmem;
    case 256: return GemmCfg<256>::kSmem;
    default: return 0;
    }
}

cudaError_t launch_gemm(const CUtensorMap *ta, const CUtensorMap *tb, const GemmParams &p, int epi, int bn,
                        int grid, cudaStream_t s)
{
    if (p.K % kBK != 0 || p.N % bn != 0 || grid < 1) return cudaErrorInvalidValue;
    CUtensorMap to, tw;
    if (!make_tmap_out(&to, p.out, (uint64_t)p.M, (uint64_t)p.N, (uint64_t)p.ldo, epi == kEpiResid))
        return cudaErrorInvalidValue;
    // split-K workspace as a [ws_units * bn / 32 * 128, 32] fp32 tensor
    // (chunk-major partial tiles); without a workspace the output map stands in
    if (p.ws) {
        if (!make_tmap_out(&tw, p.ws, (uint64_t)p.ws_units * (bn / 32) * 128, 32, 32, true))
            return cudaErrorInvalidValue;
    } else {
        tw = to;
    }
    switch (bn) {
    case 64: return launch_bn<64>(ta, tb, &to, &tw, p, epi, grid, s);
    case 128: return launch_bn<128>(ta, tb, &to, &tw, p, epi, grid, s);
    case 256: return launch_bn<256>(ta, tb, &to, &tw, p, epi, grid, s);
    default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_gemm_pair(const CUtensorMap *ta, const CUtensorMap *tb, const GemmParams &p, int epi,
                             int max_pair_tiles, cudaStream_t s)
{
    if (p.K % kPairBK != 0 || p.N % 256 != 0 || p.ws) return cudaErrorInvalidValue;
    CUtensorMap to;
    if (!make_tmap_out(&to, p.out, (uint64_t)p.M, (uint64_t)p.N, (uint64_t)p.ldo, epi == kEpiResid))
        return cudaErrorInvalidValue;
    switch (epi) {
    case kEpiBias: return launch_pair_one<kEpiBias>(ta, tb, &to, p, max_pair_tiles, s);
    case kEpiGelu: return launch_pair_one<kEpiGelu>(ta, tb, &to, p, max_pair_tiles, s);
    case kEpiResid: return launch_pair_one<kEpiResid>(ta, tb, &to, p, max_pair_tiles, s);
    case kEpiQKNorm: return launch_pair_one<kEpiQKNorm>(ta, tb, &to, p, max_pair_tiles, s);
    default: return cudaErrorInvalidValue;
    }
}

bool make_tmap_bf16(CUtensorMap *map, const void *base, uint64_t rows, uint64_t cols, uint64_t ld,
                    uint32_t box_rows, uint32_t box_cols)
{
    PFN_cuTensorMapEncodeTiled_v12000 encode = tmap_encoder();
    if (!encode || ((uintptr_t)base & 15) != 0 || (ld * 2) % 16 != 0) return false;
    CUtensorMapSwizzle swz;
    switch (box_cols * 2) {
    case 128: swz = CU_TENSOR_MAP_SWIZZLE_128B; break;
    case 64: swz = CU_TENSOR_MAP_SWIZZLE_64B; break;
    case 32: swz = CU_TENSOR_MAP_SWIZZLE_32B; break;
    default: return false;
    }
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {ld * 2};
    cuuint32_t box[2] = {box_cols, box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

}  // namespace f3dc
