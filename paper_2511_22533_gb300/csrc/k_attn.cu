// k_attn.cu -- K5 / K6: multi-head attention softmax(Q K^T / sqrt(dh)) V on
// 5th-generation tensor cores, flash style (online softmax), for
//   mode 0  self-attention of every sample among its ACTIVE tokens only
//           (Sec. 4.2: attention runs on the compacted active subset)
//   mode 1  cross-attention of the active tokens to the sample's condition
//           tokens (Supp. Sec. F cross-attention)
//   mode 2  one sequence (diagnostic entry point)
//
// Persistent kernel, one CTA per SM (320 threads), work item = (128-query
// tile, head):
//   warp 0     TMA producer: Q tile once per item, K / V tiles of 128 keys
//              into a 4-deep ring
//   warp 1     TMEM allocator + tcgen05.mma issuer:
//                S_j = Q K_j^T              (M=128, N=128, K=dh) -> TMEM S[j%2]
//                O_h += P_j,h V_j,h  h=0,1  (M=128, N=dh,  K=64) -> TMEM O_h
//              S runs two tiles ahead: S_(j+2) is issued as soon as the
//              softmax has read S_j, before P V of tile j, so the scores of
//              the next tiles are ready whenever the softmax gets to them
//   warps 2-9  softmax, two threads per query row (TMEM lane = row): the
//              thread of half h owns keys [64h, 64h + 64) of every tile and
//              runs its own online softmax over them, writing
//              P = exp2(S scale - m) as bf16 into its 64-key 128B-swizzled
//              panel (the K-major A operand of its P V MMA).  O stays in TMEM
//              for the whole item; the reference max m is only raised (and O,
//              l rescaled in place) when a tile's max exceeds it by more than
//              2^8, so most tiles need no O traffic at all.  The two halves
//              of a row are combined once per work item.  Two softmax warps per
//              SM sub-partition hide each other's exponent and TMEM latencies.
// V is the MN-major B operand of the P V MMA straight from its row-major
// TMA tile.  Keys beyond a sample's count are masked to -inf before the
// exponent; padding rows are finite by construction, so 0 * pad = 0.
#include "common.cuh"
#include "kernels.h"

namespace f3dc {

namespace {

constexpr int kAttnThreads = 320;
constexpr int kSoftmaxThreads = 256;
constexpr int kSoftmaxWarps = kSoftmaxThreads / 32;  // arrivals per phase (one per warp)
constexpr int kKVStages = 4;

template <int DH>
struct AttnCfg {
    static constexpr int kRowBytes = DH * 2;            // 128 (DH 64) or 64 (DH 32)
    static constexpr int kTileBytes = 128 * kRowBytes;  // Q, K or V tile
    static constexpr uint32_t kAtom = 8 * kRowBytes;    // 8-row swizzle atom
    static constexpr uint32_t kSwz = DH == 64 ? kSwizzle128 : kSwizzle64;
    static constexpr int kPPanel = 128 * 128;           // 64 keys x 128 rows x 2 B
    static constexpr int kPBytes = 2 * kPPanel;
    static constexpr int kCombineBytes = 128 * (DH + 2) * 4;  // half-1 (m, l, O) per row, aliases P
    static_assert(kCombineBytes <= 2 * kPBytes, "combine scratch must fit in the P buffers");
    static constexpr size_t kSmem = 1024 + kTileBytes * (1 + 2 * kKVStages) + 2 * kPBytes + 512;
    static constexpr uint32_t kTmemCols = 512;          // S0 S1 | O_0 O_1
};

struct Item {
    int q_row0, kv_row0, nk, h, store_end;
};

F3DC_DEV Item decode_item(const AttnParams &p, int w)
{
    Item it;
    const int t = w / p.heads;
    it.h = w - t * p.heads;
    it.q_row0 = t * 128;
    it.store_end = 0x7FFFFFFF;
    if (p.mode == 0) {
        const int b = p.tile_sample[t];
        it.kv_row0 = p.plan->row_off[b];
        it.nk = p.plan->n_active[b];
    } else if (p.mode == 1) {
        const int b = p.tile_sample[t];
        it.kv_row0 = b * p.nk_fixed;
        it.nk = p.nk_fixed;
    } else {
        it.kv_row0 = 0;
        it.nk = p.nk_fixed;
        it.store_end = p.q_rows;
    }
    return it;
}

F3DC_DEV bool wait_bounded(uint64_t *bar, uint32_t parity, uint64_t ns)
{
    const uint64_t t0 = globaltimer();
    while (!mbar_try_wait(bar, parity))
        if (globaltimer() - t0 > ns) return false;
    return true;
}

template <int DH>
__global__ void __launch_bounds__(kAttnThreads, 1)
    k_attn(const __grid_constant__ CUtensorMap tmq, const __grid_constant__ CUtensorMap tmk,
           const __grid_constant__ CUtensorMap tmv, const AttnParams p)
{
    using Cfg = AttnCfg<DH>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sQ = smem;
    uint8_t *sK = sQ + Cfg::kTileBytes;
    uint8_t *sV = sK + kKVStages * Cfg::kTileBytes;
    uint8_t *sP = sV + kKVStages * Cfg::kTileBytes;
    // the end-of-item combine runs when every P V of the item is done, so
    // its scratch can live in the P buffers
    float *sComb = reinterpret_cast<float *>(sP);
    uint64_t *bars = reinterpret_cast<uint64_t *>(sP + 2 * Cfg::kPBytes);
    uint64_t *q_full = bars, *q_empty = bars + 1;
    uint64_t *kv_full = bars + 2, *kv_empty = kv_full + kKVStages;
    uint64_t *s_full = kv_empty + kKVStages, *s_empty = s_full + 2;
    uint64_t *p_full = s_empty + 2, *p_empty = p_full + 2;
    // p_empty[t % 2] completes once per P V of (global) tile index t and
    // doubles as the "O holds tiles <= t" signal; o_free completes once per item
    uint64_t *o_free = p_empty + 2;
    uint64_t *drain = o_free + 1;
    uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(drain + 1);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_holder + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n_tiles = p.n_tiles_dev ? *p.n_tiles_dev : p.n_tiles;
    const int total = n_tiles * p.heads;

    if (threadIdx.x == 0) {
        mbar_init(q_full, 1);
        mbar_init(q_empty, 1);
        for (int s = 0; s < kKVStages; ++s) {
            mbar_init(&kv_full[s], 1);
            mbar_init(&kv_empty[s], 1);
        }
        for (int s = 0; s < 2; ++s) {
            mbar_init(&s_full[s], 1);
            mbar_init(&s_empty[s], kSoftmaxWarps);
            mbar_init(&p_full[s], kSoftmaxWarps);
            mbar_init(&p_empty[s], 1);
        }
        mbar_init(o_free, kSoftmaxWarps);
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

    if (warp == 0) {
        // ------------------------------------------------ TMA producer
        if (lane == 0) {
            tma_prefetch(&tmq);
            tma_prefetch(&tmk);
            tma_prefetch(&tmv);
            uint32_t kv_it = 0, item_it = 0;
            bool ok = true;
            for (int w = blockIdx.x; w < total && ok; w += gridDim.x, ++item_it) {
                const Item it = decode_item(p, w);
                if (!mbar_wait(q_empty, (item_it & 1) ^ 1, abort_flag, p.err)) break;
                mbar_arrive_expect_tx(q_full, Cfg::kTileBytes);
                tma_load_2d(sQ, &tmq, p.q_col0 + it.h * DH, it.q_row0, q_full);
                const int nkt = (it.nk + 127) / 128;
                for (int j = 0; j < nkt; ++j, ++kv_it) {
                    const int s = kv_it % kKVStages;
                    const uint32_t ph = (kv_it / kKVStages) & 1;
                    if (!mbar_wait(&kv_empty[s], ph ^ 1, abort_flag, p.err)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(&kv_full[s], 2 * Cfg::kTileBytes);
                    tma_load_2d(sK + s * Cfg::kTileBytes, &tmk, p.k_col0 + it.h * DH, it.kv_row0 + j * 128,
                                &kv_full[s]);
                    tma_load_2d(sV + s * Cfg::kTileBytes, &tmv, p.v_col0 + it.h * DH, it.kv_row0 + j * 128,
                                &kv_full[s]);
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc_s = make_idesc_bf16(128, 128, 0, 0);
            constexpr uint32_t idesc_o = make_idesc_bf16(128, DH, 0, 1);
            const uint32_t q_addr = smem_u32(sQ);
            uint32_t kv_base = 0, g_base = 0, item_it = 0;  // global tile / kv-stage counters
            bool ok = true;
            // S for tile j of the item: needs its K tile and a free S buffer
            // (the softmax has read S of tile j-2)
            auto issue_s = [&](uint32_t gt, uint32_t kvt, bool last) -> bool {
                const int s = kvt % kKVStages;
                const uint32_t sb = gt & 1;
                if (!mbar_wait(&kv_full[s], (kvt / kKVStages) & 1, abort_flag, p.err)) return false;
                if (!mbar_wait(&s_empty[sb], ((gt >> 1) & 1) ^ 1, abort_flag, p.err)) return false;
                tc_fence_after();
                const uint32_t k_addr = smem_u32(sK + s * Cfg::kTileBytes);
#pragma unroll
                for (int kk = 0; kk < DH / 16; ++kk)
                    mma_bf16(tmem + sb * 128, make_sdesc(q_addr + kk * 32, 16, Cfg::kAtom, Cfg::kSwz),
                             make_sdesc(k_addr + kk * 32, 16, Cfg::kAtom, Cfg::kSwz), idesc_s, kk > 0);
                mma_commit(&s_full[sb]);
                if (last) mma_commit(q_empty);
                return true;
            };
            // O_h (+)= P_h V_h for tile gt; the item's first tile overwrites O,
            // after the softmax has read the previous item's result
            auto issue_pv = [&](uint32_t gt, uint32_t kvt, bool first) -> bool {
                const uint32_t pb = gt & 1;
                if (!mbar_wait(&p_full[pb], (gt >> 1) & 1, abort_flag, p.err)) return false;
                if (first && !mbar_wait(o_free, (item_it & 1) ^ 1, abort_flag, p.err)) return false;
                tc_fence_after();
                const int s = kvt % kKVStages;
                const uint32_t p_addr = smem_u32(sP + pb * Cfg::kPBytes);
                const uint32_t v_addr = smem_u32(sV + s * Cfg::kTileBytes);
#pragma unroll
                for (int kk = 0; kk < 8; ++kk) {  // keys 16kk..16kk+15, half kk / 4
                    const uint64_t ad = make_sdesc(p_addr + (kk >> 2) * Cfg::kPPanel + (kk & 3) * 32, 16, 1024,
                                                   kSwizzle128);
                    const uint64_t bd = make_sdesc(v_addr + kk * 16 * Cfg::kRowBytes, Cfg::kAtom, Cfg::kAtom, Cfg::kSwz);
                    mma_bf16(tmem + 256 + (kk >> 2) * DH, ad, bd, idesc_o, !(first && (kk & 3) == 0));
                }
                mma_commit(&kv_empty[s]);
                mma_commit(&p_empty[pb]);
                return true;
            };
            // every item has at least one key tile: a sample without active
            // tokens owns no query tile, and the entry points reject nk < 1
            for (int w = blockIdx.x; w < total && ok; w += gridDim.x, ++item_it) {
                const Item it = decode_item(p, w);
                if (!mbar_wait(q_full, item_it & 1, abort_flag, p.err)) break;
                tc_fence_after();
                const uint32_t nkt = (uint32_t)((it.nk + 127) / 128);
                ok = issue_s(g_base, kv_base, nkt == 1);
                if (ok && nkt > 1) ok = issue_s(g_base + 1, kv_base + 1, nkt == 2);
                for (uint32_t j = 0; j < nkt && ok; ++j) {
                    if (j + 2 < nkt && !issue_s(g_base + j + 2, kv_base + j + 2, j + 3 == nkt)) ok = false;
                    if (ok && !issue_pv(g_base + j, kv_base + j, j == 0)) ok = false;
                }
                g_base += nkt;
                kv_base += nkt;
            }
        }
    } else {
        // ------------------------------------------------ softmax warps
        const int q = warp & 3;                  // TMEM lane quarter of this warp
        const int half = (warp - 2) >> 2;        // keys [64 half, 64 half + 64) of each tile
        const int row = q * 32 + lane;
        const uint32_t tl = (uint32_t)(q * 32) << 16;
        const uint32_t o_addr = tmem + tl + 256 + half * DH;
        uint32_t g = 0, item_it = 0;
        // P V completions are awaited strictly in order: tile t on
        // p_empty[t % 2] with parity (t / 2) % 2.  Tile g awaits P V of g - 2
        // before it reuses that P buffer, and P V of g + 1 cannot start before
        // P of g + 1 is written, so no barrier is ever more than one phase
        // past the softmax's count and a parity wait cannot confuse phases
        uint32_t pv_seen = 0;  // P V of tiles < pv_seen known complete
        auto wait_pv_through = [&](uint32_t t) -> bool {
            for (; pv_seen <= t; ++pv_seen)
                if (!mbar_wait(&p_empty[pv_seen & 1], (pv_seen >> 1) & 1, abort_flag, p.err)) return false;
            return true;
        };
        for (int w = blockIdx.x; w < total; w += gridDim.x, ++item_it) {
            const Item it = decode_item(p, w);
            const int nkt = (it.nk + 127) / 128;
            float m_ref = -INFINITY, l_run = 0.f;
            bool ok = true;
            for (int j = 0; j < nkt; ++j, ++g) {
                const uint32_t sb = g & 1, sph = (g >> 1) & 1;
                if (!mbar_wait(&s_full[sb], sph, abort_flag, p.err)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const int valid = min(128, it.nk - j * 128) - 64 * half;  // valid keys of this half
                uint32_t r0[32], r1[32];
                tmem_ld32(tmem + tl + sb * 128 + 64 * half, r0);
                tmem_ld32(tmem + tl + sb * 128 + 64 * half + 32, r1);
                tmem_wait_ld();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&s_empty[sb]);  // one arrival per warp
                float sv[64];
#pragma unroll
                for (int c = 0; c < 32; ++c) {
                    sv[c] = __uint_as_float(r0[c]);
                    sv[32 + c] = __uint_as_float(r1[c]);
                }
                if (valid < 64) {  // only the last key tile of a sequence is ragged
#pragma unroll
                    for (int c = 0; c < 64; ++c)
                        if (c >= valid) sv[c] = -INFINITY;
                }
                // four independent chains of three-input maxima
                float mx4[4];
#pragma unroll
                for (int c = 0; c < 4; ++c) mx4[c] = fmaxf(sv[c], sv[4 + c]);
#pragma unroll
                for (int c = 8; c < 64; c += 8) {
#pragma unroll
                    for (int e = 0; e < 4; ++e) mx4[e] = fmax3(mx4[e], sv[c + e], sv[c + 4 + e]);
                }
                const float mx = fmax3(mx4[0], mx4[1], fmaxf(mx4[2], mx4[3])) * p.scale_log2;
                // raise the reference max only when it grew by more than 2^8
                // (warp-uniform: TMEM loads / stores are warp-collective)
                if (__any_sync(0xffffffffu, mx > m_ref + 8.0f)) {
                    const float m_new = fmaxf(m_ref, mx);
                    if (j > 0) {  // O holds tiles < j: wait for their P V, rescale in place
                        const float alpha = exp2_fast(m_ref - m_new);
                        if (!wait_pv_through(g - 1)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
#pragma unroll
                        for (int d0 = 0; d0 < DH; d0 += 32) {
                            uint32_t r[32];
                            tmem_ld32(o_addr + d0, r);
                            tmem_wait_ld();
#pragma unroll
                            for (int d = 0; d < 32; ++d) r[d] = __float_as_uint(__uint_as_float(r[d]) * alpha);
                            tmem_st32(o_addr + d0, r);
                        }
                        tmem_wait_st();
                        l_run *= alpha;
                    }
                    m_ref = m_new;
                }
                // a half with no valid key yet keeps m = -inf: subtract 0 instead
                const float m_use = m_ref == -INFINITY ? 0.f : m_ref;
                // P[sb] may still be read by the P V MMA of tile g-2
                if (g >= 2 && !wait_pv_through(g - 2)) {
                    ok = false;
                    break;
                }
                // exponent arguments and row sums two lanes per paired instruction
                f32x2 sum0 = {0.f, 0.f}, sum1 = {0.f, 0.f};
                const f32x2 sc2 = {p.scale_log2, p.scale_log2}, nm2 = {-m_use, -m_use};
                uint8_t *panel = sP + sb * Cfg::kPBytes + half * Cfg::kPPanel + row * 128;
#pragma unroll
                for (int ch = 0; ch < 8; ++ch) {  // 16-byte chunk ch of the 128-byte row
                    float pv[8];
#pragma unroll
                    for (int e = 0; e < 8; e += 2) {
                        const f32x2 x = ffma2({sv[ch * 8 + e], sv[ch * 8 + e + 1]}, sc2, nm2);
                        pv[e] = exp2_fast(x.x);
                        pv[e + 1] = exp2_fast(x.y);
                    }
                    sum0 = fadd2(sum0, {pv[0], pv[1]});
                    sum1 = fadd2(sum1, {pv[2], pv[3]});
                    sum0 = fadd2(sum0, {pv[4], pv[5]});
                    sum1 = fadd2(sum1, {pv[6], pv[7]});
                    uint4 u;
                    u.x = pack_bf16x2(pv[0], pv[1]);
                    u.y = pack_bf16x2(pv[2], pv[3]);
                    u.z = pack_bf16x2(pv[4], pv[5]);
                    u.w = pack_bf16x2(pv[6], pv[7]);
                    *reinterpret_cast<uint4 *>(panel + ((ch ^ (row & 7)) << 4)) = u;
                }
                fence_proxy_async_smem();  // every lane orders its own P stores
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&p_full[sb]);
                l_run += (sum0.x + sum0.y) + (sum1.x + sum1.y);
            }
            if (!ok) break;
            // every P V of the item done: read this half's O, release it
            if (!wait_pv_through(g - 1)) break;
            tc_fence_after();
            float acc[DH];
#pragma unroll
            for (int d0 = 0; d0 < DH; d0 += 32) {
                uint32_t r[32];
                tmem_ld32(o_addr + d0, r);
                tmem_wait_ld();
#pragma unroll
                for (int d = 0; d < 32; ++d) acc[d0 + d] = __uint_as_float(r[d]);
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(o_free);
            // combine the two halves of each row:
            // O = (O_0 2^(m_0-m) + O_1 2^(m_1-m)) / (l_0 2^(m_0-m) + l_1 2^(m_1-m))
            float *mine = sComb + row * (DH + 2);
            if (half == 1) {
                mine[0] = m_ref;
                mine[1] = l_run;
#pragma unroll
                for (int d = 0; d < DH; ++d) mine[2 + d] = acc[d];
            }
            asm volatile("bar.sync 1, %0;" ::"n"(kSoftmaxThreads) : "memory");
            if (half == 0) {
                const float m1 = mine[0], l1 = mine[1];
                const float m = fmaxf(m_ref, m1);
                const float a0 = exp2_fast(m_ref - m), a1 = exp2_fast(m1 - m);
                const float inv = 1.0f / (l_run * a0 + l1 * a1);
                const int orow = it.q_row0 + row;
                if (orow < it.store_end) {
                    uint4 *dst = reinterpret_cast<uint4 *>(p.out + (size_t)orow * p.ldo + it.h * DH);
#pragma unroll
                    for (int d = 0; d < DH; d += 8) {
                        float o[8];
#pragma unroll
                        for (int e = 0; e < 8; ++e) o[e] = (acc[d + e] * a0 + mine[2 + d + e] * a1) * inv;
                        uint4 u;
                        u.x = pack_bf16x2(o[0], o[1]);
                        u.y = pack_bf16x2(o[2], o[3]);
                        u.z = pack_bf16x2(o[4], o[5]);
                        u.w = pack_bf16x2(o[6], o[7]);
                        dst[d / 8] = u;
                    }
                }
            }
            asm volatile("bar.sync 1, %0;" ::"n"(kSoftmaxThreads) : "memory");
        }
    }
    __syncthreads();
    if (*abort_flag) {
        if (warp == 1 && lane == 0) {
            mma_commit(drain);
            wait_bounded(drain, 0, 100000000ull);
        }
        if (threadIdx.x == 0) spin_ns(200000);
        __syncthreads();
    }
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, Cfg::kTmemCols);
    }
}

template <int DH>
cudaError_t launch_dh(const CUtensorMap *tq, const CUtensorMap *tk, const CUtensorMap *tv, const AttnParams &p,
                      int grid, cudaStream_t s)
{
    static bool attr_set = false;
    const size_t smem = AttnCfg<DH>::kSmem;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(k_attn<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    k_attn<DH><<<grid, kAttnThreads, smem, s>>>(*tq, *tk, *tv, p);
    return cudaGetLastError();
}

}  // namespace

size_t attn_smem_bytes(int dh) { return dh == 64 ? AttnCfg<64>::kSmem : AttnCfg<32>::kSmem; }

cudaError_t launch_attention(const CUtensorMap *tq, const CUtensorMap *tk, const CUtensorMap *tv,
                             const AttnParams &p, int grid, cudaStream_t s)
{
    if (grid < 1) return cudaErrorInvalidValue;
    if (p.dh == 64) return launch_dh<64>(tq, tk, tv, p, grid, s);
    if (p.dh == 32) return launch_dh<32>(tq, tk, tv, p, grid, s);
    return cudaErrorInvalidValue;
}

}  // namespace f3dc
