// k_attn_one.cu -- K5 / K6 for small launches: the attention of k_attn.cu
// with one 128-query tile per work item, for launches whose (query tile,
// head) items all fit one per CTA (the cached steps below ~1200 active
// rows).  There the pair form of k_attn.cu would leave half of those CTAs
// idle; here each item's key tiles are split by parity between two softmax
// warps per SM sub-partition, so a single query tile still has two
// independent chains.  The host picks this kernel when it knows the launch's
// tile count (f3dc_sample, f3dc_attention); both kernels compute the same
// attention for any size.  Modes 0 (self-attention over a sample's active
// tokens), 1 (cross-attention to the sample's condition) and 2 (one
// sequence) as in k_attn.cu.
//
// Persistent kernel, one CTA per SM (320 threads), work item = (128-query
// tile, head):
//   warp 0     TMA producer: Q tile once per item, K / V tiles of 128 keys
//              into a 4-deep ring
//   warp 1     TMEM allocator + tcgen05.mma issuer (the whole warp runs the
//              loop and votes on every barrier outcome; elect.sync issues):
//                S_j = Q K_j^T     (M=128, N=128, K=dh)  -> TMEM S[j%2]
//                O_e += P_j V_j    (M=128, N=dh, K=128)  -> TMEM O_e, e = j%2,
//                                   with P_j read from TMEM P_e
//              S runs two tiles ahead: S_(j+2) is issued as soon as the
//              softmax has read S_j, before P V of tile j, so the scores of
//              the next tiles are ready whenever the softmax gets to them
//   warps 2-9  softmax, two threads per query row (TMEM lane = row): the
//              thread of parity e owns the key tiles j with j%2 == e (all
//              128 keys of each) and runs its own online softmax over them,
//              writing P = exp2(S scale - m) as bf16 pairs into TMEM P_e
//              (the A operand of its P V MMA, read straight from TMEM, so P
//              costs no shared-memory bandwidth).
//              O_e stays in TMEM for the whole item; the reference max m is
//              only raised (and O_e, l rescaled in place) when a tile's max
//              exceeds it by more than 2^8, so most tiles need no O traffic.
//              The two parities of a row are combined once per work item:
//              the parity that finished first leaves its (m, l, O) in shared
//              memory (mbarrier hand-over per lane quarter) and moves on to
//              the next item's first tile, while the other combines and
//              stores, so no item boundary stalls both.
//              Because the two warps of an SM sub-partition work on
//              different tiles, one warp's TMEM load, maximum and barrier
//              phases overlap the other's exponents instead of leaving the
//              exponent unit idle.
// V is the MN-major B operand of the P V MMA straight from its row-major
// TMA tile.  Keys beyond a sample's count are masked to -inf before the
// exponent; padding rows are finite by construction, so 0 * pad = 0.
#include <atomic>

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
    static constexpr int kCombineBytes = 128 * DH * 4;  // parity-1 O, one row per softmax row
    static constexpr size_t kSmem = 1024 + kTileBytes * (2 + 2 * kKVStages) + kCombineBytes + 512 + 128 * 8;
    // TMEM columns: S_0 S_1 (fp32, 128 each) | O_0 O_1 (fp32, DH each) |
    // P_0 P_1 (bf16 pairs, 64 each)
    static constexpr uint32_t kColO = 256, kColP = 256 + 2 * DH;
    static constexpr uint32_t kTmemCols = 512;
    static_assert(kColP + 128 <= kTmemCols, "TMEM layout");
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
        it.kv_row0 = (p.kv_null_from > 0 && b >= p.kv_null_from ? p.kv_null_sample : b) * p.nk_fixed;
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

// One output row of the end-of-item combine, in parity order whichever
// parity combines: O = (O_0 a_0 + O_1 a_1) / l with a_e = 2^(m_e - m); `acc`
// is the combining thread's own O (parity 1's when SWAP), the other parity's
// row is read from its hand-over slot (float4 d4 at d4 ^ (row % (DH / 4))).
template <int DH, bool SWAP>
F3DC_DEV void combine_row(const float (&acc)[DH], const float4 *slot, int row, float a0, float a1, float inv,
                          uint4 *dst)
{
    constexpr int kV4 = DH / 4;
#pragma unroll
    for (int d = 0; d < DH; d += 8) {
        const float4 b0 = slot[(d / 4) ^ (row & (kV4 - 1))], b1 = slot[(d / 4 + 1) ^ (row & (kV4 - 1))];
        const float ob[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
        float o[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const float o0 = SWAP ? ob[e] : acc[d + e], o1 = SWAP ? acc[d + e] : ob[e];
            o[e] = __fmul_rn(__fmaf_rn(o0, a0, __fmul_rn(o1, a1)), inv);
        }
        uint4 u;
        u.x = pack_bf16x2(o[0], o[1]);
        u.y = pack_bf16x2(o[2], o[3]);
        u.z = pack_bf16x2(o[4], o[5]);
        u.w = pack_bf16x2(o[6], o[7]);
        dst[d / 8] = u;
    }
}

template <int DH>
__global__ void __launch_bounds__(kAttnThreads, 1)
    k_attn_one(const __grid_constant__ CUtensorMap tmq, const __grid_constant__ CUtensorMap tmk,
           const __grid_constant__ CUtensorMap tmv, const AttnParams p)
{
    using Cfg = AttnCfg<DH>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    // Q is double-buffered per item (item i in buffer i % 2), so the next
    // item's Q arrives while the current item's last key tiles run
    uint8_t *sQ = smem;
    uint8_t *sK = sQ + 2 * Cfg::kTileBytes;
    uint8_t *sV = sK + kKVStages * Cfg::kTileBytes;
    // the end-of-item hand-over: the parity that finishes an item first
    // leaves its O and (m, l) here for the other one, which combines
    float *sComb = reinterpret_cast<float *>(sV + kKVStages * Cfg::kTileBytes);
    uint64_t *bars = reinterpret_cast<uint64_t *>(reinterpret_cast<uint8_t *>(sComb) + Cfg::kCombineBytes);
    float2 *sML = reinterpret_cast<float2 *>(reinterpret_cast<uint8_t *>(bars) + 512);
    uint64_t *q_full = bars, *q_empty = bars + 2;
    uint64_t *kv_full = bars + 4, *kv_empty = kv_full + kKVStages;
    // Key tile g (counted over the CTA's whole run) always sits in K/V stage
    // g % kKVStages, so kv_empty[g % kKVStages] completes exactly when P V of
    // tile g does: the producer reuses the stage on it, and the softmax takes
    // it as "O_(g%2) holds tile g and P_(g%2) is free".  p_full[e] (four
    // softmax warps of parity e) certifies P of the tile and that its S was
    // read, so it also frees S buffer e.  o_free completes once per item.
    uint64_t *s_full = kv_empty + kKVStages, *p_full = s_full + 2;
    uint64_t *o_free = p_full + 2;
    uint64_t *drain = o_free + 1;
    // end-of-item hand-over of one parity's (m, l, O) to the other, per TMEM
    // lane quarter (the softmax section explains the protocol)
    uint64_t *comb_full = drain + 1, *comb_free = comb_full + 4;
    uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(comb_free + 4);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_holder + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    griddep_launch();

    if (threadIdx.x == 0) {
        for (int b = 0; b < 2; ++b) {
            mbar_init(&q_full[b], 1);
            mbar_init(&q_empty[b], 1);
        }
        for (int s = 0; s < kKVStages; ++s) {
            mbar_init(&kv_full[s], 1);
            mbar_init(&kv_empty[s], 1);
        }
        for (int s = 0; s < 2; ++s) {  // one S / P buffer per tile parity, four warps each
            mbar_init(&s_full[s], 1);
            mbar_init(&p_full[s], kSoftmaxWarps / 2);
        }
        mbar_init(o_free, kSoftmaxWarps);
        mbar_init(drain, 1);
        for (int q = 0; q < 4; ++q) {  // one arrival per thread of the quarter's warp
            mbar_init(&comb_full[q], 32);
            mbar_init(&comb_free[q], 32);
        }
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(tmem_holder, Cfg::kTmemCols);
        tmem_relinquish();
    }
    if (p.kv_prefetch_rows > 0 && warp == 0 && lane == 0) {
        // keys / values written long before this launch (the condition's):
        // pull this CTA's share into L2 while the previous kernel finishes
        const int rb = (p.kv_prefetch_rows + 127) / 128, boxes = rb * p.heads * 2;
        for (int i = blockIdx.x; i < boxes; i += gridDim.x) {
            const int r = i % rb, hk = i / rb, h = hk >> 1;
            tma_prefetch_l2_2d(hk & 1 ? &tmv : &tmk, (hk & 1 ? p.v_col0 : p.k_col0) + h * DH, r * 128);
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_holder;
    // the previous kernel's outputs (Q / K / V, the row plan) are complete
    griddep_wait();
    const int n_tiles = p.n_tiles_dev ? *p.n_tiles_dev : p.n_tiles;
    const int total = n_tiles * p.heads;

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
                // buffer qb holds items qb, qb + 2, ...: its (item_it / 2)-th use
                const uint32_t qb = item_it & 1, qph = (item_it >> 1) & 1;
                if (!mbar_wait(&q_empty[qb], qph ^ 1, abort_flag, p.err)) break;
                mbar_arrive_expect_tx(&q_full[qb], Cfg::kTileBytes);
                tma_load_2d(sQ + qb * Cfg::kTileBytes, &tmq, p.q_col0 + it.h * DH, it.q_row0, &q_full[qb]);
                const int nkt = (it.nk + 127) / 128;
                for (int j = 0; j < nkt; ++j, ++kv_it) {
                    const int s = kv_it % kKVStages;
                    const uint32_t ph = (kv_it / kKVStages) & 1;
                    if (!mbar_wait(&kv_empty[s], ph ^ 1, abort_flag, p.err)) {
                        ok = false;
                        break;
                    }
                    // fault injection (tests of the failure path): the last
                    // key tile of CTA 0's first item is never loaded, so the
                    // waits on it (and on what follows it) run out while the
                    // earlier tiles went through, and the kernel aborts
                    if (p.fault_skip_kv && blockIdx.x == 0 && item_it == 0 && j == nkt - 1) continue;
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
        // Barrier reads take a long time even when the phase is complete, so
        // each tile tests its two barriers back to back (one exposed
        // latency) and takes the bounded wait only if a test fails; the
        // steady-state loop carries no other branches.  Every lane runs the
        // loop (a converged warp keeps the descriptors warp-uniform) and
        // takes each barrier outcome as a warp vote.
        {
            constexpr uint32_t idesc_s = make_idesc_bf16(128, 128, 0, 0);
            constexpr uint32_t idesc_o = make_idesc_bf16(128, DH, 0, 1);
            // descriptors of the stage bases; a K step of 16 elements inside a
            // 128B / 64B swizzle atom advances the start address by 32 bytes,
            // i.e. the descriptor by 2
            const uint64_t q_desc0 = make_sdesc(smem_u32(sQ), 16, Cfg::kAtom, Cfg::kSwz);
            uint64_t q_desc = q_desc0;  // this item's Q buffer
            const uint64_t k_desc0 = make_sdesc(smem_u32(sK), 16, Cfg::kAtom, Cfg::kSwz);
            const uint64_t v_desc0 = make_sdesc(smem_u32(sV), Cfg::kAtom, Cfg::kAtom, Cfg::kSwz);
            constexpr uint64_t kStageStep = Cfg::kTileBytes >> 4, kVRowStep = (16 * Cfg::kRowBytes) >> 4;
            // S_gt = Q K_gt^T into S buffer gt % 2.  Only an item's first two
            // tiles commit to s_full; a later tile's S is issued just before
            // P V of the tile two back and reported by that P V's commit
            auto s_mmas = [&](uint32_t gt, bool commit) {
                const uint64_t kd = k_desc0 + (gt % kKVStages) * kStageStep;
#pragma unroll
                for (int kk = 0; kk < DH / 16; ++kk)
                    mma_bf16_elect(tmem + (gt & 1) * 128, q_desc + 2 * kk, kd + 2 * kk, idesc_s, kk > 0);
                if (commit) mma_commit_elect(&s_full[gt & 1]);
            };
            // O_e (+)= P_e V for tile gt of parity e = gt % 2, P_e read from
            // TMEM (8 columns per 16 keys); `fresh` overwrites O_e (the item's
            // first tile of each parity)
            auto pv_mmas = [&](uint32_t gt, bool fresh) {
                const uint32_t pb = gt & 1;
                const uint64_t vd = v_desc0 + (gt % kKVStages) * kStageStep;
#pragma unroll
                for (int kk = 0; kk < 8; ++kk)  // keys 16kk..16kk+15
                    mma_bf16_ts_elect(tmem + Cfg::kColO + pb * DH, tmem + Cfg::kColP + pb * 64 + kk * 8,
                                vd + kk * kVRowStep, idesc_o, !(fresh && kk == 0));
                mma_commit_elect(&kv_empty[gt % kKVStages]);
            };
            auto kv_ready = [&](uint32_t gt) { return warp_all(mbar_test(&kv_full[gt % kKVStages], (gt / kKVStages) & 1)); };
            auto kv_wait = [&](uint32_t gt) {
                return warp_all(mbar_wait(&kv_full[gt % kKVStages], (gt / kKVStages) & 1, abort_flag, p.err));
            };
            auto p_ready = [&](uint32_t gt) { return warp_all(mbar_test(&p_full[gt & 1], (gt >> 1) & 1)); };
            auto p_wait = [&](uint32_t gt) { return warp_all(mbar_wait(&p_full[gt & 1], (gt >> 1) & 1, abort_flag, p.err)); };
            uint32_t g = 0, item_it = 0;  // global key tile at the start of the item
            bool ok = true;
            // every item has at least one key tile: a sample without active
            // tokens owns no query tile, and the entry points reject nk < 1
            for (int w = blockIdx.x; w < total && ok; w += gridDim.x, ++item_it) {
                const Item it = decode_item(p, w);
                const uint32_t nkt = (uint32_t)((it.nk + 127) / 128);
                // S of the first two tiles: their S buffers were freed by the
                // previous item's P (waited on before its P V)
                const uint32_t qb = item_it & 1;
                if (!warp_all(mbar_wait(&q_full[qb], (item_it >> 1) & 1, abort_flag, p.err))) break;
                q_desc = q_desc0 + qb * (Cfg::kTileBytes >> 4);
                if (!kv_wait(g)) break;
                tc_fence_after();
                s_mmas(g, true);
                if (nkt > 1) {
                    if (!kv_wait(g + 1)) break;
                    tc_fence_after();
                    s_mmas(g + 1, true);
                }
                // O_0 / O_1 are overwritten by this item's first P V: the
                // softmax must have read the previous item's result
                if (!warp_all(mbar_wait(o_free, (item_it & 1) ^ 1, abort_flag, p.err))) break;
                // steady state: P_j ready -> S_(j+2), P V_j
                uint32_t j = 0;
                for (; j + 2 < nkt; ++j) {
                    const uint32_t gt = g + j;
                    const bool r = p_ready(gt) & kv_ready(gt + 2);
                    if (!r && !(p_wait(gt) && kv_wait(gt + 2))) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    s_mmas(gt + 2, false);
                    pv_mmas(gt, j < 2);  // its commit also reports S_(gt+2)
                }
                if (!ok) break;
                mma_commit_elect(&q_empty[qb]);  // every S of the item issued: its Q buffer may be refilled
                for (; j < nkt; ++j) {
                    const uint32_t gt = g + j;
                    if (!p_ready(gt) && !p_wait(gt)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    pv_mmas(gt, j < 2);
                }
                g += nkt;
            }
        }
    } else {
        // ------------------------------------------------ softmax warps
        const int q = warp & 3;                // TMEM lane quarter of this warp
        const int par = (warp - 2) >> 2;       // key tiles g with g % 2 == par
        const int row = q * 32 + lane;
        const uint32_t tl = (uint32_t)(q * 32) << 16;
        const uint32_t s_addr = tmem + tl + par * 128;
        const uint32_t o_addr = tmem + tl + Cfg::kColO + par * DH;
        const uint32_t p_addr = tmem + tl + Cfg::kColP + par * 64;
        uint32_t g = 0, item_it = 0;  // global key-tile counter at the start of the item
        uint32_t s_use = 0;           // s_full[par] completions consumed
        uint32_t item_k = 0;          // items finished (hand-over barrier phases)
        // S of an item's first tile of this parity completes s_full[par]
        // (once per item in which the parity has a tile; s_use counts them);
        // S of every later tile t is reported with P V of tile t - 2 on
        // kv_empty[(t - 2) % 4] (parity ((t - 2) / 4) % 2), which also frees
        // P and O for tile t.  A warp waits for P V of its previous tile
        // before it writes P again, and P V of its next tile cannot start
        // before that, so no barrier it reads is ever more than one phase
        // ahead of it.
        for (int w = blockIdx.x; w < total; w += gridDim.x, ++item_it) {
            const Item it = decode_item(p, w);
            const int nkt = (it.nk + 127) / 128;
            float m_ref = -INFINITY, l_run = 0.f;
            bool ok = true, any = false;
            uint32_t g_last = 0;
            for (int j = (int)((par - g) & 1); j < nkt; j += 2) {
                const uint32_t gt = g + (uint32_t)j;
                const bool first = j < 2;  // S reported on s_full, else with P V of tile gt - 2
                if (!warp_all(first ? mbar_wait(&s_full[par], (s_use++) & 1, abort_flag, p.err)
                                    : mbar_wait(&kv_empty[(gt - 2) % kKVStages], ((gt - 2) / kKVStages) & 1,
                                                abort_flag, p.err))) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                // pass 1: the tile's maximum (S stays in TMEM for pass 2)
                const int valid = it.nk - j * 128;  // < 128 only on the last, ragged key tile
                float mx4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
                for (int hb = 0; hb < 2; ++hb) {  // two halves of 64 keys
                    uint32_t r0[32], r1[32];
                    tmem_ld32(s_addr + 64 * hb, r0);
                    tmem_ld32(s_addr + 64 * hb + 32, r1);
                    tmem_wait_ld();
                    float sv[64];
#pragma unroll
                    for (int c = 0; c < 32; ++c) {
                        sv[c] = __uint_as_float(r0[c]);
                        sv[32 + c] = __uint_as_float(r1[c]);
                    }
                    if (valid < 128) {
#pragma unroll
                        for (int c = 0; c < 64; ++c)
                            if (64 * hb + c >= valid) sv[c] = -INFINITY;
                    }
                    // four independent chains of three-input maxima
#pragma unroll
                    for (int c = 0; c < 64; c += 8) {
#pragma unroll
                        for (int e = 0; e < 4; ++e) mx4[e] = fmax3(mx4[e], sv[c + e], sv[c + 4 + e]);
                    }
                }
                const float mx = fmax3(mx4[0], mx4[1], fmaxf(mx4[2], mx4[3])) * p.scale_log2;
                // raise the reference max only when it grew by more than 2^8
                // (warp-uniform: TMEM loads / stores are warp-collective); O
                // and l are rescaled once P V of this parity's previous tile
                // is done
                const bool raise = __any_sync(0xffffffffu, mx > m_ref + 8.0f);
                float alpha = 1.f;
                if (raise) {
                    const float m_new = fmaxf(m_ref, mx);
                    alpha = exp2_fast(m_ref - m_new);
                    m_ref = m_new;
                }
                const float m_use = m_ref == -INFINITY ? 0.f : m_ref;
                // P_par and O_par: P V of this parity's previous tile must be done
                if (first && gt >= 2 &&
                    !warp_all(mbar_wait(&kv_empty[(gt - 2) % kKVStages], ((gt - 2) / kKVStages) & 1, abort_flag,
                                        p.err))) {
                    ok = false;
                    break;
                }
                if (raise && any) {  // O_par holds this parity's earlier tiles: rescale in place
                    tc_fence_after();
#pragma unroll
                    for (int d0 = 0; d0 < DH; d0 += 16) {
                        uint32_t r[16];
                        tmem_ld16(o_addr + d0, r);
                        tmem_wait_ld();
#pragma unroll
                        for (int d = 0; d < 16; ++d) r[d] = __float_as_uint(__uint_as_float(r[d]) * alpha);
                        tmem_st16(o_addr + d0, r);
                    }
                    l_run *= alpha;
                }
                // pass 2: exponent arguments and row sums two lanes per paired
                // instruction; P goes to TMEM as bf16 pairs (keys 2c, 2c+1
                // in column c, the lower key in the low half)
                f32x2 sum0 = {0.f, 0.f}, sum1 = {0.f, 0.f};
                const f32x2 sc2 = {p.scale_log2, p.scale_log2}, nm2 = {-m_use, -m_use};
#pragma unroll
                for (int hb = 0; hb < 2; ++hb) {  // keys [64 hb, 64 hb + 64) -> columns [32 hb, 32 hb + 32)
                    float sv[64];
                    {
                        uint32_t r0[32], r1[32];
                        tmem_ld32(s_addr + 64 * hb, r0);
                        tmem_ld32(s_addr + 64 * hb + 32, r1);
                        tmem_wait_ld();
#pragma unroll
                        for (int c = 0; c < 32; ++c) {
                            sv[c] = __uint_as_float(r0[c]);
                            sv[32 + c] = __uint_as_float(r1[c]);
                        }
                    }
                    if (valid < 128) {
#pragma unroll
                        for (int c = 0; c < 64; ++c)
                            if (64 * hb + c >= valid) sv[c] = -INFINITY;
                    }
                    uint32_t pw[32];
#pragma unroll
                    for (int c = 0; c < 32; c += 2) {
                        const int k0 = 2 * c;
                        const f32x2 x0 = ffma2({sv[k0], sv[k0 + 1]}, sc2, nm2);
                        const f32x2 x1 = ffma2({sv[k0 + 2], sv[k0 + 3]}, sc2, nm2);
                        const f32x2 e0 = {exp2_fast(x0.x), exp2_fast(x0.y)};
                        const f32x2 e1 = {exp2_fast(x1.x), exp2_fast(x1.y)};
                        sum0 = fadd2(sum0, e0);
                        sum1 = fadd2(sum1, e1);
                        pw[c] = pack_bf16x2(e0.x, e0.y);
                        pw[c + 1] = pack_bf16x2(e1.x, e1.y);
                    }
                    tmem_st32(p_addr + 32 * hb, pw);
                }
                tmem_wait_st();
                l_run += (sum0.x + sum0.y) + (sum1.x + sum1.y);
                tc_fence_before();  // P (and a rescaled O) written before P V may start
                __syncwarp();
                if (lane == 0) mbar_arrive(&p_full[par]);
                any = true;
                g_last = gt;
            }
            // the parity of the item's last tile combines and stores the
            // item; the other one finished a tile earlier and only hands over
            // its (m, l, O), then goes on to the next item's first tile (which
            // is its own: tiles alternate parity across items too)
            const bool combiner = ((g + (uint32_t)nkt - 1u) & 1u) == (uint32_t)par;
            g += (uint32_t)nkt;
            // every P V of this parity done: read O_par, release it (a parity
            // without tiles in this item contributes m = -inf, l = 0, O = 0)
            float acc[DH];
#pragma unroll
            for (int d = 0; d < DH; ++d) acc[d] = 0.f;
            if (ok && any &&
                !warp_all(mbar_wait(&kv_empty[g_last % kKVStages], (g_last / kKVStages) & 1, abort_flag, p.err)))
                ok = false;
            if (ok && any) {
                tc_fence_after();
#pragma unroll
                for (int d0 = 0; d0 < DH; d0 += 32) {
                    uint32_t r[32];
                    tmem_ld32(o_addr + d0, r);
                    tmem_wait_ld();
#pragma unroll
                    for (int d = 0; d < 32; ++d) acc[d0 + d] = __uint_as_float(r[d]);
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(o_free);
            // Hand-over through shared memory, per TMEM lane quarter q (one
            // warp of each parity): comb_full[q] completes once per item when
            // the other parity's 32 rows are written, comb_free[q] once per
            // item when the combiner has read them (so the next item's
            // writer may overwrite them).  float4 d4 of row r sits at
            // r * DH + 4 (d4 ^ (r % (DH / 4))), so a warp's row-per-lane
            // accesses hit distinct banks.  Every wait is bounded; after one
            // gave up (the kernel is aborting) the warp leaves the item loop.
            const uint32_t ph = item_k & 1u;
            ++item_k;
            constexpr int kV4 = DH / 4;  // float4 slots of a row
            float4 *slot = reinterpret_cast<float4 *>(sComb + row * DH);
            if (!ok) break;
            if (!combiner) {
                if (!warp_all(mbar_wait(&comb_free[q], ph ^ 1u, abort_flag, p.err))) break;
                sML[row] = make_float2(m_ref, l_run);
#pragma unroll
                for (int d4 = 0; d4 < kV4; ++d4)
                    slot[d4 ^ (row & (kV4 - 1))] = make_float4(acc[4 * d4], acc[4 * d4 + 1], acc[4 * d4 + 2], acc[4 * d4 + 3]);
                mbar_arrive(&comb_full[q]);  // every lane: its own row is released
                continue;
            }
            if (!warp_all(mbar_wait(&comb_full[q], ph, abort_flag, p.err))) break;
            // O = (O_0 2^(m_0-m) + O_1 2^(m_1-m)) / (l_0 2^(m_0-m) + l_1 2^(m_1-m)),
            // in this order whichever parity combines
            const float2 other = sML[row];
            const float m0 = par == 0 ? m_ref : other.x, l0 = par == 0 ? l_run : other.y;
            const float m1 = par == 0 ? other.x : m_ref, l1 = par == 0 ? other.y : l_run;
            const float m = fmaxf(m0, m1);
            const float a0 = exp2_fast(m0 - m), a1 = exp2_fast(m1 - m);
            const float inv = 1.0f / (l0 * a0 + l1 * a1);
            const int orow = it.q_row0 + row;
            if (orow < it.store_end) {
                uint4 *dst = reinterpret_cast<uint4 *>(p.out + (size_t)orow * p.ldo + it.h * DH);
                if (par == 0)
                    combine_row<DH, false>(acc, slot, row, a0, a1, inv, dst);
                else
                    combine_row<DH, true>(acc, slot, row, a0, a1, inv, dst);
            }
            mbar_arrive(&comb_free[q]);  // every lane: its row was read
        }
    }
    __syncthreads();
    if (*abort_flag) {
        if (warp == 1) {
            mma_commit_elect(drain);  // the MMAs' issuing lane
            if (lane == 0) wait_bounded(drain, 0, 100000000ull);
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
    // the shared-memory attribute is per device: set it on each device's first launch
    static std::atomic<uint64_t> attr_devices{0};
    const size_t smem = AttnCfg<DH>::kSmem;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const uint64_t bit = 1ull << (dev & 63);
    if (!(attr_devices.load(std::memory_order_acquire) & bit)) {
        e = cudaFuncSetAttribute(k_attn_one<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        attr_devices.fetch_or(bit, std::memory_order_acq_rel);
    }
    launch_k(k_attn_one<DH>, dim3(grid), dim3(kAttnThreads), smem, s, *tq, *tk, *tv, p);
    return cudaGetLastError();
}

}  // namespace


cudaError_t launch_attention_one(const CUtensorMap *tq, const CUtensorMap *tk, const CUtensorMap *tv,
                                 const AttnParams &p, int grid, cudaStream_t s)
{
    if (grid < 1) return cudaErrorInvalidValue;
    if (p.dh == 64) return launch_dh<64>(tq, tk, tv, p, grid, s);
    if (p.dh == 32) return launch_dh<32>(tq, tk, tv, p, grid, s);
    return cudaErrorInvalidValue;
}

}  // namespace f3dc
