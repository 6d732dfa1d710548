// k_attn.cu -- K5 / K6: multi-head attention softmax(Q K^T / sqrt(dh)) V on
// 5th-generation tensor cores, flash style (online softmax), for
//   mode 0  self-attention of every sample among its ACTIVE tokens only
//           (Sec. 4.2: attention runs on the compacted active subset)
//   mode 1  cross-attention of the active tokens to the sample's condition
//           tokens (Supp. Sec. F cross-attention)
//   mode 2  one sequence (diagnostic entry point)
//
// Persistent kernel, one CTA per SM (320 threads).  A work item is two
// 128-query tiles A and B of one head that share their keys: the K / V tiles
// are loaded once for both, and the two tiles' score / softmax / P V chains
// run side by side, so while one tile's softmax works the tensor core serves
// the other's MMAs.
//   warp 0     TMA producer: the item's two Q tiles (double-buffered across
//              items), K / V tiles of 128 keys into a 4-deep ring
//   warp 1     TMEM allocator + tcgen05.mma issuer (the whole warp runs the
//              loop and votes on every barrier outcome; elect.sync issues).
//              Per key tile j:  S_A(j), S_B(j)   (S_t = Q_t K_j^T, N=128,
//              K=dh; each once the softmax has loaded the previous S_t),
//              then P_A V(j-1), P_B V(j-1)        (O_t += P_t V, N=dh, K=128,
//              each once P_t is written; P read straight from TMEM)
//   warps 2-5  softmax of tile A, warps 6-9 of tile B: one thread per query
//              row (TMEM lane = row), all 128 keys of each key tile, online
//              softmax with the row's running max m and sum l, in one pass
//              over the key tile's two halves of 64 keys: each half is
//              loaded once, its maximum raises the reference max m only when
//              it exceeds m by more than 2^8 (O_t, l rescaled in place; a
//              raise in the second half recomputes the first half's P), and
//              P = exp2(S scale - m) goes to TMEM P_t as bf16 pairs (once
//              P V of the previous key tile has read P_t).  The S buffer is
//              released for the next key tile's MMA as soon as its last load
//              landed.  O_t stays in TMEM for the whole item; at the item's
//              end O_t / l is stored as bf16.
// TMEM: S_A S_B (fp32, 128 columns each) | O_A O_B (dh each) | P_A P_B (64).
// V is the MN-major B operand of the P V MMA straight from its row-major
// TMA tile.  Keys beyond a sample's count are masked to -inf before the
// exponent; padding rows are finite by construction, so 0 * pad = 0.
#include <atomic>

#include "common.cuh"
#include "kernels.h"

namespace f3dc {

namespace {

constexpr int kAttnThreads = 320;  // producer, MMA issuer, 2 x 4 softmax warps
constexpr int kKVStages = 4;

template <int DH>
struct AttnCfg {
    static constexpr int kRowBytes = DH * 2;            // 128 (DH 64) or 64 (DH 32)
    static constexpr int kTileBytes = 128 * kRowBytes;  // Q, K or V tile
    static constexpr uint32_t kAtom = 8 * kRowBytes;    // 8-row swizzle atom
    static constexpr uint32_t kSwz = DH == 64 ? kSwizzle128 : kSwizzle64;
    static constexpr size_t kSmem = 1024 + kTileBytes * (4 + 2 * kKVStages) + 256;
    // TMEM columns: S_A S_B (fp32, 128 each) | O_A O_B (fp32, DH each) |
    // P_A P_B (bf16 pairs, 64 each)
    static constexpr uint32_t kColO = 256, kColP = 256 + 2 * DH;
    static constexpr uint32_t kTmemCols = 512;
    static_assert(kColP + 128 <= kTmemCols, "TMEM layout");
};

// The key rows of query tile t: the sample's active tokens (self-attention),
// the sample's condition tokens (cross-attention) or the one sequence.
F3DC_DEV void tile_keys(const AttnParams &p, int t, int &kv_row0, int &nk)
{
    if (p.mode == 0) {
        const int b = p.tile_sample[t];
        kv_row0 = p.plan->row_off[b];
        nk = p.plan->n_active[b];
    } else if (p.mode == 1) {
        const int b = p.tile_sample[t];
        kv_row0 = (p.kv_null_from > 0 && b >= p.kv_null_from ? p.kv_null_sample : b) * p.nk_fixed;
        nk = p.nk_fixed;
    } else {
        kv_row0 = 0;
        nk = p.nk_fixed;
    }
}

struct Item {
    int q_row0, kv_row0, nk, h, store_end;  // q_row0: tile A's first row (B follows)
    bool store[2];
};

// Work item w: query tiles A = 2 pt and B = 2 pt + 1 of head h, for the
// first n_pt heads items (n_pt = tile pairs).  The two tiles share the keys,
// so a pair whose tiles have different keys (two samples meet inside it)
// runs twice: the first pass with tile A's keys stores only A's rows, a
// second pass (items n_pt heads .. 2 n_pt heads - 1) with tile B's keys
// stores only B's; any other second-pass item is skipped (returns false).
// Rows of a tile beyond the tile count are computed and never stored.
F3DC_DEV bool decode_item(const AttnParams &p, int w, int n_tiles, Item &it)
{
    it.store_end = p.mode == 2 ? p.q_rows : 0x7FFFFFFF;
    const int per_pass = ((n_tiles + 1) >> 1) * p.heads;
    const int pass = w >= per_pass ? 1 : 0;
    const int w2 = w - pass * per_pass;
    const int pt = w2 / p.heads;
    it.h = w2 - pt * p.heads;
    const int t0 = 2 * pt;
    const bool has1 = t0 + 1 < n_tiles;
    int r0, n0, r1, n1;
    tile_keys(p, t0, r0, n0);
    if (has1) {
        tile_keys(p, t0 + 1, r1, n1);
    } else {
        r1 = r0;
        n1 = n0;
    }
    const bool mixed = r1 != r0 || n1 != n0;
    if (pass == 1 && !mixed) return false;
    it.kv_row0 = pass ? r1 : r0;
    it.nk = pass ? n1 : n0;
    it.q_row0 = t0 * 128;
    it.store[0] = pass == 0;
    it.store[1] = has1 && (pass == 1 || !mixed);
    return true;
}

F3DC_DEV int total_items(const AttnParams &p, int n_tiles) { return 2 * ((n_tiles + 1) >> 1) * p.heads; }

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
    // Q: two items' pairs of tiles (item i in buffer i % 2, tile A then B)
    uint8_t *sQ = smem;
    uint8_t *sK = sQ + 4 * Cfg::kTileBytes;
    uint8_t *sV = sK + kKVStages * Cfg::kTileBytes;
    uint64_t *bars = reinterpret_cast<uint64_t *>(sV + kKVStages * Cfg::kTileBytes);
    uint64_t *q_full = bars, *q_empty = bars + 2;
    uint64_t *kv_full = bars + 4, *kv_empty = kv_full + kKVStages;
    // per query tile t (0 = A, 1 = B), once per key tile: S_t written
    // (s_full), S_t read by the softmax (s_free), P_t written (p_full), P_t V
    // done (pv_done); once per item: O_t read (o_free)
    uint64_t *s_full = kv_empty + kKVStages, *s_free = s_full + 2, *p_full = s_free + 2, *pv_done = p_full + 2;
    uint64_t *o_free = pv_done + 2;
    uint64_t *drain = o_free + 2;
    uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(drain + 1);
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
        for (int t = 0; t < 2; ++t) {
            mbar_init(&s_full[t], 1);
            mbar_init(&s_free[t], 4);  // the four softmax warps of tile t
            mbar_init(&p_full[t], 4);
            mbar_init(&pv_done[t], 1);
            mbar_init(&o_free[t], 4);
        }
        mbar_init(drain, 1);
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
    const int total = total_items(p, n_tiles);

    if (warp == 0) {
        // ------------------------------------------------ TMA producer
        if (lane == 0) {
            tma_prefetch(&tmq);
            tma_prefetch(&tmk);
            tma_prefetch(&tmv);
            uint32_t kv_it = 0, item_it = 0;
            bool ok = true;
            for (int w = blockIdx.x; w < total && ok; w += gridDim.x) {
                Item it;
                if (!decode_item(p, w, n_tiles, it)) continue;
                const uint32_t my_it = item_it++;
                // Q buffer qb holds items qb, qb + 2, ...: its (my_it / 2)-th use
                const uint32_t qb = my_it & 1, qph = (my_it >> 1) & 1;
                if (!mbar_wait(&q_empty[qb], qph ^ 1, abort_flag, p.err)) break;
                mbar_arrive_expect_tx(&q_full[qb], 2 * Cfg::kTileBytes);
                for (int t = 0; t < 2; ++t)
                    tma_load_2d(sQ + (2 * qb + t) * Cfg::kTileBytes, &tmq, p.q_col0 + it.h * DH, it.q_row0 + 128 * t,
                                &q_full[qb]);
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
                    if (p.fault_skip_kv && blockIdx.x == 0 && my_it == 0 && j == nkt - 1) continue;
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
        // Every lane runs the loop (a converged warp keeps the descriptors
        // warp-uniform) and takes each barrier outcome as a warp vote;
        // elect.sync issues.  Key tile g (counted over the CTA's whole run)
        // sits in K/V stage g % kKVStages; every barrier here completes once
        // per key tile (or per item), so its phase parity follows from g.
        {
            constexpr uint32_t idesc_s = make_idesc_bf16(128, 128, 0, 0);
            constexpr uint32_t idesc_o = make_idesc_bf16(128, DH, 0, 1);
            // descriptors of the stage bases; a K step of 16 elements inside a
            // 128B / 64B swizzle atom advances the start address by 32 bytes,
            // i.e. the descriptor by 2
            const uint64_t q_desc0 = make_sdesc(smem_u32(sQ), 16, Cfg::kAtom, Cfg::kSwz);
            const uint64_t k_desc0 = make_sdesc(smem_u32(sK), 16, Cfg::kAtom, Cfg::kSwz);
            const uint64_t v_desc0 = make_sdesc(smem_u32(sV), Cfg::kAtom, Cfg::kAtom, Cfg::kSwz);
            constexpr uint64_t kStageStep = Cfg::kTileBytes >> 4, kVRowStep = (16 * Cfg::kRowBytes) >> 4;
            auto wait = [&](uint64_t *bar, uint32_t ph) { return warp_all(mbar_wait(bar, ph, abort_flag, p.err)); };
            uint32_t g = 0, item_it = 0;
            bool ok = true;
            for (int w = blockIdx.x; w < total && ok; w += gridDim.x) {
                Item it;
                if (!decode_item(p, w, n_tiles, it)) continue;
                const uint32_t my_it = item_it++;
                const uint32_t nkt = (uint32_t)((it.nk + 127) / 128);
                const uint32_t qb = my_it & 1;
                if (!wait(&q_full[qb], (my_it >> 1) & 1)) break;
                // step j: S of key tile j (j < nkt), then P V of key tile j - 1
                // (j >= 1); every item has at least one key tile (a sample
                // without active tokens owns no query tile, and the entry
                // points reject nk < 1)
                for (uint32_t j = 0; j <= nkt && ok; ++j) {
                    if (j < nkt) {
                        // S_A and S_B of key tile gt, each once the softmax
                        // has read the previous S of its tile
                        const uint32_t gt = g + j;
                        if (!wait(&kv_full[gt % kKVStages], (gt / kKVStages) & 1)) {
                            ok = false;
                            break;
                        }
                        const uint64_t kd = k_desc0 + (gt % kKVStages) * kStageStep;
                        for (int t = 0; t < 2; ++t) {
                            if (!wait(&s_free[t], (gt & 1) ^ 1)) {
                                ok = false;
                                break;
                            }
                            tc_fence_after();
                            const uint64_t qd = q_desc0 + (uint64_t)(2 * qb + t) * kStageStep;
#pragma unroll
                            for (int kk = 0; kk < DH / 16; ++kk)
                                mma_bf16_elect(tmem + t * 128, qd + 2 * kk, kd + 2 * kk, idesc_s, kk > 0);
                            mma_commit_elect(&s_full[t]);
                        }
                        if (!ok) break;
                        if (j + 1 == nkt) mma_commit_elect(&q_empty[qb]);  // every S of the item issued
                    }
                    if (j >= 1) {
                        // P_t V of key tile gp, once P_t is written
                        const uint32_t gp = g + j - 1;
                        const bool fresh = j == 1;
                        const uint64_t vd = v_desc0 + (gp % kKVStages) * kStageStep;
                        for (int t = 0; t < 2; ++t) {
                            // the item's first P V overwrites O_t: the softmax
                            // must have read the previous item's
                            if (fresh && !wait(&o_free[t], (my_it & 1) ^ 1)) {
                                ok = false;
                                break;
                            }
                            if (!wait(&p_full[t], gp & 1)) {
                                ok = false;
                                break;
                            }
                            tc_fence_after();
#pragma unroll
                            for (int kk = 0; kk < 8; ++kk)
                                mma_bf16_ts_elect(tmem + Cfg::kColO + t * DH, tmem + Cfg::kColP + t * 64 + kk * 8,
                                                  vd + kk * kVRowStep, idesc_o, !(fresh && kk == 0));
                            mma_commit_elect(&pv_done[t]);
                        }
                        if (!ok) break;
                        mma_commit_elect(&kv_empty[gp % kKVStages]);  // both tiles' S and P V of the stage issued
                    }
                }
                g += nkt;
            }
        }
    } else {
        // ------------------------------------------------ softmax warps
        const int q = warp & 3;              // TMEM lane quarter of this warp
        const int t = (warp - 2) >> 2;       // query tile: warps 2-5 A, 6-9 B
        const int row = q * 32 + lane;
        const uint32_t tl = (uint32_t)(q * 32) << 16;
        const uint32_t s_addr = tmem + tl + t * 128;
        const uint32_t o_addr = tmem + tl + Cfg::kColO + t * DH;
        const uint32_t p_addr = tmem + tl + Cfg::kColP + t * 64;
        auto wait = [&](uint64_t *bar, uint32_t ph) { return warp_all(mbar_wait(bar, ph, abort_flag, p.err)); };
        // S_t of key tile g completes s_full[t] (phase g), the four warps'
        // arrivals on s_free[t] / p_full[t] complete phase g once S_t is
        // loaded / P_t written, and P_t V of tile g completes pv_done[t]; a
        // wait that gives up (the kernel is aborting) ends this warp's loop
        uint32_t g = 0;  // key tiles of this CTA's earlier items
        for (int w = blockIdx.x; w < total; w += gridDim.x) {
            Item it;
            if (!decode_item(p, w, n_tiles, it)) continue;
            const int nkt = (it.nk + 127) / 128;
            float m_ref = -INFINITY, l_run = 0.f;
            bool ok = true;
            for (int j = 0; j < nkt; ++j) {
                const uint32_t gt = g + (uint32_t)j;
                if (!wait(&s_full[t], gt & 1)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                // one pass over the tile's two halves of 64 keys: load, take the
                // half's maximum, raise the reference max when it grew by more
                // than 2^8 (warp-uniform), then exponents against it.  A raise
                // in the second half makes the first half's P stale: its S is
                // still in TMEM (released only after this check), so it is
                // recomputed against the new max.
                const int valid = it.nk - j * 128;  // < 128 only on the last, ragged key tile
                f32x2 sum0 = {0.f, 0.f}, sum1 = {0.f, 0.f};
                bool pv_ready = gt == 0;  // P V of the previous key tile done (P_t, O_t free)
                bool o_live = j > 0;      // O_t holds this item's earlier tiles
                auto ensure_pv = [&]() {
                    if (!pv_ready) {
                        pv_ready = wait(&pv_done[t], (gt - 1) & 1);
                        if (!pv_ready) ok = false;
                    }
                    return pv_ready;
                };
                auto rescale = [&](float alpha) {
                    if (o_live) {
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
                    }
                    l_run *= alpha;
                };
                // exponents of one half against m_ref, P to TMEM as bf16 pairs
                auto emit_half = [&](int hb, const float (&sv)[64]) {
                    const float m_use = m_ref == -INFINITY ? 0.f : m_ref;
                    const f32x2 sc2 = {p.scale_log2, p.scale_log2}, nm2 = {-m_use, -m_use};
                    f32x2 s0 = {0.f, 0.f}, s1 = {0.f, 0.f};
                    uint32_t pw[32];
#pragma unroll
                    for (int c = 0; c < 32; c += 2) {
                        const int k0 = 2 * c;
                        const f32x2 x0 = ffma2({sv[k0], sv[k0 + 1]}, sc2, nm2);
                        const f32x2 x1 = ffma2({sv[k0 + 2], sv[k0 + 3]}, sc2, nm2);
                        const f32x2 e0 = {exp2_fast(x0.x), exp2_fast(x0.y)};
                        const f32x2 e1 = {exp2_fast(x1.x), exp2_fast(x1.y)};
                        s0 = fadd2(s0, e0);
                        s1 = fadd2(s1, e1);
                        pw[c] = pack_bf16x2(e0.x, e0.y);
                        pw[c + 1] = pack_bf16x2(e1.x, e1.y);
                    }
                    if (!ensure_pv()) return;
                    tmem_st32(p_addr + 32 * hb, pw);
                    if (hb == 0) {
                        sum0 = s0;
                        sum1 = s1;
                    } else {
                        sum0 = fadd2(sum0, s0);
                        sum1 = fadd2(sum1, s1);
                    }
                };
                auto load_half = [&](int hb, float (&sv)[64]) {
                    uint32_t r0[32], r1[32];
                    tmem_ld32(s_addr + 64 * hb, r0);
                    tmem_ld32(s_addr + 64 * hb + 32, r1);
                    tmem_wait_ld();
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
                };
                auto half_max = [&](const float (&sv)[64]) {
                    float mx4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
                    for (int c = 0; c < 64; c += 8) {
#pragma unroll
                        for (int e = 0; e < 4; ++e) mx4[e] = fmax3(mx4[e], sv[c + e], sv[c + 4 + e]);
                    }
                    return fmax3(mx4[0], mx4[1], fmaxf(mx4[2], mx4[3])) * p.scale_log2;
                };
                // raise m_ref to cover mx when it grew by more than 2^8; O_t and
                // l are rescaled (P V of the previous key tile must be done)
                auto maybe_raise = [&](float mx) {
                    if (!__any_sync(0xffffffffu, mx > m_ref + 8.0f)) return false;
                    const float m_new = fmaxf(m_ref, mx);
                    const float alpha = exp2_fast(m_ref - m_new);
                    m_ref = m_new;
                    if (ensure_pv()) rescale(alpha);
                    return true;
                };
                {
                    float sv[64];
                    load_half(0, sv);
                    maybe_raise(half_max(sv));
                    if (!ok) break;
                    emit_half(0, sv);
                    if (!ok) break;
                }
                {
                    float sv[64];
                    load_half(1, sv);
                    const bool raised = maybe_raise(half_max(sv));
                    if (!ok) break;
                    if (raised) {
                        // the first half's P is against the old max: redo it
                        float sv0[64];
                        load_half(0, sv0);
                        emit_half(0, sv0);
                        if (!ok) break;
                    }
                    // S_t fully read: the next key tile's S may overwrite it
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&s_free[t]);
                    emit_half(1, sv);
                    if (!ok) break;
                }
                tmem_wait_st();
                l_run += (sum0.x + sum0.y) + (sum1.x + sum1.y);
                tc_fence_before();  // P (and a rescaled O) written before P V may start
                __syncwarp();
                if (lane == 0) mbar_arrive(&p_full[t]);
            }
            if (!ok) break;
            g += (uint32_t)nkt;
            // every P V of the item done: O_t / l, stored as bf16
            if (!wait(&pv_done[t], (g - 1) & 1)) break;
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
            if (lane == 0) mbar_arrive(&o_free[t]);
            const int orow = it.q_row0 + 128 * t + row;
            if (it.store[t] && orow < it.store_end) {
                const float inv = 1.0f / l_run;
                uint4 *dst = reinterpret_cast<uint4 *>(p.out + (size_t)orow * p.ldo + it.h * DH);
#pragma unroll
                for (int d = 0; d < DH; d += 8) {
                    uint4 u;
                    u.x = pack_bf16x2(acc[d] * inv, acc[d + 1] * inv);
                    u.y = pack_bf16x2(acc[d + 2] * inv, acc[d + 3] * inv);
                    u.z = pack_bf16x2(acc[d + 4] * inv, acc[d + 5] * inv);
                    u.w = pack_bf16x2(acc[d + 6] * inv, acc[d + 7] * inv);
                    dst[d / 8] = u;
                }
            }
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
        e = cudaFuncSetAttribute(k_attn<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        attr_devices.fetch_or(bit, std::memory_order_acq_rel);
    }
    launch_k(k_attn<DH>, dim3(grid), dim3(kAttnThreads), smem, s, *tq, *tk, *tv, p);
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
