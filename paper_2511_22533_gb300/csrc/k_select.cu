// k_select.cu -- K1: Spatiotemporal Stability Criterion scoring and
// lowest-c selection (Sec. 4.1 V_i and Eq. ICE; Sec. 4.2 Eq. ssc and
// Eq. normalize; Algorithm 1 function SSC), fused with the row plan of the
// step (Sec. 4.2 index-based token compaction).
//
// One cluster of kSelCS = 8 CTAs (256 threads each) per sample; CTA r of
// the cluster owns tokens [r N / 8, (r + 1) N / 8).  Each CTA streams its
// tokens' two newest velocity slots (16 B + 16 B per token, coalesced uint4
// loads, four tokens of a thread in flight at once), keeps V and A in
// shared memory and reduces their min / max; the cluster combines the eight
// partial ranges through distributed shared memory.  Each CTA then forms
// the score in the same fp32 operation order as the definition and an
// order-preserving 32-bit key per token (in place of V), and a 4 x 8-bit
// radix select finds the c-th smallest key of the sample: every CTA counts
// its keys into a 256-bin histogram, the cluster sums the eight histograms
// bin by bin (each CTA redundantly, so all take the same digit).  Finally
// each CTA caches its keys below the threshold plus the lowest-index ties
// and compacts its active tokens in ascending order, starting from the
// counts of the lower-ranked CTAs.  With a third history slot (SSC with
// three predictions) the acceleration term is the second difference of the
// velocity and each token reads 48 B.
#include "common.cuh"
#include "kernels.h"

namespace f3dc {

namespace {

constexpr int kSelCS = 8;             // CTAs per sample (one cluster)
constexpr int kSelThreads = 256;      // one thread per histogram bin
constexpr int kSelWarps = kSelThreads / 32;
constexpr int kSelMaxTokens = 49152;  // per sample: 8 B of shared memory per token over 8 CTAs (48 KB each)
constexpr int kSelUnroll = 4;         // tokens of a thread whose loads are in flight together

// V = |v1|, A = |v1 - v2| (Sec. 4.1), or with v3 the second difference
// |(v1 - v2) - (v2 - v3)|, each channel term in that fp32 order.
F3DC_DEV void token_va(const uint4 &p, const uint4 &q, const uint4 &r, bool third, float &V, float &A)
{
    const uint32_t pw[4] = {p.x, p.y, p.z, p.w};
    const uint32_t qw[4] = {q.x, q.y, q.z, q.w};
    const uint32_t rw[4] = {r.x, r.y, r.z, r.w};
    float sv = 0.0f, sa = 0.0f;
#pragma unroll
    for (int c = 0; c < 8; ++c) {
        const uint32_t pu = (pw[c >> 1] >> ((c & 1) * 16)) & 0xFFFFu;
        const uint32_t qu = (qw[c >> 1] >> ((c & 1) * 16)) & 0xFFFFu;
        const float x = bf16_bits_to_f32(pu);
        const float y = bf16_bits_to_f32(qu);
        float d = __fsub_rn(x, y);
        if (third) d = __fsub_rn(d, __fsub_rn(y, bf16_bits_to_f32((rw[c >> 1] >> ((c & 1) * 16)) & 0xFFFFu)));
        sv = __fadd_rn(sv, __fmul_rn(x, x));
        sa = __fadd_rn(sa, __fmul_rn(d, d));
    }
    V = __fsqrt_rn(sv);
    A = __fsqrt_rn(sa);
}

// min-max normalisation; NaN stays NaN, a degenerate range gives 0.
F3DC_DEV float norm1(float x, float mn, float mx)
{
    if (isnan(x)) return x;
    if (!(mx > mn)) return 0.0f;
    return __fdiv_rn(__fsub_rn(x, mn), __fsub_rn(mx, mn));
}

// Order-preserving key: equal floats (including -0 / +0) give equal keys,
// every NaN gives the largest key (never cached before a number).
F3DC_DEV uint32_t score_key(float s)
{
    if (isnan(s)) return 0xFFFFFFFFu;
    if (s == 0.0f) s = 0.0f;
    const uint32_t u = __float_as_uint(s);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

F3DC_DEV int pad_tile(int a) { return (a + kTileRows - 1) / kTileRows * kTileRows; }

F3DC_DEV int clamp_quota(int q, int N) { return q < 0 ? 0 : (q > N ? N : q); }

// Distributed shared memory: the address of a variable in CTA `rank` of the
// cluster, and loads through it.
F3DC_DEV uint32_t dsmem_u32(const void *p, uint32_t rank) { return mapa_shared(smem_u32(p), rank); }
F3DC_DEV uint32_t ld_dsmem_u32(uint32_t addr)
{
    uint32_t v;
    asm volatile("ld.shared::cluster.u32 %0, [%1];" : "=r"(v) : "r"(addr) : "memory");
    return v;
}
F3DC_DEV float ld_dsmem_f32(uint32_t addr) { return __uint_as_float(ld_dsmem_u32(addr)); }
F3DC_DEV void cluster_arrive() { asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory"); }
F3DC_DEV void cluster_wait() { asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory"); }

// Row offset of sample b, total padded rows, and the sample's tiles.  The
// first warp sums the padded row counts of all samples (B <= 64: two per
// lane) in one round of loads.  Every CTA of the cluster computes the
// offset; only the cluster's first CTA (`writer`) writes the plan.
static_assert(kMaxBatch <= 64, "write_plan covers two samples per lane");
F3DC_DEV void write_plan(const SelectArgs &a, int b, int na, bool writer, int &off)
{
    __shared__ int s_off, s_tot_rows;
    if (threadIdx.x < 32) {
        const int lane = threadIdx.x;
        const int r0 = lane < a.B ? pad_tile(a.N - clamp_quota(a.quota[lane], a.N)) : 0;
        const int r1 = lane + 32 < a.B ? pad_tile(a.N - clamp_quota(a.quota[lane + 32], a.N)) : 0;
        int before = (lane < b ? r0 : 0) + (lane + 32 < b ? r1 : 0), tot = r0 + r1;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            before += __shfl_xor_sync(0xffffffffu, before, o);
            tot += __shfl_xor_sync(0xffffffffu, tot, o);
        }
        if (lane == 0) {
            s_off = before;
            s_tot_rows = tot;
            if (a.plan && writer) {
                a.plan->n_active[b] = na;
                a.plan->row_off[b] = before;
                if (a.cfg_dup) {  // the unguided copy of sample b
                    a.plan->n_active[a.B + b] = na;
                    a.plan->row_off[a.B + b] = tot + before;
                }
                if (b == 0) {
                    const int all = a.cfg_dup ? 2 * tot : tot;
                    a.plan->m_rows = all;
                    a.plan->n_tiles = all / kTileRows;
                }
            }
        }
    }
    __syncthreads();
    off = s_off;
    if (a.tile_sample && writer) {
        const int t0 = off / kTileRows, nt = pad_tile(na) / kTileRows;
        for (int t = threadIdx.x; t < nt; t += blockDim.x) a.tile_sample[t0 + t] = b;
        if (a.cfg_dup) {
            const int t1 = (s_tot_rows + off) / kTileRows;
            for (int t = threadIdx.x; t < nt; t += blockDim.x) a.tile_sample[t1 + t] = a.B + b;
        }
    }
}

// Inclusive scan of one value per thread over the CTA (256 threads); returns
// the inclusive prefix and leaves the total in *total.
F3DC_DEV uint32_t block_scan(uint32_t v, uint32_t *wsum, uint32_t *total)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    uint32_t incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t n = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += n;
    }
    if (lane == 31) wsum[warp] = incl;
    __syncthreads();
    uint32_t before = 0, all = 0;
#pragma unroll
    for (int w = 0; w < kSelWarps; ++w) {
        const uint32_t x = wsum[w];
        before += w < warp ? x : 0u;
        all += x;
    }
    __syncthreads();  // wsum may be reused by the next scan
    *total = all;
    return before + incl;
}

__global__ void __cluster_dims__(kSelCS, 1, 1) __launch_bounds__(kSelThreads, 4) k_ssc_select(const SelectArgs a)
{
    griddep_launch();
    griddep_wait();
    extern __shared__ float sva[];            // V, A of this CTA's tokens; the key later replaces V
    __shared__ uint32_t whist[kSelWarps / 2][256];  // one histogram per warp pair
    // this CTA's histogram of the current radix pass (read by the cluster);
    // two buffers: pass p + 1 writes the buffer that pass p - 1's readers
    // finished with before they reached pass p's cluster barrier
    __shared__ uint32_t hist[2][256];
    __shared__ float part[4];                 // this CTA's min V, max V, min A, max A (read by the cluster)
    __shared__ uint32_t cnt[2];               // this CTA's keys below / at the threshold (read by the cluster)
    __shared__ float red[4][kSelWarps];
    __shared__ float gmm[4];
    __shared__ uint32_t wsum[kSelWarps];
    __shared__ uint32_t s_digit, s_rank;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const uint32_t rk = cluster_rank();
    const int b = blockIdx.x / kSelCS;
    const int N = a.N, nl = N / kSelCS, lo = (int)rk * nl;
    const int c = clamp_quota(a.quota[b], N);
    const int na = N - c;
    const size_t base = (size_t)b * N;

    int off = 0;
    write_plan(a, b, na, rk == 0, off);
    if (a.n_active && rk == 0 && tid == 0) a.n_active[b] = na;

    // every CTA of the cluster takes the same branch here (c is per sample),
    // so none waits at a cluster barrier the others skip
    if (c == 0) {  // nothing cached: every token active, no scoring needed
        for (int i = lo + tid; i < lo + nl; i += kSelThreads) {
            a.active_idx[base + i] = i;
            if (a.mask) a.mask[base + i] = 0;
            if (a.row_of_token) a.row_of_token[base + i] = off + i;
        }
        return;
    }
    if (c == N) {  // everything cached
        for (int i = lo + tid; i < lo + nl; i += kSelThreads) {
            if (a.mask) a.mask[base + i] = 1;
            if (a.row_of_token) a.row_of_token[base + i] = -1;
        }
        return;
    }
    float *sV = sva, *sA = sva + nl;
    uint32_t *keys = reinterpret_cast<uint32_t *>(sva);  // key i overwrites V i

    // ---- V and A of this CTA's tokens, min / max (NaN never wins a comparison)
    const uint4 *g1 = reinterpret_cast<const uint4 *>(a.v1) + base + lo;
    const uint4 *g2 = reinterpret_cast<const uint4 *>(a.v2) + base + lo;
    const uint4 *g3 = a.v3 ? reinterpret_cast<const uint4 *>(a.v3) + base + lo : nullptr;
    float mnV = INFINITY, mxV = -INFINITY, mnA = INFINITY, mxA = -INFINITY;
    for (int i0 = tid; i0 < nl; i0 += kSelUnroll * kSelThreads) {
        uint4 p[kSelUnroll], q[kSelUnroll], r[kSelUnroll];
#pragma unroll
        for (int u = 0; u < kSelUnroll; ++u) {
            const int i = i0 + u * kSelThreads;
            if (i < nl) {
                p[u] = __ldg(g1 + i);
                q[u] = __ldg(g2 + i);
                r[u] = g3 ? __ldg(g3 + i) : make_uint4(0, 0, 0, 0);
            }
        }
#pragma unroll
        for (int u = 0; u < kSelUnroll; ++u) {
            const int i = i0 + u * kSelThreads;
            if (i < nl) {
                float V, A;
                token_va(p[u], q[u], r[u], g3 != nullptr, V, A);
                sV[i] = V;
                sA[i] = A;
                if (V < mnV) mnV = V;
                if (V > mxV) mxV = V;
                if (A < mnA) mnA = A;
                if (A > mxA) mxA = A;
            }
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        mnV = fminf(mnV, __shfl_xor_sync(0xffffffffu, mnV, o));
        mxV = fmaxf(mxV, __shfl_xor_sync(0xffffffffu, mxV, o));
        mnA = fminf(mnA, __shfl_xor_sync(0xffffffffu, mnA, o));
        mxA = fmaxf(mxA, __shfl_xor_sync(0xffffffffu, mxA, o));
    }
    if (lane == 0) {
        red[0][warp] = mnV;
        red[1][warp] = mxV;
        red[2][warp] = mnA;
        red[3][warp] = mxA;
    }
    __syncthreads();
    if (tid < 4) {
        float v = red[tid][0];
        for (int w = 1; w < kSelWarps; ++w) v = (tid & 1) ? fmaxf(v, red[tid][w]) : fminf(v, red[tid][w]);
        part[tid] = v;
    }
    cluster_sync();  // every CTA's partial range is in its shared memory
    if (warp == 0) {
        // lane = 4 rank + k reads entry k (min V, max V, min A, max A) of CTA rank
        float v = ld_dsmem_f32(dsmem_u32(&part[lane & 3], (uint32_t)(lane >> 2)));
#pragma unroll
        for (int o = 4; o < 32; o <<= 1) {
            const float w = __shfl_xor_sync(0xffffffffu, v, o);
            v = (lane & 1) ? fmaxf(v, w) : fminf(v, w);
        }
        if (lane < 4) gmm[lane] = v;
    }
    __syncthreads();
    mnV = gmm[0];
    mxV = gmm[1];
    mnA = gmm[2];
    mxA = gmm[3];

    // ---- C_i = w_a norm(A_i) + w_v norm(V_i) -> ordered keys, and the
    // histogram of their top byte (the first radix pass)
    for (int q = tid; q < kSelWarps / 2 * 256; q += kSelThreads) (&whist[0][0])[q] = 0;
    __syncthreads();
    for (int i = tid; i < nl; i += kSelThreads) {
        const float sc = __fadd_rn(__fmul_rn(a.wa, norm1(sA[i], mnA, mxA)), __fmul_rn(a.wv, norm1(sV[i], mnV, mxV)));
        const uint32_t k = score_key(sc);
        keys[i] = k;
        atomicAdd(&whist[warp >> 1][k >> 24], 1u);
    }
    __syncthreads();

    // ---- radix select of the c-th smallest key (1-based rank c) over the
    // cluster: each pass counts this CTA's keys matching the digits found so
    // far into its histogram; every CTA sums the eight CTAs' histograms bin by bin (thread
    // = bin), scans, and takes the digit of the bin that holds the rank
    uint32_t prefix = 0, hi_mask = 0;
    uint32_t rank = (uint32_t)c;
#pragma unroll 1
    for (int pass = 0; pass < 4; ++pass) {
        const int shift = 24 - 8 * pass;
        if (pass > 0) {
            for (int q = tid; q < kSelWarps / 2 * 256; q += kSelThreads) (&whist[0][0])[q] = 0;
            __syncthreads();
            for (int i = tid; i < nl; i += kSelThreads) {
                const uint32_t k = keys[i];
                if ((k & hi_mask) == prefix) atomicAdd(&whist[warp >> 1][(k >> shift) & 255u], 1u);
            }
            __syncthreads();
        }
        uint32_t v = 0;
#pragma unroll
        for (int w = 0; w < kSelWarps / 2; ++w) v += whist[w][tid];
        hist[pass & 1][tid] = v;
        cluster_sync();  // every CTA's histogram of this pass is complete
        uint32_t tot = 0;
#pragma unroll
        for (int r2 = 0; r2 < kSelCS; ++r2) tot += ld_dsmem_u32(dsmem_u32(&hist[pass & 1][tid], (uint32_t)r2));
        uint32_t all;
        const uint32_t incl = block_scan(tot, wsum, &all);
        const uint32_t excl = incl - tot;
        if (excl < rank && rank <= incl) {
            s_digit = (uint32_t)tid;
            s_rank = rank - excl;
        }
        __syncthreads();
        prefix |= s_digit << shift;
        hi_mask |= 255u << shift;
        rank = s_rank;
        __syncthreads();  // s_digit / s_rank are rewritten by the next pass
    }
    const uint32_t thr = prefix;  // keys below thr are cached, plus the first `rank` ties of the sample

    // ---- this CTA's keys below / at the threshold; the lower-ranked CTAs'
    // counts give the sample-wide counts before this CTA's first token
    uint32_t nlt = 0, neq = 0;
    for (int i = tid; i < nl; i += kSelThreads) {
        const uint32_t k = keys[i];
        nlt += k < thr;
        neq += k == thr;
    }
    uint32_t all_lt, all_eq;
    block_scan(nlt, wsum, &all_lt);
    block_scan(neq, wsum, &all_eq);
    if (tid == 0) {
        cnt[0] = all_lt;
        cnt[1] = all_eq;
    }
    cluster_sync();
    uint32_t run_lt = 0, run_eq = 0, sum_lt = 0, sum_eq = 0;
    if (tid < kSelCS) {
        sum_lt = ld_dsmem_u32(dsmem_u32(&cnt[0], (uint32_t)tid));
        sum_eq = ld_dsmem_u32(dsmem_u32(&cnt[1], (uint32_t)tid));
    }
    // no CTA reads another's shared memory after this: arrive now, wait at exit
    cluster_arrive();
    {
        // prefix over ranks below rk (lanes 0..7 of warp 0), broadcast
        __shared__ uint32_t s_run[4];
        if (warp == 0) {
            uint32_t bl = (uint32_t)lane < rk ? sum_lt : 0u, be = (uint32_t)lane < rk ? sum_eq : 0u;
            uint32_t tl = sum_lt, te = sum_eq;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                bl += __shfl_xor_sync(0xffffffffu, bl, o);
                be += __shfl_xor_sync(0xffffffffu, be, o);
                tl += __shfl_xor_sync(0xffffffffu, tl, o);
                te += __shfl_xor_sync(0xffffffffu, te, o);
            }
            if (lane == 0) {
                s_run[0] = bl;
                s_run[1] = be;
                s_run[2] = tl;
                s_run[3] = te;
            }
        }
        __syncthreads();
        run_lt = s_run[0];
        run_eq = s_run[1];
        if (rk == 0 && tid == 0 && (uint32_t)N - s_run[2] - min(s_run[3], rank) != (uint32_t)na)
            raise_error(a.err, kDevBadPlan);
    }

    // ---- index-ordered compaction.  For token i with L(i) smaller keys and
    // E(i) ties before it in the sample, the tie is cached iff E(i) < rank, and
    // an active token lands at position i - L(i) - min(E(i), rank).  Each
    // thread takes four consecutive tokens per round of 1024.
    for (int j0 = 0; j0 < nl; j0 += 4 * kSelThreads) {
        const int j = j0 + 4 * tid;
        uint32_t k[4];
        if (j + 3 < nl) {
            const uint4 kk = *reinterpret_cast<const uint4 *>(keys + j);
            k[0] = kk.x;
            k[1] = kk.y;
            k[2] = kk.z;
            k[3] = kk.w;
        } else {
#pragma unroll
            for (int r2 = 0; r2 < 4; ++r2) k[r2] = j + r2 < nl ? keys[j + r2] : 0u;
        }
        uint32_t ltb = 0, eqb = 0;
#pragma unroll
        for (int r2 = 0; r2 < 4; ++r2) {
            if (j + r2 < nl) {
                ltb |= (uint32_t)(k[r2] < thr) << r2;
                eqb |= (uint32_t)(k[r2] == thr) << r2;
            }
        }
        const uint32_t cnt4 = (uint32_t)__popc(ltb) | ((uint32_t)__popc(eqb) << 16);
        uint32_t tot;
        const uint32_t pre = block_scan(cnt4, wsum, &tot) - cnt4;
        uint32_t plt = run_lt + (pre & 0xFFFFu), peq = run_eq + (pre >> 16);
#pragma unroll
        for (int r2 = 0; r2 < 4; ++r2) {
            if (j + r2 >= nl) break;
            const int i = lo + j + r2;
            const bool lt = (ltb >> r2) & 1u, eq = (eqb >> r2) & 1u;
            const bool cached = lt || (eq && peq < rank);
            if (a.mask) a.mask[base + i] = cached ? 1 : 0;
            if (!cached) {
                const uint32_t pos = (uint32_t)i - plt - min(peq, rank);
                if (pos >= (uint32_t)na) raise_error(a.err, kDevBadPlan);
                else {
                    a.active_idx[base + pos] = i;
                    if (a.row_of_token) a.row_of_token[base + i] = off + (int)pos;
                }
            } else if (a.row_of_token) {
                a.row_of_token[base + i] = -1;
            }
            plt += lt;
            peq += eq;
        }
        run_lt += tot & 0xFFFFu;
        run_eq += tot >> 16;
    }
    cluster_wait();  // the other CTAs have read this CTA's shared memory
}

__global__ void k_plan_from_counts(const int32_t *n_active, int B, int N, Plan *plan, int32_t *tile_sample,
                                   uint32_t *err)
{
    griddep_launch();
    griddep_wait();
    __shared__ int offs[kMaxBatch + 1];
    if (threadIdx.x == 0) {
        int o = 0;
        for (int b = 0; b < B; ++b) {
            int na = n_active[b];
            if (na < 0 || na > N) {
                raise_error(err, kDevBadIndex);
                na = na < 0 ? 0 : N;
            }
            offs[b] = o;
            plan->n_active[b] = na;
            plan->row_off[b] = o;
            o += pad_tile(na);
        }
        offs[B] = o;
        plan->m_rows = o;
        plan->n_tiles = o / kTileRows;
    }
    __syncthreads();
    for (int b = 0; b < B; ++b) {
        const int t0 = offs[b] / kTileRows, t1 = offs[b + 1] / kTileRows;
        for (int t = t0 + threadIdx.x; t < t1; t += blockDim.x) tile_sample[t] = b;
    }
}

}  // namespace

int ssc_select_max_tokens() { return kSelMaxTokens; }

cudaError_t launch_ssc_select(const SelectArgs &a, cudaStream_t s)
{
    if (a.N > kSelMaxTokens || a.N % (4 * kSelCS) != 0 || a.B < 1 || a.B > kMaxBatch ||
        (a.cfg_dup && 2 * a.B > kMaxBatch))
        return cudaErrorInvalidValue;
    // V and A of a CTA's tokens (the key later replaces V)
    const size_t smem = (size_t)(a.N / kSelCS) * 2 * sizeof(float);
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(k_ssc_select, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
    }
    launch_k(k_ssc_select, dim3(a.B * kSelCS), dim3(kSelThreads), smem, s, a);
    return cudaGetLastError();
}

cudaError_t launch_plan_from_counts(const int32_t *n_active, const int32_t *active_idx, int B, int N,
                                    Plan *plan, int32_t *tile_sample, int32_t *row_of_token, uint32_t *err,
                                    cudaStream_t s)
{
    (void)active_idx;
    (void)row_of_token;
    if (B < 1 || B > kMaxBatch) return cudaErrorInvalidValue;
    launch_k(k_plan_from_counts, dim3(1), dim3(256), 0, s, n_active, B, N, plan, tile_sample, err);
    return cudaGetLastError();
}

}  // namespace f3dc
