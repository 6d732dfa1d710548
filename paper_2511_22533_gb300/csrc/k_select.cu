// k_select.cu -- K1: Spatiotemporal Stability Criterion scoring and
// lowest-c selection (Sec. 4.1 V_i and Eq. ICE; Sec. 4.2 Eq. ssc and
// Eq. normalize; Algorithm 1 function SSC), fused with the row plan of the
// step (Sec. 4.2 index-based token compaction).
//
// One CTA of 1024 threads per sample.  Pass 1 streams the two newest
// velocity slots (16 B + 16 B per token, coalesced uint4 loads, a thread's
// first four tokens in one round of loads) and reduces min / max of V and A;
// pass 2 takes V and A from registers (re-reading tokens beyond the first
// 4096 from L2), forms the score in the same fp32 operation order as the
// definition and stores an order-preserving 32-bit key per token in shared
// memory.  A 4 x 8-bit radix select finds the c-th smallest key; an
// index-ordered scan then caches every key below it plus the lowest-index
// ties, and compacts the active tokens in ascending order.  With a third
// history slot (SSC with three predictions) the acceleration term is the
// second difference of the velocity and pass 1 reads 48 B per token.
#include "common.cuh"
#include "kernels.h"

namespace f3dc {

namespace {

constexpr int kSelThreads = 1024;
constexpr int kSelWarps = kSelThreads / 32;
constexpr int kSelMaxTokens = 49152;  // 4-byte keys in shared memory (192 KB + 16 KB of histograms)
constexpr int kRegTok = 4;            // tokens per thread held in registers between passes 1 and 2

// V = |v1|, A = |v1 - v2| (Sec. 4.1), or with v3 the second difference
// |(v1 - v2) - (v2 - v3)|, each channel term in that fp32 order.
F3DC_DEV void load_token(const uint16_t *v1, const uint16_t *v2, const uint16_t *v3, size_t tok, float &V, float &A)
{
    const uint4 p = __ldg(reinterpret_cast<const uint4 *>(v1) + tok);
    const uint4 q = __ldg(reinterpret_cast<const uint4 *>(v2) + tok);
    const uint4 r = v3 ? __ldg(reinterpret_cast<const uint4 *>(v3) + tok) : make_uint4(0, 0, 0, 0);
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
        if (v3) d = __fsub_rn(d, __fsub_rn(y, bf16_bits_to_f32((rw[c >> 1] >> ((c & 1) * 16)) & 0xFFFFu)));
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

// Row offset of sample b, total padded rows, and the sample's tiles.  The
// first warp sums the padded row counts of all samples (B <= 64: two per
// lane) in one round of loads.
static_assert(kMaxBatch <= 64, "write_plan covers two samples per lane");
F3DC_DEV void write_plan(const SelectArgs &a, int b, int na, int &off)
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
            if (a.plan) {
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
    if (a.tile_sample) {
        const int t0 = off / kTileRows, nt = pad_tile(na) / kTileRows;
        for (int t = threadIdx.x; t < nt; t += blockDim.x) a.tile_sample[t0 + t] = b;
        if (a.cfg_dup) {
            const int t1 = (s_tot_rows + off) / kTileRows;
            for (int t = threadIdx.x; t < nt; t += blockDim.x) a.tile_sample[t1 + t] = a.B + b;
        }
    }
}

__global__ void __launch_bounds__(kSelThreads, 1) k_ssc_select(const SelectArgs a)
{
    griddep_launch();
    griddep_wait();
    extern __shared__ uint32_t keys[];
    __shared__ uint32_t whist[16][256];
    __shared__ float red[4][kSelWarps];
    __shared__ uint32_t wsum[kSelWarps], wpre[kSelWarps];
    __shared__ uint32_t s_digit, s_rank, s_tot;

    const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int N = a.N;
    const int c = clamp_quota(a.quota[b], N);
    const int na = N - c;
    const size_t base = (size_t)b * N;

    int off = 0;
    write_plan(a, b, na, off);
    if (a.n_active && tid == 0) a.n_active[b] = na;

    if (c == 0) {  // nothing cached: every token active, no scoring needed
        for (int i = tid; i < N; i += kSelThreads) {
            a.active_idx[base + i] = i;
            if (a.mask) a.mask[base + i] = 0;
            if (a.row_of_token) a.row_of_token[base + i] = off + i;
        }
        return;
    }
    if (c == N) {  // everything cached
        for (int i = tid; i < N; i += kSelThreads) {
            if (a.mask) a.mask[base + i] = 1;
            if (a.row_of_token) a.row_of_token[base + i] = -1;
        }
        return;
    }

    // ---- pass 1: min / max of V and A (NaN never wins a comparison).  The
    // first kRegTok tokens of each thread are loaded together and kept in
    // registers for pass 2; tokens beyond them are re-read there.
    float mnV = INFINITY, mxV = -INFINITY, mnA = INFINITY, mxA = -INFINITY;
    float Vr[kRegTok], Ar[kRegTok];
#pragma unroll
    for (int r = 0; r < kRegTok; ++r) {
        const int i = tid + r * kSelThreads;
        Vr[r] = Ar[r] = 0.0f;
        if (i < N) load_token(a.v1, a.v2, a.v3, base + i, Vr[r], Ar[r]);
    }
#pragma unroll
    for (int r = 0; r < kRegTok; ++r) {
        if (tid + r * kSelThreads < N) {
            if (Vr[r] < mnV) mnV = Vr[r];
            if (Vr[r] > mxV) mxV = Vr[r];
            if (Ar[r] < mnA) mnA = Ar[r];
            if (Ar[r] > mxA) mxA = Ar[r];
        }
    }
    for (int i = tid + kRegTok * kSelThreads; i < N; i += kSelThreads) {
        float V, A;
        load_token(a.v1, a.v2, a.v3, base + i, V, A);
        if (V < mnV) mnV = V;
        if (V > mxV) mxV = V;
        if (A < mnA) mnA = A;
        if (A > mxA) mxA = A;
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
    mnV = red[0][lane];
    mxV = red[1][lane];
    mnA = red[2][lane];
    mxA = red[3][lane];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        mnV = fminf(mnV, __shfl_xor_sync(0xffffffffu, mnV, o));
        mxV = fmaxf(mxV, __shfl_xor_sync(0xffffffffu, mxV, o));
        mnA = fminf(mnA, __shfl_xor_sync(0xffffffffu, mnA, o));
        mxA = fmaxf(mxA, __shfl_xor_sync(0xffffffffu, mxA, o));
    }

    // ---- pass 2: C_i = w_a norm(A_i) + w_v norm(V_i) -> ordered keys
    auto score = [&](float V, float A) {
        return __fadd_rn(__fmul_rn(a.wa, norm1(A, mnA, mxA)), __fmul_rn(a.wv, norm1(V, mnV, mxV)));
    };
#pragma unroll
    for (int r = 0; r < kRegTok; ++r) {
        const int i = tid + r * kSelThreads;
        if (i < N) keys[i] = score_key(score(Vr[r], Ar[r]));
    }
    for (int i = tid + kRegTok * kSelThreads; i < N; i += kSelThreads) {
        float V, A;
        load_token(a.v1, a.v2, a.v3, base + i, V, A);
        keys[i] = score_key(score(V, A));
    }
    __syncthreads();

    // ---- radix select: the c-th smallest key (1-based rank c).  Each pair of
    // warps counts digits into its own 256-bin histogram with plain shared-
    // memory atomics; threads 0..255 then sum the 16 histograms bin by bin
    // and scan them, and the one bin holding rank `rank` fixes the digit.
    uint32_t prefix = 0, hi_mask = 0;
    uint32_t rank = (uint32_t)c;
    for (int shift = 24; shift >= 0; shift -= 8) {
        for (int q = tid; q < 16 * 256; q += kSelThreads) (&whist[0][0])[q] = 0;
        __syncthreads();
        uint32_t *mine = whist[warp >> 1];
        for (int i = tid; i < N; i += kSelThreads) {
            const uint32_t k = keys[i];
            if ((k & hi_mask) == prefix) atomicAdd(&mine[(k >> shift) & 255u], 1u);
        }
        __syncthreads();
        uint32_t v = 0, incl = 0;
        if (tid < 256) {
#pragma unroll
            for (int w = 0; w < 16; ++w) v += whist[w][tid];
            incl = v;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const uint32_t n = __shfl_up_sync(0xffffffffu, incl, o);
                if (lane >= o) incl += n;
            }
            if (lane == 31) wsum[warp] = incl;
        }
        __syncthreads();
        if (tid < 256) {
            for (int w = 0; w < warp; ++w) incl += wsum[w];
            const uint32_t excl = incl - v;
            if (excl < rank && rank <= incl) {
                s_digit = (uint32_t)tid;
                s_rank = rank - excl;
            }
        }
        __syncthreads();
        prefix |= s_digit << shift;
        hi_mask |= 255u << shift;
        rank = s_rank;
    }
    const uint32_t thr = prefix;  // keys below thr are cached, plus the first `rank` ties

    // ---- index-ordered compaction.  For token i with L(i) smaller keys and
    // E(i) ties before it, the tie is cached iff E(i) < rank, and an active
    // token lands at position i - L(i) - min(E(i), rank).  Each thread takes
    // four consecutive tokens; one block-wide scan of the packed counts
    // (L in the low, E in the high 16 bits) per 4096 tokens.
    uint32_t run_lt = 0, run_eq = 0;
    for (int i0 = 0; i0 < N; i0 += 4 * kSelThreads) {
        const int i = i0 + 4 * tid;
        uint32_t k[4];
        if (i + 3 < N) {
            const uint4 kk = *reinterpret_cast<const uint4 *>(keys + i);
            k[0] = kk.x;
            k[1] = kk.y;
            k[2] = kk.z;
            k[3] = kk.w;
        } else {
#pragma unroll
            for (int r = 0; r < 4; ++r) k[r] = i + r < N ? keys[i + r] : 0u;
        }
        uint32_t ltb = 0, eqb = 0;
#pragma unroll
        for (int r = 0; r < 4; ++r) {
            if (i + r < N) {
                ltb |= (uint32_t)(k[r] < thr) << r;
                eqb |= (uint32_t)(k[r] == thr) << r;
            }
        }
        const uint32_t cnt = (uint32_t)__popc(ltb) | ((uint32_t)__popc(eqb) << 16);
        uint32_t incl = cnt;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t n = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += n;
        }
        if (lane == 31) wsum[warp] = incl;
        __syncthreads();
        if (warp == 0) {
            const uint32_t x = wsum[lane];
            uint32_t wi = x;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const uint32_t n = __shfl_up_sync(0xffffffffu, wi, o);
                if (lane >= o) wi += n;
            }
            wpre[lane] = wi - x;
            if (lane == 31) s_tot = wi;
        }
        __syncthreads();
        const uint32_t pre = wpre[warp] + incl - cnt;
        uint32_t plt = run_lt + (pre & 0xFFFFu), peq = run_eq + (pre >> 16);
#pragma unroll
        for (int r = 0; r < 4; ++r) {
            if (i + r >= N) break;
            const bool lt = (ltb >> r) & 1u, eq = (eqb >> r) & 1u;
            const bool cached = lt || (eq && peq < rank);
            if (a.mask) a.mask[base + i + r] = cached ? 1 : 0;
            if (!cached) {
                const uint32_t pos = (uint32_t)(i + r) - plt - min(peq, rank);
                if (pos >= (uint32_t)na) raise_error(a.err, kDevBadPlan);
                else {
                    a.active_idx[base + pos] = i + r;
                    if (a.row_of_token) a.row_of_token[base + i + r] = off + (int)pos;
                }
            } else if (a.row_of_token) {
                a.row_of_token[base + i + r] = -1;
            }
            plt += lt;
            peq += eq;
        }
        const uint32_t tot = s_tot;
        run_lt += tot & 0xFFFFu;
        run_eq += tot >> 16;
        __syncthreads();
    }
    if (tid == 0 && (uint32_t)N - run_lt - min(run_eq, rank) != (uint32_t)na) raise_error(a.err, kDevBadPlan);
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
    if (a.N > kSelMaxTokens || a.B < 1 || a.B > kMaxBatch || (a.cfg_dup && 2 * a.B > kMaxBatch))
        return cudaErrorInvalidValue;
    const size_t smem = (size_t)a.N * sizeof(uint32_t);
    cudaError_t e = cudaFuncSetAttribute(k_ssc_select, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    launch_k(k_ssc_select, dim3(a.B), dim3(kSelThreads), smem, s, a);
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
