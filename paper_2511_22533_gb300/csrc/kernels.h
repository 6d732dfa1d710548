// kernels.h -- internal launch interface between the C-ABI layer (api.cu)
// and the CUDA kernels of libf3dc.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>

namespace f3dc {

constexpr int kTileRows = 128;   // rows per tile; every sample's packed rows start on a tile
constexpr int kMaxBatch = 64;
constexpr int kChannels = 8;

typedef __nv_bfloat16 bf16;

// Per-step row plan.  Active tokens of all samples are packed row-wise,
// sample b's a_b rows starting at row_off[b] (a multiple of 128) and padded
// to a multiple of 128 with finite rows, so every 128-row tile belongs to
// one sample (tile_sample[] in a separate array).
struct Plan {
    int32_t n_tiles;               // padded rows / 128
    int32_t m_rows;                // padded rows
    int32_t n_active[kMaxBatch];   // a_b
    int32_t row_off[kMaxBatch];    // first packed row of sample b
};

// ------------------------------------------------------------ selection
struct SelectArgs {
    const uint16_t *v1, *v2;   // bf16 [B, N, 8]
    const uint16_t *v3;        // nullable: second-difference acceleration with v(t-3)
    const int32_t *quota;      // [B]
    int B, N;
    float wa, wv;              // omega and 1 - omega, fp32
    int32_t *active_idx;       // [B, N]
    int32_t *n_active;         // [B], nullable
    uint8_t *mask;             // [B, N], nullable
    int32_t *row_of_token;     // [B, N], nullable: packed row or -1 if cached
    Plan *plan;                // nullable
    int32_t *tile_sample;      // nullable
    // guided (CFG) step: the plan also lists samples B..2B-1, copies of
    // samples 0..B-1 (same active counts, rows after all of 0..B-1's)
    int cfg_dup;
    uint32_t *err;
};
cudaError_t launch_ssc_select(const SelectArgs &a, cudaStream_t s);
int ssc_select_max_tokens();

// Plan from given active lists (diagnostic forward): counts -> plan,
// tile_sample and row_of_token.
cudaError_t launch_plan_from_counts(const int32_t *n_active, const int32_t *active_idx, int B, int N,
                                    Plan *plan, int32_t *tile_sample, int32_t *row_of_token, uint32_t *err,
                                    cudaStream_t s);

// ------------------------------------------------------------ row kernels
// x[r] = in_w S[b, i] + in_b + pos[i] for packed active row r; zero pad rows.
// cfg_B > 0: plan samples b >= cfg_B read the tokens and latents of b - cfg_B.
cudaError_t launch_gather_embed(const float *S, int N, int W, const int32_t *active_idx, const Plan *plan,
                                const int32_t *tile_sample, const bf16 *in_w, const bf16 *in_b,
                                const float *pos, float *x, int max_rows, int num_sms, int cfg_B,
                                uint32_t *err, cudaStream_t s);

// Every one of `rows` rows of dst (leading dimension ld) = the bf16 row src.
cudaError_t launch_broadcast_row(bf16 *dst, size_t ld, const bf16 *src, int rows, int cols, cudaStream_t s);

// h = LN(x) (1 + scale) + shift (mode 0, fp32 mod vectors) or LN(x) g + b
// (mode 1, bf16 affine).  rows from plan->m_rows.
cudaError_t launch_layernorm(const float *x, int W, const Plan *plan, int mode, const float *shift,
                             const float *scale, const bf16 *g, const bf16 *b, bf16 *out, int max_rows,
                             int num_sms, cudaStream_t s);

// v_active[r, c] = out_w (LN(x_r)(1 + scale) + shift) + out_b  (final layer)
cudaError_t launch_final_layer(const float *x, int W, const Plan *plan, const float *shift,
                               const float *scale, const bf16 *out_w, const bf16 *out_b, float *v_active,
                               int max_rows, int num_sms, cudaStream_t s);

// Cache merge + Euler + history write (+ dynamic voxels).
struct MergeArgs {
    float *S;                     // [B, N, 8]
    const float *v_active;        // [rows, 8]
    const int32_t *row_of_token;  // [B, N]
    const uint16_t *v_prev1;      // bf16 [B, N, 8] (v_cache)
    uint16_t *v_out;              // bf16 [B, N, 8] (v_t)
    int B, N;
    float dt;
    const uint16_t *dec_w;        // bf16 [8, G]
    int G;
    int64_t *dyn;                 // nullable [B]
    int max_rows;
    // guided step (cfg_s != 0): the active velocity is v_u + cfg_s (v_c - v_u)
    // with v_c at the token's row and v_u plan->m_rows / 2 rows further
    float cfg_s;
    const Plan *plan;
    uint32_t *err;
};
cudaError_t launch_merge_euler(const MergeArgs &a, cudaStream_t s);

// Convolutional stand-in decoder of Eq. 1 on B latent grids S [B, D^3, 8]:
// occupancy bits of the (4D)^3 sub-voxels (2 D^3 words per sample) stored to
// `bits` (compare = 0) or XOR-counted against them into dyn[b] (compare = 1).
struct DecodeArgs {
    const float *S;
    int B, D;
    const uint16_t *w1, *b1, *w2, *b2, *w3, *b3;   // bf16 dc1..dc3
    float *scratch;                                // decode_scratch_floats(B, D)
    uint32_t *bits;                                // [B, 2 D^3]
    int compare;
    int64_t *dyn;                                  // [B] when compare
    int num_sms;
};
size_t decode_scratch_floats(int B, int D);
cudaError_t launch_decode_conv(const DecodeArgs &a, cudaStream_t s);

// Scatter packed rows back to sample-local positions (diagnostic forward).
cudaError_t launch_scatter_rows(const float *v_active, const Plan *plan, int B, int N, float *v_out,
                                cudaStream_t s);

// ------------------------------------------------------------ t-embedding
cudaError_t launch_time_freq(float t, float *freq, cudaStream_t s);
// freq [n, 256] for the n times t[0..n) (device)
cudaError_t launch_time_freq_many(const float *t, int n, float *freq, cudaStream_t s);
// y[n] = act_out(sum_k act_in(x[k]) w[n, k] + b[n]); act = SiLU when flag set
cudaError_t launch_gemv(const float *x, int K, const bf16 *w, const bf16 *b, float *y, int rows, int silu_in,
                        int silu_out, int num_sms, cudaStream_t s);
// the same for nv vectors x [nv, K] -> y [nv, rows]; each output equals the
// single-vector launch's bit for bit
cudaError_t launch_gemv_many(const float *x, int nv, int K, const bf16 *w, const bf16 *b, float *y, int rows,
                             int silu_in, int silu_out, int num_sms, cudaStream_t s);
// kernels one launch_gemv_many call launches (vectors in groups of 8, 4, 2, 1)
int gemv_many_kernels(int nv, int K);

// ------------------------------------------------------------ GEMM
enum GemmEpi { kEpiBias = 0, kEpiGelu = 1, kEpiResid = 2, kEpiQKNorm = 3 };

struct GemmParams {
    int M;                    // rows stored are < M
    int N, K;
    const int32_t *m_tiles_dev;   // nullable: tile count read on device
    int m_tiles;                  // used when m_tiles_dev is null
    void *out;
    int ldo;                  // elements
    const bf16 *bias;         // nullable
    const float *gate;        // nullable (RESID)
    const bf16 *qn_g, *kn_g;  // QKNORM gammas [W]
    int width, dh;            // QKNORM: columns < 2*width are normalised per dh-group
    // split-K workspace (nullable: no split).  When the tile count leaves
    // SMs idle the kernel splits each tile's K range over several CTAs, which
    // write fp32 partial tiles to ws; the last CTA of a tile (per-tile arrival
    // counter in `counters`, left at 0) sums them in split order and applies
    // the epilogue.
    float *ws;
    int32_t *counters;
    int ws_units;             // partial tiles the workspace holds
    // bn = 256 without a workspace: when the device-side tile count of
    // 256-wide tiles is below this, the kernel runs 128-wide tiles (0: never)
    int narrow_below;
    // fault injection (tests of the failure path; 0 in normal use): the
    // split-K arrival wait expects split_extra arrivals beyond the splits
    // that exist, and gives up after split_wait_ns (0: kWaitLimitNs)
    int split_extra;
    uint64_t split_wait_ns;
    uint32_t *err;
};
// bn in {64, 128, 256}.  ta: A [M, K] in boxes of 128 rows x 64 columns; tb:
// B [N, K] in boxes of gemm_b_box_rows(bn) rows x 64 columns.
cudaError_t launch_gemm(const CUtensorMap *ta, const CUtensorMap *tb, const GemmParams &p, int epi, int bn,
                        int grid, cudaStream_t s);
inline uint32_t gemm_b_box_rows(int bn) { return bn < 128 ? (uint32_t)bn : 128u; }

// 256-wide GEMM on CTA pairs (clusters of two, cta_group::2 MMAs of 256
// rows): same parameters and epilogues as launch_gemm with bn = 256, K a
// multiple of 128, no split K (p.ws null); tb in boxes of kGemmPairBBox rows
// x 64 columns.  The
// grid is min(max_pair_tiles, resident clusters) clusters.
constexpr uint32_t kGemmPairBBox = 64;
cudaError_t launch_gemm_pair(const CUtensorMap *ta, const CUtensorMap *tb, const GemmParams &p, int epi,
                             int max_pair_tiles, cudaStream_t s);
size_t gemm_smem_bytes(int bn);

// Launches a kernel of this library with programmatic stream serialization
// (programmatic dependent launch): the kernel may start while the previous
// kernel in the stream finishes and waits for it in griddep_wait().
template <typename... KArgs, typename... Args>
cudaError_t launch_k(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s, Args... args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// bytes of split-K workspace for `units` partial tiles of width bn
inline size_t gemm_ws_bytes(int bn, int units) { return (size_t)units * 128 * bn * sizeof(float); }
constexpr int kGemmMaxCounterTiles = 1024;

// Split-K rule (shared by the kernel and the host): split a tile's K range
// only when whole tiles would leave at least half of the `grid` CTAs idle,
// keeping >= 4 K blocks (of 64) per split and within `ws_units` partial tiles.
// The count is rounded so that ceil(kb_n / splits) K blocks per split leave
// no split empty (an empty split would contribute a stale accumulator).
constexpr int kGemmMaxSplits = 16;
__host__ __device__ inline int gemm_split_count(int tiles, int grid, int kb_n, int ws_units, bool have_ws)
{
    // only a long K loop (K >= 2048) saves more than the partials' round trip
    // through L2 and the in-order reduction cost
    if (!have_ws || tiles <= 0 || 2 * tiles > grid || tiles > kGemmMaxCounterTiles || kb_n < 32) return 1;
    int sp = grid / tiles;
    if (sp > kb_n / 4) sp = kb_n / 4;
    if (sp > ws_units / tiles) sp = ws_units / tiles;
    if (sp > kGemmMaxSplits) sp = kGemmMaxSplits;
    if (sp <= 1) return 1;
    const int per = (kb_n + sp - 1) / sp;
    return (kb_n + per - 1) / per;
}

// Grid of a GEMM whose tile count is known on the host: one CTA per tile,
// or every SM when few tiles leave room to split K.
inline int gemm_grid(int tiles, int sms) { return 2 * tiles <= sms ? sms : (tiles < sms ? tiles : sms); }

// ------------------------------------------------------------ attention
struct AttnParams {
    int heads, dh;
    int q_col0, k_col0, v_col0;    // column of head 0 in the q / kv buffers
    int mode;                      // 0 self (plan), 1 cross (b * nk_fixed), 2 single sequence
    const int32_t *n_tiles_dev;    // nullable
    int n_tiles;
    const int32_t *tile_sample;    // modes 0, 1
    const Plan *plan;              // mode 0
    int nk_fixed;                  // modes 1, 2
    int q_rows;                    // mode 2: rows stored are < q_rows
    bf16 *out;
    int ldo;
    float scale_log2;              // log2(e) / sqrt(dh)
    // mode 1: samples b >= kv_null_from (0: none) attend to the keys of
    // sample slot kv_null_sample (the zero condition of a guided step)
    int kv_null_from, kv_null_sample;
    // > 0: K / V rows [0, kv_prefetch_rows) are complete before the launch
    // (not written by the previous kernel) and are prefetched into L2 first
    int kv_prefetch_rows;
    // fault injection (tests; 0 in normal use): CTA 0 never loads the last
    // key tile of its first item, so the waits on it run out and the kernel
    // aborts cleanly
    int fault_skip_kv;
    uint32_t *err;
};
// grid: persistent CTAs (at most one per SM), each taking the work items
// (pair of 128-query tiles, head) in turn.
cudaError_t launch_attention(const CUtensorMap *tq, const CUtensorMap *tk, const CUtensorMap *tv,
                             const AttnParams &p, int grid, cudaStream_t s);
// The same attention with one query tile per work item (k_attn_one.cu): the
// faster kernel when every (query tile, head) item gets a CTA of its own,
// i.e. tiles * heads <= grid (attn_one_tile).
cudaError_t launch_attention_one(const CUtensorMap *tq, const CUtensorMap *tk, const CUtensorMap *tv,
                                 const AttnParams &p, int grid, cudaStream_t s);
inline bool attn_one_tile(int64_t tiles, int heads, int grid) { return tiles * heads <= grid; }
size_t attn_smem_bytes(int dh);

// ------------------------------------------------------------ host helpers
// Records the message f3dc_last_error(NULL) returns on this thread.
void set_host_error(const std::string &msg);

// Host-side fault injection for the tests of the failure paths (process
// wide; f3dc_set_fault_injection).  Nothing here faults a GPU: an allocation
// is reported as failed without being attempted, and the GEMM's split-K wait
// is given an arrival no CTA makes, so its bounded wait runs out.
struct FaultInjection {
    int fail_alloc_at = -1;        // f3dc_create's n-th device allocation fails (-1: off)
    int gemm_missing_arrivals = 0; // split-K arrivals the standalone GEMM's wait also expects
    uint64_t gemm_wait_ns = 0;     // that wait's limit (0: the default)
    int attn_missing_kv = 0;       // f3dc_attention: CTA 0 never loads its first item's last key tile
};
FaultInjection &fault_injection();

// Device address of the current device's status word of the standalone calls
// (f3dc_gemm, f3dc_gemm_noalloc, f3dc_attention; read by f3dc_gemm_status), or null if
// it cannot be resolved.  The word is a static device variable, not an
// allocation.
uint32_t *gemm_status_word();

// 2-D bf16 tensor map over a row-major [rows, cols] matrix with leading
// dimension ld (elements), box [box_rows, box_cols], 128B (box_cols = 64) or
// 64B (box_cols = 32) swizzle.  Returns false on failure.
bool make_tmap_bf16(CUtensorMap *map, const void *base, uint64_t rows, uint64_t cols, uint64_t ld,
                    uint32_t box_rows, uint32_t box_cols);

}  // namespace f3dc
