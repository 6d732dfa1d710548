// api.cu -- the C-ABI of libf3dc (include/f3dc.h): handle life cycle,
// host-side schedule logic (Supp. Sec. D time shift; Sec. 4.2 PCSC;
// Algorithm 1 phases and tau refresh), the cached step (Algorithm 1 steps
// 2-3) and the sampler (Algorithm 1), plus kernel-level diagnostic calls.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "../../include/f3dc.h"
#include "kernels.h"

using namespace f3dc;

namespace {

thread_local std::string g_last_error;

struct BlockOffsets {
    size_t mod_w, mod_b, qkv_w, qkv_b, qn_g, kn_g, o_w, o_b, ln2_g, ln2_b;
    size_t cq_w, cq_b, ckv_w, ckv_b, co_w, co_b, fc1_w, fc1_b, fc2_w, fc2_b;
};

struct Layout {
    size_t in_w, in_b, t_w1, t_b1, t_w2, t_b2, fmod_w, fmod_b, out_w, out_b, dec_w;
    size_t dc1_w, dc1_b, dc2_w, dc2_b, dc3_w, dc3_b;  // convolutional stand-in decoder
    std::vector<BlockOffsets> blk;
    size_t total;
};

// Walks the layout-v2 tensor order; each tensor starts on a 64-element
// boundary.
Layout weight_layout(const f3dc_config &c)
{
    Layout L;
    size_t pos = 0;
    const size_t W = c.width, C = c.channels, Dc = c.cond_dim, G = c.gamma_up, Wm = (size_t)c.mlp_ratio * W;
    auto take = [&](size_t n) {
        size_t o = pos;
        pos += (n + 63) / 64 * 64;
        return o;
    };
    L.in_w = take(W * C);
    L.in_b = take(W);
    L.t_w1 = take(W * 256);
    L.t_b1 = take(W);
    L.t_w2 = take(W * W);
    L.t_b2 = take(W);
    for (int l = 0; l < c.blocks; ++l) {
        BlockOffsets b;
        b.mod_w = take(6 * W * W);
        b.mod_b = take(6 * W);
        b.qkv_w = take(3 * W * W);
        b.qkv_b = take(3 * W);
        b.qn_g = take(W);
        b.kn_g = take(W);
        b.o_w = take(W * W);
        b.o_b = take(W);
        b.ln2_g = take(W);
        b.ln2_b = take(W);
        b.cq_w = take(W * W);
        b.cq_b = take(W);
        b.ckv_w = take(2 * W * Dc);
        b.ckv_b = take(2 * W);
        b.co_w = take(W * W);
        b.co_b = take(W);
        b.fc1_w = take(Wm * W);
        b.fc1_b = take(Wm);
        b.fc2_w = take(W * Wm);
        b.fc2_b = take(W);
        L.blk.push_back(b);
    }
    L.fmod_w = take(2 * W * W);
    L.fmod_b = take(2 * W);
    L.out_w = take(C * W);
    L.out_b = take(C);
    L.dec_w = take(C * G);
    L.dc1_w = take(16 * C * 27);
    L.dc1_b = take(16);
    L.dc2_w = take(8 * 16 * 27);
    L.dc2_b = take(8);
    L.dc3_w = take(8 * 27);
    L.dc3_b = take(1);
    L.total = pos;
    return L;
}

bool config_valid(const f3dc_config *c, std::string &why)
{
    if (!c) {
        why = "null config";
        return false;
    }
    const long long N = (long long)c->grid * c->grid * c->grid;
    if (c->grid < 1 || N % 32 != 0) why = "grid^3 must be a positive multiple of 32";
    else if (N > ssc_select_max_tokens()) why = "too many tokens for the selection kernel";
    else if (c->channels != kChannels) why = "channels must be 8";
    else if (c->width != 128 && c->width != 256 && c->width != 512 && c->width != 1024 && c->width != 2048)
        why = "width must be 128, 256, 512, 1024 or 2048";
    else if (c->heads < 1 || c->width % c->heads != 0) why = "width must be divisible by heads";
    else if (c->width / c->heads != 32 && c->width / c->heads != 64) why = "head dim must be 32 or 64";
    else if (c->mlp_ratio != 4) why = "mlp_ratio must be 4";
    else if (c->blocks < 1) why = "blocks must be >= 1";
    else if (c->cond_tokens < 1 || c->cond_dim < 64 || c->cond_dim % 64 != 0 || c->cond_dim > 4096)
        why = "cond_tokens >= 1 and cond_dim a multiple of 64 up to 4096";
    else if (c->steps < 1) why = "steps must be >= 1";
    else if (c->max_batch < 1 || c->max_batch > kMaxBatch) why = "max_batch must be in [1, 64]";
    else if (c->gamma_up < 1 || c->gamma_up > 512) why = "gamma_up must be in [1, 512]";
    else if (c->refresh_mode != F3DC_REFRESH_PERIOD && c->refresh_mode != F3DC_REFRESH_LITERAL)
        why = "unknown refresh_mode";
    else if (!(c->eta > 0.0) || !std::isfinite(c->mu) || !(c->omega >= 0.0 && c->omega <= 1.0) ||
             !(c->xi >= 0.0 && c->xi <= 1.0) || !(c->rho_a >= 0.0) || !(c->rho_cfg_off >= 0.0))
        why = "hyperparameter out of range";
    else if (!std::isfinite(c->cfg_strength) || c->cfg_strength < 0.0 || !std::isfinite(c->cfg_t_lo))
        why = "cfg_strength must be finite and >= 0, cfg_t_lo finite";
    else if (c->cfg_strength > 0.0 && 2 * c->max_batch > kMaxBatch)
        why = "with classifier-free guidance max_batch must be <= 32";
    else if (c->ssc_accel != 0 && c->ssc_accel != 1)
        why = "ssc_accel must be 0 or 1";
    else if ((c->decoder != 0 && c->decoder != 1) || (c->decoder == 1 && c->gamma_up != 64))
        why = "decoder must be 0, or 1 with gamma_up 64";
    else
        return true;
    return false;
}

int ceil_steps(int T, double rho) { return (int)std::ceil((double)T * rho); }

// Three-phase budget (Algorithm 1 step 1) with the PCSC forecast (Sec. 4.2).
int phase_quota(const f3dc_config &c, double sigma, int k, int *phase)
{
    const int N = c.grid * c.grid * c.grid;
    const int ka = ceil_steps(c.steps, c.rho_a), koff = ceil_steps(c.steps, c.rho_cfg_off);
    double q;
    if (k <= ka) {
        *phase = 1;
        return 0;
    }
    if (k < koff) {
        *phase = 2;
        const double forecast = sigma * std::exp(c.mu * (double)(k - ka));  // dS_hat_k
        q = std::floor((double)N - forecast / (double)c.gamma_up);
    } else {
        *phase = 3;
        const int kr = k - koff;
        if (c.f_corr > 0 && (kr + 1) % c.f_corr == 0) return 0;
        q = std::floor((double)N * c.xi);
    }
    if (!(q > 0.0)) return 0;
    if (q > (double)N) return N;
    return (int)q;
}

// Error-accumulation elimination (Sec. 4.3 Phase 2; Algorithm 1 SSC).
int tau_gate(const f3dc_config &c, int quota, int32_t *consec)
{
    if (quota > 0 && c.tau > 0) {
        const int limit = c.refresh_mode == F3DC_REFRESH_PERIOD ? c.tau - 1 : c.tau;
        if (*consec >= limit) quota = 0;
    }
    if (quota > 0) *consec += 1;
    else *consec = 0;
    return quota;
}

void time_schedule(const f3dc_config &c, float *t)
{
    for (int k = 1; k <= c.steps + 1; ++k) {
        const double tl = 1.0 - (double)(k - 1) / (double)c.steps;
        t[k - 1] = (float)(c.eta * tl / (1.0 + (c.eta - 1.0) * tl));
    }
}

// Fixed 3-D sin-cos position embedding of every token (host, fp64, once):
// per axis (d, h, w) F = W / 6 frequencies 10000^(-f/F), [sin | cos] blocks,
// the remaining W - 6F entries zero.
std::vector<float> position_table(int grid, int W)
{
    const int N = grid * grid * grid, F = W / 6;
    std::vector<float> pos((size_t)N * W, 0.0f);
    for (int i = 0; i < N; ++i) {
        const int coord[3] = {i / (grid * grid), (i / grid) % grid, i % grid};
        float *row = pos.data() + (size_t)i * W;
        for (int a = 0; a < 3; ++a)
            for (int f = 0; f < F; ++f) {
                const double w = std::pow(10000.0, -(double)f / (double)F);
                row[a * 2 * F + f] = (float)std::sin(coord[a] * w);
                row[a * 2 * F + F + f] = (float)std::cos(coord[a] * w);
            }
    }
    return pos;
}

// ---------------------------------------------------------------- profiling
enum KernelFamily {
    KF_SELECT, KF_GATHER, KF_LN, KF_GEMM, KF_ATTN_SELF, KF_ATTN_CROSS, KF_FINAL, KF_MERGE, KF_TEMB, KF_GEMM_COND,
    KF_PLAN, KF_SCATTER, KF_DECODE, KF_COUNT
};
const char *const kFamilyName[KF_COUNT] = {"ssc_select", "gather_embed", "layernorm",  "gemm",
                                           "attn_self",  "attn_cross",   "final_layer", "merge_euler",
                                           "temb_gemv",  "gemm_cond",    "plan",        "scatter",
                                           "decode_conv"};

// Algorithmic work of one launch as a function of the step's plan:
//   c_m * M + c_sq * sum_b a_b^2 + c_tok * B N + c_sel * (tokens of samples
//   that ran the selection) + c_fix, in flops or in DRAM bytes.
struct Work {
    double c_m = 0, c_sq = 0, c_tok = 0, c_sel = 0, c_fix = 0;
    bool flops = false;
};
Work wm(double c, bool flops = false)
{
    Work w;
    w.c_m = c;
    w.flops = flops;
    return w;
}
Work wfix(double c, bool flops = false)
{
    Work w;
    w.c_fix = c;
    w.flops = flops;
    return w;
}

struct ProfRecord {
    int fam;
    cudaEvent_t e0, e1;
    Work w;
};

struct Profiler {
    bool on = false;
    std::vector<cudaEvent_t> pool;
    size_t next = 0;
    std::vector<ProfRecord> pending;
    int64_t launches[KF_COUNT] = {};
    double ms[KF_COUNT] = {}, flops[KF_COUNT] = {}, bytes[KF_COUNT] = {};
    void reset()
    {
        for (int i = 0; i < KF_COUNT; ++i) {
            launches[i] = 0;
            ms[i] = flops[i] = bytes[i] = 0.0;
        }
        pending.clear();
        next = 0;
    }
};

}  // namespace

void f3dc::set_host_error(const std::string &msg) { g_last_error = msg; }

f3dc::FaultInjection &f3dc::fault_injection()
{
    static FaultInjection fi;
    return fi;
}

struct f3dc_handle {
    f3dc_config cfg;
    int N = 0, W = 0, Wm = 0, H = 0, dh = 0, L = 0, Nc = 0, Dc = 0, G = 0, T = 0;
    int max_rows = 0, max_tiles = 0, num_sms = 0, device = 0;
    size_t ckv_rows = 0;  // rows per layer of the condition K/V cache
    std::string err;
    Layout lay;

    bf16 *wblob = nullptr, *mod_w = nullptr, *mod_b = nullptr;
    int mod_rows = 0;
    // every step's time embedding and modulation, computed at the start of
    // f3dc_sample (one pass over the modulation weights per sample instead
    // of one per step); mod_pre marks a sample in progress
    float *t_all = nullptr, *freq_all = nullptr, *h1_all = nullptr, *temb_all = nullptr, *mod_all = nullptr;
    bool mod_pre = false;
    float *pos = nullptr;

    float *x = nullptr, *v_active = nullptr, *freq = nullptr, *h1 = nullptr, *temb = nullptr, *mod = nullptr;
    bf16 *h = nullptr, *qkv = nullptr, *att = nullptr, *qc = nullptr, *u = nullptr, *ckv = nullptr;
    uint16_t *ring = nullptr;
    Plan *plan = nullptr;
    int32_t *tile_sample = nullptr, *active_idx = nullptr, *row_of_token = nullptr, *n_active = nullptr;
    uint8_t *mask = nullptr;
    int32_t *quota_dev = nullptr;
    int64_t *dyn = nullptr;
    uint32_t *dev_err = nullptr;
    float *gemm_ws = nullptr;          // split-K partial tiles, one per SM
    int32_t *gemm_cnt = nullptr;       // split-K per-tile arrival counters (kept at 0)
    cudaStream_t last_stream = nullptr;
    int cond_B = 0;
    int64_t *dyn_curve = nullptr;  // [T, max_batch] for f3dc_dynamic_voxel_curve
    int32_t *zero_quota = nullptr; // [max_batch] zeros
    float *dec_scratch = nullptr;  // convolutional decoder (cfg.decoder == 1)
    uint32_t *dec_bits = nullptr;
    int cfg_B_now = 0;  // guided step in flight: samples >= cfg_B_now are the unguided copies
    // f3dc_sample's host copy of every step's quotas ([k * B + b]) while it
    // runs its steps (null otherwise), and whether the step in flight takes
    // the one-tile attention kernel (its query-tile count known on the host)
    const int32_t *hq_steps = nullptr;
    bool attn_one_now = false;
    // pinned per-step quota slots, two generations so one sampler call can
    // be enqueued while the previous one still copies from its slots
    int32_t *h_quota = nullptr;
    cudaEvent_t quota_done[2] = {nullptr, nullptr};
    unsigned calls = 0;

    Profiler prof;
    int64_t launches = 0;
    int last_B = 0;

    // CUDA graphs of sampler segments (runs of consecutive steps), replayed
    // on a library-owned stream ordered with the caller's through events
    struct SegmentGraph {
        int B, k0, k1, ka;
        float *S;
        std::vector<uint8_t> attn_one;  // per step k0..k1: the attention kernel captured
        cudaGraphExec_t exec;
        int64_t launches;
    };
    std::vector<SegmentGraph> graphs;
    bool use_graphs = true;
    cudaStream_t exec_stream = nullptr;
    cudaEvent_t ev_in = nullptr, ev_out = nullptr;

    CUtensorMap tm_h, tm_att, tm_u, tm_cond, tm_q_self, tm_q_cross;
    std::vector<CUtensorMap> tm_qkv_w, tm_o_w, tm_cq_w, tm_co_w, tm_fc1_w, tm_fc2_w, tm_ckv_w, tm_kv_cross;
    int bn_qkv = 128, bn_w = 128, bn_fc1 = 128, bn_ckv = 128;

    const bf16 *wt(size_t off) const { return wblob + off; }
};

namespace {

f3dc_status fail(f3dc_handle *h, f3dc_status st, const std::string &msg)
{
    if (h) h->err = msg;
    g_last_error = msg;
    return st;
}

#define CK(expr)                                                                                   \
    do {                                                                                           \
        cudaError_t e_ = (expr);                                                                   \
        if (e_ != cudaSuccess)                                                                     \
            return fail(h, F3DC_ERR_CUDA, std::string(#expr) + ": " + cudaGetErrorString(e_));     \
    } while (0)

cudaEvent_t prof_event(f3dc_handle *h)
{
    Profiler &P = h->prof;
    if (P.next == P.pool.size()) {
        cudaEvent_t e = nullptr;
        if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
        P.pool.push_back(e);
    }
    return P.pool[P.next++];
}

cudaEvent_t prof_begin(f3dc_handle *h, cudaStream_t s)
{
    if (!h->prof.on) return nullptr;
    cudaEvent_t e = prof_event(h);
    if (e) cudaEventRecord(e, s);
    return e;
}

void prof_end(f3dc_handle *h, cudaStream_t s, int fam, const Work &w, cudaEvent_t e0)
{
    h->launches++;
    if (!h->prof.on || !e0) return;
    cudaEvent_t e1 = prof_event(h);
    if (!e1) return;
    cudaEventRecord(e1, s);
    h->prof.pending.push_back(ProfRecord{fam, e0, e1, w});
}

// Launches one kernel through `expr`, bracketed by profiling events.
#define LAUNCH(fam, work, expr)                                                                    \
    do {                                                                                           \
        cudaEvent_t e0_ = prof_begin(h, s);                                                        \
        CK(expr);                                                                                  \
        prof_end(h, s, (fam), (work), e0_);                                                        \
    } while (0)

// Reads the pending event pairs of the last step(s); the plan on the device
// gives the active-token counts that turn each launch's Work into numbers.
f3dc_status prof_drain(f3dc_handle *h, cudaStream_t s)
{
    Profiler &P = h->prof;
    if (P.pending.empty()) return F3DC_OK;
    CK(cudaStreamSynchronize(s));
    Plan plan;
    CK(cudaMemcpy(&plan, h->plan, sizeof(Plan), cudaMemcpyDeviceToHost));
    const int B = h->last_B > 0 ? h->last_B : 1;
    double M = 0, sq = 0, sel = 0;
    for (int b = 0; b < B; ++b) {
        const double a = plan.n_active[b];
        M += a;
        sq += a * a;
        if (a > 0 && a < h->N) sel += h->N;
    }
    const double tok = (double)B * h->N;
    for (const ProfRecord &r : P.pending) {
        float ms = 0.f;
        CK(cudaEventElapsedTime(&ms, r.e0, r.e1));
        const double v = r.w.c_m * M + r.w.c_sq * sq + r.w.c_tok * tok + r.w.c_sel * sel + r.w.c_fix;
        P.launches[r.fam] += 1;
        P.ms[r.fam] += ms;
        (r.w.flops ? P.flops : P.bytes)[r.fam] += v;
    }
    P.pending.clear();
    P.next = 0;
    return F3DC_OK;
}

// f3dc_create's device allocations, numbered from 0 per call (fault injection)
int g_alloc_no = 0;

template <typename T>
cudaError_t dalloc(T **p, size_t count)
{
    const FaultInjection &fi = fault_injection();
    if (fi.fail_alloc_at >= 0 && g_alloc_no++ == fi.fail_alloc_at) return cudaErrorMemoryAllocation;
    return cudaMalloc(reinterpret_cast<void **>(p), count * sizeof(T) + 256);
}

// B-operand box rows of a step weight: 256-wide GEMMs run on CTA pairs.
uint32_t wide_b_box(int bn) { return bn == 256 ? kGemmPairBBox : gemm_b_box_rows(bn); }

// Tile width of a step GEMM: the widest that divides N.  A 128 x 256 tile
// needs 96 B of operands per clock of MMA against 128 B for 128 x 128, and
// the operand stream from L2 into each SM is what bounds these GEMMs: at 4096
// rows, width 1024 runs 9.1 us at 256 against 12.7 us at 128 (K = 1024) and
// 22.8 against 38.4 us (K = 4096), CUDA-graph timed.
int pick_bn(int N)
{
    if (N % 256 == 0) return 256;
    if (N % 128 == 0) return 128;
    return 64;
}

cudaError_t run_gemm(f3dc_handle *h, const CUtensorMap &ta, const CUtensorMap &tb, int N, int K, int bn, int epi,
                     void *out, int ldo, const bf16 *bias, const float *gate, const bf16 *qn, const bf16 *kn,
                     cudaStream_t s)
{
    GemmParams p;
    memset(&p, 0, sizeof(p));
    p.M = h->max_rows;
    p.N = N;
    p.K = K;
    p.m_tiles_dev = &h->plan->n_tiles;
    p.out = out;
    p.ldo = ldo;
    p.bias = bias;
    p.gate = gate;
    p.qn_g = qn;
    p.kn_g = kn;
    p.width = h->W;
    p.dh = h->dh;
    // split K stays off in the step: at 400-1229 active tokens it measured
    // slower than whole tiles (the partial round trip through L2 and the
    // last-arriving CTA's reduction cost more than the shorter K loop saves)
    p.ws = nullptr;
    p.counters = h->gemm_cnt;
    p.ws_units = h->num_sms;
    p.err = h->dev_err;
    // 256-wide tiles run on CTA pairs; those that would leave more than half
    // of the SMs idle (few active rows) run 128 wide
    if (bn == 256) {
        p.narrow_below = h->num_sms / 2;
        return launch_gemm_pair(&ta, &tb, p, epi, (h->max_tiles + 1) / 2 * (N / 128), s);
    }
    const int tiles = h->max_tiles * (N / bn);
    const int grid = tiles < h->num_sms ? tiles : h->num_sms;
    return launch_gemm(&ta, &tb, p, epi, bn, grid, s);
}

cudaError_t run_attention(f3dc_handle *h, int mode, const CUtensorMap &tq, const CUtensorMap &tkv, int q_col0,
                          int k_col0, int v_col0, cudaStream_t s)
{
    AttnParams p;
    memset(&p, 0, sizeof(p));
    p.heads = h->H;
    p.dh = h->dh;
    p.q_col0 = q_col0;
    p.k_col0 = k_col0;
    p.v_col0 = v_col0;
    p.mode = mode;
    p.n_tiles_dev = &h->plan->n_tiles;
    p.tile_sample = h->tile_sample;
    p.plan = h->plan;
    p.nk_fixed = h->Nc;
    p.kv_null_from = mode == 1 ? h->cfg_B_now : 0;
    p.kv_null_sample = h->cfg.max_batch;
    p.kv_prefetch_rows = mode == 1 ? h->cond_B * h->Nc : 0;  // the condition's K / V
    p.out = h->att;
    p.ldo = h->W;
    p.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)h->dh));
    p.err = h->dev_err;
    // work items: (pair of query tiles, head)
    // persistent CTAs, one per work item up to one per SM: (query tile, head)
    // items for the one-tile kernel, (pair of query tiles, head) otherwise
    const bool one = h->attn_one_now;
    const int items = one ? h->max_tiles * h->H : (h->max_tiles + 1) / 2 * h->H;
    const int grid = items < h->num_sms ? items : h->num_sms;
    return one ? launch_attention_one(&tq, &tkv, &tkv, p, grid, s) : launch_attention(&tq, &tkv, &tkv, p, grid, s);
}

// Whether step k's attention takes the one-tile kernel: only when the step's
// quotas are known on the host (f3dc_sample) and its query tiles (each
// sample's active rows padded to 128, doubled on a guided step) times the
// heads fit one item per SM.  Both kernels compute the same attention; this
// only picks the faster one.
bool step_attn_one(const f3dc_handle *h, int k, int B, bool guided)
{
    if (!h->hq_steps) return false;
    int64_t tiles = 0;
    for (int b = 0; b < B; ++b) {
        int c = h->hq_steps[(size_t)k * B + b];
        c = c < 0 ? 0 : (c > h->N ? h->N : c);
        tiles += (h->N - c + kTileRows - 1) / kTileRows;
    }
    if (guided) tiles *= 2;
    return attn_one_tile(tiles, h->H, h->num_sms);
}

bool step_guided(const f3dc_handle *h, int k)
{
    std::vector<float> t(h->T + 1);
    time_schedule(h->cfg, t.data());
    return h->cfg.cfg_strength > 0.0 && (double)t[k - 1] >= h->cfg.cfg_t_lo;
}

// The flow transformer on the packed active rows described by h->plan,
// h->tile_sample and h->active_idx (Sec. 4.2; Supp. Sec. F).
// mod_pre: nullable; this step's modulation vectors, computed beforehand
// (f3dc_sample computes every step's at its start)
f3dc_status run_dit(f3dc_handle *h, float t, const float *S, cudaStream_t s, const float *mod_pre = nullptr)
{
    const int W = h->W, L = h->L, Wm = h->Wm;
    const double dW = W, dWm = Wm;
    const Layout &ly = h->lay;
    // timestep embedding and every block's modulation (adaLN): three GEMVs
    // streaming the embedding and the repacked [L*6W + 2W, W] weights
    const Work w_temb = wfix(2.0 * ((double)h->mod_rows * W + 256.0 * W + dW * W));
    const float *mod = mod_pre;
    if (!mod) {
        LAUNCH(KF_TEMB, Work(), launch_time_freq(t, h->freq, s));
        LAUNCH(KF_TEMB, Work(), launch_gemv(h->freq, 256, h->wt(ly.t_w1), h->wt(ly.t_b1), h->h1, W, 0, 1, h->num_sms, s));
        LAUNCH(KF_TEMB, Work(), launch_gemv(h->h1, W, h->wt(ly.t_w2), h->wt(ly.t_b2), h->temb, W, 0, 0, h->num_sms, s));
        LAUNCH(KF_TEMB, w_temb, launch_gemv(h->temb, W, h->mod_w, h->mod_b, h->mod, h->mod_rows, 1, 0, h->num_sms, s));
        mod = h->mod;
    }
    // gather + embed the active tokens: 32 B latent + 4 B index in, 4W B out
    LAUNCH(KF_GATHER, wm(36.0 + 4.0 * dW),
           launch_gather_embed(S, h->N, W, h->active_idx, h->plan, h->tile_sample, h->wt(ly.in_w), h->wt(ly.in_b),
                               h->pos, h->x, h->max_rows, h->num_sms, h->cfg_B_now, h->dev_err, s));
    const Work w_ln = wm(6.0 * dW);  // fp32 row in, bf16 row out
    Work w_self;
    w_self.c_sq = 4.0 * dW;          // Q K^T and P V among each sample's active tokens
    w_self.flops = true;
    const Work w_cross = wm(4.0 * dW * h->Nc, true);
    for (int l = 0; l < L; ++l) {
        const BlockOffsets &b = ly.blk[l];
        const float *m = mod + (size_t)l * 6 * W;
        // self-attention among the active tokens
        LAUNCH(KF_LN, w_ln, launch_layernorm(h->x, W, h->plan, 0, m, m + W, nullptr, nullptr, h->h, h->max_rows,
                                             h->num_sms, s));
        LAUNCH(KF_GEMM, wm(2.0 * 3 * dW * dW, true),
               run_gemm(h, h->tm_h, h->tm_qkv_w[l], 3 * W, W, h->bn_qkv, kEpiQKNorm, h->qkv, 3 * W, h->wt(b.qkv_b),
                        nullptr, h->wt(b.qn_g), h->wt(b.kn_g), s));
        LAUNCH(KF_ATTN_SELF, w_self, run_attention(h, 0, h->tm_q_self, h->tm_q_self, 0, W, 2 * W, s));
        LAUNCH(KF_GEMM, wm(2.0 * dW * dW, true),
               run_gemm(h, h->tm_att, h->tm_o_w[l], W, W, h->bn_w, kEpiResid, h->x, W, h->wt(b.o_b), m + 2 * W,
                        nullptr, nullptr, s));
        // cross-attention to the condition
        LAUNCH(KF_LN, w_ln, launch_layernorm(h->x, W, h->plan, 1, nullptr, nullptr, h->wt(b.ln2_g), h->wt(b.ln2_b),
                                             h->h, h->max_rows, h->num_sms, s));
        LAUNCH(KF_GEMM, wm(2.0 * dW * dW, true),
               run_gemm(h, h->tm_h, h->tm_cq_w[l], W, W, h->bn_w, kEpiBias, h->qc, W, h->wt(b.cq_b), nullptr,
                        nullptr, nullptr, s));
        LAUNCH(KF_ATTN_CROSS, w_cross, run_attention(h, 1, h->tm_q_cross, h->tm_kv_cross[l], 0, 0, W, s));
        LAUNCH(KF_GEMM, wm(2.0 * dW * dW, true),
               run_gemm(h, h->tm_att, h->tm_co_w[l], W, W, h->bn_w, kEpiResid, h->x, W, h->wt(b.co_b), nullptr,
                        nullptr, nullptr, s));
        // MLP
        LAUNCH(KF_LN, w_ln, launch_layernorm(h->x, W, h->plan, 0, m + 3 * W, m + 4 * W, nullptr, nullptr, h->h,
                                             h->max_rows, h->num_sms, s));
        LAUNCH(KF_GEMM, wm(2.0 * dWm * dW, true),
               run_gemm(h, h->tm_h, h->tm_fc1_w[l], Wm, W, h->bn_fc1, kEpiGelu, h->u, Wm, h->wt(b.fc1_b), nullptr,
                        nullptr, nullptr, s));
        LAUNCH(KF_GEMM, wm(2.0 * dW * dWm, true),
               run_gemm(h, h->tm_u, h->tm_fc2_w[l], W, Wm, h->bn_w, kEpiResid, h->x, W, h->wt(b.fc2_b), m + 5 * W,
                        nullptr, nullptr, s));
    }
    const float *fm = mod + (size_t)L * 6 * W;
    LAUNCH(KF_FINAL, wm(4.0 * dW + 32.0), launch_final_layer(h->x, W, h->plan, fm, fm + W, h->wt(ly.out_w),
                                                             h->wt(ly.out_b), h->v_active, h->max_rows, h->num_sms, s));
    return F3DC_OK;
}

// Runs steps k0..k1 as one CUDA graph (captured on first use for this batch
// size, latent buffer and step range; every step reads its quota and the row
// plan from device memory, so the graph is valid for any quotas).
f3dc_status run_segment_graph(f3dc_handle *h, int B, float *S, int k0, int k1, int ka, cudaStream_t s)
{
    // the attention kernel of each step is part of the captured graph: a
    // replay whose quotas pick other kernels captures anew
    std::vector<uint8_t> one((size_t)(k1 - k0 + 1));
    for (int k = k0; k <= k1; ++k) one[(size_t)(k - k0)] = step_attn_one(h, k, B, step_guided(h, k)) ? 1 : 0;
    f3dc_handle::SegmentGraph *g = nullptr;
    for (auto &e : h->graphs)
        if (e.B == B && e.S == S && e.k0 == k0 && e.k1 == k1 && e.ka == ka && e.attn_one == one) g = &e;
    if (!g) {
        if (h->graphs.size() >= 8) {
            cudaGraphExecDestroy(h->graphs.front().exec);
            h->graphs.erase(h->graphs.begin());
        }
        const int64_t before = h->launches;
        CK(cudaStreamBeginCapture(h->exec_stream, cudaStreamCaptureModeRelaxed));
        f3dc_status st = F3DC_OK;
        for (int k = k0; k <= k1 && st == F3DC_OK; ++k)
            st = f3dc_step(h, k, B, S, h->ring, h->quota_dev + (size_t)k * B, k == ka ? h->dyn : nullptr,
                           h->exec_stream);
        cudaGraph_t graph = nullptr;
        cudaError_t e = cudaStreamEndCapture(h->exec_stream, &graph);
        const int64_t captured = h->launches - before;  // kernels per replay
        h->launches = before;
        if (st != F3DC_OK) {
            if (graph) cudaGraphDestroy(graph);
            return st;
        }
        CK(e);
        cudaGraphExec_t exec = nullptr;
        e = cudaGraphInstantiate(&exec, graph, 0);
        cudaGraphDestroy(graph);
        CK(e);
        h->graphs.push_back(f3dc_handle::SegmentGraph{B, k0, k1, ka, S, one, exec, captured});
        g = &h->graphs.back();
    }
    CK(cudaEventRecord(h->ev_in, s));
    CK(cudaStreamWaitEvent(h->exec_stream, h->ev_in, 0));
    CK(cudaGraphLaunch(g->exec, h->exec_stream));
    CK(cudaEventRecord(h->ev_out, h->exec_stream));
    CK(cudaStreamWaitEvent(s, h->ev_out, 0));
    h->launches += g->launches;
    h->last_stream = s;
    return F3DC_OK;
}

bool build_maps(f3dc_handle *h)
{
    const int W = h->W, Wm = h->Wm, dh = h->dh;
    const uint64_t R = (uint64_t)h->max_rows;
    bool ok = make_tmap_bf16(&h->tm_h, h->h, R, W, W, 128, 64) && make_tmap_bf16(&h->tm_att, h->att, R, W, W, 128, 64) &&
              make_tmap_bf16(&h->tm_u, h->u, R, Wm, Wm, 128, 64) &&
              make_tmap_bf16(&h->tm_q_self, h->qkv, R, 3 * W, 3 * W, 128, dh) &&
              make_tmap_bf16(&h->tm_q_cross, h->qc, R, W, W, 128, dh);
    if (!ok) return false;
    const int L = h->L;
    h->tm_qkv_w.resize(L);
    h->tm_o_w.resize(L);
    h->tm_cq_w.resize(L);
    h->tm_co_w.resize(L);
    h->tm_fc1_w.resize(L);
    h->tm_fc2_w.resize(L);
    h->tm_ckv_w.resize(L);
    h->tm_kv_cross.resize(L);
    for (int l = 0; l < L; ++l) {
        const BlockOffsets &b = h->lay.blk[l];
        ok = ok && make_tmap_bf16(&h->tm_qkv_w[l], h->wt(b.qkv_w), 3 * W, W, W, wide_b_box(h->bn_qkv), 64);
        ok = ok && make_tmap_bf16(&h->tm_o_w[l], h->wt(b.o_w), W, W, W, wide_b_box(h->bn_w), 64);
        ok = ok && make_tmap_bf16(&h->tm_cq_w[l], h->wt(b.cq_w), W, W, W, wide_b_box(h->bn_w), 64);
        ok = ok && make_tmap_bf16(&h->tm_co_w[l], h->wt(b.co_w), W, W, W, wide_b_box(h->bn_w), 64);
        ok = ok && make_tmap_bf16(&h->tm_fc1_w[l], h->wt(b.fc1_w), Wm, W, W, wide_b_box(h->bn_fc1), 64);
        ok = ok && make_tmap_bf16(&h->tm_fc2_w[l], h->wt(b.fc2_w), W, Wm, Wm, wide_b_box(h->bn_w), 64);
        ok = ok && make_tmap_bf16(&h->tm_ckv_w[l], h->wt(b.ckv_w), 2 * W, h->Dc, h->Dc,
                                  h->Dc % 128 == 0 ? wide_b_box(h->bn_ckv) : gemm_b_box_rows(h->bn_ckv), 64);
        ok = ok && make_tmap_bf16(&h->tm_kv_cross[l], h->ckv + (size_t)l * h->ckv_rows * 2 * W, h->ckv_rows, 2 * W,
                                  2 * W, 128, dh);
    }
    return ok;
}

void free_handle(f3dc_handle *h)
{
    void *ptrs[] = {h->wblob, h->mod_w, h->mod_b, h->pos, h->x, h->v_active, h->freq, h->h1, h->temb, h->mod,
                    h->h, h->qkv, h->att, h->qc, h->u, h->ckv, h->ring, h->plan, h->tile_sample, h->active_idx,
                    h->row_of_token, h->n_active, h->mask, h->quota_dev, h->dyn, h->dev_err, h->gemm_ws,
                    h->gemm_cnt, h->dec_scratch, h->dec_bits, h->dyn_curve, h->zero_quota, h->t_all,
                    h->freq_all, h->h1_all, h->temb_all, h->mod_all};
    for (void *p : ptrs)
        if (p) cudaFree(p);
    if (h->h_quota) cudaFreeHost(h->h_quota);
    for (cudaEvent_t ev : h->quota_done)
        if (ev) cudaEventDestroy(ev);
    for (cudaEvent_t ev : h->prof.pool) cudaEventDestroy(ev);
    for (auto &g : h->graphs) cudaGraphExecDestroy(g.exec);
    if (h->ev_in) cudaEventDestroy(h->ev_in);
    if (h->ev_out) cudaEventDestroy(h->ev_out);
    if (h->exec_stream) cudaStreamDestroy(h->exec_stream);
    delete h;
}

}  // namespace

// ============================================================================
// C-ABI
// ============================================================================
extern "C" {

f3dc_status f3dc_config_default(f3dc_config *cfg)
{
    if (!cfg) return fail(nullptr, F3DC_ERR_INVALID_ARG, "null config");
    memset(cfg, 0, sizeof(*cfg));
    cfg->grid = 16;
    cfg->channels = 8;
    cfg->width = 1024;
    cfg->blocks = 24;
    cfg->heads = 16;
    cfg->mlp_ratio = 4;
    cfg->cond_tokens = 1374;
    cfg->cond_dim = 1024;
    cfg->steps = 25;
    cfg->max_batch = 1;
    cfg->gamma_up = 64;
    cfg->tau = 3;
    cfg->f_corr = 3;
    cfg->refresh_mode = F3DC_REFRESH_PERIOD;
    cfg->eta = 3.0;
    cfg->rho_a = 0.2;
    cfg->mu = -0.07;
    cfg->omega = 0.7;
    cfg->xi = 0.7;
    cfg->rho_cfg_off = 0.75;
    cfg->cfg_strength = 0.0;
    cfg->cfg_t_lo = 0.5;
    return F3DC_OK;
}

size_t f3dc_weights_elems(const f3dc_config *cfg)
{
    std::string why;
    if (!config_valid(cfg, why)) return 0;
    return weight_layout(*cfg).total;
}

f3dc_status f3dc_time_schedule(const f3dc_config *cfg, float *t_out)
{
    std::string why;
    if (!config_valid(cfg, why)) return fail(nullptr, F3DC_ERR_INVALID_ARG, why);
    if (!t_out) return fail(nullptr, F3DC_ERR_INVALID_ARG, "null t_out");
    time_schedule(*cfg, t_out);
    return F3DC_OK;
}

f3dc_status f3dc_pcsc_quota(const f3dc_config *cfg, double sigma, int32_t k, int32_t *consec_inout,
                            int32_t *quota_out, int32_t *phase_out)
{
    std::string why;
    if (!config_valid(cfg, why)) return fail(nullptr, F3DC_ERR_INVALID_ARG, why);
    if (!quota_out) return fail(nullptr, F3DC_ERR_INVALID_ARG, "null quota_out");
    if (k < 1 || k > cfg->steps) return fail(nullptr, F3DC_ERR_INVALID_ARG, "step k outside [1, T]");
    if (std::isnan(sigma) || sigma < 0.0) return fail(nullptr, F3DC_ERR_NONFINITE, "sigma must be a non-negative number");
    int phase = 0;
    int q = phase_quota(*cfg, sigma, k, &phase);
    if (consec_inout) q = tau_gate(*cfg, q, consec_inout);
    *quota_out = q;
    if (phase_out) *phase_out = phase;
    return F3DC_OK;
}

f3dc_status f3dc_create(const f3dc_config *cfg, const f3dc_weights *w, void *stream, f3dc_handle **out)
{
    f3dc_handle *h = nullptr;
    std::string why;
    if (!out) return fail(nullptr, F3DC_ERR_INVALID_ARG, "null out");
    *out = nullptr;
    if (!config_valid(cfg, why)) return fail(nullptr, F3DC_ERR_INVALID_ARG, why);
    if (!w || w->layout_version != 2 || !w->blob) return fail(nullptr, F3DC_ERR_INVALID_ARG, "weights: need layout_version 2 and a blob");
    const Layout lay = weight_layout(*cfg);
    if (w->blob_elems != lay.total)
        return fail(nullptr, F3DC_ERR_INVALID_ARG,
                    "weights: blob_elems " + std::to_string(w->blob_elems) + " != " + std::to_string(lay.total));
    cudaStream_t s = (cudaStream_t)stream;

    h = new f3dc_handle();
    h->cfg = *cfg;
    h->lay = lay;
    h->N = cfg->grid * cfg->grid * cfg->grid;
    h->W = cfg->width;
    h->Wm = cfg->mlp_ratio * cfg->width;
    h->H = cfg->heads;
    h->dh = cfg->width / cfg->heads;
    h->L = cfg->blocks;
    h->Nc = cfg->cond_tokens;
    h->Dc = cfg->cond_dim;
    h->G = cfg->gamma_up;
    h->T = cfg->steps;
    const int B = cfg->max_batch;
    // a guided step runs every sample twice (with its condition and with the
    // zero condition, whose K/V rows sit in slot B of the condition cache)
    const bool cfg_on = cfg->cfg_strength > 0.0;
    h->max_tiles = (cfg_on ? 2 : 1) * B * ((h->N + kTileRows - 1) / kTileRows);
    h->max_rows = h->max_tiles * kTileRows;
    h->ckv_rows = ((size_t)(B + (cfg_on ? 1 : 0)) * h->Nc + 2 * kTileRows - 1) / kTileRows * kTileRows;
    h->bn_qkv = pick_bn(3 * h->W);
    h->bn_w = pick_bn(h->W);
    h->bn_fc1 = pick_bn(h->Wm);
    h->bn_ckv = pick_bn(2 * h->W);
    h->mod_rows = h->L * 6 * h->W + 2 * h->W;

    cudaError_t e;
#define CKC(expr)                                                                                  \
    do {                                                                                           \
        e = (expr);                                                                                \
        if (e != cudaSuccess) {                                                                    \
            std::string m_ = std::string(#expr) + ": " + cudaGetErrorString(e);                  \
            free_handle(h);                                                                        \
            return fail(nullptr, e == cudaErrorMemoryAllocation ? F3DC_ERR_OOM : F3DC_ERR_CUDA, m_); \
        }                                                                                          \
    } while (0)
    CKC(cudaGetDevice(&h->device));
    CKC(cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, h->device));
    int cc_major = 0, cc_minor = 0;
    CKC(cudaDeviceGetAttribute(&cc_major, cudaDevAttrComputeCapabilityMajor, h->device));
    CKC(cudaDeviceGetAttribute(&cc_minor, cudaDevAttrComputeCapabilityMinor, h->device));
    if (cc_major != 10 || cc_minor != 3) {
        free_handle(h);
        return fail(nullptr, F3DC_ERR_UNSUPPORTED, "libf3dc is built for sm_103a (GB300) only");
    }

    const size_t R = h->max_rows, W = h->W, N = h->N;
    g_alloc_no = 0;
    CKC(dalloc(&h->wblob, lay.total));
    CKC(cudaMemcpyAsync(h->wblob, w->blob, lay.total * sizeof(bf16), cudaMemcpyDeviceToDevice, s));
    // modulation weights of every block and of the final layer, repacked into
    // one [L*6W + 2W, W] matrix for a single streaming GEMV per step
    CKC(dalloc(&h->mod_w, (size_t)h->mod_rows * W));
    CKC(dalloc(&h->mod_b, (size_t)h->mod_rows));
    const bf16 *src = reinterpret_cast<const bf16 *>(w->blob);
    for (int l = 0; l < h->L; ++l) {
        CKC(cudaMemcpyAsync(h->mod_w + (size_t)l * 6 * W * W, src + lay.blk[l].mod_w, 6 * W * W * sizeof(bf16),
                            cudaMemcpyDeviceToDevice, s));
        CKC(cudaMemcpyAsync(h->mod_b + (size_t)l * 6 * W, src + lay.blk[l].mod_b, 6 * W * sizeof(bf16),
                            cudaMemcpyDeviceToDevice, s));
    }
    CKC(cudaMemcpyAsync(h->mod_w + (size_t)h->L * 6 * W * W, src + lay.fmod_w, 2 * W * W * sizeof(bf16),
                        cudaMemcpyDeviceToDevice, s));
    CKC(cudaMemcpyAsync(h->mod_b + (size_t)h->L * 6 * W, src + lay.fmod_b, 2 * W * sizeof(bf16),
                        cudaMemcpyDeviceToDevice, s));
    {
        std::vector<float> pos = position_table(cfg->grid, h->W);
        CKC(dalloc(&h->pos, pos.size()));
        CKC(cudaMemcpyAsync(h->pos, pos.data(), pos.size() * sizeof(float), cudaMemcpyHostToDevice, s));
        CKC(cudaStreamSynchronize(s));
    }
    CKC(dalloc(&h->x, R * W));
    CKC(dalloc(&h->h, R * W));
    CKC(dalloc(&h->qkv, R * 3 * W));
    CKC(dalloc(&h->att, R * W));
    CKC(dalloc(&h->qc, R * W));
    CKC(dalloc(&h->u, R * h->Wm));
    CKC(dalloc(&h->v_active, R * kChannels));
    CKC(dalloc(&h->ckv, (size_t)h->L * h->ckv_rows * 2 * W));
    CKC(cudaMemsetAsync(h->ckv, 0, (size_t)h->L * h->ckv_rows * 2 * W * sizeof(bf16), s));
    CKC(cudaMemsetAsync(h->x, 0, R * W * sizeof(float), s));
    CKC(cudaMemsetAsync(h->qkv, 0, R * 3 * W * sizeof(bf16), s));
    CKC(cudaMemsetAsync(h->qc, 0, R * W * sizeof(bf16), s));
    CKC(dalloc(&h->freq, 256));
    CKC(dalloc(&h->h1, W));
    CKC(dalloc(&h->temb, W));
    CKC(dalloc(&h->mod, (size_t)h->mod_rows));
    CKC(dalloc(&h->t_all, (size_t)h->T));
    CKC(dalloc(&h->freq_all, (size_t)h->T * 256));
    CKC(dalloc(&h->h1_all, (size_t)h->T * W));
    CKC(dalloc(&h->temb_all, (size_t)h->T * W));
    CKC(dalloc(&h->mod_all, (size_t)h->T * h->mod_rows));
    {
        std::vector<float> tt(h->T + 1);
        time_schedule(*cfg, tt.data());
        CKC(cudaMemcpy(h->t_all, tt.data(), (size_t)h->T * sizeof(float), cudaMemcpyHostToDevice));
    }
    CKC(dalloc(&h->ring, (size_t)3 * B * N * kChannels));
    CKC(dalloc(&h->plan, 1));
    CKC(cudaMemsetAsync(h->plan, 0, sizeof(Plan), s));
    CKC(dalloc(&h->tile_sample, (size_t)h->max_tiles));
    CKC(dalloc(&h->active_idx, (size_t)B * N));
    CKC(dalloc(&h->row_of_token, (size_t)B * N));
    CKC(dalloc(&h->n_active, (size_t)B));
    CKC(dalloc(&h->mask, (size_t)B * N));
    CKC(dalloc(&h->quota_dev, (size_t)(h->T + 1) * B));
    CKC(dalloc(&h->dyn, (size_t)B));
    CKC(dalloc(&h->dyn_curve, (size_t)h->T * B));
    CKC(dalloc(&h->zero_quota, (size_t)B));
    CKC(cudaMemsetAsync(h->zero_quota, 0, (size_t)B * sizeof(int32_t), s));
    if (cfg->decoder == 1) {
        CKC(dalloc(&h->dec_scratch, decode_scratch_floats(B, cfg->grid)));
        CKC(dalloc(&h->dec_bits, (size_t)B * 2 * N));
    }
    CKC(dalloc(&h->dev_err, 1));
    CKC(cudaMemsetAsync(h->dev_err, 0, sizeof(uint32_t), s));
    CKC(dalloc(&h->gemm_ws, gemm_ws_bytes(256, h->num_sms) / sizeof(float)));
    CKC(dalloc(&h->gemm_cnt, (size_t)kGemmMaxCounterTiles));
    CKC(cudaMemsetAsync(h->gemm_cnt, 0, kGemmMaxCounterTiles * sizeof(int32_t), s));
    CKC(cudaMallocHost(reinterpret_cast<void **>(&h->h_quota), (size_t)2 * (h->T + 1) * B * sizeof(int32_t)));
    CKC(cudaEventCreateWithFlags(&h->quota_done[0], cudaEventDisableTiming));
    CKC(cudaEventCreateWithFlags(&h->quota_done[1], cudaEventDisableTiming));
    CKC(cudaStreamCreateWithFlags(&h->exec_stream, cudaStreamNonBlocking));
    CKC(cudaEventCreateWithFlags(&h->ev_in, cudaEventDisableTiming));
    CKC(cudaEventCreateWithFlags(&h->ev_out, cudaEventDisableTiming));
    if (cfg_on) {
        // K/V of the zero condition: W_kv 0 + b_kv, i.e. the bias row in every
        // one of the Nc rows of slot B (what the condition GEMM gives for a
        // zero input, bf16 for bf16)
        for (int l = 0; l < h->L; ++l)
            CKC(launch_broadcast_row(h->ckv + ((size_t)l * h->ckv_rows + (size_t)B * h->Nc) * 2 * W, (size_t)2 * W,
                                     h->wt(h->lay.blk[l].ckv_b), h->Nc, 2 * W, s));
    }
#undef CKC
    if (!build_maps(h)) {
        free_handle(h);
        return fail(nullptr, F3DC_ERR_CUDA, "cuTensorMapEncodeTiled failed");
    }
    e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) {
        std::string m = std::string("create: ") + cudaGetErrorString(e);
        free_handle(h);
        return fail(nullptr, F3DC_ERR_CUDA, m);
    }
    h->last_stream = s;
    *out = h;
    return F3DC_OK;
}

f3dc_status f3dc_destroy(f3dc_handle *h)
{
    if (!h) return F3DC_OK;
    cudaDeviceSynchronize();
    free_handle(h);
    return F3DC_OK;
}

const char *f3dc_last_error(const f3dc_handle *h)
{
    if (h) return h->err.c_str();
    return g_last_error.c_str();
}

f3dc_status f3dc_device_status(f3dc_handle *h, uint32_t *status_out)
{
    if (!h || !status_out) return fail(h, F3DC_ERR_INVALID_ARG, "null argument");
    CK(cudaStreamSynchronize(h->last_stream));
    uint32_t v = 0;
    CK(cudaMemcpy(&v, h->dev_err, sizeof(v), cudaMemcpyDeviceToHost));
    CK(cudaMemset(h->dev_err, 0, sizeof(uint32_t)));
    *status_out = v;
    return F3DC_OK;
}

f3dc_status f3dc_ssc_select(f3dc_handle *h, const void *v_prev1, const void *v_prev2, int32_t B,
                            const int32_t *quota_dev, int32_t *active_idx_out, int32_t *n_active_out,
                            uint8_t *cached_mask_out, void *stream)
{
    if (!h) return fail(nullptr, F3DC_ERR_INVALID_ARG, "null handle");
    if (!v_prev1 || !v_prev2 || !quota_dev || !active_idx_out) return fail(h, F3DC_ERR_INVALID_ARG, "null pointer");
    if (B < 1 || B > h->cfg.max_batch) return fail(h, F3DC_ERR_INVALID_ARG, "B outside [1, max_batch]");
    cudaStream_t s = (cudaStream_t)stream;
    h->last_stream = s;
    SelectArgs a;
    memset(&a, 0, sizeof(a));
    a.v1 = reinterpret_cast<const uint16_t *>(v_prev1);
    a.v2 = reinterpret_cast<const uint16_t *>(v_prev2);
    a.quota = quota_dev;
    a.B = B;
    a.N = h->N;
    a.wa = (float)h->cfg.omega;
    a.wv = 1.0f - a.wa;
    a.active_idx = active_idx_out;
    a.n_active = n_active_out;
    a.mask = cached_mask_out;
    a.err = h->dev_err;
    LAUNCH(KF_SELECT, Work(), launch_ssc_select(a, s));
    return F3DC_OK;
}

f3dc_status f3dc_set_cond(f3dc_handle *h, const void *cond, int32_t B, void *stream)
{
    if (!h) return fail(nullptr, F3DC_ERR_INVALID_ARG, "null handle");
    if (!cond) return fail(h, F3DC_ERR_INVALID_ARG, "null cond");
    if (B < 1 || B > h->cfg.max_batch) return fail(h, F3DC_ERR_INVALID_ARG, "B outside [1, max_batch]");
    if (((uintptr_t)cond & 15) != 0) return fail(h, F3DC_ERR_INVALID_ARG, "cond must be 16-byte aligned");
    cudaStream_t s = (cudaStream_t)stream;
    h->last_stream = s;
    const int rows = B * h->Nc;
    if (!make_tmap_bf16(&h->tm_cond, cond, rows, h->Dc, h->Dc, 128, 64))
        return fail(h, F3DC_ERR_CUDA, "cuTensorMapEncodeTiled failed for cond");
    for (int l = 0; l < h->L; ++l) {
        GemmParams p;
        memset(&p, 0, sizeof(p));
        p.M = rows;
        p.N = 2 * h->W;
        p.K = h->Dc;
        p.m_tiles = (rows + kTileRows - 1) / kTileRows;
        p.out = h->ckv + (size_t)l * h->ckv_rows * 2 * h->W;
        p.ldo = 2 * h->W;
        p.bias = h->wt(h->lay.blk[l].ckv_b);
        p.err = h->dev_err;
        const int tiles = p.m_tiles * (p.N / h->bn_ckv);
        if (h->bn_ckv == 256 && h->Dc % 128 == 0) {
            p.narrow_below = h->num_sms / 2;
            LAUNCH(KF_GEMM_COND, wfix(2.0 * rows * p.N * (double)p.K, true),
                   launch_gemm_pair(&h->tm_cond, &h->tm_ckv_w[l], p, kEpiBias, (p.m_tiles + 1) / 2 * (p.N / 128), s));
        } else {
            LAUNCH(KF_GEMM_COND, wfix(2.0 * rows * p.N * (double)p.K, true),
                   launch_gemm(&h->tm_cond, &h->tm_ckv_w[l], p, kEpiBias, h->bn_ckv,
                               tiles < h->num_sms ? tiles : h->num_sms, s));
        }
    }
    h->cond_B = B;
    return F3DC_OK;
}

f3dc_status f3dc_step(f3dc_handle *h, int32_t k, int32_t B, float *S_inout, void *v_ring,
                      const int32_t *quota_dev, int64_t *dyn_voxels_dev, void *stream)
{
    if (!h) return fail(nullptr, F3DC_ERR_INVALID_ARG, "null handle");
    if (!S_inout || !v_ring || !quota_dev) return fail(h, F3DC_ERR_INVALID_ARG, "null pointer");
    if (k < 1 || k > h->T) return fail(h, F3DC_ERR_INVALID_ARG, "step k outside [1, T]");
    if (B < 1 || B > h->cfg.max_batch) return fail(h, F3DC_ERR_INVALID_ARG, "B outside [1, max_batch]");
    if (B > h->cond_B) return fail(h, F3DC_ERR_INVALID_ARG, "f3dc_set_cond was not called for this batch");
    cudaStream_t s = (cudaStream_t)stream;
    h->last_stream = s;
    const size_t slot = (size_t)B * h->N * kChannels;
    uint16_t *ring = reinterpret_cast<uint16_t *>(v_ring);
    uint16_t *v_new = ring + (size_t)(k % 3) * slot;
    const uint16_t *v1 = ring + (size_t)((k - 1) % 3) * slot;
    const uint16_t *v2 = ring + (size_t)(((k - 2) % 3 + 3) % 3) * slot;

    // Eq. 1 with the convolutional decoder: the grid before the step, as bits
    const bool conv_dec = dyn_voxels_dev && h->cfg.decoder == 1;
    auto decode = [&](int compare) {
        DecodeArgs d;
        memset(&d, 0, sizeof(d));
        d.S = S_inout;
        d.B = B;
        d.D = h->cfg.grid;
        d.w1 = reinterpret_cast<const uint16_t *>(h->wt(h->lay.dc1_w));
        d.b1 = reinterpret_cast<const uint16_t *>(h->wt(h->lay.dc1_b));
        d.w2 = reinterpret_cast<const uint16_t *>(h->wt(h->lay.dc2_w));
        d.b2 = reinterpret_cast<const uint16_t *>(h->wt(h->lay.dc2_b));
        d.w3 = reinterpret_cast<const uint16_t *>(h->wt(h->lay.dc3_w));
        d.b3 = reinterpret_cast<const uint16_t *>(h->wt(h->lay.dc3_b));
        d.scratch = h->dec_scratch;
        d.bits = h->dec_bits;
        d.compare = compare;
        d.dyn = dyn_voxels_dev;
        d.num_sms = h->num_sms;
        return launch_decode_conv(d, s);
    };
    // (4D)^3 outputs of the last layer plus (2D)^3 x 8 and D^3 x 16 before it
    const Work w_dec = wfix(2.0 * 27 * (double)h->N * B * (8 * 16 + 64 * 16 * 8 / 8 + 64 * 8), true);
    if (conv_dec) LAUNCH(KF_DECODE, w_dec, decode(0));

    // classifier-free guidance when t_k lies in the CFG interval (Supp. Sec. D)
    std::vector<float> t(h->T + 1);
    time_schedule(h->cfg, t.data());
    const bool guided = h->cfg.cfg_strength > 0.0 && (double)t[k - 1] >= h->cfg.cfg_t_lo;

    // SSC selection + row plan (Algorithm 1 step 2, first line); a guided
    // step's plan adds an unguided copy of every sample
    SelectArgs a;
    memset(&a, 0, sizeof(a));
    a.cfg_dup = guided ? 1 : 0;
    a.v1 = v1;
    a.v2 = v2;
    // v(t-3) still sits in the slot this step overwrites (zeros before step 3)
    a.v3 = h->cfg.ssc_accel ? v_new : nullptr;
    a.quota = quota_dev;
    a.B = B;
    a.N = h->N;
    a.wa = (float)h->cfg.omega;
    a.wv = 1.0f - a.wa;
    a.active_idx = h->active_idx;
    a.n_active = h->n_active;
    a.mask = h->mask;
    a.row_of_token = h->row_of_token;
    a.plan = h->plan;
    a.tile_sample = h->tile_sample;
    a.err = h->dev_err;
    h->last_B = B;
    Work w_sel;
    w_sel.c_sel = 33.0;  // two bf16 history slots (32 B) and the mask byte per token
    w_sel.c_m = 4.0;     // one index per active token
    LAUNCH(KF_SELECT, w_sel, launch_ssc_select(a, s));

    // FlowTransformer on the active tokens at t_k
    h->cfg_B_now = guided ? B : 0;
    h->attn_one_now = step_attn_one(h, k, B, guided);
    f3dc_status st = run_dit(h, t[k - 1], S_inout, s,
                             h->mod_pre ? h->mod_all + (size_t)(k - 1) * h->mod_rows : nullptr);
    h->cfg_B_now = 0;
    h->attn_one_now = false;
    if (st != F3DC_OK) return st;

    // merge + Euler + history (Algorithm 1 step 3)
    MergeArgs m;
    memset(&m, 0, sizeof(m));
    m.S = S_inout;
    m.v_active = h->v_active;
    m.row_of_token = h->row_of_token;
    m.v_prev1 = v1;
    m.v_out = v_new;
    m.B = B;
    m.N = h->N;
    m.dt = t[k - 1] - t[k];
    m.dec_w = reinterpret_cast<const uint16_t *>(h->wt(h->lay.dec_w));
    m.G = h->G;
    m.dyn = conv_dec ? nullptr : dyn_voxels_dev;  // the linear decoder is fused into the merge
    m.max_rows = h->max_rows;
    m.cfg_s = guided ? (float)h->cfg.cfg_strength : 0.0f;
    m.plan = h->plan;
    m.err = h->dev_err;
    Work w_merge;
    w_merge.c_tok = 96.0;  // S in/out (32 + 32 B), cached velocity in, v_t out (16 + 16 B)
    w_merge.c_m = 32.0;    // fresh fp32 velocity of each active token
    LAUNCH(KF_MERGE, w_merge, launch_merge_euler(m, s));
    if (conv_dec) LAUNCH(KF_DECODE, w_dec, decode(1));  // the grid after the step, XOR-counted
    if (h->prof.on) return prof_drain(h, s);
    return F3DC_OK;
}

static f3dc_status sample_run(f3dc_handle *h, float *S_inout, const void *cond, int32_t B, const double *sigma_override,
                       const int32_t *quota_schedule, int32_t *quota_log, double *sigma_out, void *stream);

f3dc_status f3dc_sample(f3dc_handle *h, float *S_inout, const void *cond, int32_t B, const double *sigma_override,
                        const int32_t *quota_schedule, int32_t *quota_log, double *sigma_out, void *stream)
{
    if (!h) return fail(nullptr, F3DC_ERR_INVALID_ARG, "null handle");
    // the time embedding and the modulation of all T steps depend only on
    // t_k and the weights: computed once here, in four passes per 8 steps
    // over the modulation weights, and read by each step
    const int W = h->W;
    const Layout &ly = h->lay;
    cudaStream_t s = (cudaStream_t)stream;
    const Work w_pre = wfix(2.0 * ((double)h->mod_rows * W + 256.0 * W + (double)W * W) * ((h->T + 7) / 8));
    LAUNCH(KF_TEMB, Work(), launch_time_freq_many(h->t_all, h->T, h->freq_all, s));
    LAUNCH(KF_TEMB, Work(), launch_gemv_many(h->freq_all, h->T, 256, h->wt(ly.t_w1), h->wt(ly.t_b1), h->h1_all, W, 0, 1,
                                             h->num_sms, s));
    LAUNCH(KF_TEMB, Work(), launch_gemv_many(h->h1_all, h->T, W, h->wt(ly.t_w2), h->wt(ly.t_b2), h->temb_all, W, 0, 0,
                                             h->num_sms, s));
    LAUNCH(KF_TEMB, w_pre, launch_gemv_many(h->temb_all, h->T, W, h->mod_w, h->mod_b, h->mod_all, h->mod_rows, 1, 0,
                                            h->num_sms, s));
    // each of the three calls above launches one kernel per group of vectors
    h->launches += (gemv_many_kernels(h->T, 256) - 1) + 2 * (gemv_many_kernels(h->T, W) - 1);
    h->mod_pre = true;
    const f3dc_status st = sample_run(h, S_inout, cond, B, sigma_override, quota_schedule, quota_log, sigma_out, stream);
    h->mod_pre = false;
    return st;
}

static f3dc_status sample_run(f3dc_handle *h, float *S_inout, const void *cond, int32_t B, const double *sigma_override,
                       const int32_t *quota_schedule, int32_t *quota_log, double *sigma_out, void *stream)
{
    if (!h) return fail(nullptr, F3DC_ERR_INVALID_ARG, "null handle");
    if (!S_inout || !cond) return fail(h, F3DC_ERR_INVALID_ARG, "null pointer");
    if (B < 1 || B > h->cfg.max_batch) return fail(h, F3DC_ERR_INVALID_ARG, "B outside [1, max_batch]");
    if (sigma_override)
        for (int b = 0; b < B; ++b)
            if (std::isnan(sigma_override[b]) || sigma_override[b] < 0.0)
                return fail(h, F3DC_ERR_NONFINITE, "sigma_override must be non-negative numbers");
    cudaStream_t s = (cudaStream_t)stream;
    const int T = h->T, N = h->N;
    const int ka = ceil_steps(T, h->cfg.rho_a);
    f3dc_status st = f3dc_set_cond(h, cond, B, stream);
    if (st != F3DC_OK) return st;
    CK(cudaMemsetAsync(h->ring, 0, (size_t)3 * B * N * kChannels * sizeof(uint16_t), s));
    CK(cudaMemsetAsync(h->dyn, 0, (size_t)B * sizeof(int64_t), s));

    const unsigned gen = h->calls++ & 1u;
    CK(cudaEventSynchronize(h->quota_done[gen]));  // slots of the call before last are free
    int32_t *hq = h->h_quota + (size_t)gen * (T + 1) * B;
    std::vector<double> sigma(B, 0.0), measured(B, 0.0);
    if (sigma_override)
        for (int b = 0; b < B; ++b) sigma[b] = sigma_override[b];
    std::vector<int32_t> consec(B, 0);
    const bool need_measure = !quota_schedule && !sigma_override && ka >= 1 && ka < T;
    bool have_measured = false;
    // effective quotas (phase rule or caller schedule, then tau) of steps k0..k1
    auto fill = [&](int k0, int k1) {
        for (int k = k0; k <= k1; ++k)
            for (int b = 0; b < B; ++b) {
                int phase = 0;
                int c = quota_schedule ? quota_schedule[(size_t)(k - 1) * B + b]
                                       : phase_quota(h->cfg, sigma[b], k, &phase);
                c = c < 0 ? 0 : (c > N ? N : c);
                hq[(size_t)k * B + b] = tau_gate(h->cfg, c, &consec[b]);
                if (quota_log) quota_log[(size_t)(k - 1) * B + b] = hq[(size_t)k * B + b];
            }
    };
    // the steps' quotas stay readable on the host while they run (kernel choice)
    struct HostQuotas {
        f3dc_handle *h;
        HostQuotas(f3dc_handle *hh, const int32_t *q) : h(hh) { h->hq_steps = q; }
        ~HostQuotas() { h->hq_steps = nullptr; }
    };
    auto run = [&](int k0, int k1) -> f3dc_status {
        HostQuotas hq_guard(h, hq);
        CK(cudaMemcpyAsync(h->quota_dev + (size_t)k0 * B, hq + (size_t)k0 * B, (size_t)(k1 - k0 + 1) * B * sizeof(int32_t),
                           cudaMemcpyHostToDevice, s));
        if (h->use_graphs && !h->prof.on) return run_segment_graph(h, B, S_inout, k0, k1, ka, s);
        for (int k = k0; k <= k1; ++k) {
            f3dc_status r = f3dc_step(h, k, B, S_inout, h->ring, h->quota_dev + (size_t)k * B,
                                      k == ka ? h->dyn : nullptr, stream);
            if (r != F3DC_OK) return r;
        }
        return F3DC_OK;
    };
    if (need_measure) {
        // Phase 1 up to the anchor, read sigma (Eq. 1 at k_a), then the rest
        fill(1, ka);
        if ((st = run(1, ka)) != F3DC_OK) return st;
        std::vector<int64_t> d(B);
        CK(cudaMemcpyAsync(d.data(), h->dyn, (size_t)B * sizeof(int64_t), cudaMemcpyDeviceToHost, s));
        CK(cudaStreamSynchronize(s));
        for (int b = 0; b < B; ++b) sigma[b] = measured[b] = (double)d[b];
        have_measured = true;
        fill(ka + 1, T);
        if ((st = run(ka + 1, T)) != F3DC_OK) return st;
    } else {
        fill(1, T);
        if ((st = run(1, T)) != F3DC_OK) return st;
    }
    h->last_stream = s;
    if (sigma_out) {
        if (!have_measured && ka >= 1 && ka <= T) {
            std::vector<int64_t> d(B);
            CK(cudaMemcpyAsync(d.data(), h->dyn, (size_t)B * sizeof(int64_t), cudaMemcpyDeviceToHost, s));
            CK(cudaStreamSynchronize(s));
            for (int b = 0; b < B; ++b) measured[b] = (double)d[b];
        }
        for (int b = 0; b < B; ++b) sigma_out[b] = measured[b];
    }
    CK(cudaEventRecord(h->quota_done[gen], s));
    if (quota_log) CK(cudaStreamSynchronize(s));
    return F3DC_OK;
}

f3dc_status f3dc_dynamic_voxel_curve(f3dc_handle *h, float *S_inout, const void *cond, int32_t B,
                                     int64_t *curve_out, void *stream)
{
    if (!h) return fail(nullptr, F3DC_ERR_INVALID_ARG, "null handle");
    if (!S_inout || !cond || !curve_out) return fail(h, F3DC_ERR_INVALID_ARG, "null pointer");
    if (B < 1 || B > h->cfg.max_batch) return fail(h, F3DC_ERR_INVALID_ARG, "B outside [1, max_batch]");
    cudaStream_t s = (cudaStream_t)stream;
    f3dc_status st = f3dc_set_cond(h, cond, B, stream);
    if (st != F3DC_OK) return st;
    CK(cudaMemsetAsync(h->ring, 0, (size_t)3 * B * h->N * kChannels * sizeof(uint16_t), s));
    CK(cudaMemsetAsync(h->dyn_curve, 0, (size_t)h->T * B * sizeof(int64_t), s));
    for (int k = 1; k <= h->T; ++k) {
        st = f3dc_step(h, k, B, S_inout, h->ring, h->zero_quota, h->dyn_curve + (size_t)(k - 1) * B, stream);
        if (st != F3DC_OK) return st;
    }
    CK(cudaMemcpyAsync(curve_out, h->dyn_curve, (size_t)h->T * B * sizeof(int64_t), cudaMemcpyDeviceToHost, s));
    CK(cudaStreamSynchronize(s));
    h->last_stream = s;
    return F3DC_OK;
}

f3dc_status f3dc_fit_mu(const double *curves, int32_t n, int32_t T, int32_t k_lo, int32_t k_hi, double tol,
                        double min_frac, double *mu_out, double *slopes_out, int32_t *kept_out)
{
    if (!curves || !mu_out || n < 0 || T < 1 || k_lo < 1 || k_hi < k_lo || !(tol >= 0.0) ||
        !(min_frac >= 0.0 && min_frac <= 1.0))
        return fail(nullptr, F3DC_ERR_INVALID_ARG, "fit_mu: bad arguments");
    std::vector<double> kept_slopes;
    for (int i = 0; i < n; ++i) {
        // the window's points (k, ln dS_k), zero counts left out
        std::vector<double> x, y;
        for (int k = k_lo; k <= k_hi && k <= T; ++k) {
            const double d = curves[(size_t)i * T + (k - 1)];
            if (d > 0.0) {
                x.push_back((double)k);
                y.push_back(std::log(d));
            }
        }
        const int m = (int)x.size();
        double slope = std::nan("");
        bool keep = false;
        if (m >= 3) {
            // exhaustive hypotheses: the line through every pair of points
            int best_in = -1;
            double best_sse = INFINITY, ba = 0.0, bb = 0.0;
            for (int p = 0; p < m; ++p)
                for (int q = p + 1; q < m; ++q) {
                    const double b = (y[q] - y[p]) / (x[q] - x[p]);
                    const double a = y[p] - b * x[p];
                    int in = 0;
                    double sse = 0.0;
                    for (int j = 0; j < m; ++j) {
                        const double r = y[j] - (a + b * x[j]);
                        if (std::fabs(r) <= tol) {
                            ++in;
                            sse += r * r;
                        }
                    }
                    if (in > best_in || (in == best_in && sse < best_sse)) {
                        best_in = in;
                        best_sse = sse;
                        ba = a;
                        bb = b;
                    }
                }
            // least-squares slope over the winning line's inliers
            double sx = 0.0, sy = 0.0, sxx = 0.0, sxy = 0.0;
            int c = 0;
            for (int j = 0; j < m; ++j)
                if (std::fabs(y[j] - (ba + bb * x[j])) <= tol) {
                    sx += x[j];
                    sy += y[j];
                    sxx += x[j] * x[j];
                    sxy += x[j] * y[j];
                    ++c;
                }
            const double den = c * sxx - sx * sx;
            slope = den != 0.0 ? (c * sxy - sx * sy) / den : bb;
            keep = (double)best_in >= min_frac * (double)m;
        }
        if (slopes_out) slopes_out[i] = slope;
        if (kept_out) kept_out[i] = keep ? 1 : 0;
        if (keep) kept_slopes.push_back(slope);
    }
    double mu = std::nan("");
    if (!kept_slopes.empty()) {
        std::sort(kept_slopes.begin(), kept_slopes.end());
        const size_t c = kept_slopes.size();
        mu = (c % 2) ? kept_slopes[c / 2] : 0.5 * (kept_slopes[c / 2 - 1] + kept_slopes[c / 2]);
    }
    *mu_out = mu;
    return F3DC_OK;
}

f3dc_status f3dc_forward(f3dc_handle *h, float t, int32_t B, const float *S, const int32_t *active_idx,
                         const int32_t *n_active, float *v_out, void *stream)
{
    if (!h) return fail(nullptr, F3DC_ERR_INVALID_ARG, "null handle");
    if (!S || !active_idx || !n_active || !v_out) return fail(h, F3DC_ERR_INVALID_ARG, "null pointer");
    if (B < 1 || B > h->cfg.max_batch) return fail(h, F3DC_ERR_INVALID_ARG, "B outside [1, max_batch]");
    if (B > h->cond_B) return fail(h, F3DC_ERR_INVALID_ARG, "f3dc_set_cond was not called for this batch");
    cudaStream_t s = (cudaStream_t)stream;
    h->last_stream = s;
    CK(cudaMemcpyAsync(h->active_idx, active_idx, (size_t)B * h->N * sizeof(int32_t), cudaMemcpyDeviceToDevice, s));
    h->last_B = B;
    LAUNCH(KF_PLAN, Work(), launch_plan_from_counts(n_active, h->active_idx, B, h->N, h->plan, h->tile_sample,
                                                    nullptr, h->dev_err, s));
    f3dc_status st = run_dit(h, t, S, s);
    if (st != F3DC_OK) return st;
    LAUNCH(KF_SCATTER, wm(64.0), launch_scatter_rows(h->v_active, h->plan, B, h->N, v_out, s));
    if (h->prof.on) return prof_drain(h, s);
    return F3DC_OK;
}

f3dc_status f3dc_profile(f3dc_handle *h, int32_t enable)
{
    if (!h) return fail(nullptr, F3DC_ERR_INVALID_ARG, "null handle");
    CK(cudaStreamSynchronize(h->last_stream));
    h->prof.reset();
    h->prof.on = enable != 0;
    return F3DC_OK;
}

f3dc_status f3dc_profile_read(f3dc_handle *h, f3dc_kernel_stats *out, int32_t capacity, int32_t *count)
{
    if (!h || !count || (capacity > 0 && !out)) return fail(h, F3DC_ERR_INVALID_ARG, "null argument");
    f3dc_status st = prof_drain(h, h->last_stream);
    if (st != F3DC_OK) return st;
    int n = 0;
    for (int f = 0; f < KF_COUNT; ++f) {
        if (h->prof.launches[f] == 0) continue;
        if (n < capacity) {
            f3dc_kernel_stats &o = out[n];
            memset(&o, 0, sizeof(o));
            strncpy(o.name, kFamilyName[f], sizeof(o.name) - 1);
            o.launches = h->prof.launches[f];
            o.total_ms = h->prof.ms[f];
            o.flops = h->prof.flops[f];
            o.bytes = h->prof.bytes[f];
        }
        ++n;
    }
    *count = n;
    return F3DC_OK;
}

f3dc_status f3dc_set_graphs(f3dc_handle *h, int32_t enable)
{
    if (!h) return fail(nullptr, F3DC_ERR_INVALID_ARG, "null handle");
    h->use_graphs = enable != 0;
    return F3DC_OK;
}

f3dc_status f3dc_launch_count(const f3dc_handle *h, int64_t *count)
{
    if (!h || !count) return fail(nullptr, F3DC_ERR_INVALID_ARG, "null argument");
    *count = h->launches;
    return F3DC_OK;
}

f3dc_status f3dc_gemm(const void *A, const void *B, const void *bias, const float *gate, void *out, int32_t M,
                      int32_t N, int32_t K, int32_t epilogue, void *stream)
{
    f3dc_handle *h = nullptr;
    if (!A || !B || !out) return fail(nullptr, F3DC_ERR_INVALID_ARG, "null pointer");
    if (M < 1 || N < 64 || N % 64 != 0 || K < 64 || K % 64 != 0)
        return fail(nullptr, F3DC_ERR_INVALID_ARG, "need M >= 1, N and K positive multiples of 64");
    if (epilogue < F3DC_EPI_BIAS || epilogue > F3DC_EPI_RESID) return fail(nullptr, F3DC_ERR_INVALID_ARG, "bad epilogue");
    if (((uintptr_t)out & 15) || (bias && ((uintptr_t)bias & 15)) || (gate && ((uintptr_t)gate & 15)))
        return fail(nullptr, F3DC_ERR_INVALID_ARG, "pointers must be 16-byte aligned");
    const int bn = N % 256 == 0 ? 256 : (N % 128 == 0 ? 128 : 64);
    int dev = 0, sms = 0;
    CK(cudaGetDevice(&dev));
    CK(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
    const int m_tiles = (M + kTileRows - 1) / kTileRows;
    // 256-wide tiles without split K run on CTA pairs
    const bool pair = bn == 256 && K % 128 == 0 && gemm_split_count(m_tiles * (N / bn), gemm_grid(m_tiles * (N / bn), sms), K / 64,
                                                    sms, true) == 1;
    CUtensorMap ta, tb;
    if (!make_tmap_bf16(&ta, A, M, K, K, 128, 64) ||
        !make_tmap_bf16(&tb, B, N, K, K, pair ? kGemmPairBBox : gemm_b_box_rows(bn), 64))
        return fail(nullptr, F3DC_ERR_INVALID_ARG, "cuTensorMapEncodeTiled rejected A or B (alignment?)");
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
    // a bounded wait that runs out is recorded here (read by f3dc_gemm_status)
    p.err = gemm_status_word();
    if (!p.err) return fail(nullptr, F3DC_ERR_CUDA, "cannot resolve the GEMM status word");
    const int tiles = p.m_tiles * (N / bn);
    const int epi = epilogue == F3DC_EPI_BIAS ? kEpiBias : (epilogue == F3DC_EPI_GELU ? kEpiGelu : kEpiResid);
    cudaStream_t s = (cudaStream_t)stream;
    if (pair) {
        p.narrow_below = sms / 2;
        CK(launch_gemm_pair(&ta, &tb, p, epi, (m_tiles + 1) / 2 * (N / 128), s));
        return F3DC_OK;
    }
    // split-K workspace: allocated once per device on first use and kept for
    // the life of the process
    static std::mutex ws_lock;
    static std::vector<std::pair<int, void *>> ws_per_device;
    void *ws = nullptr;
    {
        std::lock_guard<std::mutex> g(ws_lock);
        for (auto &e : ws_per_device)
            if (e.first == dev) ws = e.second;
        if (!ws) {
            CK(cudaMalloc(&ws, gemm_ws_bytes(256, sms) + kGemmMaxCounterTiles * sizeof(int32_t)));
            CK(cudaMemset(reinterpret_cast<char *>(ws) + gemm_ws_bytes(256, sms), 0,
                          kGemmMaxCounterTiles * sizeof(int32_t)));
            ws_per_device.push_back({dev, ws});
        }
    }
    p.ws = reinterpret_cast<float *>(ws);
    p.counters = reinterpret_cast<int32_t *>(reinterpret_cast<char *>(ws) + gemm_ws_bytes(256, sms));
    p.ws_units = sms;
    p.split_extra = fault_injection().gemm_missing_arrivals;
    p.split_wait_ns = fault_injection().gemm_wait_ns;
    // a launch whose split wait ran out leaves its tile counters raised: they
    // start at zero for every launch
    CK(cudaMemsetAsync(p.counters, 0, kGemmMaxCounterTiles * sizeof(int32_t), s));
    CK(launch_gemm(&ta, &tb, p, epi, bn, gemm_grid(tiles, sms), s));
    return F3DC_OK;
}

f3dc_status f3dc_set_fault_injection(const f3dc_fault_injection *fi)
{
    FaultInjection &f = fault_injection();
    if (!fi) {
        f = FaultInjection();
        return F3DC_OK;
    }
    if (fi->fail_alloc_at < -1 || fi->gemm_missing_arrivals < 0 || fi->gemm_missing_arrivals > 1024 ||
        fi->gemm_wait_ns < 0 || (fi->attn_missing_kv != 0 && fi->attn_missing_kv != 1))
        return fail(nullptr, F3DC_ERR_INVALID_ARG, "fault injection: values out of range");
    f.fail_alloc_at = fi->fail_alloc_at;
    f.gemm_missing_arrivals = fi->gemm_missing_arrivals;
    f.gemm_wait_ns = (uint64_t)fi->gemm_wait_ns;
    f.attn_missing_kv = fi->attn_missing_kv;
    return F3DC_OK;
}

f3dc_status f3dc_attention(const void *q, int32_t ldq, const void *k, const void *v, int32_t ldkv, void *out,
                           int32_t nq, int32_t nk, int32_t heads, int32_t dh, void *stream)
{
    f3dc_handle *h = nullptr;
    if (!q || !k || !v || !out) return fail(nullptr, F3DC_ERR_INVALID_ARG, "null pointer");
    if (nq < 1 || nk < 1 || heads < 1 || (dh != 32 && dh != 64) || ldq % 8 || ldkv % 8 || ldq < heads * dh ||
        ldkv < heads * dh)
        return fail(nullptr, F3DC_ERR_INVALID_ARG, "bad attention shape");
    CUtensorMap tq, tk, tv;
    if (!make_tmap_bf16(&tq, q, nq, ldq, ldq, 128, dh) || !make_tmap_bf16(&tk, k, nk, ldkv, ldkv, 128, dh) ||
        !make_tmap_bf16(&tv, v, nk, ldkv, ldkv, 128, dh))
        return fail(nullptr, F3DC_ERR_INVALID_ARG, "cuTensorMapEncodeTiled rejected q / k / v (alignment?)");
    AttnParams p;
    memset(&p, 0, sizeof(p));
    p.heads = heads;
    p.dh = dh;
    p.mode = 2;
    p.n_tiles = (nq + 127) / 128;
    p.nk_fixed = nk;
    p.q_rows = nq;
    p.out = reinterpret_cast<bf16 *>(out);
    p.ldo = heads * dh;
    p.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)dh));
    // a bounded wait that runs out is recorded here (read by f3dc_gemm_status)
    p.err = gemm_status_word();
    if (!p.err) return fail(nullptr, F3DC_ERR_CUDA, "cannot resolve the status word");
    p.fault_skip_kv = fault_injection().attn_missing_kv;
    int dev = 0, sms = 0;
    CK(cudaGetDevice(&dev));
    CK(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
    // one-tile items when each gets an SM of its own, pairs of query tiles otherwise
    if (attn_one_tile(p.n_tiles, heads, sms)) {
        CK(launch_attention_one(&tq, &tk, &tv, p, p.n_tiles * heads, (cudaStream_t)stream));
    } else {
        const int items = (p.n_tiles + 1) / 2 * heads;  // (pair of query tiles, head)
        CK(launch_attention(&tq, &tk, &tv, p, items < sms ? items : sms, (cudaStream_t)stream));
    }
    return F3DC_OK;
}

}  // extern "C"
