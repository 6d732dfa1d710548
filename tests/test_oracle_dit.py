"""Oracle pins for the flow transformer on an active subset (Sec. 4.2,
Supp. Sec. F) and for the whole sampler (Algorithm 1)."""
import numpy as np
import pytest

from paper_2511_22533_gb300 import synth

TINY = synth.SHAPES["tiny"]


@pytest.fixture(scope="module")
def tiny(orc):
    blob = synth.weights_blob(TINY, 0)
    m = orc.Model(TINY, blob)
    cond = synth.cond_tokens(TINY, 2, 0)
    S = synth.latents(TINY, 2, 0)
    kv = m.cond_kv(cond[0])
    return dict(model=m, blob=blob, cond=cond, S=S, kv=kv)


def test_forward_shapes_and_finite(tiny):
    m, S, kv = tiny["model"], tiny["S"][0], tiny["kv"]
    v = m.forward(S, np.arange(TINY.tokens), 0.8, kv)
    assert v.shape == (TINY.tokens, TINY.channels) and np.isfinite(v).all()
    assert 0.05 < v.std() < 20


def test_forward_permutation_equivariant(tiny):
    # attention is permutation-equivariant over the active set: reordering the
    # active list reorders the outputs and changes nothing else
    m, S, kv = tiny["model"], tiny["S"][0], tiny["kv"]
    rng = np.random.default_rng(0)
    idx = np.sort(rng.choice(TINY.tokens, 200, replace=False)).astype(np.int32)
    p = rng.permutation(200)
    v = m.forward(S, idx, 0.7, kv)
    vp = m.forward(S, idx[p], 0.7, kv)
    np.testing.assert_allclose(vp, v[p], rtol=1e-5, atol=1e-5)


def test_forward_ignores_cached_tokens(tiny):
    # self-attention runs among the active tokens only (Sec. 4.2): the latent
    # of a token outside I_active cannot influence any active output
    m, S, kv = tiny["model"], tiny["S"][0].copy(), tiny["kv"]
    idx = np.arange(0, TINY.tokens, 3, dtype=np.int32)
    v = m.forward(S, idx, 0.6, kv)
    S[1] += 100.0
    S[TINY.tokens - 1] -= 50.0
    v2 = m.forward(S, idx, 0.6, kv)
    np.testing.assert_array_equal(v, v2)


def test_forward_depends_on_active_neighbours(tiny):
    m, S, kv = tiny["model"], tiny["S"][0].copy(), tiny["kv"]
    idx = np.arange(0, 64, dtype=np.int32)
    v = m.forward(S, idx, 0.6, kv)
    S[5] += 1.0
    v2 = m.forward(S, idx, 0.6, kv)
    assert np.abs(v2 - v)[np.arange(64) != 5].max() > 0  # coupling through attention


def test_zeroed_branches_make_block_identity(orc):
    # with every modulation of a block zero (gates 0) and its cross-attention
    # output projection zero, the block passes the residual stream through:
    # an L=2 model with block 1 zeroed equals the L=1 model sharing block 0.
    s2 = synth.ModelShape(4, 8, 48, 2, 2, 4, 5, 48, 4, 8)
    s1 = synth.ModelShape(4, 8, 48, 1, 2, 4, 5, 48, 4, 8)
    b2 = synth.weights_blob(s2, 3)
    for name in ("mod_w", "mod_b", "co_w", "co_b"):
        synth.set_weight(b2, s2, name, 1, 0.0)
    b1 = synth.weights_blob(s1, 3)
    offs2, _ = synth.weight_offsets(s2)
    offs1, _ = synth.weight_offsets(s1)
    for (name, blk), (off1, dims) in offs1.items():
        off2, _ = offs2[(name, blk)]
        n = int(np.prod(dims))
        b1[off1:off1 + n] = b2[off2:off2 + n]
    m1, m2 = orc.Model(s1, b1), orc.Model(s2, b2)
    rng = np.random.default_rng(1)
    S = rng.standard_normal((64, 8)).astype(np.float32)
    cond = synth.cond_tokens(s2, 1, 2)[0]
    idx = np.arange(64, dtype=np.int32)
    v1 = m1.forward(S, idx, 0.5, m1.cond_kv(cond))
    v2 = m2.forward(S, idx, 0.5, m2.cond_kv(cond))
    np.testing.assert_allclose(v2, v1, rtol=1e-6, atol=1e-6)
    # and a nonzero gate does change the output
    b3 = b2.copy()
    synth.set_weight(b3, s2, "mod_b", 1, 0.5)
    m3 = orc.Model(s2, b3)
    v3 = m3.forward(S, idx, 0.5, m3.cond_kv(cond))
    assert np.abs(v3 - v2).max() > 1e-3


def test_identity_blocks_leave_embedding_and_final_layer(orc):
    # with every block an identity (zero modulation: gates 0; zero
    # cross-attention output), the forward is the final layer applied to the
    # input embedding: v_i = W_out (LN(x_i) (1 + scale) + shift) + b_out,
    # x_i = W_in S_i + b_in + pos(i), (shift, scale) = Linear(SiLU(temb)).
    # At t = 0 the timestep sinusoid is [1]*128 + [0]*128, so the expected
    # value is plain NumPy on the blob's weights (plus the position table,
    # pinned by its closed form); this fixes the embedding and final-layer
    # wiring: operand orientation, the shift / scale order and the 1 + scale.
    s = synth.ModelShape(4, 8, 64, 2, 2, 4, 5, 64, 4, 8)
    blob = synth.weights_blob(s, 7)
    for l in range(s.blocks):
        for name in ("mod_w", "mod_b", "co_w", "co_b"):
            synth.set_weight(blob, s, name, l, 0.0)
    offs, _ = synth.weight_offsets(s)

    def w(name):
        off, dims = offs[(name, -1)]
        return synth.bf16_bits_to_f32(blob[off:off + int(np.prod(dims))]).astype(np.float64).reshape(dims)

    def silu(z):
        return z / (1.0 + np.exp(-z))

    m = orc.Model(s, blob)
    rng = np.random.default_rng(5)
    S = rng.standard_normal((s.tokens, 8)).astype(np.float32)
    idx = np.sort(rng.choice(s.tokens, 40, replace=False)).astype(np.int32)
    cond = synth.cond_tokens(s, 1, 4)[0]
    got = m.forward(S, idx, 0.0, m.cond_kv(cond)).astype(np.float64)

    freq = np.concatenate([np.ones(128), np.zeros(128)])
    temb = w("t_w2") @ silu(w("t_w1") @ freq + w("t_b1")) + w("t_b2")
    mod = w("fmod_w") @ silu(temb) + w("fmod_b")
    shift, scale = mod[:s.width], mod[s.width:]
    pos = np.stack([orc.pos_embed(s.grid, s.width, int(i)) for i in idx]).astype(np.float64)
    x = S[idx].astype(np.float64) @ w("in_w").T + w("in_b") + pos
    xh = (x - x.mean(axis=1, keepdims=True)) / np.sqrt(x.var(axis=1, keepdims=True) + 1e-6)
    ref = (xh * (1.0 + scale) + shift) @ w("out_w").T + w("out_b")
    np.testing.assert_allclose(got, ref, rtol=2e-4, atol=2e-5)


def _numpy_head_tail(s, blob):
    """NumPy input embedding and t = 0 final layer on the blob's weights."""
    offs, _ = synth.weight_offsets(s)

    def w(name, blk=-1):
        off, dims = offs[(name, blk)]
        return synth.bf16_bits_to_f32(blob[off:off + int(np.prod(dims))]).astype(np.float64).reshape(dims)

    def silu(z):
        return z / (1.0 + np.exp(-z))

    def ln(x):
        return (x - x.mean(axis=1, keepdims=True)) / np.sqrt(x.var(axis=1, keepdims=True) + 1e-6)

    freq = np.concatenate([np.ones(128), np.zeros(128)])
    temb = w("t_w2") @ silu(w("t_w1") @ freq + w("t_b1")) + w("t_b2")
    fmod = w("fmod_w") @ silu(temb) + w("fmod_b")

    def tail(x):
        return (ln(x) * (1.0 + fmod[s.width:]) + fmod[:s.width]) @ w("out_w").T + w("out_b")

    return w, ln, tail


def _one_branch_model(orc, gate_slot, seed):
    # blocks are identities except block 0's branch `gate_slot` (2: the
    # self-attention gate, 5: the MLP gate), whose modulation is the constant
    # bias shift = 0.25, scale = 0.125, gate = 0.5 (exact in bf16)
    s = synth.ModelShape(4, 8, 64, 2, 2, 4, 5, 64, 4, 8)
    blob = synth.weights_blob(s, seed)
    for l in range(s.blocks):
        for name in ("mod_w", "mod_b", "co_w", "co_b"):
            synth.set_weight(blob, s, name, l, 0.0)
    mb = np.zeros(6 * s.width, np.float32)
    base = (gate_slot - 2) * s.width  # shift of the same branch
    mb[base:base + s.width] = 0.25
    mb[base + s.width:base + 2 * s.width] = 0.125
    mb[base + 2 * s.width:base + 3 * s.width] = 0.5
    synth.set_weight(blob, s, "mod_b", 0, mb)
    return s, blob


def test_single_token_self_attention_branch(orc):
    # one active token attends to itself only (softmax over one key is 1),
    # so block 0's self-attention branch reduces to its value and output
    # projections: x += gate1 (W_o (W_v h + b_v) + b_o), h = LN(x)(1 +
    # scale1) + shift1 -- pins the value rows of the QKV projection, the
    # output projection and the (shift, scale, gate) order of the modulation
    s, blob = _one_branch_model(orc, 2, 11)
    w, ln, tail = _numpy_head_tail(s, blob)
    m = orc.Model(s, blob)
    S = np.random.default_rng(6).standard_normal((s.tokens, 8)).astype(np.float32)
    cond = synth.cond_tokens(s, 1, 4)[0]
    i = 37
    got = m.forward(S, np.array([i], np.int32), 0.0, m.cond_kv(cond)).astype(np.float64)
    W = s.width
    x = S[[i]].astype(np.float64) @ w("in_w").T + w("in_b") + orc.pos_embed(s.grid, W, i).astype(np.float64)
    h = ln(x) * 1.125 + 0.25
    qkv = h @ w("qkv_w", 0).T + w("qkv_b", 0)
    y = qkv[:, 2 * W:] @ w("o_w", 0).T + w("o_b", 0)
    ref = tail(x + 0.5 * y)
    np.testing.assert_allclose(got, ref, rtol=2e-4, atol=2e-5)


def test_mlp_branch(orc):
    # block 0's MLP branch alone: x += gate2 fc2(GELU_tanh(fc1(LN(x)(1 +
    # scale2) + shift2))) on every active token independently
    s, blob = _one_branch_model(orc, 5, 12)
    w, ln, tail = _numpy_head_tail(s, blob)
    m = orc.Model(s, blob)
    S = np.random.default_rng(7).standard_normal((s.tokens, 8)).astype(np.float32)
    cond = synth.cond_tokens(s, 1, 4)[0]
    idx = np.array([3, 17, 40, 63], np.int32)
    got = m.forward(S, idx, 0.0, m.cond_kv(cond)).astype(np.float64)
    W = s.width
    pos = np.stack([orc.pos_embed(s.grid, W, int(i)) for i in idx]).astype(np.float64)
    x = S[idx].astype(np.float64) @ w("in_w").T + w("in_b") + pos
    h = ln(x) * 1.125 + 0.25
    u = h @ w("fc1_w", 0).T + w("fc1_b", 0)
    g = 0.5 * u * (1.0 + np.tanh(np.sqrt(2.0 / np.pi) * (u + 0.044715 * u ** 3)))
    y = g @ w("fc2_w", 0).T + w("fc2_b", 0)
    ref = tail(x + 0.5 * y)
    np.testing.assert_allclose(got, ref, rtol=2e-4, atol=2e-5)


def test_single_condition_token_cross_attention_branch(orc):
    # with one condition token every query's cross-attention weight is 1, so
    # block 0's cross-attention branch (no gate) adds W_co V_c + b_co with
    # V_c the value half of the condition projection: pins the K/V split of
    # that projection, the output projection and the ungated residual
    s = synth.ModelShape(4, 8, 64, 2, 2, 4, 1, 64, 4, 8)
    blob = synth.weights_blob(s, 13)
    for l in range(s.blocks):
        for name in ("mod_w", "mod_b"):
            synth.set_weight(blob, s, name, l, 0.0)
    for name in ("co_w", "co_b"):
        synth.set_weight(blob, s, name, 1, 0.0)
    w, ln, tail = _numpy_head_tail(s, blob)
    m = orc.Model(s, blob)
    S = np.random.default_rng(8).standard_normal((s.tokens, 8)).astype(np.float32)
    cond = synth.cond_tokens(s, 1, 9)[0]
    idx = np.array([0, 21, 50], np.int32)
    got = m.forward(S, idx, 0.0, m.cond_kv(cond)).astype(np.float64)
    W = s.width
    pos = np.stack([orc.pos_embed(s.grid, W, int(i)) for i in idx]).astype(np.float64)
    x = S[idx].astype(np.float64) @ w("in_w").T + w("in_b") + pos
    c = synth.bf16_bits_to_f32(np.asarray(cond).reshape(-1)).astype(np.float64)
    kv = w("ckv_w", 0) @ c + w("ckv_b", 0)
    y = w("co_w", 0) @ kv[W:] + w("co_b", 0)
    ref = tail(x + y)
    np.testing.assert_allclose(got, ref, rtol=2e-4, atol=2e-5)


def test_qk_rmsnorm_invariance(orc):
    # per-head RMSNorm of Q and K (Supp. Sec. F self-attention): scaling the
    # query or key projection (rows and bias, by powers of two, exact in
    # bf16) leaves the block unchanged, while scaling the norm's gain does
    # not -- pins that both are normalised before the scores, gain after
    s, blob = _one_branch_model(orc, 2, 14)
    W = s.width
    offs, _ = synth.weight_offsets(s)
    S = np.random.default_rng(9).standard_normal((s.tokens, 8)).astype(np.float32)
    cond = synth.cond_tokens(s, 1, 4)[0]
    idx = np.arange(0, s.tokens, 5, dtype=np.int32)

    def run(b):
        m = orc.Model(s, b)
        return m.forward(S, idx, 0.0, m.cond_kv(cond)).astype(np.float64)

    def scaled(b, name, lo, hi, f):
        out = b.copy()
        off, dims = offs[(name, 0)]
        cols = dims[1] if len(dims) > 1 else 1
        seg = synth.bf16_bits_to_f32(out[off + lo * cols:off + hi * cols]) * np.float32(f)
        out[off + lo * cols:off + hi * cols] = synth.f32_to_bf16_bits(seg)
        return out

    base = run(blob)
    for lo, hi, f in ((0, W, 2.0), (W, 2 * W, 4.0)):  # Q rows, K rows
        b = scaled(scaled(blob, "qkv_w", lo, hi, f), "qkv_b", lo, hi, f)
        np.testing.assert_allclose(run(b), base, rtol=1e-5, atol=1e-5)
    assert np.abs(run(scaled(blob, "qn_g", 0, W, 2.0)) - base).max() > 1e-3
    assert np.abs(run(scaled(blob, "kn_g", 0, W, 2.0)) - base).max() > 1e-3


def test_sample_quota_zero_is_plain_euler(tiny, orc):
    # quota 0 at every step must reproduce the uncached sampler exactly
    m, S, cond = tiny["model"], tiny["S"][:1], tiny["cond"][:1]
    T = 4
    out = m.sample(S, cond, T=T, quota_schedule=np.zeros((T, 1), np.int32), tau=0)
    t = orc.time_schedule(T, 3.0)
    x = S[0].copy()
    kv = m.cond_kv(cond[0])
    vc = np.zeros((TINY.tokens, 8), np.uint16)
    for k in range(T):
        v = m.forward(x, np.arange(TINY.tokens), float(t[k]), kv)
        x, vc = orc.merge_euler(x, np.arange(TINY.tokens, dtype=np.int32), v, vc, float(t[k] - t[k + 1]))
    np.testing.assert_array_equal(out["S"][0], x)
    assert np.all(out["n_active"] == TINY.tokens)


def test_sample_cached_tokens_carry_velocity(tiny, orc):
    # a token cached at step k keeps v_t = v_(t-1) bit for bit, so its
    # acceleration A_i is exactly 0 at step k+1
    m, S, cond = tiny["model"], tiny["S"][:1], tiny["cond"][:1]
    T = 4
    q = np.array([[0], [0], [0], [300]], np.int32)
    out = m.sample(S, cond, T=T, quota_schedule=q, tau=0)
    vcache, vprev = out["v_hist"][0, 0], out["v_hist"][1, 0]
    same = np.all(vcache == vprev, axis=1)
    assert same.sum() == 300
    assert out["n_active"][3, 0] == TINY.tokens - 300


def test_sample_batch_members_independent(tiny):
    m, S, cond = tiny["model"], tiny["S"], tiny["cond"]
    q = np.tile(np.array([[0], [0], [0], [256], [256]], np.int32), (1, 2))
    both = m.sample(S, cond, T=5, quota_schedule=q, tau=0)
    one = m.sample(S[1:], cond[1:], T=5, quota_schedule=q[:, 1:], tau=0)
    np.testing.assert_array_equal(both["S"][1], one["S"][0])


def test_sample_pcsc_anchor_and_log(tiny, orc):
    # Algorithm 1 with PCSC: sigma is measured at the anchor step k_a (Eq. 1)
    # and the forecast uses it; sigma_override replaces it in the forecast
    m, S, cond = tiny["model"], tiny["S"][:1], tiny["cond"][:1]
    T = 8
    out = m.sample(S, cond, T=T, tau=3)
    ka = orc.ceil_steps(T, 0.2)
    assert np.all(out["quota"][:ka] == 0)
    assert out["sigma"][0] >= 0
    gate = orc.TauGate(3, 0)
    for k in range(1, T + 1):
        c, _ = orc.phase_quota(TINY.tokens, T, 0.2, 0.75, -0.07, 0.7, 3, TINY.gamma_up,
                               float(out["sigma"][0]), k)
        assert out["quota"][k - 1, 0] == gate(c)
    assert np.all(out["n_active"] == TINY.tokens - out["quota"])
    ov = m.sample(S, cond, T=T, tau=3, sigma_override=np.array([64.0 * 100]))
    assert ov["sigma"][0] == out["sigma"][0]
    c6, _ = orc.phase_quota(TINY.tokens, T, 0.2, 0.75, -0.07, 0.7, 3, TINY.gamma_up, 6400.0, ka + 1)
    assert ov["quota"][ka, 0] == c6


def test_time_embedding_closed_form_at_t0(orc):
    # at t = 0 every frequency has argument 0: the 256-dim sinusoid is
    # [cos 0]*128 + [sin 0]*128 = [1]*128 + [0]*128, so the embedding reduces
    # to Linear(SiLU(Linear(that vector))) with library-checked linear layers
    shape = synth.ModelShape(4, 8, 48, 1, 2, 4, 5, 48, 4, 8)
    blob = synth.weights_blob(shape, 9)
    m = orc.Model(shape, blob)
    freq = np.concatenate([np.ones(128), np.zeros(128)]).astype(np.float32)[None]
    w1, b1 = synth.weight_view(blob, shape, "t_w1"), synth.weight_view(blob, shape, "t_b1")
    w2, b2 = synth.weight_view(blob, shape, "t_w2"), synth.weight_view(blob, shape, "t_b2")
    h1 = freq.astype(np.float64) @ w1.T.astype(np.float64) + b1
    h1 = h1 / (1.0 + np.exp(-h1))
    ref = h1 @ w2.T.astype(np.float64) + b2
    np.testing.assert_allclose(m.time_embed(0.0), ref[0], rtol=1e-5, atol=1e-6)
    # and t enters only through the sinusoid: two different times differ
    assert np.abs(m.time_embed(0.5) - m.time_embed(0.0)).max() > 1e-3


def test_modulation_is_linear_of_silu(orc):
    shape = synth.ModelShape(4, 8, 48, 2, 2, 4, 5, 48, 4, 8)
    blob = synth.weights_blob(shape, 10)
    m = orc.Model(shape, blob)
    temb = np.random.default_rng(0).standard_normal(48).astype(np.float32)
    s = temb.astype(np.float64) / (1.0 + np.exp(-temb.astype(np.float64)))
    for blk, name in ((1, "mod"), (-1, "fmod")):
        w = synth.weight_view(blob, shape, name + "_w", blk).astype(np.float64)
        b = synth.weight_view(blob, shape, name + "_b", blk).astype(np.float64)
        np.testing.assert_allclose(m.modulation(temb, blk), w @ s + b, rtol=1e-5, atol=1e-6)


def test_cross_attention_query_path_multi_token(orc):
    # block 0's cross-attention branch alone (every modulation zero, so the
    # gated self-attention and MLP branches add exactly 0; block 1's output
    # projection zero) with five condition tokens, so the softmax weights
    # depend on the query: y = W_co softmax_h(q_h K_h^T / sqrt(dh)) V_h + b_co
    # with q = W_cq (LN(x) g2 + b2) + b_cq and [K | V] = W_ckv c + b_ckv, added
    # ungated.  LN2's gain and bias are drawn wide so that dropping either,
    # applying the bias before the gain, projecting x instead of LN2(x) or
    # swapping the key and value halves moves the output far beyond the
    # tolerance (checked below against NumPy variants with each mistake).
    s = synth.ModelShape(4, 8, 64, 2, 2, 4, 5, 64, 4, 8)
    blob = synth.weights_blob(s, 15)
    for l in range(s.blocks):
        for name in ("mod_w", "mod_b"):
            synth.set_weight(blob, s, name, l, 0.0)
    for name in ("co_w", "co_b"):
        synth.set_weight(blob, s, name, 1, 0.0)
    rng = np.random.default_rng(21)
    W = s.width
    synth.set_weight(blob, s, "ln2_g", 0, (1.0 + 0.5 * rng.standard_normal(W)).astype(np.float32))
    synth.set_weight(blob, s, "ln2_b", 0, (0.5 * rng.standard_normal(W)).astype(np.float32))
    # a sharper query projection makes the attention weights far from uniform
    cq = synth.weight_view(blob, s, "cq_w", 0) * np.float32(4.0)
    synth.set_weight(blob, s, "cq_w", 0, cq)
    w, ln, tail = _numpy_head_tail(s, blob)
    m = orc.Model(s, blob)
    S = rng.standard_normal((s.tokens, 8)).astype(np.float32)
    cond = synth.cond_tokens(s, 1, 17)[0]
    idx = np.array([2, 9, 26, 41, 58, 63], np.int32)
    got = m.forward(S, idx, 0.0, m.cond_kv(cond)).astype(np.float64)

    pos = np.stack([orc.pos_embed(s.grid, W, int(i)) for i in idx]).astype(np.float64)
    x = S[idx].astype(np.float64) @ w("in_w").T + w("in_b") + pos
    c = synth.bf16_bits_to_f32(np.asarray(cond).reshape(s.cond_tokens, s.cond_dim)).astype(np.float64)
    kv = c @ w("ckv_w", 0).T + w("ckv_b", 0)
    dh = W // s.heads

    def branch(h_in, k_half=0):
        q = h_in @ w("cq_w", 0).T + w("cq_b", 0)
        K, V = kv[:, k_half * W:(k_half + 1) * W], kv[:, (1 - k_half) * W:(2 - k_half) * W]
        o = np.empty_like(q)
        for hd in range(s.heads):
            sl = slice(hd * dh, (hd + 1) * dh)
            sc = q[:, sl] @ K[:, sl].T / np.sqrt(dh)
            p = np.exp(sc - sc.max(axis=1, keepdims=True))
            p /= p.sum(axis=1, keepdims=True)
            o[:, sl] = p @ V[:, sl]
        return o @ w("co_w", 0).T + w("co_b", 0)

    g2, b2 = w("ln2_g", 0), w("ln2_b", 0)
    ref = tail(x + branch(ln(x) * g2 + b2))
    np.testing.assert_allclose(got, ref, rtol=2e-4, atol=2e-5)

    # the pin separates each plausible slip from the right reading
    scale = np.abs(ref).max()
    wrong = {
        "no LN2 bias": ln(x) * g2,
        "no LN2 gain": ln(x) + b2,
        "bias before gain": (ln(x) + b2) * g2,
        "query from x": x,
    }
    for what, h_in in wrong.items():
        assert np.abs(tail(x + branch(h_in)) - ref).max() > 100 * (2e-5 + 2e-4 * scale), what
    assert np.abs(tail(x + branch(ln(x) * g2 + b2, k_half=1)) - ref).max() > 100 * (2e-5 + 2e-4 * scale)
