"""Pins of the oracle's routers (no GPU).

The paper prints no router weights or outputs, so router parity against the
paper is unpinned; what is pinned here: the parameter count the paper states
for LBS ("600k", App. C.1), the zero-weight closed form (all weights zero but
the head bias c gives O = c at every row), the layer structure against
PyTorch's own nn.TransformerEncoderLayer / LayerNorm / GELU (post-norm for
LBS, pre-norm for LPS), both whole routers against torch.nn modules assembled
from the sizes and the order of App. C.1 (F_ent, the [e ; t] fusion, E_pos
after W_combine) and App. D.1 (Linear, LayerNorm, GELU input layer), and
permutation equivariance where the architecture has no positional table.
"""
import numpy as np
import pytest
import torch

import synth
from oracle import ebd_oracle as o


def _W(seed=11, d_base=64, L=32):
    return o.weights_f64(synth.router_weights(seed, d_base, L))


def test_parameter_counts():
    lay = synth.router_layout(4096, 512)
    assert lay.count("lbs.") == 613761           # "600k" (App. C.1)
    assert synth.router_layout(4096, 256).count("lbs.") == 580993
    assert lay.count("lps.") == 17377            # stated dims of App. D.1


def test_zero_weights_closed_form():
    W = {k: np.zeros_like(v) for k, v in _W().items()}
    W["lbs.head.b"][:] = 0.75
    W["lps.head.b"][:] = -1.25
    emb = synth.f32_to_bf16_bits(np.random.default_rng(0).standard_normal((50, 64)))
    O = o.lbs_router(np.linspace(0, 1, 9), np.arange(9), emb, W)
    np.testing.assert_allclose(O, 0.75, atol=1e-15)
    Op = o.lps_router(np.random.default_rng(1).random((7, 5)), W)
    np.testing.assert_allclose(Op, -1.25, atol=1e-15)


def _torch_layer(W, p, d, nhead, ff, norm_first):
    layer = torch.nn.TransformerEncoderLayer(d, nhead, ff, dropout=0.0,
                                             activation="gelu", batch_first=True,
                                             norm_first=norm_first, dtype=torch.float64)
    sd = {
        "self_attn.in_proj_weight": W[p + ".qkv.w"], "self_attn.in_proj_bias": W[p + ".qkv.b"],
        "self_attn.out_proj.weight": W[p + ".out.w"], "self_attn.out_proj.bias": W[p + ".out.b"],
        "linear1.weight": W[p + ".ff1.w"], "linear1.bias": W[p + ".ff1.b"],
        "linear2.weight": W[p + ".ff2.w"], "linear2.bias": W[p + ".ff2.b"],
        "norm1.weight": W[p + ".ln1.g"], "norm1.bias": W[p + ".ln1.b"],
        "norm2.weight": W[p + ".ln2.g"], "norm2.bias": W[p + ".ln2.b"],
    }
    layer.load_state_dict({k: torch.from_numpy(np.array(v)) for k, v in sd.items()})
    layer.eval()
    return layer


def _perturb_ln(W):
    """LayerNorm gains/biases are 1/0 at init; perturb them so that a wrong
    gain/bias placement would show."""
    rng = np.random.default_rng(4)
    W = dict(W)
    for k in list(W):
        if ".ln" in k:
            W[k] = W[k] + rng.standard_normal(W[k].shape) * 0.3
    return W


def test_lbs_layer_matches_torch_post_norm():
    W = _perturb_ln(_W())
    x = np.random.default_rng(2).standard_normal((11, 128))
    layer = _torch_layer(W, "lbs.l0", 128, 4, 256, norm_first=False)
    with torch.no_grad():
        ref = layer(torch.from_numpy(x)[None])[0].numpy()
    np.testing.assert_allclose(o.lbs_encoder_layer(x, W, "lbs.l0"), ref, rtol=1e-10, atol=1e-10)


def test_lps_block_matches_torch_pre_norm():
    W = _perturb_ln(_W())
    x = np.random.default_rng(3).standard_normal((9, 32))
    layer = _torch_layer(W, "lps.l1", 32, 4, 64, norm_first=True)
    with torch.no_grad():
        ref = layer(torch.from_numpy(x)[None])[0].numpy()
    np.testing.assert_allclose(o.lps_block(x, W, "lps.l1"), ref, rtol=1e-10, atol=1e-10)


def test_elementary_layers_match_torch():
    x = np.random.default_rng(8).standard_normal((5, 64)) * 3
    g = np.random.default_rng(9).standard_normal(64)
    b = np.random.default_rng(10).standard_normal(64)
    ref = torch.nn.functional.layer_norm(torch.from_numpy(x), (64,), torch.from_numpy(g),
                                         torch.from_numpy(b), eps=1e-5).numpy()
    np.testing.assert_allclose(o.layer_norm(x, g, b), ref, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(o.gelu(x), torch.nn.functional.gelu(torch.from_numpy(x)).numpy(),
                               rtol=1e-12, atol=1e-14)


def test_lps_permutation_equivariant():
    W = _W()
    f = np.random.default_rng(12).random((10, 5))
    perm = np.random.default_rng(13).permutation(10)
    np.testing.assert_allclose(o.lps_router(f[perm], W), o.lps_router(f, W)[perm], atol=1e-12)


def test_lbs_rank_positional_table():
    """With E_pos zeroed the LBS router is permutation-equivariant; with it,
    the output of a row depends on its rank (compacted index, Reading R11)."""
    W = _W()
    emb = synth.f32_to_bf16_bits(np.random.default_rng(14).standard_normal((40, 64)))
    h = np.random.default_rng(15).random(8)
    x = np.random.default_rng(16).integers(0, 40, 8)
    perm = np.random.default_rng(17).permutation(8)
    W0 = dict(W); W0["lbs.pos"] = np.zeros_like(W["lbs.pos"])
    np.testing.assert_allclose(o.lbs_router(h[perm], x[perm], emb, W0),
                               o.lbs_router(h, x, emb, W0)[perm], atol=1e-12)
    assert not np.allclose(o.lbs_router(h[perm], x[perm], emb, W),
                           o.lbs_router(h, x, emb, W)[perm], atol=1e-6)


def test_lbs_token_branch_uses_embedding_row():
    """Changing the embedding row of a token that is not predicted leaves O
    unchanged; changing a predicted one changes it."""
    W = _W()
    emb = synth.f32_to_bf16_bits(np.random.default_rng(18).standard_normal((40, 64)))
    h = np.random.default_rng(19).random(5)
    x = np.array([3, 7, 7, 20, 1])
    base = o.lbs_router(h, x, emb, W)
    e2 = emb.copy(); e2[30] ^= 0x0040
    np.testing.assert_array_equal(o.lbs_router(h, x, e2, W), base)
    e3 = emb.copy(); e3[20] = synth.f32_to_bf16_bits(np.full(64, 2.0, np.float32))
    assert np.abs(o.lbs_router(h, x, e3, W) - base).max() > 1e-6


def test_router_init_generator_properties():
    """Init values lie in [-bound, bound], are bf16-exact and are not
    constant; LayerNorm gains are exactly 1."""
    w = synth.router_weights(3, 64, 32)
    f = {k: synth.bf16_to_f32(v) for k, v in w.items()}
    assert np.all(np.abs(f["lbs.l0.ff2.w"]) <= 1 / 16)
    assert np.all(f["lbs.l1.ln1.g"] == 1.0) and np.all(f["lps.in_ln.b"] == 0.0)
    assert np.all(np.abs(f["lbs.pos"]) <= 0.02 * np.sqrt(3) * (1 + 2 ** -8))  # bf16 rounding
    assert f["lbs.tok.w"].std() > 0
    u = synth.splitmix64_uniform(0, 0, 100000)
    assert 0.49 < u.mean() < 0.51 and u.min() >= 0 and u.max() < 1


def test_splitmix64_published_vectors():
    """SplitMix64 outputs for state 0 and for seed 1234567, as published with
    the generator's reference implementation."""
    from synth import router_init as r
    G = 0x9E3779B97F4A7C15
    assert [r._mix_int((k * G) % 2 ** 64) for k in (1, 2, 3)] == \
        [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]
    assert [r._mix_int((1234567 + k * G) % 2 ** 64) for k in (1, 2, 3)] == \
        [6457827717110365317, 3203168211198807973, 9817491932198370423]


def _lin(W, name, fan_in, fan_out):
    m = torch.nn.Linear(fan_in, fan_out, dtype=torch.float64)
    m.load_state_dict({"weight": torch.from_numpy(np.array(W[name + ".w"])),
                       "bias": torch.from_numpy(np.array(W[name + ".b"]))})
    return m


def _ln(W, name, width):
    m = torch.nn.LayerNorm(width, eps=1e-5, dtype=torch.float64)
    m.load_state_dict({"weight": torch.from_numpy(np.array(W[name + ".g"])),
                       "bias": torch.from_numpy(np.array(W[name + ".b"]))})
    return m


def torch_lps_router(feats, W):
    """The LPS router of App. D.1 assembled from torch.nn modules at the
    stated sizes: Linear(5 -> 32) -> LayerNorm -> GELU, two pre-norm encoder
    blocks (4 heads, FFN 64, GELU), Linear(32 -> 1)."""
    net = torch.nn.Sequential(_lin(W, "lps.in", 5, 32), _ln(W, "lps.in_ln", 32),
                              torch.nn.GELU(),
                              _torch_layer(W, "lps.l0", 32, 4, 64, norm_first=True),
                              _torch_layer(W, "lps.l1", 32, 4, 64, norm_first=True),
                              _lin(W, "lps.head", 32, 1))
    net.eval()
    with torch.no_grad():
        return net(torch.from_numpy(np.asarray(feats, np.float64))[None])[0, :, 0].numpy()


def torch_lbs_router(ent_norm_seq, xhat_seq, w_emb, W):
    """The LBS router of App. C.1 assembled from torch.nn modules at the
    stated sizes: F_ent = Linear(1 -> 64) -> GELU -> Linear(64 -> 64) ->
    LayerNorm; token branch W_tok W_e(x_hat) with W_e a frozen nn.Embedding;
    Z = W_combine [F_ent ; token] + E_pos (Eq. lbs_feat); two post-norm
    encoder layers (4 heads, FFN 256, GELU); Linear(128 -> 1)."""
    d_base = w_emb.shape[1]
    f_ent = torch.nn.Sequential(_lin(W, "lbs.ent1", 1, 64), torch.nn.GELU(),
                                _lin(W, "lbs.ent2", 64, 64), _ln(W, "lbs.ent_ln", 64))
    emb = torch.nn.Embedding.from_pretrained(torch.from_numpy(o.bf16(w_emb)), freeze=True)
    tok = _lin(W, "lbs.tok", d_base, 64)
    comb = _lin(W, "lbs.comb", 128, 128)
    enc = torch.nn.Sequential(_torch_layer(W, "lbs.l0", 128, 4, 256, norm_first=False),
                              _torch_layer(W, "lbs.l1", 128, 4, 256, norm_first=False))
    enc.eval()
    head = _lin(W, "lbs.head", 128, 1)
    h = torch.from_numpy(np.asarray(ent_norm_seq, np.float64))[:, None]
    x = torch.from_numpy(np.asarray(xhat_seq, np.int64))
    with torch.no_grad():
        z = comb(torch.cat([f_ent(h), tok(emb(x))], dim=-1))
        z = z + torch.from_numpy(np.array(W["lbs.pos"]))[:len(x)]
        return head(enc(z[None])[0])[:, 0].numpy()


def test_lps_router_matches_torch_modules():
    """The whole LPS router, input layer order included (Linear, then
    LayerNorm, then GELU), against torch.nn modules built from App. D.1."""
    W = _perturb_ln(_W())
    f = np.random.default_rng(21).random((7, 5)) * np.array([1, 1, 1, 1, 1.6])
    np.testing.assert_allclose(o.lps_router(f, W), torch_lps_router(f, W), rtol=1e-10, atol=1e-10)


def test_lbs_router_matches_torch_modules():
    """The whole LBS router, Eq. lbs_feat included (F_ent's order, the [e ; t]
    concatenation, E_pos added after W_combine), against torch.nn modules
    built from App. C.1."""
    W = _perturb_ln(_W())
    emb = synth.f32_to_bf16_bits(np.random.default_rng(22).standard_normal((60, 64)))
    h = np.random.default_rng(23).random(13)
    x = np.random.default_rng(24).integers(0, 60, 13)
    np.testing.assert_allclose(o.lbs_router(h, x, emb, W), torch_lbs_router(h, x, emb, W),
                               rtol=1e-10, atol=1e-10)
