"""Pins of the oracle's forward pass against things other than itself.

Each check ties one building block of the Llama block (Sec. 3.1's f_{0->k},
f_{k->L}) to a library routine, a closed form or an invariant, so that a
dropped term, a wrong sign, a wrong GQA index or a transposed weight fails.
"""
import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import OracleModel, rmsnorm, rope, softmax, log_softmax, silu
from workloads import make_weights, workload, tiny_shape

pytestmark = pytest.mark.filterwarnings("ignore::DeprecationWarning")


def _rng(seed=0):
    return np.random.default_rng(seed)


def test_rmsnorm_matches_torch():
    x = _rng().standard_normal((5, 64))
    g = _rng(1).standard_normal(64)
    ref = F.rms_norm(torch.from_numpy(x), (64,), torch.from_numpy(g), eps=1e-5).numpy()
    np.testing.assert_allclose(rmsnorm(x, g, 1e-5), ref, rtol=1e-12, atol=1e-12)


def test_rmsnorm_scale_invariant_and_unit_rms():
    x = _rng().standard_normal((3, 32))
    y = rmsnorm(x, np.ones(32), 0.0)
    np.testing.assert_allclose(np.mean(y * y, axis=-1), 1.0, rtol=1e-12)
    np.testing.assert_allclose(rmsnorm(7.5 * x, np.ones(32), 0.0), y, rtol=1e-12)


@pytest.mark.parametrize("hd", [2, 8, 64])
def test_rope_equals_complex_rotation(hd):
    """Rotate-half RoPE == multiplying (x_i + i x_{i+hd/2}) by exp(i pos theta^(-2i/hd))."""
    R, H, theta = 6, 3, 10000.0
    x = _rng().standard_normal((R, H, hd))
    pos = np.array([0, 1, 2, 17, 300, 4099])
    half = hd // 2
    z = x[..., :half] + 1j * x[..., half:]
    freq = np.array([theta ** (-(2 * i) / hd) for i in range(half)])
    rot = np.exp(1j * np.outer(pos, freq))[:, None, :]
    zr = z * rot
    ref = np.concatenate([zr.real, zr.imag], axis=-1)
    np.testing.assert_allclose(rope(x, pos, theta), ref, rtol=1e-10, atol=1e-12)


def test_rope_identity_at_zero_and_relative_positions():
    x = _rng().standard_normal((1, 2, 16))
    np.testing.assert_allclose(rope(x, np.array([0]), 1e4), x, atol=0)
    q = _rng(2).standard_normal((1, 1, 16))
    k = _rng(3).standard_normal((1, 1, 16))
    d1 = np.sum(rope(q, np.array([9]), 1e4) * rope(k, np.array([4]), 1e4))
    d2 = np.sum(rope(q, np.array([105]), 1e4) * rope(k, np.array([100]), 1e4))
    assert abs(d1 - d2) < 1e-12


def test_softmax_logsoftmax_silu_against_torch():
    z = _rng().standard_normal((4, 50)) * 30
    t = torch.from_numpy(z)
    np.testing.assert_allclose(softmax(z), torch.softmax(t, -1).numpy(), rtol=1e-12, atol=1e-300)
    np.testing.assert_allclose(log_softmax(z), torch.log_softmax(t, -1).numpy(), rtol=1e-12)
    np.testing.assert_allclose(silu(z), F.silu(t).numpy(), rtol=1e-12)


def _model(shape=None, seed=0, dtype=np.float64):
    w = workload("tiny").with_(shape=shape or tiny_shape(), weight_seed=seed)
    return OracleModel(make_weights(w, threads=2), w.shape, 1.0, dtype), w


@pytest.mark.parametrize("hkv", [4, 2, 1])
def test_layer_matches_torch_sdpa_block(hkv):
    """One layer on a causal block vs torch's rms_norm / SDPA (GQA) / silu."""
    shape = tiny_shape(d_model=64, n_heads=4, n_kv_heads=hkv, head_dim=16, d_ffn=96,
                       vocab=64, n_layers=2)
    m, _ = _model(shape)
    R = 7
    x = _rng(5).standard_normal((R, 64))
    cache = m.new_cache(16)
    out = m.layer(0, x.copy(), 0, cache)

    w = {k: torch.from_numpy(v) for k, v in m.layers[0].items()}
    X = torch.from_numpy(x)
    n1 = F.rms_norm(X, (64,), w["attn_norm"], eps=1e-5)
    q = (n1 @ w["wq"].T).view(R, 4, 16).transpose(0, 1)
    k = (n1 @ w["wk"].T).view(R, hkv, 16).transpose(0, 1)
    v = (n1 @ w["wv"].T).view(R, hkv, 16).transpose(0, 1)
    # rotary embedding as complex multiplication, independent of oracle.rope
    pos = torch.arange(R, dtype=torch.float64)
    freq = 1e4 ** (-torch.arange(0, 16, 2, dtype=torch.float64) / 16)
    rot = torch.polar(torch.ones(R, 8, dtype=torch.float64), pos[:, None] * freq[None, :])

    def rotate(t):
        c = torch.complex(t[..., :8], t[..., 8:]) * rot
        return torch.cat([c.real, c.imag], -1)

    q, k = rotate(q), rotate(k)
    k = k.repeat_interleave(4 // hkv, dim=0)
    v = v.repeat_interleave(4 // hkv, dim=0)
    o = F.scaled_dot_product_attention(q[None], k[None], v[None], is_causal=True)[0]
    h = X + o.transpose(0, 1).reshape(R, 64) @ w["wo"].T
    n2 = F.rms_norm(h, (64,), w["ffn_norm"], eps=1e-5)
    ref = h + (F.silu(n2 @ w["w_gate"].T) * (n2 @ w["w_up"].T)) @ w["w_down"].T
    np.testing.assert_allclose(out, ref.numpy(), rtol=1e-10, atol=1e-12)


def test_incremental_decode_equals_full_recompute():
    """KV-cached one-row steps == one causal pass over the whole sequence (fp64)."""
    m, w = _model()
    L = w.shape.n_layers
    toks = _rng(7).integers(0, w.shape.vocab, 20)
    full = m.layers_range(0, L, m.embed(toks), 0, m.new_cache(32))
    c = m.new_cache(32)
    rows = [m.layers_range(0, L, m.embed(toks[i:i + 1]), i, c)[0] for i in range(20)]
    np.testing.assert_allclose(np.stack(rows), full, rtol=1e-12, atol=1e-12)


def test_block_causal_block_equals_rowwise_after_prefix():
    """A block of K rows on top of a cached prefix == the same rows one by one."""
    m, w = _model()
    L = w.shape.n_layers
    toks = _rng(8).integers(0, w.shape.vocab, 15)
    c1, c2 = m.new_cache(32), m.new_cache(32)
    m.layers_range(0, L, m.embed(toks[:10]), 0, c1)
    m.layers_range(0, L, m.embed(toks[:10]), 0, c2)
    blk = m.layers_range(0, L, m.embed(toks[10:]), 10, c1)
    one = [m.layers_range(0, L, m.embed(toks[i:i + 1]), i, c2)[0] for i in range(10, 15)]
    np.testing.assert_allclose(blk, np.stack(one), rtol=1e-12, atol=1e-12)


def test_split_factorization_composes():
    """f_{k->L}(f_{0->k}(x)) == f_{0->L}(x) for every split k (Sec. 3.1)."""
    m, w = _model()
    L = w.shape.n_layers
    toks = _rng(9).integers(0, w.shape.vocab, 6)
    ref = m.layers_range(0, L, m.embed(toks), 0, m.new_cache(8))
    for k in range(1, L):
        c = m.new_cache(8)
        hk = m.layers_range(0, k, m.embed(toks), 0, c)
        np.testing.assert_allclose(m.layers_range(k, L, hk, 0, c), ref, rtol=1e-12, atol=1e-12)


def test_heads_match_definitions():
    """p_phi uses W^V on RMSNorm_final(h_L); p_theta uses W^S + gamma A B."""
    m, w = _model()
    h = _rng(3).standard_normal((3, w.shape.d_model))
    m.lora_a = _rng(4).standard_normal(m.lora_a.shape)
    m.gamma = 0.7
    u = F.rms_norm(torch.from_numpy(h), (h.shape[1],), torch.from_numpy(m.final_g), eps=1e-5).numpy()
    Weff = m.w_s + 0.7 * m.lora_a @ m.lora_b
    np.testing.assert_allclose(m.drafter_logits(h), u @ Weff.T, rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(m.verifier_logits(h), u @ m.w_v.T, rtol=1e-10, atol=1e-12)


def test_to_bf16_matches_torch_rounding():
    """to_bf16 == torch's float32 -> bfloat16 conversion (round to nearest even), ties included."""
    from oracle.model import to_bf16
    r = _rng(21)
    x = np.concatenate([r.standard_normal(4096) * 10.0 ** r.integers(-6, 6, 4096),
                        -r.standard_normal(512) * 1e-3]).astype(np.float32)
    # exact ties: low 16 bits 0x8000 on both even and odd kept parts
    ties = (r.integers(0x3F000000, 0x40800000, 256, dtype=np.uint32) & np.uint32(0xFFFF0000)) | np.uint32(0x8000)
    x = np.concatenate([x, ties.view(np.float32), -ties.view(np.float32)])
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float32).numpy()
    np.testing.assert_array_equal(to_bf16(x), ref)


def test_bf16_kv_cache_rows_and_incremental_decode():
    """kv_dtype='bf16': cached rows are bfloat16 values, cached decode == full recompute,
    and the logits move by no more than bf16 storage noise."""
    from oracle.model import to_bf16
    m, w = _model()
    mb = OracleModel(make_weights(w), w.shape, w.lora_gamma, kv_dtype="bf16")
    L = w.shape.n_layers
    toks = _rng(7).integers(0, w.shape.vocab, 20)
    cf = mb.new_cache(32)
    full = mb.layers_range(0, L, mb.embed(toks), 0, cf)
    assert np.array_equal(to_bf16(cf.k[:, :20]).astype(np.float64), cf.k[:, :20])
    assert np.array_equal(to_bf16(cf.v[:, :20]).astype(np.float64), cf.v[:, :20])
    c = mb.new_cache(32)
    rows = [mb.layers_range(0, L, mb.embed(toks[i:i + 1]), i, c)[0] for i in range(20)]
    np.testing.assert_allclose(np.stack(rows), full, rtol=1e-12, atol=1e-12)
    ref = m.verifier_logits(m.layers_range(0, L, m.embed(toks), 0, m.new_cache(32)))
    diff = np.abs(mb.verifier_logits(full) - ref).max()
    assert 0.0 < diff < 2.0 ** -8 * np.abs(ref).max()
