"""Pins of the oracle's time/step conditioning (Sec. 3.1, App. A).

The conditioned block is checked against facts fixed outside the oracle: the
sinusoidal features' closed forms, torch re-implementations of the embedding
MLPs and the modulator, reductions to the unconditioned backbone (which
test_oracle_pins.py pins to a textbook transformer) when the modulator is
constant, and properties of the uniform trajectory that isolate the time and
step embeddings. Planted mistakes in the oracle must each fail a pin.
"""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import tlf_oracle as O
from paper_2609_15160_gb300 import synth

from test_oracle_pins import _random_norm_gains, _textbook_logits


def _cond_tiny(T=10, seed_tokens=4, **kw):
    cfg = synth.tiny_config(conditioning=True, **kw)
    w = _random_norm_gains(synth.make_weights(cfg))
    w["embedding"] = w["embedding"] * 40.0     # O(1) activations so every term matters
    for k in ("wq", "wk", "wv", "wo", "w_gate", "w_up", "w_down"):
        w[k] = w[k] * 15.0
    toks = np.random.default_rng(seed_tokens).integers(0, cfg.vocab, size=T)
    return cfg, w, toks


def _constant_modulator(cfg, w, a_msa, a_mlp, g_msa, g_mlp):
    """Modulator with zero weights: every token and loop gets the bias (alpha_msa, alpha_mlp, gamma_msa, gamma_mlp)."""
    w = dict(w)
    d, J = cfg.d_model, cfg.n_layers
    w["mod_w"] = np.zeros((J, 4 * d, d), dtype=np.float64)
    b = np.concatenate([np.broadcast_to(np.asarray(x, dtype=np.float64), (d,)) for x in (a_msa, a_mlp, g_msa, g_mlp)])
    w["mod_b"] = np.tile(b, (J, 1))
    return w


def _plain(w):
    return {k: v for k, v in w.items() if not (k.startswith("cond_") or k.startswith("mod_"))}


def _all_logits(cfg, w, toks, m):
    """Logits of every position from the three formulations (they must agree)."""
    model = O.OracleModel.from_config(cfg, w)
    full = O.forward_masked(model, toks, m)
    seq = O.OracleSequence(model)
    dec = np.stack([O.decode_token(model, seq, int(x), forced=int(m[t]))[0] for t, x in enumerate(toks)])
    seq_g = O.OracleSequence(model)
    last, _ = O.prefill_gathered(model, seq_g, toks, forced=m)
    return full, dec, last


def _torch_fourier(tau, width=256):
    K = width // 2
    w = torch.exp(-torch.arange(K, dtype=torch.float64) * (math.log(10000.0) / K))
    return torch.stack([torch.cos(tau * w), torch.sin(tau * w)], dim=1).reshape(-1)


def _torch_phi(w, which, tau):
    t = lambda a: torch.tensor(np.asarray(a, dtype=np.float64))
    hdn = F.silu(F.linear(_torch_fourier(tau), t(w[f"cond_{which}_w1"]), t(w[f"cond_{which}_b1"])))
    return F.linear(hdn, t(w[f"cond_{which}_w2"]), t(w[f"cond_{which}_b2"]))


# ----------------------------------------------------------------------------

def test_fourier_features_closed_forms():
    f0 = O.fourier_features(0.0)
    np.testing.assert_array_equal(f0[0::2], 1.0)      # cos 0
    np.testing.assert_array_equal(f0[1::2], 0.0)      # sin 0
    for tau in (0.3, 1.0, 7.5):
        f = O.fourier_features(tau)
        assert f.shape == (256,)
        np.testing.assert_allclose(np.sum(f ** 2), 128.0, rtol=1e-13)   # one unit pair per frequency
        np.testing.assert_allclose(f[:2], [math.cos(tau), math.sin(tau)], rtol=1e-15)  # first frequency is 1
        # the slowest frequency is 10^4^(-127/128)
        wl = 10000.0 ** (-127.0 / 128.0)
        np.testing.assert_allclose(f[-2:], [math.cos(tau * wl), math.sin(tau * wl)], rtol=1e-13, atol=1e-15)
        np.testing.assert_allclose(f, _torch_fourier(tau).numpy(), rtol=1e-13, atol=1e-15)


def test_embedding_and_modulator_match_torch():
    cfg, w, _ = _cond_tiny(max_loops=4)
    model = O.OracleModel.from_config(cfg, w)
    t = lambda a: torch.tensor(np.asarray(a, dtype=np.float64))
    d = cfg.d_model
    for which in ("t", "dt"):
        for tau in (0.0, 0.25, 1.0):
            np.testing.assert_allclose(model.phi(which, tau), _torch_phi(w, which, tau).numpy(), rtol=1e-12, atol=1e-12)
    for (m, i) in ((1, 1), (3, 2), (4, 4)):
        c = _torch_phi(w, "t", (i - 1) / m) + _torch_phi(w, "dt", 1.0 / m)
        for j in range(cfg.n_layers):
            v = F.linear(F.silu(c), t(w["mod_w"][j]), t(w["mod_b"][j])).numpy()
            got = np.concatenate(model.modulation(j, m, i))
            np.testing.assert_allclose(got, v, rtol=1e-12, atol=1e-12)
            assert got[:d].std() > 0 and got[2 * d:].std() > 0


def test_uniform_trajectory_schedule():
    """Loop i of a depth-m token uses t = (i-1)/m and Delta = 1/m (the embeddings isolated in turn)."""
    cfg, w, _ = _cond_tiny(max_loops=4)
    z = lambda a: np.zeros_like(a)
    only_dt = dict(w, cond_t_w2=z(w["cond_t_w2"]), cond_t_b2=z(w["cond_t_b2"]))
    only_t = dict(w, cond_dt_w2=z(w["cond_dt_w2"]), cond_dt_b2=z(w["cond_dt_b2"]))
    mdt = O.OracleModel.from_config(cfg, only_dt)
    mt = O.OracleModel.from_config(cfg, only_t)
    full = O.OracleModel.from_config(cfg, w)
    for m in range(1, 5):
        for i in range(1, m + 1):
            # the step embedding alone depends on the depth, not on the loop
            np.testing.assert_allclose(mdt.conditioning(m, i), mdt.conditioning(m, 1), rtol=0, atol=0)
            # the two embeddings add
            np.testing.assert_allclose(full.conditioning(m, i), mt.conditioning(m, i) + mdt.conditioning(m, i),
                                       rtol=1e-14, atol=1e-14)
        # the first loop of every depth starts at time 0
        np.testing.assert_allclose(mt.conditioning(m, 1), mt.conditioning(1, 1), rtol=0, atol=0)
    np.testing.assert_allclose(mt.conditioning(4, 3), mt.conditioning(2, 2), rtol=0, atol=0)   # t = 1/2
    assert np.abs(mt.conditioning(4, 2) - mt.conditioning(4, 3)).max() > 1e-3
    assert np.abs(mdt.conditioning(2, 1) - mdt.conditioning(3, 1)).max() > 1e-3


def test_constant_unit_gates_reduce_to_the_backbone():
    """alpha = 1, gamma = 0 for every token: the unconditioned model (itself pinned to a textbook decoder)."""
    cfg, w, toks = _cond_tiny(max_loops=3)
    wc = _constant_modulator(cfg, w, 1.0, 1.0, 0.0, 0.0)
    m = np.array([1, 3, 2, 2, 3, 1, 3, 2, 1, 3], dtype=np.int32)
    for got, ref in zip(_all_logits(cfg, wc, toks, m), _all_logits(cfg, _plain(w), toks, m)):
        np.testing.assert_allclose(got, ref, rtol=1e-11, atol=1e-11)
    full = _all_logits(cfg, wc, toks, np.full(len(toks), 2, np.int32))[0]
    np.testing.assert_allclose(full, _textbook_logits(cfg, _plain(w), toks, 2), rtol=1e-9, atol=1e-9)


def test_zero_gates_switch_the_block_off():
    """alpha = 0: every state stays h^(0), so the logits are the LM head of the embedding."""
    cfg, w, toks = _cond_tiny(max_loops=3)
    wc = _constant_modulator(cfg, w, 0.0, 0.0, 0.3, -0.2)
    m = np.array([1, 3, 2, 2, 3, 1, 3, 2, 1, 3], dtype=np.int32)
    t = lambda a: torch.tensor(np.asarray(a, dtype=np.float64))
    x = t(w["embedding"])[torch.as_tensor(toks)]
    ref = F.linear(F.rms_norm(x, (cfg.d_model,), weight=t(w["final_norm"]), eps=cfg.norm_eps), t(w["embedding"]))
    for got in _all_logits(cfg, wc, toks, m)[:2]:
        np.testing.assert_allclose(got, ref.numpy(), rtol=1e-11, atol=1e-11)


def test_gamma_acts_as_a_norm_gain():
    """gamma constant per feature = the backbone with its norm gains multiplied by (1 + gamma)."""
    cfg, w, toks = _cond_tiny(max_loops=3)
    rng = np.random.default_rng(11)
    g1, g2 = 0.4 * rng.standard_normal(cfg.d_model), 0.4 * rng.standard_normal(cfg.d_model)
    wc = _constant_modulator(cfg, w, 1.0, 1.0, g1, g2)
    wp = _plain(w)
    wp["attn_norm"] = wp["attn_norm"] * (1.0 + g1)
    wp["mlp_norm"] = wp["mlp_norm"] * (1.0 + g2)
    got = _all_logits(cfg, wc, toks, np.full(len(toks), 2, np.int32))[0]
    np.testing.assert_allclose(got, _textbook_logits(cfg, wp, toks, 2), rtol=1e-9, atol=1e-9)


def test_alpha_scales_the_branch_outputs():
    """alpha constant per feature = the backbone with the rows of W_o and W_down scaled by alpha."""
    cfg, w, toks = _cond_tiny(max_loops=3)
    rng = np.random.default_rng(12)
    a1, a2 = 1.0 + 0.5 * rng.standard_normal(cfg.d_model), 1.0 + 0.5 * rng.standard_normal(cfg.d_model)
    wc = _constant_modulator(cfg, w, a1, a2, 0.0, 0.0)
    wp = _plain(w)
    wp["wo"] = wp["wo"] * a1[None, :, None]
    wp["w_down"] = wp["w_down"] * a2[None, :, None]
    got = _all_logits(cfg, wc, toks, np.full(len(toks), 3, np.int32))[0]
    np.testing.assert_allclose(got, _textbook_logits(cfg, wp, toks, 3), rtol=1e-9, atol=1e-9)


def test_conditioned_formulations_agree():
    """Cached decode = gathered prefill = masked brute force with per-token (depth, loop) conditioning."""
    cfg, w, toks = _cond_tiny(T=12, max_loops=3)
    m = np.array([1, 3, 2, 1, 3, 3, 1, 2, 2, 3, 1, 2], dtype=np.int32)
    full, dec, last = _all_logits(cfg, w, toks, m)
    np.testing.assert_allclose(dec, full, rtol=1e-10, atol=1e-10)
    np.testing.assert_allclose(last, full[-1], rtol=1e-10, atol=1e-10)
    # and the conditioning changes the result
    ref = _all_logits(cfg, _plain(w), toks, m)[0]
    assert np.abs(full - ref).max() > 1e-3


# ----------------------------------------------------------------------------
# planted mistakes
# ----------------------------------------------------------------------------

def _attn_out_one_plus(self, j, o, mod=None):
    lead = o.shape[:-2]
    y = o.reshape(*lead, self.n_heads * self.head_dim) @ self.w["wo"][j].T
    return y if mod is None else (1.0 + mod[0].reshape(y.shape)) * y


def _attn_out_swapped_gate(self, j, o, mod=None):
    lead = o.shape[:-2]
    y = o.reshape(*lead, self.n_heads * self.head_dim) @ self.w["wo"][j].T
    return y if mod is None else mod[1].reshape(y.shape) * y


def _qkv_gamma_before_norm(self, j, h, mod=None):
    x = h if mod is None else h * (1.0 + mod[2].reshape(h.shape))
    a = O.rms_norm(x, self.w["attn_norm"][j], self.norm_eps)
    lead = h.shape[:-1]
    return ((a @ self.w["wq"][j].T).reshape(*lead, self.n_heads, self.head_dim),
            (a @ self.w["wk"][j].T).reshape(*lead, self.n_kv_heads, self.head_dim),
            (a @ self.w["wv"][j].T).reshape(*lead, self.n_kv_heads, self.head_dim))


def _trajectory_shifted(m, i):
    return i / m, 1.0 / m


def _fourier_sin_first(tau, width=256, max_period=10000.0):
    f = O.__dict__["_orig_fourier"](tau, width, max_period)
    g = np.empty_like(f)
    g[0::2], g[1::2] = f[1::2], f[0::2]
    return g


def _modulation_no_silu(self, j, m, i):
    v = self.w["mod_w"][j] @ self.conditioning(m, i) + self.w["mod_b"][j]
    d = self.d_model
    return (v[:d], v[d:2 * d], v[2 * d:3 * d], v[3 * d:])


COND_PLANTS = {
    "gate_one_plus_alpha": ("OracleModel.attn_out", _attn_out_one_plus),
    "gate_swapped": ("OracleModel.attn_out", _attn_out_swapped_gate),
    "gamma_before_norm": ("OracleModel.qkv", _qkv_gamma_before_norm),
    "trajectory_shifted": ("trajectory", _trajectory_shifted),
    "fourier_sin_first": ("fourier_features", _fourier_sin_first),
    "modulator_no_silu": ("OracleModel.modulation", _modulation_no_silu),
}


def _all_cond_pins_pass():
    tests = [test_fourier_features_closed_forms, test_embedding_and_modulator_match_torch,
             test_uniform_trajectory_schedule, test_constant_unit_gates_reduce_to_the_backbone,
             test_zero_gates_switch_the_block_off, test_gamma_acts_as_a_norm_gain,
             test_alpha_scales_the_branch_outputs, test_conditioned_formulations_agree]
    for t in tests:
        try:
            t()
        except AssertionError:
            return False
    return True


@pytest.mark.parametrize("name", sorted(COND_PLANTS))
def test_conditioning_planted_mistakes(name, monkeypatch):
    target, fn = COND_PLANTS[name]
    monkeypatch.setitem(O.__dict__, "_orig_fourier", O.fourier_features)
    if "." in target:
        cls, attr = target.split(".")
        monkeypatch.setattr(getattr(O, cls), attr, fn)
    else:
        monkeypatch.setattr(O, target, fn)
    assert not _all_cond_pins_pass(), f"planted mistake {name} went unnoticed"


def test_unplanted_oracle_passes_conditioning_pins():
    assert _all_cond_pins_pass()
