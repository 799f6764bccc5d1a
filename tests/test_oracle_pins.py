"""Pins of the CPU oracle against facts fixed outside it.

Each test checks the oracle against something other than itself: values
worked by hand from the routing rule (Eq. 3-5), closed forms of RMSNorm /
RoPE / softmax attention, an independent textbook transformer built from
torch library routines (the fixed-depth special case, which the paper calls
Base-Loop), the brute-force masked recomputation (Eq. 7, Eq. 10 with mu) and
invariants of the recursion-wise cache (Sec. 3.3). ``test_planted_mistakes``
plants plausible bugs in the oracle and checks that a pin catches each one.
"""
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import tlf_oracle as O
from paper_2609_15160_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ----------------------------------------------------------------------------
# helpers
# ----------------------------------------------------------------------------

def _model(cfg=None, **kw):
    cfg = cfg or synth.tiny_config(**kw)
    return cfg, O.OracleModel.from_config(cfg, synth.make_weights(cfg))


def _textbook_logits(cfg, w, tokens, loops):
    """A plain pre-norm RoPE/SwiGLU decoder from torch library routines.

    The shared J-layer block is applied ``loops`` times to every token with
    ordinary causal attention: the fixed-depth looped transformer. RoPE is
    applied as a complex rotation of (x_k + i x_{k+hd/2}).
    """
    t = lambda a: torch.tensor(np.asarray(a, dtype=np.float64))
    E = t(w["embedding"])
    x = E[torch.as_tensor(np.asarray(tokens, dtype=np.int64))]
    T, d, hd = x.shape[0], cfg.d_model, cfg.head_dim
    half = hd // 2
    freqs = cfg.rope_base ** (-2.0 * torch.arange(half, dtype=torch.float64) / hd)
    rot = torch.polar(torch.ones(T, half, dtype=torch.float64),
                      torch.arange(T, dtype=torch.float64)[:, None] * freqs)

    def rope_c(a):  # [T, H, hd]
        c = torch.complex(a[..., :half], a[..., half:]) * rot[:, None, :]
        return torch.cat([c.real, c.imag], dim=-1)

    for _ in range(loops):
        for j in range(cfg.n_layers):
            a = F.rms_norm(x, (d,), weight=t(w["attn_norm"][j]), eps=cfg.norm_eps)
            q = rope_c(F.linear(a, t(w["wq"][j])).view(T, cfg.n_heads, hd))
            k = rope_c(F.linear(a, t(w["wk"][j])).view(T, cfg.n_kv_heads, hd))
            v = F.linear(a, t(w["wv"][j])).view(T, cfg.n_kv_heads, hd)
            o = F.scaled_dot_product_attention(q.transpose(0, 1), k.transpose(0, 1), v.transpose(0, 1),
                                               is_causal=True, enable_gqa=True)
            x = x + F.linear(o.transpose(0, 1).reshape(T, -1), t(w["wo"][j]))
            b = F.rms_norm(x, (d,), weight=t(w["mlp_norm"][j]), eps=cfg.norm_eps)
            x = x + F.linear(F.silu(F.linear(b, t(w["w_gate"][j]))) * F.linear(b, t(w["w_up"][j])),
                             t(w["w_down"][j]))
    return F.linear(F.rms_norm(x, (d,), weight=t(w["final_norm"]), eps=cfg.norm_eps), E).numpy()


def _random_norm_gains(w, seed=5):
    """Non-unit gains so that a dropped or misplaced gain is visible."""
    rng = np.random.default_rng(seed)
    w = dict(w)
    for k in ("attn_norm", "mlp_norm"):
        w[k] = (1.0 + 0.3 * rng.standard_normal(w[k].shape)).astype(np.float32)
    w["final_norm"] = (1.0 + 0.3 * rng.standard_normal(w["final_norm"].shape)).astype(np.float32)
    return w


def _tiny(seed_tokens=3, T=11, **kw):
    cfg = synth.tiny_config(**kw)
    w = _random_norm_gains(synth.make_weights(cfg))
    w["embedding"] = w["embedding"] * 40.0     # O(1) activations so every term matters
    for k in ("wq", "wk", "wv", "wo", "w_gate", "w_up", "w_down"):
        w[k] = w[k] * 15.0
    model = O.OracleModel.from_config(cfg, w)
    toks = np.random.default_rng(seed_tokens).integers(0, cfg.vocab, size=T)
    return cfg, w, model, toks


# ----------------------------------------------------------------------------
# elementary operations
# ----------------------------------------------------------------------------

def test_rms_norm_closed_forms():
    x = np.array([3.0, -3.0, 3.0, -3.0])
    np.testing.assert_allclose(O.rms_norm(x, None, 0.0), [1, -1, 1, -1], rtol=0, atol=1e-15)
    rng = np.random.default_rng(0)
    y = rng.standard_normal((5, 32))
    out = O.rms_norm(y, None, 0.0)
    np.testing.assert_allclose(np.sqrt(np.mean(out ** 2, axis=-1)), 1.0, rtol=1e-14)
    np.testing.assert_allclose(O.rms_norm(7.5 * y, None, 0.0), out, rtol=1e-13)
    g = rng.standard_normal(32)
    np.testing.assert_allclose(O.rms_norm(y, g, 0.0), out * g, rtol=1e-14)
    # eps enters as mean(x^2) + eps: a constant row c gives c / sqrt(c^2 + eps)
    np.testing.assert_allclose(O.rms_norm(np.full(8, 0.01), None, 1e-4), 0.01 / np.sqrt(1e-4 + 1e-4))


def test_softmax_and_silu_match_torch():
    z = np.random.default_rng(1).standard_normal((4, 9)) * 3
    np.testing.assert_allclose(O.softmax(z), torch.softmax(torch.tensor(z), -1).numpy(), rtol=1e-14)
    np.testing.assert_allclose(O.silu(z), F.silu(torch.tensor(z)).numpy(), rtol=1e-13)


def test_rope_closed_forms():
    hd, base = 16, 10000.0
    rng = np.random.default_rng(2)
    q, k = rng.standard_normal(hd), rng.standard_normal(hd)
    # position 0 is the identity; rotations preserve norms
    np.testing.assert_allclose(O.rope(q, 0, base), q, rtol=0, atol=0)
    np.testing.assert_allclose(np.linalg.norm(O.rope(q, 37, base)), np.linalg.norm(q), rtol=1e-14)
    # scores depend only on the relative offset
    for t1, t2, s in [(5, 2, 11), (0, 9, 100), (1000, 3, 7)]:
        a = O.rope(q, t1, base) @ O.rope(k, t2, base)
        b = O.rope(q, t1 + s, base) @ O.rope(k, t2 + s, base)
        np.testing.assert_allclose(a, b, rtol=1e-10)
    # a unit vector in dimension kk turns into the pair (kk, kk + hd/2) at angle pos * base^(-2kk/hd)
    for kk in (0, 3, 7):
        e = np.zeros(hd)
        e[kk] = 1.0
        pos = 13
        ang = pos * base ** (-2.0 * kk / hd)
        want = np.zeros(hd)
        want[kk], want[kk + hd // 2] = np.cos(ang), np.sin(ang)
        np.testing.assert_allclose(O.rope(e, pos, base), want, atol=1e-15)


def test_attention_closed_forms_and_library():
    rng = np.random.default_rng(3)
    hq, hkv, hd = 4, 2, 8
    q = rng.standard_normal((hq, hd))
    kv = rng.standard_normal((1, hkv, hd))
    np.testing.assert_allclose(O.attention(q, kv, kv * 2), np.repeat(kv[0] * 2, 2, axis=0), rtol=1e-14)
    same_k = np.repeat(rng.standard_normal((1, hkv, hd)), 6, axis=0)
    v = rng.standard_normal((6, hkv, hd))
    np.testing.assert_allclose(O.attention(q, same_k, v), np.repeat(v.mean(0), 2, axis=0), rtol=1e-13)
    k = rng.standard_normal((9, hkv, hd))
    v = rng.standard_normal((9, hkv, hd))
    ref = F.scaled_dot_product_attention(torch.tensor(q)[:, None, :], torch.tensor(k).permute(1, 0, 2),
                                         torch.tensor(v).permute(1, 0, 2), enable_gqa=True)[:, 0, :]
    np.testing.assert_allclose(O.attention(q, k, v), ref.numpy(), rtol=1e-12, atol=1e-14)


# ----------------------------------------------------------------------------
# router (Eq. 2-5)
# ----------------------------------------------------------------------------

def _golden_rows():
    rows = []
    with open(os.path.join(GOLDEN, "router_worked_examples.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            rule, vals, m, margin = [s.strip() for s in line.split("|")]
            rows.append((rule, np.array([float(x) for x in vals.split()]), int(m), float(margin)))
    return rows


@pytest.mark.parametrize("row", _golden_rows(), ids=lambda r: f"{r[0]}-{len(r[1])}")
def test_router_worked_examples(row):
    rule, vals, m_want, margin_want = row
    cfg, model = _model(max_loops=len(vals), exit_rule=rule)
    z = np.log(vals) if rule == "survival" else vals
    m, margin = O.loop_counts(model, z[None, :])
    assert int(m[0]) == m_want
    np.testing.assert_allclose(margin[0], margin_want, atol=2e-7)


def test_survival_rule_nesting_and_median():
    """A_1 holds every token, the sets nest, and m is the upper weighted median."""
    cfg, model = _model(max_loops=6, exit_rule="survival")
    z = np.random.default_rng(4).standard_normal((500, 6)) * 2
    m, _ = O.loop_counts(model, z)
    pi = O.softmax(z.astype(np.float32).astype(np.float64))
    for t in range(z.shape[0]):
        p = np.cumsum(pi[t][::-1])[::-1]
        act = p > 0.5
        assert act[0]
        assert np.all(act[:-1] >= act[1:])                   # nested active sets
        assert m[t] == act.sum()
        # brute force: the largest i with P(depth >= i) > 1/2
        assert m[t] == max(i for i in range(1, 7) if pi[t][i - 1:].sum() > 0.5)
    assert m.min() >= 1 and m.max() <= 6


def _mlp_router_model(d=16, hidden=24, M=4, seed=9):
    cfg = synth.tiny_config(router_hidden=hidden, max_loops=M)
    return cfg, synth.make_weights(cfg)


def test_gelu_matches_torch():
    x = np.linspace(-8, 8, 401)
    np.testing.assert_allclose(O.gelu(x), F.gelu(torch.tensor(x), approximate="none").numpy(), rtol=1e-14, atol=1e-15)


def test_mlp_router_matches_torch():
    """The two-layer MLP router (Sec. 3.2) against torch library routines."""
    cfg, w = _mlp_router_model()
    model = O.OracleModel.from_config(cfg, w)
    toks = np.arange(cfg.vocab)
    t = lambda a: torch.tensor(np.asarray(a, dtype=np.float64))
    x = F.rms_norm(t(w["embedding"])[torch.as_tensor(toks)], (cfg.d_model,), eps=cfg.norm_eps)
    z = F.linear(F.gelu(F.linear(x, t(w["router_w1"]), t(w["router_b1"]))), t(w["router_w"]), t(w["router_b"]))
    np.testing.assert_allclose(O.router_logits(model, toks), z.numpy(), rtol=1e-12, atol=1e-12)


def test_mlp_router_reduces_to_the_linear_router():
    """W_1 = I and a large b_1 make GELU the identity shifted by b_1: the linear router with bias b_r + b_1 W_r 1."""
    cfg, w = _mlp_router_model(hidden=16)
    d = cfg.d_model
    wm = dict(w, router_w1=np.eye(d), router_b1=np.full(d, 40.0))
    lin = {k: v for k, v in w.items() if k not in ("router_w1", "router_b1")}
    lin["router_b"] = w["router_b"].astype(np.float64) + 40.0 * w["router_w"].astype(np.float64).sum(axis=1)
    toks = np.arange(cfg.vocab)
    z_mlp = O.router_logits(O.OracleModel.from_config(cfg, wm), toks)
    z_lin = O.router_logits(O.OracleModel.from_config(cfg, lin), toks)
    np.testing.assert_allclose(z_mlp, z_lin, rtol=1e-12, atol=1e-10)


def test_router_reads_only_the_embedding():
    """The loop count is a function of the token id (R2 reading)."""
    cfg, w, model, toks = _tiny(max_loops=4)
    table, _ = O.depth_table(model)
    seq = O.OracleSequence(model)
    ms = [O.decode_token(model, seq, int(x))[1] for x in toks]
    assert list(ms) == [int(table[x]) for x in toks]


# ----------------------------------------------------------------------------
# whole-model pins
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("k", [1, 2, 3])
def test_fixed_depth_equals_textbook_looped_transformer(k):
    """Every token forced to k loops = a k-times-looped plain decoder."""
    cfg, w, model, toks = _tiny(T=9)
    ref = _textbook_logits(cfg, w, toks, k)
    forced = [k] * len(toks)
    full = O.forward_masked(model, toks, forced)
    np.testing.assert_allclose(full, ref, rtol=1e-9, atol=1e-9)
    seq = O.OracleSequence(model)
    for t, x in enumerate(toks):
        lg, m, _ = O.decode_token(model, seq, int(x), forced=k)
        assert m == k
        np.testing.assert_allclose(lg, ref[t], rtol=1e-9, atol=1e-9)
    seq2 = O.OracleSequence(model)
    lg, _ = O.prefill_gathered(model, seq2, toks, forced=forced)
    np.testing.assert_allclose(lg, ref[-1], rtol=1e-9, atol=1e-9)


def test_three_formulations_agree_with_routed_depths():
    """Cached decode (Eq. 8-11) = gathered prefill (Eq. 6-7) = masked brute force (Eq. 10 with mu)."""
    cfg, w, model, toks = _tiny(T=14, max_loops=3)
    m = np.array([1, 3, 2, 1, 3, 3, 1, 2, 2, 3, 1, 1, 2, 3], dtype=np.int32)
    full = O.forward_masked(model, toks, m)
    seq = O.OracleSequence(model)
    for t, x in enumerate(toks):
        lg, mm, _ = O.decode_token(model, seq, int(x), forced=int(m[t]))
        np.testing.assert_allclose(lg, full[t], rtol=1e-10, atol=1e-10)
    for T in (5, 14):
        seq_g = O.OracleSequence(model)
        lg, mg = O.prefill_gathered(model, seq_g, toks[:T], forced=m[:T])
        np.testing.assert_allclose(lg, full[T - 1], rtol=1e-10, atol=1e-10)
    # the two cache-building paths hold the same entries
    for i in range(cfg.max_loops):
        for j in range(cfg.n_layers):
            p1, k1, v1 = seq.caches[i][j].view()
            p2, k2, v2 = seq_g.caches[i][j].view()
            np.testing.assert_array_equal(p1, p2)
            np.testing.assert_allclose(k1, k2, rtol=1e-11, atol=1e-12)
            np.testing.assert_allclose(v1, v2, rtol=1e-11, atol=1e-12)


def test_routed_prefill_uses_router_depths():
    cfg, w, model, toks = _tiny(T=12, max_loops=4)
    table, _ = O.depth_table(model)
    seq = O.OracleSequence(model)
    lg, m = O.prefill_gathered(model, seq, toks)
    np.testing.assert_array_equal(m, table[toks])
    full = O.forward_masked(model, toks, m)
    np.testing.assert_allclose(lg, full[-1], rtol=1e-10, atol=1e-10)


def test_cache_content_invariant():
    """Cache (i, j) holds exactly the positions with m_t >= i, in order."""
    cfg, w, model, toks = _tiny(T=17, max_loops=4)
    m = np.random.default_rng(9).integers(1, 5, size=17)
    seq = O.OracleSequence(model)
    for t, x in enumerate(toks):
        O.decode_token(model, seq, int(x), forced=int(m[t]))
    total = 0
    for i in range(1, 5):
        want = np.nonzero(m >= i)[0]
        for j in range(cfg.n_layers):
            np.testing.assert_array_equal(seq.caches[i - 1][j].view()[0], want)
        total += seq.cache_len(i)
    assert total == m.sum()


def test_depth_locality():
    """A token's output ignores caches deeper than its own loop count and the value of M."""
    cfg, w, model, toks = _tiny(T=8, max_loops=3)
    m = np.array([3, 1, 2, 3, 2, 1, 3, 2])
    seq = O.OracleSequence(model)
    for t, x in enumerate(toks[:-1]):
        O.decode_token(model, seq, int(x), forced=int(m[t]))
    import copy
    seq_b = copy.deepcopy(seq)
    seq_b.caches[2][0].k[:seq_b.caches[2][0].n] += 5.0          # perturb loop-3 caches
    seq_b.caches[2][1].v[:seq_b.caches[2][1].n] -= 2.0
    la, _, _ = O.decode_token(model, seq, int(toks[-1]), forced=2)
    lb, _, _ = O.decode_token(model, seq_b, int(toks[-1]), forced=2)
    np.testing.assert_array_equal(la, lb)
    # a larger M (extra, unused loops) changes nothing when depths are fixed
    cfg5 = synth.tiny_config(max_loops=5)
    w5 = dict(w)
    w5["router_w"] = np.concatenate([w["router_w"], w["router_w"][:2]])
    w5["router_b"] = np.zeros(5, dtype=np.float32)
    model5 = O.OracleModel.from_config(cfg5, w5)
    np.testing.assert_allclose(O.forward_masked(model5, toks, m), O.forward_masked(model, toks, m),
                               rtol=0, atol=0)


def test_exited_token_leaves_deeper_caches_untouched():
    cfg, w, model, toks = _tiny(T=6, max_loops=3)
    seq = O.OracleSequence(model)
    for x in toks:
        O.decode_token(model, seq, int(x), forced=3)
    before = [seq.cache_len(i) for i in (1, 2, 3)]
    O.decode_token(model, seq, int(toks[0]), forced=1)
    assert [seq.cache_len(i) for i in (1, 2, 3)] == [before[0] + 1, before[1], before[2]]


def test_batch_invariance():
    cfg, w, model, toks = _tiny(T=10)
    seqs = [O.OracleSequence(model) for _ in range(3)]
    solo = [O.OracleSequence(model) for _ in range(3)]
    rng = np.random.default_rng(11)
    for step in range(4):
        batch_toks = rng.integers(0, cfg.vocab, size=3)
        lg, m, _ = O.decode_step(model, seqs, batch_toks)
        for b in range(3):
            l1, m1, _ = O.decode_token(model, solo[b], int(batch_toks[b]))
            np.testing.assert_array_equal(lg[b], l1)
            assert m[b] == m1


def test_prefill_then_decode_equals_longer_prefill():
    cfg, w, model, toks = _tiny(T=13, max_loops=3)
    seq = O.OracleSequence(model)
    O.prefill_gathered(model, seq, toks[:-1])
    lg_dec, _, _ = O.decode_token(model, seq, int(toks[-1]))
    seq2 = O.OracleSequence(model)
    lg_all, _ = O.prefill_gathered(model, seq2, toks)
    np.testing.assert_allclose(lg_dec, lg_all, rtol=1e-10, atol=1e-10)


def test_snapshot_round_trip():
    cfg = synth.tiny_config(max_loops=3, dtype="bf16")
    w = synth.make_weights(cfg)
    model = O.OracleModel.from_config(cfg, w)
    snap = synth.make_cache_snapshot(cfg, 20, seed=4)
    seq = O.load_snapshot(model, snap)
    for i in range(3):
        assert seq.cache_len(i + 1) == int((snap["depths"] >= i + 1).sum())
        for j in range(cfg.n_layers):
            p, k, v = seq.caches[i][j].view()
            np.testing.assert_array_equal(p, snap["positions"][i])
            np.testing.assert_array_equal(k, snap["k"][i][:, j])
    lg, m, _ = O.decode_token(model, seq, 5)
    assert lg.shape == (cfg.vocab,) and seq.n_tokens == 21


# ----------------------------------------------------------------------------
# planted mistakes: each must make at least one pin fail
# ----------------------------------------------------------------------------

def _rope_sign(x, pos, base):
    x = np.asarray(x, dtype=np.float64)
    hd = x.shape[-1]; half = hd // 2
    ang = np.asarray(pos, dtype=np.float64)[..., None] * base ** (-2.0 * np.arange(half) / hd)
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * np.cos(ang) + x2 * np.sin(ang), -x1 * np.sin(ang) + x2 * np.cos(ang)], -1)


def _rope_interleaved(x, pos, base):
    x = np.asarray(x, dtype=np.float64)
    hd = x.shape[-1]
    y = x.copy()
    ang = np.asarray(pos, dtype=np.float64)[..., None] * base ** (-2.0 * np.arange(hd // 2) / hd)
    a, b = x[..., 0::2], x[..., 1::2]
    y[..., 0::2] = a * np.cos(ang) - b * np.sin(ang)
    y[..., 1::2] = a * np.sin(ang) + b * np.cos(ang)
    return y


def _attention_noscale(q, k, v):
    return _orig_attention(q * np.sqrt(q.shape[-1]), k, v)


def _attention_gqa_mod(q, k, v):
    hq = q.shape[0]
    hkv = k.shape[1]
    return np.stack([_orig_attention(q[h:h + 1], k[:, [h % hkv]], v[:, [h % hkv]])[0] for h in range(hq)])


_orig_attention = O.attention
_orig_mlp = O.OracleModel.mlp
_orig_qkv = O.OracleModel.qkv


def _mlp_swapped(self, j, h, mod=None):
    b = O.rms_norm(h, self.w["mlp_norm"][j], self.norm_eps)
    return (O.silu(b @ self.w["w_up"][j].T) * (b @ self.w["w_gate"][j].T)) @ self.w["w_down"][j].T


def _qkv_transposed(self, j, h, mod=None):
    a = O.rms_norm(h, self.w["attn_norm"][j], self.norm_eps)
    lead = h.shape[:-1]
    return ((a @ self.w["wq"][j]).reshape(*lead, self.n_heads, self.head_dim),
            (a @ self.w["wk"][j].T).reshape(*lead, self.n_kv_heads, self.head_dim),
            (a @ self.w["wv"][j].T).reshape(*lead, self.n_kv_heads, self.head_dim))


def _qkv_no_gain(self, j, h, mod=None):
    a = O.rms_norm(h, None, self.norm_eps)
    lead = h.shape[:-1]
    return ((a @ self.w["wq"][j].T).reshape(*lead, self.n_heads, self.head_dim),
            (a @ self.w["wk"][j].T).reshape(*lead, self.n_kv_heads, self.head_dim),
            (a @ self.w["wv"][j].T).reshape(*lead, self.n_kv_heads, self.head_dim))


def _decode_attend_before_append(model, seq, token, forced=None):
    """Mistake: the token attends to the cache before writing its own entry."""
    pos = seq.n_tokens
    m = int(forced) if forced else int(O.loop_counts(model, O.router_logits(model, [token]))[0][0])
    h = model.w["embedding"][token].astype(np.float64)
    for i in range(1, m + 1):
        for j in range(model.n_layers):
            q, k, v = model.qkv(j, h)
            q, k = O.rope(q, pos, model.rope_base), O.rope(k, pos, model.rope_base)
            c = seq.caches[i - 1][j]
            if c.n:
                _, kc, vc = c.view()
                o = O.attention(q, kc, vc)
            else:
                o = np.zeros_like(q)
            c.append(pos, k, v)
            h = h + model.attn_out(j, o)
            h = h + model.mlp(j, h)
    seq.n_tokens += 1
    return model.logits(h), m, 0.0


def _decode_shared_cache(model, seq, token, forced=None):
    """Mistake: every loop reads and writes the loop-1 cache (no recursion-wise cache)."""
    pos = seq.n_tokens
    m = int(forced) if forced else int(O.loop_counts(model, O.router_logits(model, [token]))[0][0])
    h = model.w["embedding"][token].astype(np.float64)
    for i in range(1, m + 1):
        for j in range(model.n_layers):
            q, k, v = model.qkv(j, h)
            q, k = O.rope(q, pos, model.rope_base), O.rope(k, pos, model.rope_base)
            c = seq.caches[0][j]
            c.append(pos, k, v)
            _, kc, vc = c.view()
            h = h + model.attn_out(j, O.attention(q, kc, vc))
            h = h + model.mlp(j, h)
    seq.n_tokens += 1
    return model.logits(h), m, 0.0


def _gelu_tanh(x):
    return 0.5 * x * (1.0 + np.tanh(np.sqrt(2.0 / np.pi) * (x + 0.044715 * x ** 3)))


def _router_no_hidden_bias(model, tokens):
    h0 = model.w["embedding"][np.asarray(tokens, dtype=np.int64)]
    x = O.rms_norm(h0, None, model.norm_eps)
    if "router_w1" in model.w:
        x = O.gelu(x @ model.w["router_w1"].T)
    return x @ model.w["router_w"].T + model.w["router_b"]


def _loop_counts_off_by_one(model, z):
    m, g = _orig_loop_counts(model, z)
    return np.minimum(m + 1, model.max_loops).astype(np.int32), g


_orig_loop_counts = O.loop_counts


def _loop_counts_ge(model, z):
    """Mistake: survival rule with >= instead of > (and argmax ties to the larger depth)."""
    z32 = np.atleast_2d(np.asarray(z, dtype=np.float32).astype(np.float64))
    m = np.empty(len(z32), dtype=np.int32)
    for t in range(len(z32)):
        if model.exit_rule == "argmax":
            m[t] = len(z32[t]) - int(np.argmax(z32[t][::-1]))
        else:
            pi = O.softmax(z32[t])
            m[t] = sum(1 for i in range(len(pi)) if pi[i:].sum() >= model.threshold)
    return m, np.zeros(len(z32))


PLANTS = {
    "rope_sign": ("rope", _rope_sign),
    "rope_pairs": ("rope", _rope_interleaved),
    "attn_scale": ("attention", _attention_noscale),
    "gqa_map": ("attention", _attention_gqa_mod),
    "mlp_swap": ("OracleModel.mlp", _mlp_swapped),
    "qkv_transpose": ("OracleModel.qkv", _qkv_transposed),
    "norm_gain_dropped": ("OracleModel.qkv", _qkv_no_gain),
    "attend_before_append": ("decode_token", _decode_attend_before_append),
    "shared_cache": ("decode_token", _decode_shared_cache),
    "depth_off_by_one": ("loop_counts", _loop_counts_off_by_one),
    "threshold_ge": ("loop_counts", _loop_counts_ge),
    "gelu_tanh": ("gelu", _gelu_tanh),
    "router_hidden_bias_dropped": ("router_logits", _router_no_hidden_bias),
}


def _all_pins_pass():
    tests = [
        lambda: [test_fixed_depth_equals_textbook_looped_transformer(k) for k in (1, 2)],
        test_three_formulations_agree_with_routed_depths,
        lambda: [test_router_worked_examples(r) for r in _golden_rows()],
        test_routed_prefill_uses_router_depths,
        test_cache_content_invariant,
        test_exited_token_leaves_deeper_caches_untouched,
        test_gelu_matches_torch,
        test_mlp_router_matches_torch,
        test_mlp_router_reduces_to_the_linear_router,
    ]
    for t in tests:
        try:
            t()
        except (AssertionError, ValueError, IndexError):
            return False
    return True


@pytest.mark.parametrize("name", sorted(PLANTS))
def test_planted_mistakes(name, monkeypatch):
    target, fn = PLANTS[name]
    if "." in target:
        cls, attr = target.split(".")
        monkeypatch.setattr(getattr(O, cls), attr, fn)
    else:
        monkeypatch.setattr(O, target, fn)
    assert not _all_pins_pass(), f"planted mistake {name} went unnoticed"


def test_unplanted_oracle_passes_all_pins():
    assert _all_pins_pass()
