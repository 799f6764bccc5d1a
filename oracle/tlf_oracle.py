"""Plain float64 CPU oracle of the T-LoopFormer decode step.

TEST INFRASTRUCTURE. Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
module. It shares no code with the CUDA library and imports nothing from it;
the two meet only through the seeded inputs of ``synth``.

What it computes, in the paper's notation (T-LoopFormer, Sec. 3):

* Router (Sec. 3.2, Eq. 2-5): the initial state h^(0) = E[x] of each token is
  mapped to M router logits; the loop count m is read off those logits.
* Gather-scatter (Eq. 6-7): loop i runs the shared block Phi_J only on the
  active set A_i = {tau : m_tau >= i}; exited tokens keep h^(m).
* Recursion-wise KV cache (Sec. 3.3, Eq. 8-11): each (loop i, layer j) keeps
  its own cache; a token writes its k, v into cache (i, j) only when it runs
  loop i, and its loop-i query attends only to cache (i, j) -- the validity
  mask mu^(i) of Eq. 10.
* Final normalisation and the tied LM head on h^(m) (end of Sec. 3.3).

Three formulations are given, so that they can be checked against each other:

``decode_token``       one token at a time with caches (Eq. 8-11);
``prefill_gathered``   a whole prompt, loop by loop, on the gathered rows
                       with a causal mask among them, writing caches at the
                       original positions rho^(i) (Eq. 6-7, App. B);
``forward_masked``     a whole sequence with no gather: every row is computed
                       at every loop, attention uses the mask
                       [t' <= t] * mu^(i)_{t'}, and Eq. 7 keeps the rows of
                       exited tokens (the brute-force reading).

Readings where the paper is open or inconsistent (all follow the workload
definitions the implementation is built for):

* Block: pre-norm layer with RMSNorm (with a stored gain, all ones), multi-head
  attention with rotary position embedding (base 10000, rotate-half pairs
  (k, k + hd/2), theta_k = base^(-2k/hd), at the token's original 0-based
  position), and a SwiGLU MLP. The paper's block has learned absolute
  positions and a GELU MLP (App. A); the workloads replace both.
* Grouped-query attention: query head h reads kv head h // (Hq / Hkv).
* Eq. 7's "Block(H) + H" is the residual stream of the pre-norm layers, not
  an extra outer residual.
* A decoding token appends its own k, v to cache (i, j) and then attends to
  every entry of that cache, itself included (Eq. 10 writes K_{<t}, Eq. 11
  appends k_t; the softmax set is never empty).
* Router input: RMSNorm (no gain) of h^(0) = E[x] followed by a linear map
  with bias, d -> M; or, with router weights router_w1 / router_b1, the
  paper's two-layer MLP: a hidden layer of width H_r with the exact GELU (the
  activation of the paper's block MLP; the router's own is unstated), then
  the linear map H_r -> M. (The paper's router is a two-layer MLP on E + E_pos; the
  workloads use RoPE, so the router sees only the token embedding and the
  loop count is a function of the token id.)
* Exit rule "argmax": m = 1 + argmax_l z_l, ties to the smaller depth,
  margin = z_(1) - z_(2). Exit rule "survival" (Eq. 3-5): pi = softmax(z),
  p^(i) = sum_{l >= i} pi_l, m = max{i : p^(i) > threshold}, margin =
  min(p^(m) - threshold, threshold - p^(m+1)) with p^(M+1) = 0. The decision
  is taken on the logits rounded to float32 (the precision in which the GPU
  takes it); everything else is float64.
* RMSNorm eps = 1e-5 (unstated in the paper).
* Nothing is written to caches deeper than m (Eq. 11 and the text after it).
* Time/step conditioning (Sec. 3.1, App. A; only when the weights carry the
  conditioning MLPs): a token of depth m follows the uniform trajectory of
  length m, so at loop i it is conditioned on the cumulative time
  t = c_{i-1} = (i-1)/m and the step Delta = 1/m. Each scalar goes through
  sinusoidal Fourier features (width 256, max period 10^4; cos and sin of each
  frequency, in that order) and its own two-layer SiLU MLP; the two results
  are summed into c. Layer j's modulator maps SiLU(c) linearly to
  (alpha_msa, alpha_mlp, gamma_msa, gamma_mlp), and the layer computes
  x <- x + alpha_msa * MHSA(RMSNorm(x) * g * (1 + gamma_msa)) and
  x <- x + alpha_mlp * FFN(RMSNorm(x) * g * (1 + gamma_mlp)), the gates
  applied as the equation in App. A writes them (the stored gains g are kept;
  the paper's norms have none, which gains of one reproduce).
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List, Optional, Sequence, Tuple

import numpy as np

__all__ = [
    "OracleModel", "OracleSequence", "RecursionCache",
    "rms_norm", "silu", "softmax", "rope", "attention",
    "router_logits", "loop_counts", "decode_token", "decode_step",
    "prefill_sequential", "prefill_gathered", "forward_masked", "load_snapshot",
    "depth_table", "fourier_features", "trajectory", "gelu",
]


# ----------------------------------------------------------------------------
# Elementary operations
# ----------------------------------------------------------------------------

def rms_norm(x: np.ndarray, gain: Optional[np.ndarray], eps: float) -> np.ndarray:
    """RMSNorm over the last axis: x / sqrt(mean(x^2) + eps), times gain if given."""
    x = np.asarray(x, dtype=np.float64)
    y = x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps)
    return y if gain is None else y * gain


def silu(x: np.ndarray) -> np.ndarray:
    return x / (1.0 + np.exp(-x))


def gelu(x: np.ndarray) -> np.ndarray:
    """x * Phi(x), Phi the standard normal CDF (the exact GELU)."""
    from scipy.special import erf
    return 0.5 * x * (1.0 + erf(x / np.sqrt(2.0)))


def fourier_features(tau: float, width: int = 256, max_period: float = 10000.0) -> np.ndarray:
    """[cos(tau w_1), sin(tau w_1), ..., cos(tau w_K), sin(tau w_K)], K = width / 2,
    w_k = exp(-(k - 1) / K * ln(max_period)) (App. A conditioning embedding)."""
    K = width // 2
    w = np.exp(-np.arange(K, dtype=np.float64) / K * np.log(max_period))
    out = np.empty(width, dtype=np.float64)
    out[0::2] = np.cos(tau * w)
    out[1::2] = np.sin(tau * w)
    return out


def trajectory(m: int, i: int) -> Tuple[float, float]:
    """(cumulative time c_{i-1}, step Delta_i) of loop i for a token of depth m: the uniform
    trajectory of length m (Sec. 3.1: the full trajectory of L loops has Delta_i = 1/L)."""
    return (i - 1) / m, 1.0 / m


def softmax(z: np.ndarray, axis: int = -1) -> np.ndarray:
    z = np.asarray(z, dtype=np.float64)
    e = np.exp(z - np.max(z, axis=axis, keepdims=True))
    return e / np.sum(e, axis=axis, keepdims=True)


def rope(x: np.ndarray, pos, base: float) -> np.ndarray:
    """Rotary embedding on the last axis (length hd) at integer position(s) pos.

    Pair (k, k + hd/2) is rotated by the angle pos * base^(-2k/hd).
    ``pos`` is a scalar or broadcasts against x's leading axes.
    """
    x = np.asarray(x, dtype=np.float64)
    hd = x.shape[-1]
    half = hd // 2
    theta = base ** (-2.0 * np.arange(half, dtype=np.float64) / hd)
    ang = np.asarray(pos, dtype=np.float64)[..., None] * theta
    c, s = np.cos(ang), np.sin(ang)
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c - x2 * s, x1 * s + x2 * c], axis=-1)


def attention(q: np.ndarray, k: np.ndarray, v: np.ndarray) -> np.ndarray:
    """One query per head against a list of keys (Eq. 10 on a valid-only cache).

    q [Hq, hd]; k, v [L, Hkv, hd]; returns o [Hq, hd].
    """
    hq, hd = q.shape
    group = hq // k.shape[1]
    o = np.empty((hq, hd), dtype=np.float64)
    for h in range(hq):
        kh = k[:, h // group, :].astype(np.float64)
        vh = v[:, h // group, :].astype(np.float64)
        p = softmax(kh @ q[h] / np.sqrt(hd))
        o[h] = p @ vh
    return o


# ----------------------------------------------------------------------------
# Model
# ----------------------------------------------------------------------------

@dataclasses.dataclass
class OracleModel:
    """Weights widened to float64 plus the shape constants."""
    vocab: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    n_layers: int
    ffn_hidden: int
    max_loops: int
    rope_base: float
    norm_eps: float
    exit_rule: str
    threshold: float
    w: Dict[str, np.ndarray]

    @classmethod
    def from_config(cls, cfg, weights: Dict[str, np.ndarray]) -> "OracleModel":
        """cfg: any object with the ModelConfig attribute names."""
        w = {k: np.asarray(v, dtype=np.float64) for k, v in weights.items()}
        return cls(vocab=cfg.vocab, d_model=cfg.d_model, n_heads=cfg.n_heads,
                   n_kv_heads=cfg.n_kv_heads, head_dim=cfg.head_dim, n_layers=cfg.n_layers,
                   ffn_hidden=cfg.ffn_hidden, max_loops=cfg.max_loops, rope_base=cfg.rope_base,
                   norm_eps=cfg.norm_eps, exit_rule=cfg.exit_rule, threshold=cfg.threshold, w=w)

    # -- time/step conditioning (Sec. 3.1, App. A) ----------------------------
    @property
    def conditioned(self) -> bool:
        return "mod_w" in self.w

    def phi(self, which: str, tau: float) -> np.ndarray:
        """Embedding of one scalar: Fourier features, then a two-layer SiLU MLP."""
        f = fourier_features(tau)
        hdn = silu(self.w[f"cond_{which}_w1"] @ f + self.w[f"cond_{which}_b1"])
        return self.w[f"cond_{which}_w2"] @ hdn + self.w[f"cond_{which}_b2"]

    def conditioning(self, m: int, i: int) -> np.ndarray:
        """c = phi_t(c_{i-1}) + phi_Delta(Delta_i) for a token of depth m at loop i."""
        t, dt = trajectory(m, i)
        return self.phi("t", t) + self.phi("dt", dt)

    def modulation(self, j: int, m: int, i: int):
        """(alpha_msa, alpha_mlp, gamma_msa, gamma_mlp) of layer j, each [d]."""
        key = (j, m, i)
        cache = self.__dict__.setdefault("_mod_cache", {})
        if key not in cache:
            v = self.w["mod_w"][j] @ silu(self.conditioning(m, i)) + self.w["mod_b"][j]
            d = self.d_model
            cache[key] = (v[:d], v[d:2 * d], v[2 * d:3 * d], v[3 * d:])
        return cache[key]

    def mods(self, j: int, m, i: int):
        """Per-row modulation for rows of depths m at loop i (None without conditioning).

        Rows with m < i are not run at loop i; they get the vectors of depth i so that
        vectorised formulations stay finite (their results are discarded).
        """
        if not self.conditioned:
            return None
        m = np.atleast_1d(np.asarray(m))
        parts = [self.modulation(j, max(int(mm), i), i) for mm in m]
        return tuple(np.stack([p[q] for p in parts]) for q in range(4))

    # -- pieces of one layer of the shared block --------------------------------
    def qkv(self, j: int, h: np.ndarray, mod=None):
        """Eq. 9: q, k, v of layer j from the incoming states h [..., d]."""
        a = rms_norm(h, self.w["attn_norm"][j], self.norm_eps)
        if mod is not None:
            a = a * (1.0 + mod[2].reshape(a.shape))
        q = a @ self.w["wq"][j].T
        k = a @ self.w["wk"][j].T
        v = a @ self.w["wv"][j].T
        lead = h.shape[:-1]
        return (q.reshape(*lead, self.n_heads, self.head_dim),
                k.reshape(*lead, self.n_kv_heads, self.head_dim),
                v.reshape(*lead, self.n_kv_heads, self.head_dim))

    def attn_out(self, j: int, o: np.ndarray, mod=None) -> np.ndarray:
        lead = o.shape[:-2]
        y = o.reshape(*lead, self.n_heads * self.head_dim) @ self.w["wo"][j].T
        return y if mod is None else mod[0].reshape(y.shape) * y

    def mlp(self, j: int, h: np.ndarray, mod=None) -> np.ndarray:
        b = rms_norm(h, self.w["mlp_norm"][j], self.norm_eps)
        if mod is not None:
            b = b * (1.0 + mod[3].reshape(b.shape))
        g = b @ self.w["w_gate"][j].T
        u = b @ self.w["w_up"][j].T
        y = (silu(g) * u) @ self.w["w_down"][j].T
        return y if mod is None else mod[1].reshape(y.shape) * y

    def logits(self, h: np.ndarray) -> np.ndarray:
        """Final normalisation and tied LM head on h^(m)."""
        return rms_norm(h, self.w["final_norm"], self.norm_eps) @ self.w["embedding"].T


# ----------------------------------------------------------------------------
# Router (Sec. 3.2, Eq. 2-5)
# ----------------------------------------------------------------------------

def router_logits(model: OracleModel, tokens) -> np.ndarray:
    """z = W_r RMSNorm(h^(0)) + b_r with h^(0) = E[x]; returns [n, M] float64.

    With the two-layer MLP router of Sec. 3.2 (weights router_w1 [H_r, d], router_b1 [H_r]):
    z = W_r GELU(W_1 RMSNorm(h^(0)) + b_1) + b_r, router_w then [M, H_r].
    """
    h0 = model.w["embedding"][np.asarray(tokens, dtype=np.int64)]
    x = rms_norm(h0, None, model.norm_eps)
    if "router_w1" in model.w:
        x = gelu(x @ model.w["router_w1"].T + model.w["router_b1"])
    return x @ model.w["router_w"].T + model.w["router_b"]


def loop_counts(model: OracleModel, z: np.ndarray) -> Tuple[np.ndarray, np.ndarray]:
    """Loop count m in 1..M and decision margin for each row of router logits z.

    The decision is taken on z rounded to float32 (see the module docstring).
    """
    z32 = np.asarray(z, dtype=np.float64).astype(np.float32).astype(np.float64)
    z32 = np.atleast_2d(z32)
    n, M = z32.shape
    m = np.empty(n, dtype=np.int32)
    margin = np.empty(n, dtype=np.float64)
    for t in range(n):
        if model.exit_rule == "argmax":
            top = int(np.argmax(z32[t]))              # first maximum: ties go to the smaller depth
            rest = np.delete(z32[t], top)
            m[t] = top + 1
            margin[t] = z32[t, top] - (rest.max() if rest.size else np.inf)
        elif model.exit_rule == "survival":
            pi = softmax(z32[t])                        # Eq. 2
            p = np.array([pi[i:].sum() for i in range(M)] + [0.0])   # Eq. 3, p^(M+1) = 0
            active = [i + 1 for i in range(M) if p[i] > model.threshold]   # Eq. 4
            m[t] = max(active) if active else 1         # Eq. 5 (p^(1) = 1 keeps A_1 full)
            mi = m[t]
            margin[t] = min(p[mi - 1] - model.threshold, model.threshold - p[mi])
        else:
            raise ValueError(model.exit_rule)
    return m, margin


def depth_table(model: OracleModel, chunk: int = 4096) -> Tuple[np.ndarray, np.ndarray]:
    """Loop count and margin of every token id (the router reads only E[x])."""
    ms, gs = [], []
    for s in range(0, model.vocab, chunk):
        m, g = loop_counts(model, router_logits(model, np.arange(s, min(model.vocab, s + chunk))))
        ms.append(m)
        gs.append(g)
    return np.concatenate(ms), np.concatenate(gs)


# ----------------------------------------------------------------------------
# Recursion-wise KV cache (Sec. 3.3, Eq. 8 and 11)
# ----------------------------------------------------------------------------

class RecursionCache:
    """Cache of one (sequence, loop i, layer j): original positions, K and V rows."""

    def __init__(self, n_kv_heads: int, head_dim: int, dtype=np.float64, capacity: int = 16):
        self.n = 0
        self.pos = np.zeros(capacity, dtype=np.int64)
        self.k = np.zeros((capacity, n_kv_heads, head_dim), dtype=dtype)
        self.v = np.zeros((capacity, n_kv_heads, head_dim), dtype=dtype)

    def _grow(self, need: int):
        cap = self.pos.shape[0]
        if need <= cap:
            return
        new = max(need, 2 * cap)
        self.pos = np.resize(self.pos, new)
        self.k = np.concatenate([self.k, np.zeros((new - cap,) + self.k.shape[1:], self.k.dtype)])
        self.v = np.concatenate([self.v, np.zeros((new - cap,) + self.v.shape[1:], self.v.dtype)])

    def append(self, pos: int, k: np.ndarray, v: np.ndarray):
        """Eq. 11: write (k, v) of the token at position pos."""
        self._grow(self.n + 1)
        self.pos[self.n] = pos
        self.k[self.n] = k
        self.v[self.n] = v
        self.n += 1

    def extend(self, pos: np.ndarray, k: np.ndarray, v: np.ndarray):
        c = len(pos)
        self._grow(self.n + c)
        self.pos[self.n:self.n + c] = pos
        self.k[self.n:self.n + c] = k
        self.v[self.n:self.n + c] = v
        self.n += c

    def view(self):
        return self.pos[:self.n], self.k[:self.n], self.v[:self.n]


class OracleSequence:
    """All M x J caches of one sequence plus its token count."""

    def __init__(self, model: OracleModel, cache_dtype=np.float64):
        self.n_tokens = 0
        self.caches: List[List[RecursionCache]] = [
            [RecursionCache(model.n_kv_heads, model.head_dim, cache_dtype) for _ in range(model.n_layers)]
            for _ in range(model.max_loops)]

    def cache_len(self, i: int) -> int:
        """Length of the loop-i caches (1-based i); all J layers share it."""
        return self.caches[i - 1][0].n


# ----------------------------------------------------------------------------
# Decode (Eq. 9-11 for one token)
# ----------------------------------------------------------------------------

def decode_token(model: OracleModel, seq: OracleSequence, token: int,
                 forced: Optional[int] = None):
    """Process one token of one sequence; returns (logits [V], m, margin).

    ``forced`` (1..M) replaces the router's loop count (fixed-depth runs).
    """
    pos = seq.n_tokens
    z = router_logits(model, [token])
    m_arr, margin = loop_counts(model, z)
    m = int(m_arr[0]) if forced is None or forced < 1 else int(forced)
    h = model.w["embedding"][token].astype(np.float64)            # h^(0)
    for i in range(1, m + 1):                                      # loops 1..m (early exit after m)
        for j in range(model.n_layers):
            mod = model.modulation(j, m, i) if model.conditioned else None
            q, k, v = model.qkv(j, h, mod)                         # Eq. 9
            q = rope(q, pos, model.rope_base)
            k = rope(k, pos, model.rope_base)
            cache = seq.caches[i - 1][j]
            cache.append(pos, k, v)                                # Eq. 11
            _, kc, vc = cache.view()
            o = attention(q, kc, vc)                               # Eq. 10 (cache i holds only valid entries)
            h = h + model.attn_out(j, o, mod)
            h = h + model.mlp(j, h, mod)
    seq.n_tokens += 1
    return model.logits(h), m, float(margin[0])


def decode_step(model: OracleModel, seqs: Sequence[OracleSequence], tokens: Sequence[int],
                forced: Optional[Sequence[int]] = None):
    """A decode step over a batch of independent sequences (one token each)."""
    outs = [decode_token(model, s, int(t), None if forced is None else int(forced[b]))
            for b, (s, t) in enumerate(zip(seqs, tokens))]
    logits = np.stack([o[0] for o in outs])
    m = np.array([o[1] for o in outs], dtype=np.int32)
    margin = np.array([o[2] for o in outs], dtype=np.float64)
    return logits, m, margin


def prefill_sequential(model: OracleModel, seq: OracleSequence, tokens: Sequence[int],
                       forced: Optional[Sequence[int]] = None):
    """Prompt processed token by token with decode_token; returns (last logits, m [T])."""
    ms = []
    logits = None
    for t, x in enumerate(tokens):
        logits, m, _ = decode_token(model, seq, int(x), None if forced is None else int(forced[t]))
        ms.append(m)
    return logits, np.array(ms, dtype=np.int32)


# ----------------------------------------------------------------------------
# Batched prefill with gather-scatter (Eq. 6-7, App. B)
# ----------------------------------------------------------------------------

def _causal_attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, allowed: np.ndarray) -> np.ndarray:
    """q [T, Hq, hd], k/v [S, Hkv, hd], allowed [T, S] bool -> o [T, Hq, hd]."""
    T, hq, hd = q.shape
    group = hq // k.shape[1]
    o = np.empty_like(q)
    for h in range(hq):
        s = q[:, h, :] @ k[:, h // group, :].T / np.sqrt(hd)
        s = np.where(allowed, s, -np.inf)
        o[:, h, :] = softmax(s, axis=-1) @ v[:, h // group, :]
    return o


def prefill_gathered(model: OracleModel, seq: OracleSequence, tokens: Sequence[int],
                     forced: Optional[Sequence[int]] = None, row_block: int = 1024):
    """Whole prompt on an empty sequence, loop by loop on the gathered rows.

    Loop i gathers A_i (sorted, Eq. 6), runs the J layers on the gathered
    rows with a causal mask among them, writes each layer's k, v into cache
    (i, j) at the original positions rho^(i) = sort(A_i), and scatters the
    rows back (Eq. 7). Returns (logits of the last prompt token, m [T]).
    """
    if seq.n_tokens != 0:
        raise ValueError("prefill_gathered expects an empty sequence")
    tokens = np.asarray(tokens, dtype=np.int64)
    T = tokens.size
    m, _ = loop_counts(model, router_logits(model, tokens))
    if forced is not None:
        f = np.asarray(forced)
        m = np.where(f >= 1, f, m).astype(np.int32)
    H = model.w["embedding"][tokens].astype(np.float64)
    for i in range(1, model.max_loops + 1):
        rho = np.nonzero(m >= i)[0]                                  # sorted A_i
        if rho.size == 0:
            break
        X = H[rho]                                                   # Eq. 6
        for j in range(model.n_layers):
            mod = model.mods(j, m[rho], i)
            q, k, v = model.qkv(j, X, mod)
            q = rope(q, rho[:, None], model.rope_base)
            k = rope(k, rho[:, None], model.rope_base)
            seq.caches[i - 1][j].extend(rho, k, v)                   # written at rho^(i)
            o = np.empty_like(q)
            for r0 in range(0, rho.size, row_block):                 # causal among gathered rows
                r1 = min(rho.size, r0 + row_block)
                allowed = rho[None, :] <= rho[r0:r1, None]
                o[r0:r1] = _causal_attention(q[r0:r1], k[:r1], v[:r1], allowed[:, :r1])
            X = X + model.attn_out(j, o, mod)
            X = X + model.mlp(j, X, mod)
        H[rho] = X                                                   # Eq. 7 scatter
    seq.n_tokens = T
    return model.logits(H[-1]), m


# ----------------------------------------------------------------------------
# Brute force without gather (Eq. 7 and Eq. 10 with the mask mu)
# ----------------------------------------------------------------------------

def forward_masked(model: OracleModel, tokens: Sequence[int], m: Sequence[int]) -> np.ndarray:
    """Logits at every position of a sequence with given loop counts m.

    Every row is computed at every loop; attention at loop i uses the mask
    [t' <= t] * [m_{t'} >= i]; after each layer only rows with m_t >= i take
    the new state (Eq. 7). For small inputs only.
    """
    tokens = np.asarray(tokens, dtype=np.int64)
    m = np.asarray(m)
    T = tokens.size
    pos = np.arange(T)
    H = model.w["embedding"][tokens].astype(np.float64)
    for i in range(1, model.max_loops + 1):
        mu = m >= i                                                  # validity indicator mu^(i)
        if not mu.any():
            break
        allowed = (pos[None, :] <= pos[:, None]) & mu[None, :]
        for j in range(model.n_layers):
            mod = model.mods(j, m, i)
            q, k, v = model.qkv(j, H, mod)
            q = rope(q, pos[:, None], model.rope_base)
            k = rope(k, pos[:, None], model.rope_base)
            rows = mu.copy()
            safe = allowed.copy()
            safe[~rows] = False
            safe[~rows, 0] = True                                    # rows that are discarded anyway
            o = _causal_attention(q, k, v, safe)
            Hn = H + model.attn_out(j, o, mod)
            Hn = Hn + model.mlp(j, Hn, mod)
            H = np.where(rows[:, None], Hn, H)
    return model.logits(H)


# ----------------------------------------------------------------------------
# Cache snapshots
# ----------------------------------------------------------------------------

def load_snapshot(model: OracleModel, snapshot: dict, cache_dtype=np.float64) -> OracleSequence:
    """A sequence whose caches hold a given snapshot.

    snapshot: dict(positions: list over loops of [n_i], k, v: list over loops
    of [n_i, J, Hkv, hd]); positions of loop 1 must be 0..L-1.
    """
    seq = OracleSequence(model, cache_dtype)
    pos = snapshot["positions"]
    L = len(pos[0])
    if not np.array_equal(pos[0], np.arange(L)):
        raise ValueError("loop-1 cache must hold every position")
    for i in range(model.max_loops):
        for j in range(model.n_layers):
            seq.caches[i][j].extend(np.asarray(pos[i]), snapshot["k"][i][:, j], snapshot["v"][i][:, j])
    seq.n_tokens = L
    return seq
