"""Seeded synthetic inputs for the T-LoopFormer decode step.

This module serves both the CUDA library and the oracle. It holds the five
workload configurations, the weight generator, the router-bias calibration,
the prompt / decode-token generators and synthetic recursion-wise cache
snapshots. It holds none of the method's arithmetic: it never evaluates the
router, a norm, a projection or attention on a token.

Everything here stands in for the paper's FineWeb-Edu workload and trained
checkpoints (Sec. 4), neither of which is available: weights are N(0, 0.02),
prompts and decode tokens are uniform random ids, and the router bias is
chosen so that the loop-count distribution over the vocabulary is long-tailed
like the one reported for FineWeb-Edu (Fig. 1b, mean 3.69).

Random streams: every tensor is drawn from numpy's PCG64 generator seeded with
``SeedSequence([seed, stream_id])`` so that any tensor can be regenerated on
its own. Matrices are stored row-major with the output dimension first
(``y = W @ x``).
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, List, Optional, Sequence, Tuple

import numpy as np

__all__ = [
    "ModelConfig", "WorkloadConfig", "CONFIGS", "get_config",
    "make_weights", "round_to_bf16", "bf16_bits", "calibrate_router_bias",
    "make_prompts", "make_decode_tokens", "make_cache_snapshot",
    "sample_depths", "tiny_config",
]


@dataclasses.dataclass(frozen=True)
class ModelConfig:
    """Shapes and numerics of one looped LM (shared block of ``n_layers``)."""
    vocab: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    n_layers: int
    ffn_hidden: int
    max_loops: int
    dtype: str = "bf16"            # "f32" or "bf16": storage of matrices, activations and KV
    rope_base: float = 10000.0
    norm_eps: float = 1e-5
    exit_rule: str = "argmax"      # "argmax" or "survival" (Eq. 3-5)
    threshold: float = 0.5         # survival threshold (Eq. 4)
    depth_probs: Optional[Tuple[float, ...]] = None  # target P(m = 1..M); None = no bias
    weight_seed: int = 0
    init_std: float = 0.02
    conditioning: bool = False     # time/step AdaLN conditioning (Sec. 3.1, App. A)
    router_hidden: int = 0         # > 0: the two-layer MLP router of Sec. 3.2 with this hidden width

    @property
    def q_dim(self) -> int:
        return self.n_heads * self.head_dim

    @property
    def kv_dim(self) -> int:
        return self.n_kv_heads * self.head_dim

    def layer_params(self) -> int:
        d, f = self.d_model, self.ffn_hidden
        return d * (self.q_dim + 2 * self.kv_dim) + self.q_dim * d + 3 * d * f


@dataclasses.dataclass(frozen=True)
class WorkloadConfig:
    """A model plus the batch / prompt / decode shape it is run on."""
    name: str
    model: ModelConfig
    batch: int
    prompt_len: Tuple[int, int]    # (lo, hi) inclusive; lo == hi for fixed length
    decode_steps: int
    greedy: bool                   # greedy decode (teacher-forced from the oracle) vs random tokens
    prompt_seed: int = 1
    token_seed: int = 2
    forced_loops: Optional[int] = None  # fixed-depth baseline (every token runs this many loops)
    batch_sweep: Tuple[int, ...] = ()

    def with_batch(self, b: int) -> "WorkloadConfig":
        return dataclasses.replace(self, batch=b)


# Target depth distributions. C3's is given; C2 and C4 only give a mean and a
# maximum, so a long-tailed distribution with that mean is chosen.
_P_C2 = (0.10, 0.15, 0.40, 0.35)                                  # mean 3.00, M = 4
_P_C3 = (0.10, 0.12, 0.22, 0.24, 0.14, 0.09, 0.06, 0.03)          # mean 3.86, M = 8
_P_C4 = (0.10, 0.12, 0.22, 0.24, 0.18, 0.14)                      # mean 3.70, M = 6

_M1 = ModelConfig(vocab=256, d_model=64, n_heads=4, n_kv_heads=4, head_dim=16, n_layers=1,
                  ffn_hidden=176, max_loops=4, dtype="f32", depth_probs=None)
_M2 = ModelConfig(vocab=32000, d_model=512, n_heads=8, n_kv_heads=8, head_dim=64, n_layers=2,
                  ffn_hidden=1376, max_loops=4, dtype="bf16", depth_probs=_P_C2)
_M3 = ModelConfig(vocab=50304, d_model=1024, n_heads=16, n_kv_heads=16, head_dim=64, n_layers=4,
                  ffn_hidden=2752, max_loops=8, dtype="bf16", depth_probs=_P_C3)
_M4 = ModelConfig(vocab=32000, d_model=2048, n_heads=16, n_kv_heads=8, head_dim=128, n_layers=2,
                  ffn_hidden=5504, max_loops=6, dtype="bf16", depth_probs=_P_C4)

CONFIGS: Dict[str, WorkloadConfig] = {
    # Tiny fp32 LM: batch 1, 32-token prompt, greedy decode of 16 tokens.
    "c1": WorkloadConfig("c1", _M1, batch=1, prompt_len=(32, 32), decode_steps=16, greedy=True),
    # Small bf16 LM: batch 8, 512-token prompts, greedy decode of 128 tokens.
    "c2": WorkloadConfig("c2", _M2, batch=8, prompt_len=(512, 512), decode_steps=128, greedy=True),
    # Mid-size bf16 LM: batch 64, 2048-token prompts, 256 decode steps.
    "c3": WorkloadConfig("c3", _M3, batch=64, prompt_len=(2048, 2048), decode_steps=256, greedy=False),
    # Long-context GQA stress: batch 16, 32768-token prompts, 64 decode steps.
    "c4": WorkloadConfig("c4", _M4, batch=16, prompt_len=(32768, 32768), decode_steps=64, greedy=False),
    # Ragged serving sweep on the C3 model; prompt lengths uniform in [128, 8192].
    "c5": WorkloadConfig("c5", _M3, batch=32, prompt_len=(128, 8192), decode_steps=128, greedy=False,
                         prompt_seed=3, batch_sweep=(1, 8, 32, 128, 256)),
}
CONFIGS["c5f"] = dataclasses.replace(CONFIGS["c5"], name="c5f", forced_loops=8)
# The C2 and C3 workloads on models with the paper's time/step conditioning (Sec. 3.1, App. A).
CONFIGS["c2c"] = dataclasses.replace(CONFIGS["c2"], name="c2c", model=dataclasses.replace(_M2, conditioning=True))
CONFIGS["c3c"] = dataclasses.replace(CONFIGS["c3"], name="c3c", model=dataclasses.replace(_M3, conditioning=True))


def get_config(name: str) -> WorkloadConfig:
    return CONFIGS[name]


def tiny_config(**kw) -> ModelConfig:
    """A very small model for exhaustive oracle tests."""
    base = dict(vocab=37, d_model=16, n_heads=4, n_kv_heads=2, head_dim=4, n_layers=2,
                ffn_hidden=24, max_loops=3, dtype="f32", depth_probs=None)
    base.update(kw)
    return ModelConfig(**base)


# ----------------------------------------------------------------------------
# bf16 storage helpers (input quantisation, not part of the method)
# ----------------------------------------------------------------------------

def round_to_bf16(x: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bfloat16 (ties to even); returns float32."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    r = ((u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000).astype(np.uint32)
    return r.view(np.float32)


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """uint16 bit patterns of float32 values that are already bf16-exact."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32)
    if np.any(u & 0xFFFF):
        raise ValueError("values are not bf16-exact; call round_to_bf16 first")
    return (u >> 16).astype(np.uint16)


def _rng(seed: int, stream: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, stream])))


def _normal(seed: int, stream: int, shape, std: float, dtype: str) -> np.ndarray:
    a = _rng(seed, stream).standard_normal(size=shape, dtype=np.float32)
    a *= np.float32(std)
    return round_to_bf16(a) if dtype == "bf16" else a


# ----------------------------------------------------------------------------
# Weights
# ----------------------------------------------------------------------------

# Stream ids: 0 embedding, 1 router weight, 2 router-calibration draws,
# 100 + 10 * layer + k for the k-th matrix of a layer.
_LAYER_MATS = ("wq", "wk", "wv", "wo", "w_gate", "w_up", "w_down")


def calibrate_router_bias(router_w: np.ndarray, depth_probs: Sequence[float], init_std: float,
                          norm_eps: float, seed: int, n_samples: int = 200_000,
                          iters: int = 300) -> np.ndarray:
    """Pick a router bias b so that argmax(u + b) has the target distribution.

    The router reads RMSNorm(E[x]) for an embedding row E[x] with i.i.d.
    N(0, init_std^2) entries, so over the vocabulary the router's linear part
    u = W_r x is close to N(0, c W_r W_r^T) with c = s / (s + eps), s = init_std^2.
    The bias is fitted against draws from that Gaussian by the multiplicative
    update b_l += 0.5 (log P*_l - log P_hat_l); no token is ever routed here.
    The distribution realised over the vocabulary is reported by the tests.
    """
    p = np.asarray(depth_probs, dtype=np.float64)
    if p.ndim != 1 or p.size != router_w.shape[0] or np.any(p <= 0) or abs(p.sum() - 1) > 1e-9:
        raise ValueError("depth_probs must be a positive distribution over the loop counts")
    w = router_w.astype(np.float64)
    s = init_std ** 2
    cov = (s / (s + norm_eps)) * (w @ w.T)
    chol = np.linalg.cholesky(cov + 1e-12 * np.eye(cov.shape[0]))
    u = _rng(seed, 2).standard_normal((n_samples, p.size)) @ chol.T
    b = np.log(p)
    for _ in range(iters):
        freq = np.bincount(np.argmax(u + b, axis=1), minlength=p.size) / n_samples
        step = np.log(p) - np.log(np.maximum(freq, 1.0 / n_samples))
        if np.max(np.abs(step)) < 1e-3:
            break
        b += 0.5 * step
        b -= b.mean()
    return b.astype(np.float32)


def make_weights(m: ModelConfig) -> Dict[str, np.ndarray]:
    """All parameters as float32 arrays (bf16-exact values for bf16 models).

    Shapes: embedding [V, d] (tied LM head); router_w [M, d]; router_b [M];
    per-layer stacks wq [J, Hq*hd, d], wk/wv [J, Hkv*hd, d], wo [J, d, Hq*hd],
    w_gate/w_up [J, ff, d], w_down [J, d, ff]; norm gains attn_norm/mlp_norm
    [J, d] and final_norm [d] (all ones: the paper's RMSNorm has no learned
    gain, the gains are kept so a trained checkpoint could be loaded).
    """
    seed, std, dt = m.weight_seed, m.init_std, m.dtype
    d, J = m.d_model, m.n_layers
    w: Dict[str, np.ndarray] = {}
    w["embedding"] = _normal(seed, 0, (m.vocab, d), std, dt)
    if m.router_hidden > 0:
        # two-layer MLP router: hidden pre-activations of order one, logits spread over a few units
        # so that the depth decisions are well separated; no bias fit (the distribution is whatever
        # these seeded weights give)
        w["router_w1"] = _normal(seed, 2, (m.router_hidden, d), 1.0 / d ** 0.5, dt)
        w["router_b1"] = _normal(seed, 3, (m.router_hidden,), 0.5, "f32")
        w["router_w"] = _normal(seed, 1, (m.max_loops, m.router_hidden), 3.0 / m.router_hidden ** 0.5, dt)
        w["router_b"] = np.zeros(m.max_loops, dtype=np.float32)
    else:
        w["router_w"] = _normal(seed, 1, (m.max_loops, d), std, dt)
        if m.depth_probs is None:
            w["router_b"] = np.zeros(m.max_loops, dtype=np.float32)
        else:
            w["router_b"] = calibrate_router_bias(w["router_w"], m.depth_probs, std, m.norm_eps, seed)
    shapes = {
        "wq": (m.q_dim, d), "wk": (m.kv_dim, d), "wv": (m.kv_dim, d), "wo": (d, m.q_dim),
        "w_gate": (m.ffn_hidden, d), "w_up": (m.ffn_hidden, d), "w_down": (d, m.ffn_hidden),
    }
    for k, name in enumerate(_LAYER_MATS):
        w[name] = np.stack([_normal(seed, 100 + 10 * j + k, shapes[name], std, dt) for j in range(J)])
    w["attn_norm"] = np.ones((J, d), dtype=np.float32)
    w["mlp_norm"] = np.ones((J, d), dtype=np.float32)
    w["final_norm"] = np.ones(d, dtype=np.float32)
    if m.conditioning:
        w.update(make_conditioning_weights(m))
    return w


COND_FOURIER = 256  # width of the sinusoidal features of the conditioning scalars (App. A)


def make_conditioning_weights(m: ModelConfig) -> Dict[str, np.ndarray]:
    """Float32 weights of the time/step conditioning (App. A), for each scalar t and dt:
    cond_{t,dt}_w1 [d, 256], _b1 [d], _w2 [d, d], _b2 [d]; the modulators mod_w [J, 4d, d],
    mod_b [J, 4d] with outputs ordered (alpha_msa, alpha_mlp, gamma_msa, gamma_mlp).

    The paper zero-initialises the modulator for training; these stand in for trained
    weights instead: the gate biases are one and the scale biases zero, and the weights
    are scaled so that the embeddings are of order one and alpha and gamma move by
    about 0.2 with (t, dt), so that every (depth, loop) pair has its own modulation.
    """
    seed, d, J = m.weight_seed, m.d_model, m.n_layers
    w: Dict[str, np.ndarray] = {}
    for k, which in enumerate(("t", "dt")):
        w[f"cond_{which}_w1"] = _normal(seed, 500 + 10 * k, (d, COND_FOURIER), (2.0 / COND_FOURIER) ** 0.5, "f32")
        w[f"cond_{which}_b1"] = np.zeros(d, dtype=np.float32)
        w[f"cond_{which}_w2"] = _normal(seed, 501 + 10 * k, (d, d), 1.7 / d ** 0.5, "f32")
        w[f"cond_{which}_b2"] = np.zeros(d, dtype=np.float32)
    w["mod_w"] = np.stack([_normal(seed, 600 + j, (4 * d, d), 0.28 / d ** 0.5, "f32") for j in range(J)])
    b = np.zeros(4 * d, dtype=np.float32)
    b[:2 * d] = 1.0
    w["mod_b"] = np.tile(b, (J, 1))
    return w


# ----------------------------------------------------------------------------
# Prompts, decode tokens, depth samples, cache snapshots
# ----------------------------------------------------------------------------

def make_prompts(wl: WorkloadConfig, batch: Optional[int] = None) -> List[np.ndarray]:
    """Uniform random token ids; lengths uniform in prompt_len (seeded)."""
    b = wl.batch if batch is None else batch
    rng = _rng(wl.prompt_seed, 0)
    lo, hi = wl.prompt_len
    lens = rng.integers(lo, hi + 1, size=b) if hi > lo else np.full(b, lo)
    rng_t = _rng(wl.prompt_seed, 1)
    return [rng_t.integers(0, wl.model.vocab, size=int(n), dtype=np.int64).astype(np.int32) for n in lens]


def make_decode_tokens(wl: WorkloadConfig, steps: Optional[int] = None,
                       batch: Optional[int] = None) -> np.ndarray:
    """[steps, batch] uniform random decode tokens (for the throughput configs)."""
    s = wl.decode_steps if steps is None else steps
    b = wl.batch if batch is None else batch
    return _rng(wl.token_seed, 0).integers(0, wl.model.vocab, size=(s, b), dtype=np.int64).astype(np.int32)


def sample_depths(probs: Optional[Sequence[float]], max_loops: int, n: int, seed: int) -> np.ndarray:
    """n loop counts in 1..M drawn from probs (uniform when probs is None)."""
    p = np.full(max_loops, 1.0 / max_loops) if probs is None else np.asarray(probs, dtype=np.float64)
    return (_rng(seed, 7).choice(max_loops, size=n, p=p / p.sum()) + 1).astype(np.int32)


def make_cache_snapshot(m: ModelConfig, length: int, seed: int,
                        depths: Optional[np.ndarray] = None) -> dict:
    """A synthetic recursion-wise KV cache for one sequence of ``length`` tokens.

    Past tokens get loop counts from the model's target distribution; cache r
    holds the positions t with depth_t >= r in increasing order (so the caches
    nest like the paper's active sets, Eq. 4-5). K and V entries are multiples
    of 1/64 in [-2, 2), exactly representable in bf16 and fp32.

    Returns dict(depths [L], positions: list over r of int32 [n_r],
    k, v: list over r of float32 [n_r, J, Hkv, hd]).
    """
    if depths is None:
        depths = sample_depths(m.depth_probs, m.max_loops, length, seed)
    rng = _rng(seed, 8)
    pos, ks, vs = [], [], []
    for r in range(1, m.max_loops + 1):
        p = np.nonzero(depths >= r)[0].astype(np.int32)
        shape = (p.size, m.n_layers, m.n_kv_heads, m.head_dim)
        ks.append(rng.integers(-128, 128, size=shape, dtype=np.int16).astype(np.float32) / 64.0)
        vs.append(rng.integers(-128, 128, size=shape, dtype=np.int16).astype(np.float32) / 64.0)
        pos.append(p)
    return {"depths": np.asarray(depths, dtype=np.int32), "positions": pos, "k": ks, "v": vs}


def make_cache_positions(m: ModelConfig, length: int, seed: int,
                         depths: Optional[np.ndarray] = None) -> dict:
    """Only the positions of a cache snapshot (values to be filled on the device)."""
    if depths is None:
        depths = sample_depths(m.depth_probs, m.max_loops, length, seed)
    return {"depths": np.asarray(depths, dtype=np.int32),
            "positions": [np.nonzero(depths >= r)[0].astype(np.int32) for r in range(1, m.max_loops + 1)]}


def make_attn_problem(n: int, lens, hq: int, hkv: int, hd: int, n_layers: int = 2, layer: int = 1,
                      dtype: str = "bf16", seed: int = 0, spare_pages: int = 3, page_size: int = 64) -> dict:
    """Inputs of the kernel-level attention operation on paged caches.

    q [n, hq, hd] float32 (already rotated); pool [n_pages, J, 2, hkv, page, hd]
    with values that are multiples of 1/64 in [-2, 2) (exact in bf16 and fp32);
    page_table [n, max_pages] giving every row distinct, randomly placed pages.
    """
    rng = _rng(seed, 9)
    lens = np.asarray(lens, dtype=np.int32)
    if lens.size != n:
        raise ValueError("one length per row")
    need = [(int(L) + page_size - 1) // page_size for L in lens]
    max_pages = max(need)
    n_pages = sum(need) + spare_pages
    perm = rng.permutation(n_pages)
    pt = np.full((n, max_pages), -1, dtype=np.int32)
    o = 0
    for b in range(n):
        pt[b, :need[b]] = perm[o:o + need[b]]
        o += need[b]
    pool = rng.integers(-128, 128, size=(n_pages, n_layers, 2, hkv, page_size, hd), dtype=np.int16)
    pool = pool.astype(np.float32) / 64.0
    q = rng.standard_normal((n, hq, hd), dtype=np.float32)
    return dict(n=n, lens=lens, hq=hq, hkv=hkv, hd=hd, n_layers=n_layers, layer=layer, dtype=dtype,
                q=q, pool=pool, page_table=pt, max_pages=max_pages, n_pages=n_pages, page_size=page_size)


def expected_mean_depth(probs: Sequence[float]) -> float:
    return float(sum((i + 1) * p for i, p in enumerate(probs)))


def describe(wl: WorkloadConfig) -> dict:
    m = wl.model
    return {"workload": wl.name, "vocab": m.vocab, "d_model": m.d_model, "n_heads": m.n_heads,
            "n_kv_heads": m.n_kv_heads, "head_dim": m.head_dim, "n_layers": m.n_layers,
            "ffn_hidden": m.ffn_hidden, "max_loops": m.max_loops, "dtype": m.dtype,
            "batch": wl.batch, "prompt_len": list(wl.prompt_len), "decode_steps": wl.decode_steps,
            "forced_loops": wl.forced_loops}


if __name__ == "__main__":  # pragma: no cover
    for k, v in CONFIGS.items():
        print(k, describe(v), "params/layer", v.model.layer_params(),
              "mean depth target", None if v.model.depth_probs is None else expected_mean_depth(v.model.depth_probs))

