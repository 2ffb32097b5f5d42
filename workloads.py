"""Seeded synthetic inputs for one TAPS decoding round.

This module is shared by the tests, the benchmark and the oracle's callers. It
draws random numbers and lays them out; it holds none of the method's
arithmetic (no softmax, no top-K, no scoring, no selection, no attention).

The paper evaluates on public datasets with Qwen3-4B/8B and LLaMA targets and a
DFlash drafter (Sec. 5.1, Table 1). None of those weights or datasets is used
here: every input is drawn from a seeded generator with the shapes of those
workloads (vocab 151936, draft block 16, 36 layers, 32 query heads, 8 KV heads,
head dim 128, paged bf16 KV cache with 16-token pages).

Recipes (one per named workload):

* ``tiny``      B=1, L=8, V=32000, fp32 logits ~ N(0,1)*3 with 1-2 spike
                tokens per position raised by +10; K=4, budget 16; one layer
                with 8 q heads, 2 KV heads, D=64, context 512.
* ``qwen3_4b``  B=1, L=16, V=151936, bf16 logits x[v] = -1.1*ln(rank(v)) +
                Gumbel(0,1) with a seeded rank permutation per position; K=8,
                budget 64; 36 layers, 32/8 heads, D=128, context 2048.
* ``qwen3_8b``  as qwen3_4b but each position's logits divided by a
                temperature rising linearly 0.6 -> 1.4 over the block; budget
                64 (the sweep uses 32/64/128/256); context 4096.
* ``batched``   qwen3_8b logits per request, B=32, budget 64, context lengths
                uniform in [512, 8192].
* ``long``      B=8, K=16, budget 256, context 32768; every third position
                carries two tokens of probability ~0.45 each (bimodal top-2).

Target-model greedy tokens: for each request a continuation y_1..y_{L+1} is
drawn, y_d from the drafter's softmax at position d (Gumbel-max sampling), and
y_{L+1} uniformly. A tree node at depth k whose path spells y_1..y_k receives
target token y_{k+1}; the acceptance walk only ever visits such nodes, so every
node simply receives y_{depth+1} (``target_tokens_for_tree``).
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

SEED_BASE = 20260487
PAGE = 16


@dataclasses.dataclass(frozen=True)
class RoundConfig:
    name: str
    B: int
    L: int
    V: int
    K: int
    n_max: int
    logits_kind: str          # gauss_spike | zipf | zipf_temp | bimodal
    logits_dtype: str         # f32 | bf16
    layers: int
    Hq: int
    Hkv: int
    D: int
    ctx: int | tuple          # fixed context, or (lo, hi) uniform per request
    page: int = PAGE
    emb_dim: int = 16
    hidden: int = 32
    lambda1: float = 1.0
    lambda2: float = 0.1
    tau: float = 0.0
    config_id: int = 0

    def with_(self, **kw) -> "RoundConfig":
        return dataclasses.replace(self, **kw)


CONFIGS = {
    "tiny": RoundConfig("tiny", B=1, L=8, V=32000, K=4, n_max=16, logits_kind="gauss_spike",
                        logits_dtype="f32", layers=1, Hq=8, Hkv=2, D=64, ctx=512, config_id=0),
    "qwen3_4b": RoundConfig("qwen3_4b", B=1, L=16, V=151936, K=8, n_max=64, logits_kind="zipf",
                            logits_dtype="bf16", layers=36, Hq=32, Hkv=8, D=128, ctx=2048,
                            config_id=1),
    "qwen3_8b": RoundConfig("qwen3_8b", B=1, L=16, V=151936, K=8, n_max=64,
                            logits_kind="zipf_temp", logits_dtype="bf16", layers=36, Hq=32,
                            Hkv=8, D=128, ctx=4096, config_id=2),
    "batched": RoundConfig("batched", B=32, L=16, V=151936, K=8, n_max=64,
                           logits_kind="zipf_temp", logits_dtype="bf16", layers=36, Hq=32,
                           Hkv=8, D=128, ctx=(512, 8192), config_id=3),
    "long": RoundConfig("long", B=8, L=16, V=151936, K=16, n_max=256, logits_kind="bimodal",
                        logits_dtype="bf16", layers=36, Hq=32, Hkv=8, D=128, ctx=32768,
                        config_id=4),
    # LLaMA-3.1-8B-Instruct target: draft block 10, vocabulary 128256, 32 layers
    # of 32 query / 8 KV heads of dimension 128
    "llama31_8b": RoundConfig("llama31_8b", B=1, L=10, V=128256, K=8, n_max=64,
                              logits_kind="zipf_temp", logits_dtype="bf16", layers=32, Hq=32,
                              Hkv=8, D=128, ctx=4096, config_id=5),
}


def rng_for(cfg: RoundConfig, *stream) -> np.random.Generator:
    """Independent PCG64 stream for (config, stream tags...)."""
    return np.random.default_rng([SEED_BASE, cfg.config_id, *[int(s) for s in stream]])


# stream tags
_S_LOGITS, _S_SCORER, _S_CTX, _S_ROOT, _S_TARGET, _S_KV, _S_Q, _S_PAGES = range(1, 9)


def round_to_bf16(x: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bfloat16 (ties to even); returns float32.

    Works on the uint32 bit patterns in place: adding 0x7FFF plus the lowest
    kept bit cannot overflow 32 bits for any non-NaN value (the inputs here
    never hold NaN)."""
    bits = np.array(x, dtype=np.float32, copy=True).view(np.uint32)
    flat = bits.reshape(-1)
    step = 1 << 22
    for a in range(0, flat.size, step):
        c = flat[a:a + step]
        lsb = (c >> 16) & 1
        c += np.uint32(0x7FFF)
        c += lsb
        c &= np.uint32(0xFFFF0000)
    return bits.view(np.float32)


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """uint16 bit patterns of float32 values that are already bf16-representable."""
    return (np.ascontiguousarray(x, dtype=np.float32).view(np.uint32) >> 16).astype(np.uint16)


# ---------------------------------------------------------------------------
# drafter logits
# ---------------------------------------------------------------------------

def _logits_row(cfg: RoundConfig, rng: np.random.Generator, d: int) -> np.ndarray:
    V = cfg.V
    if cfg.logits_kind == "gauss_spike":
        x = rng.standard_normal(V).astype(np.float32) * 3.0
        n_spike = 1 + int(rng.integers(0, 2))
        spikes = rng.choice(V, size=n_spike, replace=False)
        x[spikes] += 10.0
        return x
    # Zipf-shaped logits over a seeded rank permutation, plus Gumbel noise
    rank = rng.permutation(V).astype(np.float64) + 1.0
    g = rng.gumbel(size=V)
    x = -1.1 * np.log(rank) + g
    if cfg.logits_kind in ("zipf_temp", "bimodal"):
        T = 0.6 + 0.8 * d / max(cfg.L - 1, 1)
        x = x / T
    if cfg.logits_kind == "bimodal" and (d + 1) % 3 == 0:
        top2 = rng.choice(V, size=2, replace=False)
        rest = np.ones(V, bool)
        rest[top2] = False
        m = x[rest].max()
        z_rest = m + math.log(np.exp(x[rest] - m).sum())
        x[top2] = z_rest + math.log(4.5)      # p ~ 0.45 each, 0.1 left for the rest
    return x.astype(np.float32)


def make_logits(cfg: RoundConfig, B: int | None = None) -> np.ndarray:
    """Drafter marginal logits [B, L, V] as float32 (bf16-representable if bf16)."""
    B = cfg.B if B is None else B
    out = np.empty((B, cfg.L, cfg.V), np.float32)
    for b in range(B):
        rng = rng_for(cfg, _S_LOGITS, b)
        for d in range(cfg.L):
            out[b, d] = _logits_row(cfg, rng, d)
    if cfg.logits_dtype == "bf16":
        out = round_to_bf16(out)
    return out


def make_root_tokens(cfg: RoundConfig, B: int | None = None) -> np.ndarray:
    B = cfg.B if B is None else B
    return rng_for(cfg, _S_ROOT).integers(0, cfg.V, size=B).astype(np.int32)


def make_ctx_lens(cfg: RoundConfig, B: int | None = None) -> np.ndarray:
    B = cfg.B if B is None else B
    if isinstance(cfg.ctx, tuple):
        lo, hi = cfg.ctx
        return rng_for(cfg, _S_CTX).integers(lo, hi + 1, size=B).astype(np.int32)
    return np.full(B, cfg.ctx, np.int32)


# ---------------------------------------------------------------------------
# scorer weights (random init; the paper's trained weights are not published)
# ---------------------------------------------------------------------------

def scorer_layout(V: int, max_depth: int, E: int, H: int) -> dict:
    """Offsets (in floats) of each tensor in the packed scorer weight buffer.

    Order: tok_emb[V][E], dep_emb[max_depth][E], W1[H][3E+2], b1[H], w2[H], w_lp.
    """
    F = 3 * E + 2
    off = {}
    o = 0
    for name, n in (("tok_emb", V * E), ("dep_emb", max_depth * E), ("W1", H * F),
                    ("b1", H), ("w2", H), ("w_lp", 1)):
        off[name] = (o, n)
        o += n
    off["total"] = o
    return off


def make_scorer_weights(cfg: RoundConfig, max_depth: int | None = None) -> dict:
    """Random-init weights of the edge scorer, as float32 arrays plus a packed buffer."""
    E, H = cfg.emb_dim, cfg.hidden
    max_depth = cfg.L + 1 if max_depth is None else max_depth
    F = 3 * E + 2
    rng = rng_for(cfg, _S_SCORER)
    w = {
        "tok_emb": (rng.standard_normal((cfg.V, E)) * 0.5).astype(np.float32),
        "dep_emb": (rng.standard_normal((max_depth, E)) * 0.5).astype(np.float32),
        "W1": (rng.standard_normal((H, F)) / math.sqrt(F)).astype(np.float32),
        "b1": (rng.standard_normal(H) * 0.1).astype(np.float32),
        "w2": (rng.standard_normal(H) * 0.5 / math.sqrt(H)).astype(np.float32),
        "w_lp": np.array([1.0], np.float32),
    }
    lay = scorer_layout(cfg.V, max_depth, E, H)
    packed = np.empty(lay["total"], np.float32)
    for name in ("tok_emb", "dep_emb", "W1", "b1", "w2", "w_lp"):
        o, n = lay[name]
        packed[o:o + n] = w[name].reshape(-1)
    w["packed"] = packed
    w["E"], w["H"], w["V"], w["max_depth"] = E, H, cfg.V, max_depth
    return w


# ---------------------------------------------------------------------------
# target-model greedy continuation (stand-in for the target model)
# ---------------------------------------------------------------------------

def make_target_sequence(cfg: RoundConfig, logits: np.ndarray) -> np.ndarray:
    """y[b, 0..L]: y[b, d] ~ softmax(logits[b, d]) for d < L, y[b, L] uniform.

    Sampling uses the Gumbel-max trick on the float64-widened logits.
    """
    B = logits.shape[0]
    y = np.empty((B, cfg.L + 1), np.int32)
    for b in range(B):
        rng = rng_for(cfg, _S_TARGET, b)
        for d in range(cfg.L):
            g = rng.gumbel(size=cfg.V)
            y[b, d] = int(np.argmax(logits[b, d].astype(np.float64) + g))
        y[b, cfg.L] = int(rng.integers(0, cfg.V))
    return y


def target_tokens_for_tree(y: np.ndarray, depth: np.ndarray, n_nodes: np.ndarray) -> np.ndarray:
    """target_tok[b, i] = y[b, depth[b, i]] for i < n_nodes[b], else -1 (pure indexing)."""
    B, N = depth.shape
    out = np.full((B, N), -1, np.int32)
    for b in range(B):
        n = int(n_nodes[b])
        out[b, :n] = y[b, depth[b, :n]]
    return out


# ---------------------------------------------------------------------------
# paged KV cache and tree queries
# ---------------------------------------------------------------------------

def pages_needed(ctx_lens: np.ndarray, n_max: int, page: int = PAGE) -> np.ndarray:
    return (ctx_lens.astype(np.int64) + n_max + page - 1) // page


def make_block_table(cfg: RoundConfig, ctx_lens: np.ndarray, n_max: int | None = None,
                     spare_pages: int = 3):
    """Seeded random physical placement of every request's logical pages.

    Returns (block_table [B, max_pages] int32 padded with -1, num_pages).
    """
    n_max = cfg.n_max if n_max is None else n_max
    need = pages_needed(ctx_lens, n_max, cfg.page)
    total = int(need.sum()) + spare_pages
    perm = rng_for(cfg, _S_PAGES).permutation(total).astype(np.int32)
    max_pages = int(need.max())
    bt = np.full((len(ctx_lens), max_pages), -1, np.int32)
    o = 0
    for b, n in enumerate(need):
        bt[b, :n] = perm[o:o + n]
        o += int(n)
    return bt, total


def make_kv_numpy(cfg: RoundConfig, num_pages: int, layer: int = 0):
    """K and V caches [num_pages, Hkv, page, D], bf16-representable float32 ~ N(0,1)."""
    rng = rng_for(cfg, _S_KV, layer)
    shape = (num_pages, cfg.Hkv, cfg.page, cfg.D)
    k = round_to_bf16(rng.standard_normal(shape, dtype=np.float32))
    v = round_to_bf16(rng.standard_normal(shape, dtype=np.float32))
    return k, v


def make_q_numpy(cfg: RoundConfig, B: int, n_max: int, layer: int = 0) -> np.ndarray:
    """Tree-node queries [B, n_max, Hq, D], bf16-representable float32 ~ N(0,1)."""
    rng = rng_for(cfg, _S_Q, layer)
    return round_to_bf16(rng.standard_normal((B, n_max, cfg.Hq, cfg.D), dtype=np.float32))


def make_kv_torch(cfg: RoundConfig, num_pages: int, layer: int, device):
    """Device-side K/V caches for workloads too large to draw on the host (bf16 N(0,1))."""
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(SEED_BASE * 1000 + cfg.config_id * 100 + layer)
    shape = (num_pages, cfg.Hkv, cfg.page, cfg.D)
    k = torch.randn(shape, generator=g, device=device, dtype=torch.float32).to(torch.bfloat16)
    v = torch.randn(shape, generator=g, device=device, dtype=torch.float32).to(torch.bfloat16)
    return k, v


def make_q_torch(cfg: RoundConfig, B: int, n_max: int, layer: int, device):
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(SEED_BASE * 1000 + 50000 + cfg.config_id * 100 + layer)
    return torch.randn((B, n_max, cfg.Hq, cfg.D), generator=g, device=device,
                       dtype=torch.float32).to(torch.bfloat16)


def make_verify_logits_torch(cfg: RoundConfig, target_tok, device, seed_offset: int = 0):
    """Target verify logits [B, n_max, V] bf16 on the device, drawn N(0, 4), with
    the value 24 (12 standard deviations) planted at target_tok[b, i] for every
    row whose token is >= 0, so the row's greedy token is the stand-in
    target's token."""
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(SEED_BASE * 1000 + 90000 + cfg.config_id * 100 + seed_offset)
    B, N = target_tok.shape
    x = torch.randn((B, N, cfg.V), generator=g, device=device, dtype=torch.float32) * 2.0
    tt = target_tok.to(device=device, dtype=torch.int64)
    b, i = torch.nonzero(tt >= 0, as_tuple=True)
    x[b, i, tt[b, i]] = 24.0
    return x.to(torch.bfloat16)
