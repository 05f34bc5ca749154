"""Seeded synthetic inputs shaped like the paper's serving workloads.

This module is the only code shared by the CUDA path's harness and the CPU
oracle. It draws random numbers and rounds them to the storage format; it holds
none of the selection method's arithmetic (no softmax, no top-K, no network).

Shapes follow the paper's setup (Sec. 3.1-3.2, App. A, Table "hparams"): a
drafter emits per-slot logits over a Qwen3-sized vocabulary (V = 151936), the
scoring head sees drafter hidden states of width H, five captured target layers
of width H, and a frozen token-embedding table [V, H]. The paper's datasets and
trained weights are not available, so every tensor is drawn from a seeded
distribution; the recipe per workload is stated in ``Workload.logit_kind``.

Draw order per sequence (one ``numpy.random.Generator(PCG64(seed))`` each):
logits [L, V], planted ids [L] (when the workload plants a token), drafter
hidden [L, H], target hidden [5, H]. Head weights come from their own seed in
blob order; the embedding table from a third seed, in chunks of rows.
"""
from __future__ import annotations

import concurrent.futures as _cf
import dataclasses
import os
from typing import Dict, List, Optional, Sequence, Tuple

import numpy as np

WEIGHT_SEED = 1_000_003
EMBED_SEED = 1_000_033
EMBED_CHUNK_ROWS = 2048
N_TGT_LAYERS = 5       # captured target layers (App. A "Architecture")
N_LAYERS = 2           # scoring Transformer layers (Table "hparams")
N_HEADS = 8            # attention heads (Table "hparams")
WEIGHT_STD = 0.02
UNIT_EMBED_STD = 1.0   # the wide-margin parity case: token embeddings at the hidden states' scale


@dataclasses.dataclass(frozen=True)
class Workload:
    """One synthetic workload: shapes, dtype and the logit recipe."""
    name: str
    B: int              # sequences per call
    L: int              # drafted slots carrying logits
    V: int              # vocabulary
    K: int              # candidates kept per slot
    d: int              # in/out vector dimension d_e
    H: int              # drafter / target hidden width
    dtype: str          # "f32" or "bf16": logits, hidden states and weights
    logit_kind: str     # see _draw_logits
    logit_param: Tuple[float, ...]
    seed_base: int
    tiers: Tuple[float, ...] = ()   # Gumbel temperatures, one batch of B per tier
    blocks: int = 1                 # independent calls (batch-1 latency runs)

    @property
    def D(self) -> int:         # head width (= d, the paper's D = d_e ratio)
        return self.d

    @property
    def F(self) -> int:         # feed-forward width (= 2 D, the paper's 2048/1024)
        return 2 * self.d

    @property
    def n_heads(self) -> int:
        return N_HEADS

    @property
    def n_layers(self) -> int:
        return N_LAYERS

    @property
    def n_tgt(self) -> int:
        return N_TGT_LAYERS

    def seeds(self, tier: int = 0) -> List[int]:
        """Per-sequence seeds of one batch (``tier`` selects the Gumbel tier)."""
        if self.tiers:
            return [self.seed_base + 100 * tier + b for b in range(self.B)]
        return [self.seed_base + b for b in range(self.B)]

    def block_seeds(self) -> List[int]:
        """Seeds of the ``blocks`` repeated batch-1 calls (seed_base .. +blocks-1)."""
        return [self.seed_base + i for i in range(self.blocks)]


WORKLOADS: Dict[str, Workload] = {
    # fp32 block small enough for the oracle to brute-force all 4^8 paths.
    "tiny_f32": Workload("tiny_f32", B=1, L=8, V=32000, K=4, d=64, H=256, dtype="f32",
                         logit_kind="normal_planted", logit_param=(2.0, 6.0), seed_base=0),
    # Single request, the paper's block shape at Qwen3-8B vocabulary/width.
    "single_request": Workload("single_request", B=1, L=16, V=151936, K=8, d=256, H=4096,
                               dtype="bf16", logit_kind="normal_planted",
                               logit_param=(3.0, 8.0), seed_base=1, blocks=1000),
    # 32 concurrent sequences, per-sequence logit scale ~ U[1, 5] mixes entropies.
    "serving_b32": Workload("serving_b32", B=32, L=16, V=151936, K=8, d=256, H=4096,
                            dtype="bf16", logit_kind="scaled_normal", logit_param=(1.0, 5.0),
                            seed_base=2000),
    # Gumbel noise / tau, three entropy tiers of 64 sequences each.
    "entropy_tiers_b64": Workload("entropy_tiers_b64", B=64, L=16, V=151936, K=16, d=256,
                                  H=4096, dtype="bf16", logit_kind="gumbel", logit_param=(),
                                  seed_base=3000, tiers=(0.3, 1.0, 3.0)),
    # 256 sequences, logits on a 0.25 grid so top-K ties are frequent.
    "ties_b256": Workload("ties_b256", B=256, L=16, V=151936, K=16, d=512, H=4096,
                          dtype="bf16", logit_kind="quantised_normal", logit_param=(2.0, 0.25),
                          seed_base=4000),
}

WORKLOAD_ORDER = ["tiny_f32", "single_request", "serving_b32", "entropy_tiers_b64", "ties_b256"]


# --------------------------------------------------------------------------- bf16 storage
def round_to_bf16(a: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bf16 (ties to even); returns float32."""
    return bf16_bits_to_f32(bf16_bits(a))


def bf16_bits(a: np.ndarray) -> np.ndarray:
    """float32 -> bf16 bit patterns (uint16), round to nearest even. No NaN/inf expected."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    u = a.view(np.uint32)
    r = (u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)
    return r.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """bf16 bit patterns (uint16) -> float32 values (exact)."""
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def _store(a: np.ndarray, dtype: str) -> np.ndarray:
    return round_to_bf16(a) if dtype == "bf16" else np.asarray(a, dtype=np.float32)


# --------------------------------------------------------------------------- per-sequence draws
def _draw_logits(wl: Workload, rng: np.random.Generator, tier: int) -> Tuple[np.ndarray, Optional[np.ndarray]]:
    L, V = wl.L, wl.V
    kind = wl.logit_kind
    planted = None
    if kind == "normal_planted":          # N(0, std) plus `boost` on one seeded id per slot
        std, boost = wl.logit_param
        x = rng.standard_normal((L, V), dtype=np.float32) * np.float32(std)
        planted = rng.integers(0, V, size=L, dtype=np.int64)
        x[np.arange(L), planted] += np.float32(boost)
    elif kind == "scaled_normal":         # a_b * N(0, 1), a_b ~ U[lo, hi] per sequence
        lo, hi = wl.logit_param
        a = np.float32(rng.uniform(lo, hi))
        x = rng.standard_normal((L, V), dtype=np.float32) * a
    elif kind == "gumbel":                # Gumbel(0, 1) / tau
        tau = wl.tiers[tier]
        x = (rng.gumbel(0.0, 1.0, size=(L, V)) / tau).astype(np.float32)
    elif kind == "quantised_normal":      # q * round(N(0, std) / q): exact in bf16, many ties
        std, q = wl.logit_param
        z = rng.standard_normal((L, V), dtype=np.float32) * np.float32(std / q)
        x = (np.round(z) * np.float32(q)).astype(np.float32)
    else:
        raise ValueError(kind)
    return _store(x, wl.dtype), planted


def sequence_inputs(wl: Workload, seed: int, tier: int = 0) -> Dict[str, np.ndarray]:
    """Inputs of one sequence: logits [L,V], hidden [L,H], target [5,H] (float32 values
    exactly representable in ``wl.dtype``) and ``planted`` ids [L] (or None)."""
    rng = np.random.default_rng(np.random.PCG64(seed))
    logits, planted = _draw_logits(wl, rng, tier)
    hidden = _store(rng.standard_normal((wl.L, wl.H), dtype=np.float32), wl.dtype)
    target = _store(rng.standard_normal((wl.n_tgt, wl.H), dtype=np.float32), wl.dtype)
    return {"logits": logits, "planted": planted, "hidden": hidden, "target": target}


def _threads() -> int:
    return max(1, min(16, os.cpu_count() or 1))


def batch_inputs(wl: Workload, seeds: Sequence[int], tier: int = 0) -> Dict[str, np.ndarray]:
    """Stacked inputs of several sequences: logits [B,L,V], hidden [B,L,H], target [B,5,H]."""
    with _cf.ThreadPoolExecutor(_threads()) as ex:
        seqs = list(ex.map(lambda s: sequence_inputs(wl, s, tier), seeds))
    out = {k: np.stack([s[k] for s in seqs]) for k in ("logits", "hidden", "target")}
    out["planted"] = (np.stack([s["planted"] for s in seqs]) if seqs[0]["planted"] is not None
                      else None)
    return out


# --------------------------------------------------------------------------- head weights
def head_param_shapes(H: int, D: int, d: int, F: int, n_heads: int, L: int, K: int,
                      n_layers: int = N_LAYERS) -> List[Tuple[str, Tuple[int, ...]]]:
    """Named parameter tensors of the scoring head, in weight-blob order.

    Linear weights are [out, in]. Names: ``emb_*`` token-embedding projection,
    ``hid_*`` drafter-state projection, ``conf*`` confidence MLP over the 5
    features, ``slot``/``rank`` tables, ``tgt_*`` target-state norm and
    projection, ``l{i}.*`` Transformer layers (``an`` attention norm, ``fn`` FFN
    norm, ``dist``/``same`` attention biases), ``final_norm``, ``fuse_*`` the one
    3D -> D concatenation layer, ``out_*``/``in_*``/``anc_*`` vector heads.
    """
    s: List[Tuple[str, Tuple[int, ...]]] = [
        ("emb_w", (D, H)), ("emb_b", (D,)),
        ("hid_w", (D, H)), ("hid_b", (D,)),
        ("conf1_w", (D, 5)), ("conf1_b", (D,)), ("conf2_w", (D, D)), ("conf2_b", (D,)),
        ("slot", (L, D)), ("rank", (K, D)),
        ("tgt_norm", (H,)), ("tgt_w", (D, H)), ("tgt_b", (D,)),
    ]
    for i in range(n_layers):
        p = f"l{i}."
        s += [(p + "an", (D,)),
              (p + "wq", (D, D)), (p + "bq", (D,)), (p + "wk", (D, D)), (p + "bk", (D,)),
              (p + "wv", (D, D)), (p + "bv", (D,)), (p + "wo", (D, D)), (p + "bo", (D,)),
              (p + "dist", (n_heads, 2 * L - 1)), (p + "same", (n_heads,)),
              (p + "fn", (D,)),
              (p + "w1", (F, D)), (p + "b1", (F,)), (p + "w2", (D, F)), (p + "b2", (D,))]
    s += [("final_norm", (D,)),
          ("fuse_w", (D, 3 * D)), ("fuse_b", (D,)),
          ("out_w", (d, D)), ("out_b", (d,)),
          ("in_w", (d, D)), ("in_b", (d,)),
          ("anc_w", (d, D)), ("anc_b", (d,))]
    return s


def _is_norm_gain(name: str) -> bool:
    return name in ("tgt_norm", "final_norm") or name.endswith(".an") or name.endswith(".fn")


def head_weights(wl: Workload, seed: int = WEIGHT_SEED) -> Dict[str, np.ndarray]:
    """Random-init head weights: N(0, 0.02) for matrices, biases and tables; RMSNorm
    gains 1 + N(0, 0.02). Values are rounded to ``wl.dtype``. Ordered as the blob."""
    rng = np.random.default_rng(np.random.PCG64(seed))
    out: Dict[str, np.ndarray] = {}
    for name, shape in head_param_shapes(wl.H, wl.D, wl.d, wl.F, wl.n_heads, wl.L, wl.K,
                                         wl.n_layers):
        a = rng.standard_normal(shape, dtype=np.float32) * np.float32(WEIGHT_STD)
        if _is_norm_gain(name):
            a = a + np.float32(1.0)
        out[name] = _store(a, wl.dtype)
    return out


# --------------------------------------------------------------------------- embedding table
def _embed_chunk(V: int, H: int, c: int, seed: int, std: float = WEIGHT_STD) -> np.ndarray:
    r0 = c * EMBED_CHUNK_ROWS
    n = min(EMBED_CHUNK_ROWS, V - r0)
    rng = np.random.default_rng(np.random.PCG64([seed, c]))
    return rng.standard_normal((n, H), dtype=np.float32) * np.float32(std)


_EMBED_CACHE: Dict[Tuple[int, int, str, int, float], np.ndarray] = {}


def embed_table(V: int, H: int, dtype: str, seed: int = EMBED_SEED,
                std: float = WEIGHT_STD) -> np.ndarray:
    """Frozen token-embedding table [V, H] ~ N(0, std) (std 0.02 by default, like the
    head's weights; ``UNIT_EMBED_STD`` for the wide-margin parity case).

    Returned as bf16 bit patterns (uint16) for ``dtype == "bf16"`` and float32
    otherwise. Rows are drawn in chunks of EMBED_CHUNK_ROWS with per-chunk seeds,
    so ``embed_rows`` can regenerate any row without the full table. The last
    table built is cached in-process.
    """
    key = (V, H, dtype, seed, float(std))
    if key in _EMBED_CACHE:
        return _EMBED_CACHE[key]
    nchunks = (V + EMBED_CHUNK_ROWS - 1) // EMBED_CHUNK_ROWS
    out = np.empty((V, H), dtype=np.uint16 if dtype == "bf16" else np.float32)

    def fill(c: int) -> None:
        a = _embed_chunk(V, H, c, seed, std)
        r0 = c * EMBED_CHUNK_ROWS
        out[r0:r0 + a.shape[0]] = bf16_bits(a) if dtype == "bf16" else a

    with _cf.ThreadPoolExecutor(_threads()) as ex:
        list(ex.map(fill, range(nchunks)))
    _EMBED_CACHE.clear()
    _EMBED_CACHE[key] = out
    return out


def embed_rows(V: int, H: int, dtype: str, ids: np.ndarray, seed: int = EMBED_SEED,
               std: float = WEIGHT_STD) -> np.ndarray:
    """Rows ``ids`` of the embedding table as float32 values, regenerated per chunk."""
    ids = np.asarray(ids, dtype=np.int64).reshape(-1)
    key = (V, H, dtype, seed, float(std))
    if key in _EMBED_CACHE:
        t = _EMBED_CACHE[key][ids]
        return bf16_bits_to_f32(t) if dtype == "bf16" else t.astype(np.float32)
    rows = np.empty((ids.size, H), dtype=np.float32)
    for c in np.unique(ids // EMBED_CHUNK_ROWS):
        a = _embed_chunk(V, H, int(c), seed, std)
        a = round_to_bf16(a) if dtype == "bf16" else a
        sel = np.nonzero(ids // EMBED_CHUNK_ROWS == c)[0]
        rows[sel] = a[ids[sel] - c * EMBED_CHUNK_ROWS]
    return rows
