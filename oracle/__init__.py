"""CPU oracle of the LiLiCorr per-block draft-selection path.

TEST INFRASTRUCTURE ONLY. Nothing on the product path may import, call or link
this package: only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline
leg of ``bench.py`` use it. It shares no code with the CUDA library; the only
module both sides use is ``workloads`` (seeded input draws, no method
arithmetic).

Everything here is plain, slow and in float64, written from the paper:

* top-K + log-normaliser per slot (Sec. 3.2 "top-K candidate tokens"; App. A
  "Serving" fuses top-K extraction with vocabulary-wide normalisation): the
  plain definition, a full log-sum-exp over V and a full stable sort.
* the scoring network (Sec. 3.2; App. A "Architecture"; Table "hparams"):
  restated step by step with library matmuls, no fusion or reordering.
* pair scores (Eq. "pair"; Sec. 3.5), the greedy walk (Sec. 3.5), the path score
  (Eq. "pathscore") and the exact Viterbi maximiser (App. E).
* the local next-candidate distributions (Eq. "localar") and decision gaps
  (Eq. "margin") along a path; coverage, oracle prefix and prefix acceptance
  against ground-truth tokens (Sec. 3.3 "Oracle-prefix supervision"; Sec. 3.1).

Pinned by ``tests/test_oracle_*.py`` against closed forms, brute force,
library routines and the paper's printed parameter counts. The scoring network's
numeric values are **parity unpinned** against any paper number: the paper
publishes no weights or worked example for it. Its architecture is pinned by the
parameter-count closed form (Table "hparams": 36.76 M / 32.04 M), and its pieces
by library special cases (RMSNorm, attention, SiLU MLP) in the tests.

Readings where the paper is silent (also listed in the design notes):
  L       = drafted slots carrying logits (the paper's block size is L + 1).
  D = d   head width equals the in/out dimension; F = 2 D; 8 heads.
  biases  every Linear has a bias; confidence MLP is 5 -> D -> D with SiLU.
  target  the 5 captured layers are averaged, RMSNorm'ed over H, projected to D.
  norms   RMSNorm with gain, eps = 1e-6, pre-norm blocks, a final norm.
  FFN     W2 SiLU(W1 x + b1) + b2 (not gated).
  biases  attention logits get dist[h, s_j - s_i + L - 1] + same[h] * 1{s_i = s_j}.
  gap     feature 3 is logp_top1 - logp_k (>= 0); rank feature k / (K - 1), 0 if K = 1.
  anchor  o_0 = normalise(W_a t + b_a) from the projected target state t.
  ties    top-K: larger logit first, then lower token id; -0.0 equals +0.0.
          walk: lower candidate index first.
  unit    v / max(||v||, 1e-12).
"""
from __future__ import annotations

import itertools
from typing import Callable, Dict, List, Optional, Sequence, Tuple

import numpy as np

RMS_EPS = 1e-6
NORM_EPS = 1e-12
N_CONF_FEATURES = 5
SIGMA = 8.0            # cosine scale sigma (Table "hparams"); never changes an argmax


# =========================================================================== architecture
def param_shapes(H: int, D: int, d: int, F: int, n_heads: int, L: int, K: int,
                 n_layers: int = 2) -> Dict[str, Tuple[int, ...]]:
    """Every learned tensor of the head, as this oracle reads App. A.

    Node terms (App. A, four summed terms): emb_* projects the frozen target
    embedding, hid_* the drafter state, conf* is the two-layer network over the 5
    confidence scalars, slot/rank are the learned tables. Target state: tgt_norm
    (RMSNorm gain over H) and tgt_*. Per layer: attention norm, Q/K/V/O with bias,
    the signed-slot-distance and same-slot bias tables, FFN norm, W1/W2 with bias.
    Then final_norm, the one concatenation layer fuse_* (3D -> D), and the out,
    in and anchor heads (D -> d).
    """
    s: Dict[str, Tuple[int, ...]] = {
        "emb_w": (D, H), "emb_b": (D,), "hid_w": (D, H), "hid_b": (D,),
        "conf1_w": (D, N_CONF_FEATURES), "conf1_b": (D,), "conf2_w": (D, D), "conf2_b": (D,),
        "slot": (L, D), "rank": (K, D),
        "tgt_norm": (H,), "tgt_w": (D, H), "tgt_b": (D,),
    }
    for i in range(n_layers):
        p = f"l{i}."
        s.update({p + "an": (D,), p + "wq": (D, D), p + "bq": (D,), p + "wk": (D, D),
                  p + "bk": (D,), p + "wv": (D, D), p + "bv": (D,), p + "wo": (D, D),
                  p + "bo": (D,), p + "dist": (n_heads, 2 * L - 1), p + "same": (n_heads,),
                  p + "fn": (D,), p + "w1": (F, D), p + "b1": (F,), p + "w2": (D, F),
                  p + "b2": (D,)})
    s.update({"final_norm": (D,), "fuse_w": (D, 3 * D), "fuse_b": (D,),
              "out_w": (d, D), "out_b": (d,), "in_w": (d, D), "in_b": (d,),
              "anc_w": (d, D), "anc_b": (d,)})
    return s


def param_count(H: int, D: int, d: int, F: int, n_heads: int, L: int, K: int,
                n_layers: int = 2) -> int:
    """Total learned parameters (Table "hparams" prints 36.76 M at H = 4096 and
    32.04 M at H = 2560 for D = d = 1024, F = 2048, 8 heads, K = 8, 15 slots)."""
    return int(sum(np.prod(v) for v in param_shapes(H, D, d, F, n_heads, L, K,
                                                   n_layers).values()))


# =========================================================================== step a1
def topk_lse(x: np.ndarray, K: int) -> Tuple[np.ndarray, np.ndarray, float]:
    """Top-K candidates and log-normaliser of one slot's logits (Sec. 3.2; App. A
    "Serving": top-K extraction fused with vocabulary-wide normalisation).

    lse = log sum_v exp(x_v), computed as m + log sum exp(x - m) over all V;
    ids = first K of a full stable sort by (logit descending, token id ascending);
    logp = x[ids] - lse. Returns (ids int64[K], logp float64[K], lse float).
    """
    x = np.asarray(x, dtype=np.float64)
    V = x.shape[0]
    if not (1 <= K <= V):
        raise ValueError("need 1 <= K <= V")
    if np.isnan(x).any() or not np.isfinite(x.max()):
        raise ValueError("row has NaN, +inf, or is all -inf")
    m = x.max()
    lse = float(m + np.log(np.sum(np.exp(x - m))))
    order = np.lexsort((np.arange(V), -x))      # primary -x ascending, then id ascending
    ids = order[:K].astype(np.int64)
    return ids, x[ids] - lse, lse


def topk_lse_partial(x: np.ndarray, K: int, id_offset: int):
    """One vocabulary shard's summary of a slot row (the vocabulary-sharded step (1) of a
    tensor-parallel LM head): the shard's maximum m, s = sum exp(x - m) over the shard,
    and its K largest logits with their vocabulary ids (column + id_offset) by the same
    full stable sort as topk_lse, padded with (-inf, -1) when the shard is narrower than
    K. m = -inf and s = 0 for a shard holding only -inf. Returns (m, s, vals[K], ids[K])."""
    x = np.asarray(x, dtype=np.float64)
    V = x.shape[0]
    m = float(x.max()) if V else -np.inf
    s = float(np.sum(np.exp(x - m))) if np.isfinite(m) else 0.0
    order = np.lexsort((np.arange(V), -x))[:K]
    vals = np.full(K, -np.inf)
    ids = np.full(K, -1, dtype=np.int64)
    vals[:len(order)] = x[order]
    ids[:len(order)] = order + id_offset
    return m, s, vals, ids


def merge_partials(parts, K: int) -> Tuple[np.ndarray, np.ndarray, float]:
    """Combine shard summaries (any order) into topk_lse's result for the whole row:
    lse = M + log sum_p s_p exp(m_p - M) with M = max_p m_p, and the K largest of the
    union of the shards' candidates by (value descending, id ascending)."""
    ms = np.array([p[0] for p in parts], dtype=np.float64)
    ss = np.array([p[1] for p in parts], dtype=np.float64)
    M = ms.max()
    if not np.isfinite(M):
        raise ValueError("row has NaN, +inf, or is all -inf")
    lse = float(M + np.log(np.sum(ss * np.exp(ms - M))))
    vals = np.concatenate([p[2] for p in parts])
    ids = np.concatenate([p[3] for p in parts])
    keep = ids >= 0
    vals, ids = vals[keep], ids[keep]
    order = np.lexsort((ids, -vals))[:K]
    return ids[order].astype(np.int64), vals[order] - lse, lse


def lm_head_topk(hidden: np.ndarray, w_vocab: np.ndarray, K: int):
    """The LM-head projection followed by step (1) (the projection that produces the
    drafter's logits, Table "cost"): logits = w_vocab @ hidden in fp64 (a library matmul),
    then topk_lse of those logits. hidden [H], w_vocab [V, H]. Returns topk_lse's
    (ids, logp, lse) and the logits."""
    x = np.asarray(w_vocab, dtype=np.float64) @ np.asarray(hidden, dtype=np.float64)
    ids, logp, lse = topk_lse(x, K)
    return ids, logp, lse, x


# =========================================================================== step a2
def confidence_features(logp: np.ndarray) -> np.ndarray:
    """Five confidence scalars per candidate of one slot (App. A "Architecture"):
    log-probability, probability, gap to the slot's most likely candidate,
    rank normalised to [0, 1], indicator of the top choice. logp is in rank order."""
    logp = np.asarray(logp, dtype=np.float64)
    K = logp.shape[0]
    k = np.arange(K, dtype=np.float64)
    rank01 = k / (K - 1) if K > 1 else np.zeros(K)
    return np.stack([logp, np.exp(logp), logp[0] - logp, rank01,
                     (k == 0).astype(np.float64)], axis=1)


def rms_norm(x: np.ndarray, g: np.ndarray, eps: float = RMS_EPS) -> np.ndarray:
    """RMSNorm over the last axis with gain g (App. A: "using RMSNorm")."""
    x = np.asarray(x, dtype=np.float64)
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * np.asarray(g, np.float64)


def silu(z: np.ndarray) -> np.ndarray:
    """SiLU(z) = z * sigmoid(z) (App. A: "SiLU activations")."""
    return z / (1.0 + np.exp(-z))


def linear(x: np.ndarray, w: np.ndarray, b: np.ndarray) -> np.ndarray:
    """y = x W^T + b with W stored [out, in]."""
    return np.asarray(x, np.float64) @ np.asarray(w, np.float64).T + np.asarray(b, np.float64)


def target_state(T: np.ndarray, W: Dict[str, np.ndarray]) -> np.ndarray:
    """Target state t in R^D (App. A): the target's hidden states at the last
    verified token, collapsed across the 5 captured layers (mean), normalised
    (RMSNorm over H) and projected to the head width."""
    T = np.asarray(T, dtype=np.float64)
    return linear(rms_norm(T.mean(axis=0), W["tgt_norm"]), W["tgt_w"], W["tgt_b"])


def nodes(ids: np.ndarray, logp: np.ndarray, hidden: np.ndarray, emb_rows: np.ndarray,
          W: Dict[str, np.ndarray]) -> np.ndarray:
    """Node vectors [L*K, D], slot-major (node j = s*K + k), Sec. 3.2 / App. A: the sum
    of four equal-width terms, (1) projected frozen embedding of the token,
    (2) projected drafter hidden state of the slot (shared by its K candidates),
    (3) a two-layer network over the confidence features, (4) slot and rank tables.

    ids/logp [L, K] in rank order, hidden [L, H], emb_rows [L, K, H]."""
    L, K = ids.shape
    n = np.zeros((L, K, W["emb_b"].shape[0]))
    for s in range(L):
        f = confidence_features(logp[s])
        emb = linear(emb_rows[s], W["emb_w"], W["emb_b"])                # (1)
        hid = linear(hidden[s], W["hid_w"], W["hid_b"])                  # (2)
        conf = linear(silu(linear(f, W["conf1_w"], W["conf1_b"])),       # (3)
                      W["conf2_w"], W["conf2_b"])
        n[s] = emb + hid[None, :] + conf + W["slot"][s][None, :] + W["rank"][:K]   # (4)
    return n.reshape(L * K, -1)


# =========================================================================== step a3
def attention(x: np.ndarray, W: Dict[str, np.ndarray], p: str, L: int, K: int,
              n_heads: int) -> np.ndarray:
    """Bidirectional multi-head self-attention over all L*K nodes (App. A): no mask;
    per-head learned biases added to the logits, one by signed slot distance
    s_j - s_i, one for pairs in the same slot. Q/K/V/O are linear with bias."""
    N, D = x.shape
    hd = D // n_heads
    q = linear(x, W[p + "wq"], W[p + "bq"])
    k = linear(x, W[p + "wk"], W[p + "bk"])
    v = linear(x, W[p + "wv"], W[p + "bv"])
    slot = np.arange(N) // K
    delta = slot[None, :] - slot[:, None]                 # s_j - s_i, row i = query
    same = (delta == 0).astype(np.float64)
    heads = []
    for h in range(n_heads):
        sl = slice(h * hd, (h + 1) * hd)
        logits = q[:, sl] @ k[:, sl].T / np.sqrt(hd)
        logits = logits + W[p + "dist"][h][delta + L - 1] + W[p + "same"][h] * same
        logits = logits - logits.max(axis=1, keepdims=True)
        a = np.exp(logits)
        a = a / a.sum(axis=1, keepdims=True)
        heads.append(a @ v[:, sl])
    return linear(np.concatenate(heads, axis=1), W[p + "wo"], W[p + "bo"])


def transformer(x: np.ndarray, W: Dict[str, np.ndarray], L: int, K: int, n_heads: int,
                n_layers: int) -> np.ndarray:
    """The scoring Transformer (App. A; Table "hparams": 2 layers, 8 heads, FFN 2D):
    pre-norm residual blocks x += Attn(RMSNorm x); x += W2 SiLU(W1 RMSNorm x),
    then a final RMSNorm."""
    x = np.asarray(x, dtype=np.float64)
    for i in range(n_layers):
        p = f"l{i}."
        x = x + attention(rms_norm(x, W[p + "an"]), W, p, L, K, n_heads)
        h = silu(linear(rms_norm(x, W[p + "fn"]), W[p + "w1"], W[p + "b1"]))
        x = x + linear(h, W[p + "w2"], W[p + "b2"])
    return rms_norm(x, W["final_norm"])


# =========================================================================== step a4
def unit(v: np.ndarray) -> np.ndarray:
    """v / max(||v||, 1e-12) along the last axis (out/in vectors are unit norm, Sec. 3.2)."""
    n = np.sqrt(np.sum(v * v, axis=-1, keepdims=True))
    return v / np.maximum(n, NORM_EPS)


def fuse_and_heads(x: np.ndarray, t: np.ndarray, W: Dict[str, np.ndarray], L: int,
                   K: int) -> Tuple[np.ndarray, np.ndarray, np.ndarray]:
    """Target fusion and vector heads (Sec. 3.2; App. A): u = SiLU(W_f [x; t; x*t] + b_f),
    the head's one concatenation; out = unit(W_o u + b_o), in = unit(W_i u + b_i);
    the anchor's out vector o_0 = unit(W_a t + b_a). Returns out, in [L, K, d], o_0 [d]."""
    N, D = x.shape
    tt = np.broadcast_to(t[None, :], (N, D))
    u = silu(linear(np.concatenate([x, tt, x * tt], axis=1), W["fuse_w"], W["fuse_b"]))
    out = unit(linear(u, W["out_w"], W["out_b"])).reshape(L, K, -1)
    inn = unit(linear(u, W["in_w"], W["in_b"])).reshape(L, K, -1)
    anc = unit(linear(t, W["anc_w"], W["anc_b"]))
    return out, inn, anc


def head_forward(ids: np.ndarray, logp: np.ndarray, hidden: np.ndarray, target: np.ndarray,
                 emb_rows: np.ndarray, W: Dict[str, np.ndarray], n_heads: int = 8,
                 n_layers: int = 2) -> Tuple[np.ndarray, np.ndarray, np.ndarray]:
    """One pass of the scoring head for one sequence (steps a2-a4): candidates ->
    out, in [L, K, d] and anchor out [d], all unit norm."""
    L, K = ids.shape
    H = hidden.shape[1]
    D = W["emb_b"].shape[0]
    d = W["out_b"].shape[0]
    F = W["l0.b1"].shape[0]
    want = param_shapes(H, D, d, F, n_heads, L, K, n_layers)
    for name, shape in want.items():
        if tuple(W[name].shape) != shape:
            raise ValueError(f"weight {name}: shape {W[name].shape}, expected {shape}")
    Wd = {k: np.asarray(v, dtype=np.float64) for k, v in W.items()}
    x = nodes(ids, logp, np.asarray(hidden, np.float64), np.asarray(emb_rows, np.float64), Wd)
    x = transformer(x, Wd, L, K, n_heads, n_layers)
    t = target_state(target, Wd)
    return fuse_and_heads(x, t, Wd, L, K)


# =========================================================================== step a5
def cosine(a: np.ndarray, b: np.ndarray) -> float:
    """cos(a, b) = <a, b> / (||a|| ||b||)."""
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.dot(a, b) / (max(np.linalg.norm(a), NORM_EPS) * max(np.linalg.norm(b), NORM_EPS)))


def pair_scores(out: np.ndarray, inn: np.ndarray, anchor: np.ndarray) -> Tuple[np.ndarray, np.ndarray]:
    """Matching terms of Eq. "pair" without the scale sigma (Sec. 3.5 counts
    (L-1) K^2 + K of them): anchor row A[k] = cos(o_0, i_{1,k}) and
    P[s, k, k'] = cos(o_{s,k}, i_{s+1,k'}) for consecutive drafted slots.
    out/inn [L, K, d], anchor [d] -> A [K], P [L-1, K, K]."""
    L, K, _ = out.shape
    A = np.array([cosine(anchor, inn[0, k]) for k in range(K)])
    P = np.zeros((max(L - 1, 0), K, K))
    for s in range(L - 1):
        for k in range(K):
            for k2 in range(K):
                P[s, k, k2] = cosine(out[s, k], inn[s + 1, k2])
    return A, P


# =========================================================================== step a6
def _argmax_first(v: np.ndarray) -> int:
    """Index of the maximum, lowest index among equal maxima."""
    best = 0
    for i in range(1, len(v)):
        if v[i] > v[best]:
            best = i
    return best


def _margin(v: np.ndarray) -> float:
    """Best minus second-best score of one walk step (inf when K = 1)."""
    if len(v) < 2:
        return float("inf")
    s = np.sort(np.asarray(v, np.float64))
    return float(s[-1] - s[-2])


def greedy_walk(A: np.ndarray, P: np.ndarray) -> Tuple[np.ndarray, np.ndarray]:
    """Greedy left-to-right commit (Sec. 3.5): c_1 = argmax_k A[k],
    c_s = argmax_k P[s-1, c_{s-1}, k]. Returns choices [L] and per-step margins
    (top1 - top2 of the row the step maximised over)."""
    L = P.shape[0] + 1
    c = np.zeros(L, dtype=np.int64)
    marg = np.zeros(L)
    c[0] = _argmax_first(A)
    marg[0] = _margin(A)
    for s in range(1, L):
        row = P[s - 1, c[s - 1]]
        c[s] = _argmax_first(row)
        marg[s] = _margin(row)
    return c, marg


def path_score(A: np.ndarray, P: np.ndarray, c: Sequence[int], sigma: float = SIGMA) -> float:
    """g(c) = sum_s phi(s-1, c_{s-1}, c_s), Eq. "pathscore" (phi = sigma * cos)."""
    g = A[c[0]]
    for s in range(1, len(c)):
        g += P[s - 1, c[s - 1], c[s]]
    return float(sigma * g)


def viterbi(A: np.ndarray, P: np.ndarray, sigma: float = SIGMA) -> Tuple[np.ndarray, float]:
    """Exact maximiser of g (App. E): sweep left to right keeping, per candidate, the
    score of the best path ending there and its predecessor; trace back from the
    best final candidate. Ties go to the lower index."""
    L = P.shape[0] + 1
    K = A.shape[0]
    best = sigma * np.asarray(A, np.float64)
    back = np.zeros((L, K), dtype=np.int64)
    for s in range(1, L):
        nxt = np.empty(K)
        for k2 in range(K):
            cand = best + sigma * P[s - 1, :, k2]
            back[s, k2] = _argmax_first(cand)
            nxt[k2] = cand[back[s, k2]]
        best = nxt
    c = np.zeros(L, dtype=np.int64)
    c[-1] = _argmax_first(best)
    for s in range(L - 1, 0, -1):
        c[s - 1] = back[s, c[s]]
    return c, float(best[c[-1]])


def brute_force_paths(A: np.ndarray, P: np.ndarray, sigma: float = SIGMA):
    """All K^L paths with their scores g (tiny lattices only)."""
    L = P.shape[0] + 1
    K = A.shape[0]
    for c in itertools.product(range(K), repeat=L):
        yield c, path_score(A, P, c, sigma)


# =========================================================================== diagnostics
def local_softmax(A: np.ndarray, P: np.ndarray, sigma: float = SIGMA) -> Tuple[np.ndarray, np.ndarray]:
    """Eq. "localar": P(c_s = k | c_{s-1}) = softmax_k(z_s[k]) with node scores
    z_s[k] = phi(s-1, c_{s-1}, k) = sigma * cos. Returns the anchor row's distribution
    [K] (predecessor: the anchor) and, for every slot pair and predecessor k, the
    distribution over successors [L-1, K, K] (last axis sums to 1)."""
    def softmax(z):
        z = np.asarray(z, np.float64)
        e = np.exp(z - z.max())
        return e / e.sum()
    A = np.asarray(A, np.float64)
    P = np.asarray(P, np.float64)
    pa = softmax(sigma * A)
    pp = np.zeros_like(P)
    for s in range(P.shape[0]):
        for k in range(P.shape[1]):
            pp[s, k] = softmax(sigma * P[s, k])
    return pa, pp


def path_probs(A: np.ndarray, P: np.ndarray, c: Sequence[int], sigma: float = SIGMA):
    """Along the path c: prob[s] = P(c_s | c_{s-1}) of Eq. "localar" (the anchor before
    slot 0), gap[s] = z_s[c_s] - max_{k != c_s} z_s[k] (the decision gap of Eq. "margin";
    +inf when K = 1) and log_prob = sum_s log prob[s]."""
    pa, pp = local_softmax(A, P, sigma)
    L = len(c)
    prob = np.zeros(L)
    gap = np.zeros(L)
    for s in range(L):
        z = sigma * (np.asarray(A, np.float64) if s == 0 else np.asarray(P[s - 1, c[s - 1]], np.float64))
        prob[s] = pa[c[0]] if s == 0 else pp[s - 1, c[s - 1], c[s]]
        others = np.delete(z, c[s])
        gap[s] = z[c[s]] - others.max() if others.size else np.inf
    return prob, gap, float(np.sum(np.log(prob)))


def block_acceptance(ids: np.ndarray, tokens: np.ndarray, truth: np.ndarray):
    """Against ground-truth tokens truth [L]: covered[s] = truth[s] is among slot s's K
    candidates; the oracle prefix is the longest leading run of covered slots; the
    accepted length is the longest leading run of slots whose chosen token equals the
    truth (prefix acceptance: the verifier keeps tokens up to the first mismatch)."""
    L = len(truth)
    covered = np.array([int(truth[s] in set(int(x) for x in ids[s])) for s in range(L)])
    oracle_prefix = 0
    while oracle_prefix < L and covered[oracle_prefix]:
        oracle_prefix += 1
    accepted = 0
    while accepted < L and int(tokens[accepted]) == int(truth[accepted]):
        accepted += 1
    return covered, oracle_prefix, accepted


# =========================================================================== whole path
def select_sequence(logits: np.ndarray, hidden: np.ndarray, target: np.ndarray,
                    embed_rows: Callable[[np.ndarray], np.ndarray], W: Dict[str, np.ndarray],
                    K: int, n_heads: int = 8, n_layers: int = 2) -> Dict[str, np.ndarray]:
    """The whole per-block selection for one sequence: logits [L, V], hidden [L, H],
    target [5, H] -> chosen tokens [L] plus every intermediate.
    ``embed_rows(ids)`` returns the frozen embedding rows [n, H] of token ids."""
    L = logits.shape[0]
    ids = np.zeros((L, K), dtype=np.int64)
    logp = np.zeros((L, K))
    lse = np.zeros(L)
    for s in range(L):
        ids[s], logp[s], lse[s] = topk_lse(logits[s], K)
    emb = np.asarray(embed_rows(ids.reshape(-1)), np.float64).reshape(L, K, -1)
    out, inn, anc = head_forward(ids, logp, hidden, target, emb, W, n_heads, n_layers)
    A, P = pair_scores(out, inn, anc)
    choice, margin = greedy_walk(A, P)
    tokens = ids[np.arange(L), choice]
    return {"ids": ids, "logp": logp, "lse": lse, "out": out, "in": inn, "anchor": anc,
            "A": A, "P": P, "choice": choice, "margin": margin, "tokens": tokens}
