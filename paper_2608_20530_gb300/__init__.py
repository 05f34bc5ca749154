"""Python binding of the LiLiCorr per-block draft-selection library (sm_103a).

Argument marshalling only: every step of the path runs in the CUDA library
``lib/liblilicorr.so`` through its C ABI (``include/lilicorr.h``). PyTorch
supplies device memory and the current stream. There is no CPU fallback: if the
library is missing, every call raises.

Names follow the C ABI: ``topk_lse``, ``embed_in_out``, ``pair_scores``,
``greedy_walk``, ``select_block``, plus ``Head`` (an uploaded scoring head) and
``Workspace`` (caller-owned scratch).
"""
from __future__ import annotations

import ctypes
import os
from typing import Dict, Mapping, Optional, Sequence, Tuple

import numpy as np
import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "lib", "liblilicorr.so")

F32, BF16 = 0, 1
STATUS = {0: "ok", 1: "invalid argument", 2: "unsupported or inconsistent shape",
          3: "unsupported dtype", 4: "CUDA error", 5: "non-finite logit row",
          6: "device wait timed out", 7: "workspace too small"}
ERR_ARG, ERR_SHAPE, ERR_NONFINITE = 1, 2, 5
MAX_K = 32


class LilicorrError(RuntimeError):
    def __init__(self, status: int, where: str):
        super().__init__(f"{where}: {STATUS.get(status, status)} (status {status})")
        self.status = status


class HeadDesc(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int) for n in
                ("H", "D", "d", "n_heads", "ffn", "n_layers", "L", "K", "V", "n_tgt")] + \
               [("dtype", ctypes.c_int)]


_LIB: Optional[ctypes.CDLL] = None
_P = ctypes.c_void_p
_I = ctypes.c_int
_S = ctypes.c_size_t

_SIGS = {
    "lilicorr_status_str": (ctypes.c_char_p, [_I]),
    "lilicorr_version": (_I, []),
    "lilicorr_head_param_count": (_S, [ctypes.POINTER(HeadDesc)]),
    "lilicorr_head_create": (_I, [ctypes.POINTER(HeadDesc), _P, _P, ctypes.POINTER(_P)]),
    "lilicorr_head_destroy": (_I, [_P]),
    "lilicorr_workspace_init": (_I, [_P, _S, _P]),
    "lilicorr_topk_lse_workspace_bytes": (_S, [_I, _I, _I]),
    "lilicorr_topk_lse": (_I, [_P, _I, _I, _I, _I, _P, _P, _P, _P, _S, _P]),
    "lilicorr_workspace_bytes": (_S, [_P, _I]),
    "lilicorr_embed_in_out": (_I, [_P, _I, _P, _P, _P, _P, _P, _P, _P, _P, _S, _P]),
    "lilicorr_pair_scores": (_I, [_I, _I, _I, _I, _P, _P, _P, _P, _P, _P]),
    "lilicorr_greedy_walk": (_I, [_I, _I, _I, _P, _P, _P, _P, _P, _P, _P]),
    "lilicorr_select_block": (_I, [_P, _I, _P, _P, _P, _P, _P, _S, _P]),
    "lilicorr_best_path": (_I, [_I, _I, _I, _P, _P, _P, ctypes.c_float, _P, _P, _P, _P]),
    "lilicorr_select_block_walk": (_I, [_P, _I, _P, _P, _P, _I, _P, _P, _S, _P]),
    "lilicorr_local_softmax": (_I, [_I, _I, _I, _P, _P, ctypes.c_float, _P, _P, _P]),
    "lilicorr_path_probs": (_I, [_I, _I, _I, _P, _P, _P, ctypes.c_float, _P, _P, _P, _P]),
    "lilicorr_block_acceptance": (_I, [_I, _I, _I, _P, _P, _P, _P, _P, _P, _P]),
    "lilicorr_select_block_intermediates": (_I, [_P, _I, _P, _S] + [ctypes.POINTER(_P)] * 6),
    "lilicorr_get_device_status": (_I, [_P, _P]),
    "lilicorr_launch_count": (ctypes.c_uint64, []),
    "lilicorr_test_fused_path": (_I, [_P, _I]),
    "lilicorr_test_attention_path": (_I, [_I]),
    "lilicorr_topk_lse_noalloc_max_bytes": (_S, []),
    "lilicorr_topk_partial_bytes": (_S, [_I]),
    "lilicorr_lm_head_topk_workspace_bytes": (_S, [_I, _I, _I, _I]),
    "lilicorr_lm_head_topk": (_I, [_P, _P, _I, _I, _I, _I, _P, _P, _P, _P, _S, _P]),
    "lilicorr_topk_lse_partial_workspace_bytes": (_S, [_I, _I, _I]),
    "lilicorr_topk_lse_partial": (_I, [_P, _I, _I, _I, _I, _I, _P, _P, _S, _P]),
    "lilicorr_topk_lse_merge": (_I, [_P, _I, _I, _I, _P, _P, _P, _P, _P]),
    "lilicorr_topk_lse_noalloc": (_I, [_P, _I, _I, _I, _I, _P, _P, _P, _P]),
    "lilicorr_test_linear": (_I, [_P, _I, _I, _P, _I, _I, _P, _I, _I, _I, _I, _I, _P, _P, _I, _I,
                                  _P, _P]),
    "lilicorr_test_linear_timeout": (_I, [_P, _P, _P, _I, _I, _I, ctypes.c_longlong, _P, _P]),
}


def lib() -> ctypes.CDLL:
    """The loaded CUDA library (raises if it has not been built)."""
    global _LIB
    if _LIB is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"CUDA library not built ({LIB_PATH}); run __graft_entry__.build()")
        so = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            f = getattr(so, name)
            f.restype = res
            f.argtypes = args
        _LIB = so
    return _LIB


def _check(status: int, where: str) -> None:
    if status != 0:
        raise LilicorrError(status, where)


def _stream() -> int:
    return torch.cuda.current_stream().cuda_stream


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    return None if t is None else t.data_ptr()


def _dev(t: torch.Tensor, name: str) -> torch.Tensor:
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return t


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return F32
    if t.dtype == torch.bfloat16:
        return BF16
    raise ValueError(f"unsupported dtype {t.dtype}")


def launch_count() -> int:
    """Kernel launches the library has enqueued in this process (graph replays excluded)."""
    return int(lib().lilicorr_launch_count())


# --------------------------------------------------------------------------- workspace
class Workspace:
    """Caller-owned device scratch, zero-filled once (the library's counters start at 0)."""

    def __init__(self, nbytes: int, device=None):
        self.nbytes = int(max(nbytes, 256))
        self.buf = torch.zeros(self.nbytes, dtype=torch.uint8, device=device or "cuda")

    @property
    def ptr(self) -> int:
        return self.buf.data_ptr()

    def status(self) -> int:
        """Read and clear the device status word (synchronises the current stream)."""
        return int(lib().lilicorr_get_device_status(self.ptr, _stream()))


# --------------------------------------------------------------------------- head
def blob_order(H: int, D: int, d: int, F: int, n_heads: int, L: int, K: int,
               n_layers: int) -> Sequence[Tuple[str, Tuple[int, ...]]]:
    """Tensor names and shapes in the weight-blob order of ``lilicorr.h``."""
    s = [("emb_w", (D, H)), ("emb_b", (D,)), ("hid_w", (D, H)), ("hid_b", (D,)),
         ("conf1_w", (D, 5)), ("conf1_b", (D,)), ("conf2_w", (D, D)), ("conf2_b", (D,)),
         ("slot", (L, D)), ("rank", (K, D)), ("tgt_norm", (H,)), ("tgt_w", (D, H)),
         ("tgt_b", (D,))]
    for i in range(n_layers):
        p = f"l{i}."
        s += [(p + "an", (D,)), (p + "wq", (D, D)), (p + "bq", (D,)), (p + "wk", (D, D)),
              (p + "bk", (D,)), (p + "wv", (D, D)), (p + "bv", (D,)), (p + "wo", (D, D)),
              (p + "bo", (D,)), (p + "dist", (n_heads, 2 * L - 1)), (p + "same", (n_heads,)),
              (p + "fn", (D,)), (p + "w1", (F, D)), (p + "b1", (F,)), (p + "w2", (D, F)),
              (p + "b2", (D,))]
    s += [("final_norm", (D,)), ("fuse_w", (D, 3 * D)), ("fuse_b", (D,)), ("out_w", (d, D)),
          ("out_b", (d,)), ("in_w", (d, D)), ("in_b", (d,)), ("anc_w", (d, D)), ("anc_b", (d,))]
    return s


def _as_storage(a: np.ndarray, dtype: int) -> np.ndarray:
    """float32 values -> contiguous storage of the head dtype (bf16 as uint16 bits,
    round to nearest even; exact for values already representable in bf16)."""
    if dtype == F32:
        return np.ascontiguousarray(a, dtype=np.float32)
    if a.dtype == np.uint16:
        return np.ascontiguousarray(a)
    t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


class Head:
    """A scoring head uploaded to the current CUDA device (lilicorr_head_create)."""

    def __init__(self, *, H: int, D: int, d: int, n_heads: int, ffn: int, n_layers: int, L: int,
                 K: int, V: int, n_tgt: int, dtype: str, weights: Mapping[str, np.ndarray],
                 embed_table: np.ndarray):
        self.dtype_code = BF16 if dtype == "bf16" else F32
        self.desc = HeadDesc(H, D, d, n_heads, ffn, n_layers, L, K, V, n_tgt, self.dtype_code)
        self.L, self.K, self.V, self.H, self.d, self.D, self.n_tgt = L, K, V, H, d, D, n_tgt
        order = blob_order(H, D, d, ffn, n_heads, L, K, n_layers)
        parts = []
        for name, shape in order:
            w = np.asarray(weights[name])
            if tuple(w.shape) != tuple(shape):
                raise ValueError(f"{name}: shape {w.shape}, expected {shape}")
            parts.append(_as_storage(w, self.dtype_code).reshape(-1))
        blob = np.concatenate(parts)
        n = lib().lilicorr_head_param_count(ctypes.byref(self.desc))
        if n == 0 or n != blob.size:
            raise LilicorrError(2, f"head_param_count ({n} vs blob {blob.size})")
        emb = _as_storage(embed_table, self.dtype_code)
        if emb.shape != (V, H):
            raise ValueError(f"embed_table shape {emb.shape}, expected {(V, H)}")
        h = _P()
        _check(lib().lilicorr_head_create(ctypes.byref(self.desc), blob.ctypes.data,
                                          emb.ctypes.data, ctypes.byref(h)), "head_create")
        self._h = h
        self.torch_dtype = torch.bfloat16 if self.dtype_code == BF16 else torch.float32

    @classmethod
    def from_workload(cls, wl, weights, embed_table) -> "Head":
        return cls(H=wl.H, D=wl.D, d=wl.d, n_heads=wl.n_heads, ffn=wl.F, n_layers=wl.n_layers,
                   L=wl.L, K=wl.K, V=wl.V, n_tgt=wl.n_tgt, dtype=wl.dtype, weights=weights,
                   embed_table=embed_table)

    @property
    def handle(self) -> int:
        return self._h.value

    def workspace_bytes(self, B: int) -> int:
        return int(lib().lilicorr_workspace_bytes(self._h, B))

    def workspace(self, B: int) -> Workspace:
        return Workspace(self.workspace_bytes(B))

    def close(self) -> None:
        if getattr(self, "_h", None) is not None and self._h.value:
            _check(lib().lilicorr_head_destroy(self._h), "head_destroy")
            self._h = _P()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


# --------------------------------------------------------------------------- calls
def topk_lse(logits: torch.Tensor, K: int, ws: Optional[Workspace] = None):
    """Top-K ids [rows, K] int32, log-probs [rows, K] fp32 and log-normaliser [rows] fp32
    of logit rows [..., V] (fp32 or bf16)."""
    _dev(logits, "logits")
    V = logits.shape[-1]
    rows = logits.numel() // V if V else 0
    need = int(lib().lilicorr_topk_lse_workspace_bytes(rows, V, K))
    if ws is None:
        ws = Workspace(need, logits.device)
    lead = tuple(logits.shape[:-1])
    ids = torch.empty(lead + (K,), dtype=torch.int32, device=logits.device)
    logp = torch.empty(lead + (K,), dtype=torch.float32, device=logits.device)
    lse = torch.empty(lead, dtype=torch.float32, device=logits.device)
    _check(lib().lilicorr_topk_lse(logits.data_ptr(), _dtype_code(logits), rows, V, K,
                                   ids.data_ptr(), logp.data_ptr(), lse.data_ptr(), ws.ptr,
                                   ws.nbytes, _stream()), "topk_lse")
    return ids, logp, lse


def topk_lse_noalloc(logits: torch.Tensor, K: int):
    """topk_lse without a caller workspace: the library's fixed device scratch is used
    instead (for callers that cannot allocate device memory; see lilicorr.h). Calls that
    overlap on the GPU race on that scratch."""
    _dev(logits, "logits")
    V = logits.shape[-1]
    rows = logits.numel() // V if V else 0
    lead = tuple(logits.shape[:-1])
    ids = torch.empty(lead + (K,), dtype=torch.int32, device=logits.device)
    logp = torch.empty(lead + (K,), dtype=torch.float32, device=logits.device)
    lse = torch.empty(lead, dtype=torch.float32, device=logits.device)
    _check(lib().lilicorr_topk_lse_noalloc(logits.data_ptr(), _dtype_code(logits), rows, V, K,
                                           ids.data_ptr(), logp.data_ptr(), lse.data_ptr(),
                                           _stream()), "topk_lse_noalloc")
    return ids, logp, lse


def lm_head_topk(hidden: torch.Tensor, w_vocab: torch.Tensor, K: int,
                 ws: Optional[Workspace] = None):
    """Top-K ids [rows, K] int32, log-probs [rows, K] and log-normaliser [rows] of the
    logits hidden [rows, H] @ w_vocab[V, H]^T (bf16), which are never written out."""
    _dev(hidden, "hidden")
    _dev(w_vocab, "w_vocab")
    if hidden.dtype != torch.bfloat16 or w_vocab.dtype != torch.bfloat16:
        raise ValueError("hidden and w_vocab must be bf16")
    rows, H = hidden.shape
    V = w_vocab.shape[0]
    need = int(lib().lilicorr_lm_head_topk_workspace_bytes(rows, H, V, K))
    if need == 0 and rows > 0:
        raise LilicorrError(ERR_SHAPE, "lm_head_topk")
    if ws is None:
        ws = Workspace(need, hidden.device)
    dev = hidden.device
    ids = torch.empty((rows, K), dtype=torch.int32, device=dev)
    logp = torch.empty((rows, K), dtype=torch.float32, device=dev)
    lse = torch.empty((rows,), dtype=torch.float32, device=dev)
    _check(lib().lilicorr_lm_head_topk(hidden.data_ptr(), w_vocab.data_ptr(), rows, H, V, K,
                                       ids.data_ptr(), logp.data_ptr(), lse.data_ptr(), ws.ptr,
                                       ws.nbytes, _stream()), "lm_head_topk")
    return ids, logp, lse


def topk_partial_bytes(K: int) -> int:
    """Bytes of one row's partial record of a vocabulary shard (8 + 8K)."""
    return 8 + 8 * int(K)


def topk_lse_partial(logits: torch.Tensor, K: int, id_offset: int,
                     ws: Optional[Workspace] = None) -> torch.Tensor:
    """Partial records [rows, 8 + 8K] (uint8) of a vocabulary shard: logits [..., V_shard]
    whose column 0 is vocabulary id ``id_offset`` (see lilicorr_topk_lse_partial)."""
    _dev(logits, "logits")
    V = logits.shape[-1]
    rows = logits.numel() // V if V else 0
    need = int(lib().lilicorr_topk_lse_partial_workspace_bytes(rows, V, K))
    if ws is None:
        ws = Workspace(need, logits.device)
    rec = torch.empty((rows, topk_partial_bytes(K)), dtype=torch.uint8, device=logits.device)
    _check(lib().lilicorr_topk_lse_partial(logits.data_ptr(), _dtype_code(logits), rows, V, K,
                                           int(id_offset), rec.data_ptr(), ws.ptr, ws.nbytes,
                                           _stream()), "topk_lse_partial")
    return rec


def topk_lse_merge(partials: torch.Tensor, K: int, status: Optional[torch.Tensor] = None):
    """Merge the shards' records [P, rows, 8 + 8K] into (ids [rows, K] int32, logp [rows, K],
    lse [rows]) as topk_lse computes them on whole rows."""
    _dev(partials, "partials")
    if partials.dim() != 3 or partials.shape[2] != topk_partial_bytes(K):
        raise ValueError("partials must be [P, rows, 8 + 8K] bytes")
    P, rows = partials.shape[0], partials.shape[1]
    dev = partials.device
    ids = torch.empty((rows, K), dtype=torch.int32, device=dev)
    logp = torch.empty((rows, K), dtype=torch.float32, device=dev)
    lse = torch.empty((rows,), dtype=torch.float32, device=dev)
    _check(lib().lilicorr_topk_lse_merge(partials.contiguous().data_ptr(), P, rows, K,
                                         ids.data_ptr(), logp.data_ptr(), lse.data_ptr(),
                                         _ptr(status), _stream()), "topk_lse_merge")
    return ids, logp, lse


def embed_in_out(head: Head, ids: torch.Tensor, logp: torch.Tensor, hidden: torch.Tensor,
                 target: torch.Tensor, ws: Optional[Workspace] = None):
    """Unit out/in vectors [B, L, K, d] and anchor out vectors [B, d] (fp32)."""
    B = ids.shape[0]
    for t, n in ((ids, "ids"), (logp, "logp"), (hidden, "hidden"), (target, "target")):
        _dev(t, n)
    if hidden.dtype != head.torch_dtype or target.dtype != head.torch_dtype:
        raise ValueError("hidden/target dtype must match the head dtype")
    ws = ws or head.workspace(B)
    dev = ids.device
    out = torch.empty((B, head.L, head.K, head.d), dtype=torch.float32, device=dev)
    inn = torch.empty_like(out)
    anc = torch.empty((B, head.d), dtype=torch.float32, device=dev)
    _check(lib().lilicorr_embed_in_out(head._h, B, ids.data_ptr(), logp.data_ptr(),
                                       hidden.data_ptr(), target.data_ptr(), out.data_ptr(),
                                       inn.data_ptr(), anc.data_ptr(), ws.ptr, ws.nbytes,
                                       _stream()), "embed_in_out")
    return out, inn, anc


def pair_scores(out_vec: torch.Tensor, in_vec: torch.Tensor, anchor_out: torch.Tensor):
    """Anchor row [B, K] and pair matrices [B, L-1, K, K] of cosines (no sigma)."""
    B, L, K, d = out_vec.shape
    for t, n in ((out_vec, "out_vec"), (in_vec, "in_vec"), (anchor_out, "anchor_out")):
        _dev(t, n)
    A = torch.empty((B, K), dtype=torch.float32, device=out_vec.device)
    P = torch.empty((B, max(L - 1, 0), K, K), dtype=torch.float32, device=out_vec.device)
    _check(lib().lilicorr_pair_scores(B, L, K, d, out_vec.data_ptr(), in_vec.data_ptr(),
                                      anchor_out.data_ptr(), A.data_ptr(),
                                      P.data_ptr() if P.numel() else None, _stream()),
           "pair_scores")
    return A, P


def greedy_walk(A: torch.Tensor, P: torch.Tensor, ids: torch.Tensor):
    """Greedy walk: choice [B, L], tokens [B, L] (int32) and margins [B, L] (fp32)."""
    B, K = A.shape
    L = P.shape[1] + 1
    for t, n in ((A, "anchor_scores"), (P, "pair_scores"), (ids, "ids")):
        _dev(t, n)
    choice = torch.empty((B, L), dtype=torch.int32, device=A.device)
    tokens = torch.empty_like(choice)
    margin = torch.empty((B, L), dtype=torch.float32, device=A.device)
    _check(lib().lilicorr_greedy_walk(B, L, K, A.data_ptr(), P.data_ptr() if P.numel() else None,
                                      ids.data_ptr(), choice.data_ptr(), tokens.data_ptr(),
                                      margin.data_ptr(), _stream()), "greedy_walk")
    return choice, tokens, margin


SIGMA = 8.0
WALKS = {"greedy": 0, "viterbi": 1}


def best_path(A: torch.Tensor, P: torch.Tensor, ids: torch.Tensor, sigma: float = SIGMA):
    """Exact best path (App. E): choice [B, L], tokens [B, L] (int32) and path score
    g [B] (fp32, scaled by sigma)."""
    B, K = A.shape
    L = P.shape[1] + 1
    for t, n in ((A, "anchor_scores"), (P, "pair_scores"), (ids, "ids")):
        _dev(t, n)
    choice = torch.empty((B, L), dtype=torch.int32, device=A.device)
    tokens = torch.empty_like(choice)
    score = torch.empty((B,), dtype=torch.float32, device=A.device)
    _check(lib().lilicorr_best_path(B, L, K, A.data_ptr(), P.data_ptr() if P.numel() else None,
                                    ids.data_ptr(), float(sigma), choice.data_ptr(),
                                    tokens.data_ptr(), score.data_ptr(), _stream()), "best_path")
    return choice, tokens, score


def local_softmax(A: torch.Tensor, P: torch.Tensor, sigma: float = SIGMA):
    """Local next-candidate distributions (Eq. "localar"): anchor [B, K] and, per slot
    pair and predecessor, over successors [B, L-1, K, K] (fp32)."""
    B, K = A.shape
    L = P.shape[1] + 1
    for t, n in ((A, "anchor_scores"), (P, "pair_scores")):
        _dev(t, n)
    pa = torch.empty_like(A)
    pp = torch.empty_like(P)
    _check(lib().lilicorr_local_softmax(B, L, K, A.data_ptr(), P.data_ptr() if P.numel() else None,
                                        float(sigma), pa.data_ptr(),
                                        pp.data_ptr() if pp.numel() else None, _stream()),
           "local_softmax")
    return pa, pp


def path_probs(A: torch.Tensor, P: torch.Tensor, choice: torch.Tensor, sigma: float = SIGMA):
    """Along the path `choice` [B, L]: P(c_s | c_{s-1}) [B, L], decision gaps [B, L] and the
    path's log-probability [B] (fp32)."""
    B, K = A.shape
    L = P.shape[1] + 1
    for t, n in ((A, "anchor_scores"), (P, "pair_scores"), (choice, "choice")):
        _dev(t, n)
    prob = torch.empty((B, L), dtype=torch.float32, device=A.device)
    gap = torch.empty_like(prob)
    lp = torch.empty((B,), dtype=torch.float32, device=A.device)
    _check(lib().lilicorr_path_probs(B, L, K, A.data_ptr(), P.data_ptr() if P.numel() else None,
                                     choice.data_ptr(), float(sigma), prob.data_ptr(),
                                     gap.data_ptr(), lp.data_ptr(), _stream()), "path_probs")
    return prob, gap, lp


def block_acceptance(ids: torch.Tensor, tokens: torch.Tensor, truth: torch.Tensor):
    """Coverage [B, L], oracle prefix [B] and accepted prefix length [B] (int32) of chosen
    tokens against ground-truth tokens."""
    B, L, K = ids.shape
    for t, n in ((ids, "ids"), (tokens, "tokens"), (truth, "truth")):
        _dev(t, n)
    covered = torch.empty((B, L), dtype=torch.int32, device=ids.device)
    prefix = torch.empty((B,), dtype=torch.int32, device=ids.device)
    acc = torch.empty_like(prefix)
    _check(lib().lilicorr_block_acceptance(B, L, K, ids.data_ptr(), tokens.data_ptr(),
                                           truth.data_ptr(), covered.data_ptr(), prefix.data_ptr(),
                                           acc.data_ptr(), _stream()), "block_acceptance")
    return covered, prefix, acc


def select_block(head: Head, logits: torch.Tensor, hidden: torch.Tensor, target: torch.Tensor,
                 ws: Optional[Workspace] = None, tokens: Optional[torch.Tensor] = None,
                 walk: str = "greedy"):
    """The fused path: logits [B, L, V], hidden [B, L, H], target [B, n_tgt, H] (head dtype,
    on the device) -> chosen token ids [B, L] int32. walk: "greedy" (Sec. 3.5) or
    "viterbi" (the exact best path, App. E)."""
    B = logits.shape[0]
    for t, n in ((logits, "logits"), (hidden, "hidden"), (target, "target")):
        _dev(t, n)
        if t.dtype != head.torch_dtype:
            raise ValueError(f"{n} dtype must match the head dtype")
    ws = ws or head.workspace(B)
    if tokens is None:
        tokens = torch.empty((B, head.L), dtype=torch.int32, device=logits.device)
    if walk == "greedy":
        _check(lib().lilicorr_select_block(head._h, B, logits.data_ptr(), hidden.data_ptr(),
                                           target.data_ptr(), tokens.data_ptr(), ws.ptr,
                                           ws.nbytes, _stream()), "select_block")
    else:
        _check(lib().lilicorr_select_block_walk(head._h, B, logits.data_ptr(), hidden.data_ptr(),
                                                target.data_ptr(), WALKS[walk], tokens.data_ptr(),
                                                ws.ptr, ws.nbytes, _stream()), "select_block_walk")
    return tokens


def test_linear(A: torch.Tensor, W: torch.Tensor, out_dtype=torch.float32, bias=None,
                residual=None, act: int = 0, path: int = 0, status: Optional[torch.Tensor] = None):
    """Test hook: one linear layer C = act(A W^T + bias) + residual through kernel `path`
    (0 auto, 1 tiled CUDA cores, 2 few-row CUDA cores, 3 tensor cores, 4 tensor cores for one
    tile of rows, 5 row-block CUDA cores for fp32 A)."""
    M, Kd = A.shape
    N = W.shape[0]
    C = torch.empty((M, N), dtype=out_dtype, device=A.device)
    _check(lib().lilicorr_test_linear(A.data_ptr(), _dtype_code(A), A.stride(0), W.data_ptr(),
                                      _dtype_code(W), W.stride(0), C.data_ptr(), _dtype_code(C),
                                      C.stride(0), M, N, Kd, _ptr(bias), _ptr(residual), act,
                                      path, _ptr(status), _stream()), "test_linear")
    return C


def test_linear_timeout(A: torch.Tensor, W: torch.Tensor, wait_cycles: int,
                        status: torch.Tensor) -> torch.Tensor:
    """Test hook: the tensor-core linear layer with its copies withheld, so its bounded
    waits run out after ``wait_cycles`` SM cycles and it records the timeout status in
    ``status`` (a device int32/uint32 word) instead of hanging. Returns C (unspecified)."""
    M, Kd = A.shape
    N = W.shape[0]
    C = torch.empty((M, N), dtype=torch.float32, device=A.device)
    _check(lib().lilicorr_test_linear_timeout(A.data_ptr(), W.data_ptr(), C.data_ptr(), M, N, Kd,
                                              int(wait_cycles), status.data_ptr(), _stream()),
           "test_linear_timeout")
    return C


def test_attention_path(mode: int) -> int:
    """Test hook: the chain's attention core on tcgen05 where supported (1), on the
    mma.sync kernel (0), or by shape (2, the default); returns the previous mode."""
    return int(lib().lilicorr_test_attention_path(int(mode)))


def test_fused_path(head: Optional[Head], mode: int) -> bool:
    """Test hook: the fused scoring-network kernel for every head in the process is used
    never (0), from 8 sequences on (1, the default) or always (2); returns whether
    ``head`` can take it."""
    h = head._h if head is not None else _P()
    return bool(lib().lilicorr_test_fused_path(h, int(mode)))


def select_block_intermediates(head: Head, B: int, ws: Workspace) -> Dict[str, torch.Tensor]:
    """Views of the last select_block call's intermediates inside ``ws``."""
    ptrs = [_P() for _ in range(6)]
    _check(lib().lilicorr_select_block_intermediates(head._h, B, ws.ptr, ws.nbytes,
                                                     *[ctypes.byref(p) for p in ptrs]),
           "select_block_intermediates")
    base = ws.buf.data_ptr()
    L, K = head.L, head.K

    def view(p, shape, dtype):
        n = int(np.prod(shape))
        off = p.value - base
        es = 4
        return ws.buf[off: off + n * es].view(dtype).reshape(shape)

    return {"ids": view(ptrs[0], (B, L, K), torch.int32),
            "logp": view(ptrs[1], (B, L, K), torch.float32),
            "lse": view(ptrs[2], (B, L), torch.float32),
            "A": view(ptrs[3], (B, K), torch.float32),
            "P": view(ptrs[4], (B, max(L - 1, 0), K, K), torch.float32),
            "choice": view(ptrs[5], (B, L), torch.int32)}
