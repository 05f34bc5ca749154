"""Pins of the oracle's scoring network (Sec. 3.2; App. A; Table "hparams").

The network's values are parity unpinned against any paper number (no weights or
worked example are published). What is pinned: the architecture, by the
parameter counts the paper prints; each component, by an independent library
implementation (torch RMSNorm, multi-head attention, SiLU); and structural
properties the paper states (shared hidden term per slot, bidirectional
attention, unit-norm out/in vectors, cosine range)."""
import json
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as Fn

import oracle
import workloads

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def test_param_count_matches_paper():
    g = json.load(open(os.path.join(GOLD, "param_counts.json")))
    for c in g["cases"]:
        n = oracle.param_count(c["H"], c["D"], c["d"], c["F"], c["n_heads"], c["L"], c["K"],
                               c["n_layers"])
        assert round(n / 1e6, 2) == c["millions"], n


def test_alternative_readings_miss_the_paper_count():
    # a gated FFN, concatenated target layers or bias-free linears all miss 36.76M
    base = oracle.param_count(4096, 1024, 1024, 2048, 8, 15, 8)
    gated = base + 2 * (1024 * 2048 + 2048)
    concat5 = base + 4 * 4096 * 1024 + 4 * 4096
    n_lin_bias = 4 + 2 + 2 * 6 + 1 + 3
    assert round(base / 1e6, 2) == 36.76
    for alt in (gated, concat5):
        assert round(alt / 1e6, 2) != 36.76
    assert round((base - n_lin_bias * 1024 - 2 * 1024) / 1e6, 2) != 36.76


def test_generator_shapes_follow_oracle_architecture():
    for name in workloads.WORKLOAD_ORDER:
        wl = workloads.WORKLOADS[name]
        gen = dict(workloads.head_param_shapes(wl.H, wl.D, wl.d, wl.F, wl.n_heads, wl.L, wl.K))
        want = oracle.param_shapes(wl.H, wl.D, wl.d, wl.F, wl.n_heads, wl.L, wl.K)
        assert gen == want


def test_confidence_features_golden():
    g = json.load(open(os.path.join(GOLD, "conf_features.json")))
    f = oracle.confidence_features(np.array(g["logp"]))
    assert np.allclose(f, np.array(g["features"]), atol=1e-15)
    f1 = oracle.confidence_features(np.array([-0.7]))
    assert np.allclose(f1, [[-0.7, np.exp(-0.7), 0.0, 0.0, 1.0]])


def test_rms_norm_matches_torch():
    rng = np.random.default_rng(0)
    x = rng.standard_normal((9, 64)) * 3
    g = 1 + 0.1 * rng.standard_normal(64)
    want = Fn.rms_norm(torch.from_numpy(x), (64,), weight=torch.from_numpy(g), eps=1e-6)
    assert np.allclose(oracle.rms_norm(x, g), want.numpy(), atol=1e-13)


def test_silu_matches_torch():
    z = np.linspace(-30, 30, 1001)
    assert np.allclose(oracle.silu(z), Fn.silu(torch.from_numpy(z)).numpy(), atol=1e-14)


def _rand_layer(rng, D, nh, L, scale=0.3):
    W = {}
    for n in ("wq", "wk", "wv", "wo"):
        W["l0." + n] = rng.standard_normal((D, D)) * scale
    for n in ("bq", "bk", "bv", "bo"):
        W["l0." + n] = rng.standard_normal(D) * scale
    W["l0.dist"] = rng.standard_normal((nh, 2 * L - 1))
    W["l0.same"] = rng.standard_normal(nh)
    return W


def test_attention_matches_torch_multi_head_attention():
    rng = np.random.default_rng(1)
    L, K, D, nh = 5, 3, 32, 8
    N = L * K
    W = _rand_layer(rng, D, nh, L)
    x = rng.standard_normal((N, D))
    got = oracle.attention(x, W, "l0.", L, K, nh)
    slot = np.arange(N) // K
    mask = np.zeros((nh, N, N))
    for h in range(nh):
        for i in range(N):
            for j in range(N):
                mask[h, i, j] = W["l0.dist"][h, slot[j] - slot[i] + L - 1] + \
                    (W["l0.same"][h] if slot[i] == slot[j] else 0.0)
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a))
    xq = t(x)[:, None, :]
    want, _ = Fn.multi_head_attention_forward(
        xq, xq, xq, D, nh,
        in_proj_weight=t(np.concatenate([W["l0.wq"], W["l0.wk"], W["l0.wv"]])),
        in_proj_bias=t(np.concatenate([W["l0.bq"], W["l0.bk"], W["l0.bv"]])),
        bias_k=None, bias_v=None, add_zero_attn=False, dropout_p=0.0,
        out_proj_weight=t(W["l0.wo"]), out_proj_bias=t(W["l0.bo"]),
        training=False, need_weights=False, attn_mask=t(mask))
    assert np.allclose(got, want[:, 0, :].numpy(), atol=1e-11)


def test_attention_is_bidirectional_and_bias_sensitive():
    rng = np.random.default_rng(2)
    L, K, D, nh = 4, 2, 16, 8
    W = _rand_layer(rng, D, nh, L)
    x = rng.standard_normal((L * K, D))
    y = oracle.attention(x, W, "l0.", L, K, nh)
    x2 = x.copy()
    x2[-1] += 1.0                                  # last node of the last slot
    y2 = oracle.attention(x2, W, "l0.", L, K, nh)
    assert not np.allclose(y[0], y2[0])            # first node sees it: no causal mask
    W2 = dict(W)
    W2["l0.dist"] = W["l0.dist"].copy()
    W2["l0.dist"][:, L - 1 + 2] += 1.0             # only pairs with s_j - s_i = +2
    y3 = oracle.attention(x, W2, "l0.", L, K, nh)
    assert not np.allclose(y[0], y3[0])            # slot 0 has a slot 2 to its right
    assert np.allclose(y[-1], y3[-1])              # last slot has no slot at +2


def _tiny():
    wl = workloads.WORKLOADS["tiny_f32"]
    W = workloads.head_weights(wl)
    inp = workloads.sequence_inputs(wl, wl.seeds()[0])
    emb = lambda ids: workloads.embed_rows(wl.V, wl.H, wl.dtype, ids)
    return wl, W, inp, emb


def test_hidden_term_is_shared_by_the_slot():
    wl, W, inp, emb = _tiny()
    L, K = 3, wl.K
    ids = np.tile(np.arange(K), (L, 1))
    logp = np.tile(-np.arange(K, dtype=float), (L, 1))
    E = emb(ids.reshape(-1)).reshape(L, K, -1)
    Wd = {k: v.astype(np.float64) for k, v in W.items()}
    h = inp["hidden"][:L].astype(np.float64)
    n1 = oracle.nodes(ids, logp, h, E, Wd).reshape(L, K, -1)
    n2 = oracle.nodes(ids, logp, h + 1.0, E, Wd).reshape(L, K, -1)
    diff = n2 - n1
    assert np.allclose(diff, diff[:, :1, :])                     # same shift for all K
    assert np.allclose(diff[0, 0], Wd["hid_w"].sum(axis=1))      # = W_h applied to ones


def test_tiny_workload_end_to_end_properties():
    wl, W, inp, emb = _tiny()
    r = oracle.select_sequence(inp["logits"], inp["hidden"], inp["target"], emb, W, wl.K)
    assert r["tokens"].shape == (wl.L,)
    for s in range(wl.L):
        assert r["tokens"][s] == r["ids"][s, r["choice"][s]]
    assert np.allclose(np.linalg.norm(r["out"], axis=-1), 1)
    assert np.allclose(np.linalg.norm(r["in"], axis=-1), 1)
    assert abs(np.linalg.norm(r["anchor"]) - 1) < 1e-12
    assert np.all(np.abs(r["P"]) <= 1) and np.all(np.abs(r["A"]) <= 1)
    # brute force over all K^L = 4^8 paths: greedy = lexicographic maximiser, Viterbi = max
    A, P = r["A"], r["P"]
    best_vec, best_path = None, None
    gmax = -np.inf
    import itertools
    for c in itertools.product(range(wl.K), repeat=wl.L):
        vec = [A[c[0]]] + [P[s - 1, c[s - 1], c[s]] for s in range(1, wl.L)]
        if best_vec is None or vec > best_vec:
            best_vec, best_path = vec, c
        gmax = max(gmax, oracle.SIGMA * sum(vec))
    assert tuple(r["choice"]) == best_path
    _, gv = oracle.viterbi(A, P)
    assert abs(gv - gmax) < 1e-9


def test_fusion_with_zero_target_reduces_to_first_block():
    rng = np.random.default_rng(3)
    D, d, L, K = 8, 6, 2, 2
    W = {"fuse_w": rng.standard_normal((D, 3 * D)), "fuse_b": rng.standard_normal(D),
         "out_w": rng.standard_normal((d, D)), "out_b": rng.standard_normal(d),
         "in_w": rng.standard_normal((d, D)), "in_b": rng.standard_normal(d),
         "anc_w": rng.standard_normal((d, D)), "anc_b": rng.standard_normal(d)}
    x = rng.standard_normal((L * K, D))
    out, inn, anc = oracle.fuse_and_heads(x, np.zeros(D), W, L, K)
    u = Fn.silu(Fn.linear(torch.from_numpy(x), torch.from_numpy(W["fuse_w"][:, :D]),
                          torch.from_numpy(W["fuse_b"]))).numpy()
    o = u @ W["out_w"].T + W["out_b"]
    assert np.allclose(out.reshape(L * K, d), o / np.linalg.norm(o, axis=1, keepdims=True))
    a = W["anc_b"] / np.linalg.norm(W["anc_b"])
    assert np.allclose(anc, a)


def test_transformer_matches_torch_encoder_stack():
    """The whole pre-norm stack (App. A) against torch's own encoder layers with RMSNorm
    swapped in, SiLU as the FFN activation and the bias tables as a per-head additive mask:
    pins the order of norm, residual and FFN that the per-component pins leave open."""
    rng = np.random.default_rng(4)
    L, K, D, F, nh, nl = 4, 3, 32, 64, 8, 2
    N = L * K
    W = {}
    for i in range(nl):
        p = f"l{i}."
        for n in ("wq", "wk", "wv", "wo"):
            W[p + n] = rng.standard_normal((D, D)) * 0.3
        for n in ("bq", "bk", "bv", "bo", "b2"):
            W[p + n] = rng.standard_normal(D) * 0.3
        W[p + "w1"] = rng.standard_normal((F, D)) * 0.3
        W[p + "b1"] = rng.standard_normal(F) * 0.3
        W[p + "w2"] = rng.standard_normal((D, F)) * 0.3
        W[p + "an"] = 1 + 0.2 * rng.standard_normal(D)
        W[p + "fn"] = 1 + 0.2 * rng.standard_normal(D)
        W[p + "dist"] = rng.standard_normal((nh, 2 * L - 1))
        W[p + "same"] = rng.standard_normal(nh)
    W["final_norm"] = 1 + 0.2 * rng.standard_normal(D)
    x = rng.standard_normal((N, D))
    got = oracle.transformer(x, W, L, K, nh, nl)

    t = lambda a: torch.from_numpy(np.ascontiguousarray(a))
    slot = np.arange(N) // K
    rel = slot[None, :] - slot[:, None] + L - 1
    y = t(x)[None]
    with torch.no_grad():
        for i in range(nl):
            p = f"l{i}."
            layer = torch.nn.TransformerEncoderLayer(D, nh, F, dropout=0.0, activation=Fn.silu,
                                                     batch_first=True, norm_first=True)
            layer.norm1 = torch.nn.RMSNorm(D, eps=1e-6)
            layer.norm2 = torch.nn.RMSNorm(D, eps=1e-6)
            layer = layer.double().eval()
            layer.self_attn.in_proj_weight.copy_(t(np.concatenate([W[p + "wq"], W[p + "wk"],
                                                                   W[p + "wv"]])))
            layer.self_attn.in_proj_bias.copy_(t(np.concatenate([W[p + "bq"], W[p + "bk"],
                                                                 W[p + "bv"]])))
            layer.self_attn.out_proj.weight.copy_(t(W[p + "wo"]))
            layer.self_attn.out_proj.bias.copy_(t(W[p + "bo"]))
            layer.linear1.weight.copy_(t(W[p + "w1"]))
            layer.linear1.bias.copy_(t(W[p + "b1"]))
            layer.linear2.weight.copy_(t(W[p + "w2"]))
            layer.linear2.bias.copy_(t(W[p + "b2"]))
            layer.norm1.weight.copy_(t(W[p + "an"]))
            layer.norm2.weight.copy_(t(W[p + "fn"]))
            mask = W[p + "dist"][:, rel] + W[p + "same"][:, None, None] * (rel == L - 1)
            y = layer(y, src_mask=t(mask))
        fin = torch.nn.RMSNorm(D, eps=1e-6).double()
        fin.weight.copy_(t(W["final_norm"]))
        want = fin(y)[0].numpy()
    assert np.allclose(got, want, atol=1e-11)


def _zero_node_weights(H, D, L, K):
    return {"emb_w": np.zeros((D, H)), "emb_b": np.zeros(D), "hid_w": np.zeros((D, H)),
            "hid_b": np.zeros(D), "conf1_w": np.zeros((D, 5)), "conf1_b": np.zeros(D),
            "conf2_w": np.zeros((D, D)), "conf2_b": np.zeros(D), "slot": np.zeros((L, D)),
            "rank": np.zeros((K, D))}


def test_nodes_decompose_into_the_four_terms():
    """Sec. 3.2: each node is the sum of four terms. Switching all but one family of
    weights off isolates each term, so a swapped slot/rank index, a token paired with the
    wrong embedding row or a missing SiLU in the confidence network fails here."""
    rng = np.random.default_rng(5)
    H, D, L, K = 12, 6, 3, 4                        # L != K so slot and rank cannot swap
    ids = rng.integers(0, 50, (L, K))
    logp = -np.sort(rng.random((L, K)) * 4, axis=1)
    hidden = rng.standard_normal((L, H))
    E = rng.standard_normal((L, K, H))
    base = _zero_node_weights(H, D, L, K)

    W = dict(base, slot=rng.standard_normal((L, D)), rank=rng.standard_normal((K, D)))
    n = oracle.nodes(ids, logp, hidden, E, W).reshape(L, K, D)
    assert np.allclose(n, W["slot"][:, None, :] + W["rank"][None, :, :], atol=0)

    W = dict(base, emb_w=rng.standard_normal((D, H)), emb_b=rng.standard_normal(D))
    n = oracle.nodes(ids, logp, hidden, E, W).reshape(L, K, D)
    for s in range(L):
        for k in range(K):
            assert np.allclose(n[s, k], W["emb_w"] @ E[s, k] + W["emb_b"])

    W = dict(base, conf1_w=rng.standard_normal((D, 5)), conf1_b=rng.standard_normal(D),
             conf2_w=rng.standard_normal((D, D)), conf2_b=rng.standard_normal(D))
    n = oracle.nodes(ids, logp, hidden, E, W).reshape(L, K, D)
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a))
    mlp = torch.nn.Sequential(torch.nn.Linear(5, D), torch.nn.SiLU(),
                              torch.nn.Linear(D, D)).double()
    with torch.no_grad():
        mlp[0].weight.copy_(t(W["conf1_w"])); mlp[0].bias.copy_(t(W["conf1_b"]))
        mlp[2].weight.copy_(t(W["conf2_w"])); mlp[2].bias.copy_(t(W["conf2_b"]))
        for s in range(L):
            lp = logp[s]
            feats = np.stack([lp, np.exp(lp), lp[0] - lp, np.arange(K) / (K - 1),
                              (np.arange(K) == 0).astype(float)], axis=1)
            assert np.allclose(n[s], mlp(t(feats)).numpy(), atol=1e-13)


def test_target_state_reads_the_mean_of_the_captured_layers():
    """App. A: the five captured target layers are averaged before the RMSNorm over H, so
    their order does not matter, a uniform positive scale cancels in the norm (up to its
    epsilon), and five equal layers reduce to one."""
    rng = np.random.default_rng(6)
    H, D = 16, 8
    W = {"tgt_norm": 1 + 0.1 * rng.standard_normal(H), "tgt_w": rng.standard_normal((D, H)),
         "tgt_b": rng.standard_normal(D)}
    T = rng.standard_normal((5, H))
    t0 = oracle.target_state(T, W)
    assert np.allclose(oracle.target_state(T[::-1], W), t0, atol=1e-13)
    assert np.allclose(oracle.target_state(7.0 * T, W), t0, atol=1e-6)
    one = T[2]
    want = W["tgt_w"] @ (one / np.sqrt(np.mean(one * one) + 1e-6) * W["tgt_norm"]) + W["tgt_b"]
    assert np.allclose(oracle.target_state(np.tile(one, (5, 1)), W), want, atol=1e-12)
    # the mean, not the first or last layer: moving one layer moves t
    T2 = T.copy()
    T2[4] += 1.0
    assert not np.allclose(oracle.target_state(T2, W), t0)


def test_heads_are_scale_free_and_the_anchor_ignores_the_nodes():
    """Sec. 3.2: out/in vectors are unit-normalised, so a positive scale of a head's
    weights and bias leaves them unchanged; the anchor's vector depends on t alone."""
    rng = np.random.default_rng(7)
    D, d, L, K = 8, 6, 3, 2
    W = {"fuse_w": rng.standard_normal((D, 3 * D)), "fuse_b": rng.standard_normal(D),
         "out_w": rng.standard_normal((d, D)), "out_b": rng.standard_normal(d),
         "in_w": rng.standard_normal((d, D)), "in_b": rng.standard_normal(d),
         "anc_w": rng.standard_normal((d, D)), "anc_b": rng.standard_normal(d)}
    x = rng.standard_normal((L * K, D))
    t = rng.standard_normal(D)
    out, inn, anc = oracle.fuse_and_heads(x, t, W, L, K)
    W2 = dict(W, out_w=3 * W["out_w"], out_b=3 * W["out_b"], in_w=0.5 * W["in_w"],
              in_b=0.5 * W["in_b"])
    out2, inn2, anc2 = oracle.fuse_and_heads(x, t, W2, L, K)
    assert np.allclose(out, out2, atol=1e-14) and np.allclose(inn, inn2, atol=1e-14)
    _, _, anc3 = oracle.fuse_and_heads(rng.standard_normal((L * K, D)), t, W, L, K)
    assert np.allclose(anc, anc3, atol=0)
    # the x*t block: with x = 0 only the t block and bias remain, the same for every node
    out0, _, _ = oracle.fuse_and_heads(np.zeros((L * K, D)), t, W, L, K)
    u = Fn.silu(torch.from_numpy(W["fuse_w"][:, D:2 * D] @ t + W["fuse_b"])).numpy()
    o = W["out_w"] @ u + W["out_b"]
    assert np.allclose(out0.reshape(L * K, d), o / np.linalg.norm(o))
