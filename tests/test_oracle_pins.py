"""Pins of the fp64 oracle against what the paper and the mathematics fix.

Nothing here compares the oracle with itself: each check is a closed form, a
special case that reduces to a textbook or library routine (numpy / scipy),
brute-force enumeration on tiny inputs, an invariant stated in the paper
(Sec. 3.2 losslessness, mask sums) or a value the paper prints (Tables 1, 3).
"""
import itertools
import math
import os

import numpy as np
import pytest
import scipy.special

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "kv_fractions.txt")


def haar(rng, n):
    q, r = np.linalg.qr(rng.standard_normal((n, n)))
    return q * np.sign(np.diag(r))[None, :]


def rnd_problem(rng, H=2, dh=16, G=4, C=3, F=8, n_tok=((5, 3, 0, 0),), k=((4, 4, 4, 4),), n_q=(4,),
                R=None):
    E = len(n_tok)
    d = H * dh
    rows = int(np.sum(n_tok))
    qrows = int(np.sum(n_q))
    p = dict(H=H, dh=dh, G=G, C=C, F=F, n_tok=np.array(n_tok), k=np.array(k), n_q=np.array(n_q))
    p["h"] = rng.standard_normal((rows, d))
    p["v"] = rng.standard_normal((rows, d))
    p["K"] = rng.standard_normal((rows, d))
    p["q"] = rng.standard_normal((qrows, d))
    p["R"] = np.stack([haar(rng, dh) for _ in range(H)]) if R is None else R
    p["W_re"] = 0.3 * rng.standard_normal((C, d))
    p["b_re"] = 0.3 * rng.standard_normal(C)
    p["W1"] = 0.3 * rng.standard_normal((F, 2 * d + C))
    p["b1"] = 0.3 * rng.standard_normal(F)
    p["W2"] = 0.3 * rng.standard_normal((G, F))
    p["b2"] = 0.3 * rng.standard_normal(G)
    p["E"] = E
    return p


def run(oracle, p, alpha_role=0.1, alpha_lang=0.1, idx_force=None, scale=0.0):
    spec = oracle.Spec(p["H"], p["dh"], p["G"], p["C"], p["F"], p["n_tok"], p["k"], p["n_q"])
    c = oracle.compress_layer(spec, p["h"], p["v"], p["R"], p["W_re"], p["b_re"], p["W1"], p["b1"],
                              p["W2"], p["b2"], alpha_role, alpha_lang, idx_force=idx_force)
    o = oracle.attend_layer(spec, p["q"], p["K"], c["packed"], c["idx"], p["R"], scale=scale)
    return spec, c, o


def dense_attention(p, vtil_fn=None, scale=None):
    """Textbook softmax(q K^T * scale) V per episode and head, numpy only."""
    H, dh = p["H"], p["dh"]
    scale = 1.0 / math.sqrt(dh) if scale is None else scale
    ep_row = np.concatenate([[0], np.cumsum(np.sum(p["n_tok"], 1))])
    ep_q = np.concatenate([[0], np.cumsum(p["n_q"])])
    o = np.zeros_like(p["q"])
    for e in range(p["E"]):
        r0, r1 = ep_row[e], ep_row[e + 1]
        q0, q1 = ep_q[e], ep_q[e + 1]
        for h in range(H):
            sl = slice(h * dh, (h + 1) * dh)
            if r1 == r0:
                continue
            s = p["q"][q0:q1, sl] @ p["K"][r0:r1, sl].T * scale
            P = scipy.special.softmax(s, axis=1)
            V = p["v"][r0:r1, sl] if vtil_fn is None else vtil_fn(e, h, r0, r1)
            o[q0:q1, sl] = P @ V
    return o


def rel_err(a, b, dh):
    """max |a-b| per (row, head) relative to the row norm of b."""
    a = a.reshape(a.shape[0], -1, dh)
    b = b.reshape(b.shape[0], -1, dh)
    nrm = np.linalg.norm(b, axis=2, keepdims=True)
    return float(np.max(np.abs(a - b) / np.maximum(nrm, 1e-300)))


# ---------------------------------------------------------------------------
# Layout and accounting
# ---------------------------------------------------------------------------

def test_layout_offsets_hand_computed(oracle):
    n_tok = [[3, 2, 0, 0], [1, 0, 0, 2]]
    k = [[2, 4, 4, 4], [0, 4, 1, 4]]
    lay = oracle.layout(n_tok, k, H=2, dh=8, G=4)   # d_s = 2
    # packed sizes H*n*k*ds: 24, 32, 0, 0 | 0, 0, 0, 32
    assert list(lay["packed_off"]) == [0, 24, 56, 56, 56, 56, 56, 56]
    assert lay["packed_elems"] == 88
    assert list(lay["idx_off"]) == [0, 6, 14, 14, 14, 14, 14, 14]
    assert lay["idx_bytes"] == 22
    assert list(lay["row_off"]) == [0, 3, 5, 5, 5, 6, 6, 6]
    assert lay["rows"] == 8


def half_up(x, nd=2):
    """Round half away from zero, the way the paper's tables print."""
    f = 10 ** nd
    return math.floor(x * f + 0.5 + 1e-9) / f


def _golden():
    vis, lang = [], []
    for line in open(GOLDEN):
        line = line.split("#")[0].split()
        if not line:
            continue
        if line[0] == "vis":
            vis.append((int(line[1]), int(line[2]), int(line[3]), float(line[4])))
        else:
            lang.append((int(line[1]), float(line[2]), float(line[3])))
    return vis, lang


def test_kv_fractions_reproduce_tables_1_and_3(oracle):
    H, dh, G = 32, 128, 16
    d = H * dh
    vis, lang = _golden()
    assert len(vis) == 9 and len(lang) == 4
    for n_keep, n_total, K, pct in vis:
        lay = oracle.layout([[n_keep, 0, 0, 0]], [[K, G, G, G]], H, dh, G)
        kv = (n_keep * d + lay["packed_elems"]) / (2.0 * n_total * d)
        assert half_up(100 * kv) == pytest.approx(pct, abs=1e-9), (n_keep, K)
    for K, vpct, kvpct in lang:
        n = 40
        lay = oracle.layout([[0, n, 0, 0]], [[G, K, G, G]], H, dh, G)
        v_frac = lay["packed_elems"] / (n * d)
        kv = (n * d + lay["packed_elems"]) / (2.0 * n * d)
        assert half_up(100 * v_frac) == pytest.approx(vpct, abs=1e-9)
        assert half_up(100 * kv) == pytest.approx(kvpct, abs=1e-9)


# ---------------------------------------------------------------------------
# Router pieces
# ---------------------------------------------------------------------------

def test_lang_pool_mean_closed_form(oracle):
    n, d = 7, 5
    h = np.arange(1, n + 1, dtype=float)[:, None] * np.ones((1, d))
    assert np.array_equal(oracle.lang_pool(h), np.full(d, (n + 1) / 2.0))
    assert np.array_equal(oracle.lang_pool(np.zeros((0, d))), np.zeros(d))


def test_role_is_softmax(oracle):
    rng = np.random.default_rng(1)
    C, d = 16, 40
    W = rng.standard_normal((C, d))
    b = rng.standard_normal(C)
    h = rng.standard_normal(d)
    a = oracle.role(W, b, h)
    ref = scipy.special.softmax(W @ h + b)
    assert np.max(np.abs(a - ref)) < 1e-15
    assert abs(a.sum() - 1.0) < 1e-14
    # zero network -> uniform role vector, exactly 1/C
    assert np.array_equal(oracle.role(np.zeros((C, d)), np.zeros(C), h), np.full(C, 1.0 / C))
    # large logits do not overflow (max-subtracted)
    a = oracle.role(W * 1e4, b, h)
    assert np.all(np.isfinite(a)) and abs(a.sum() - 1.0) < 1e-12


def test_router_token_block_alone(oracle):
    rng = np.random.default_rng(2)
    d, C = 6, 3
    F = G = d
    W1 = np.zeros((F, 2 * d + C))
    W1[:, :d] = np.eye(d)
    h = rng.standard_normal(d)
    g = oracle.router_score(W1, np.zeros(F), np.eye(G), np.zeros(G), h, rng.random(C),
                            rng.standard_normal(d), 0.7, 0.9)
    assert np.array_equal(g, np.maximum(h, 0.0))


def test_router_role_block_alone(oracle):
    rng = np.random.default_rng(3)
    d, C = 6, 4
    F = G = C
    W1 = np.zeros((F, 2 * d + C))
    W1[:, d:d + C] = np.eye(C)
    W_re = rng.standard_normal((C, d))
    b_re = rng.standard_normal(C)
    h = rng.standard_normal(d)
    a = oracle.role(W_re, b_re, h)
    g = oracle.router_score(W1, np.zeros(F), np.eye(G), np.zeros(G), h, a, rng.standard_normal(d),
                            0.25, 0.9)
    assert np.max(np.abs(g - 0.25 * scipy.special.softmax(W_re @ h + b_re))) < 1e-16


def test_router_language_block_alone(oracle):
    rng = np.random.default_rng(4)
    d, C = 6, 3
    F = G = d
    W1 = np.zeros((F, 2 * d + C))
    W1[:, d + C:] = np.eye(d)
    h_lang = rng.random((5, d)) + 0.1      # positive: ReLU is the identity
    c = oracle.lang_pool(h_lang)
    g = oracle.router_score(W1, np.zeros(F), np.eye(G), np.zeros(G), rng.standard_normal(d),
                            rng.random(C), c, 0.7, 0.125)
    assert np.max(np.abs(g - 0.125 * h_lang.mean(0))) < 1e-16


def test_router_biases_and_output_layer(oracle):
    rng = np.random.default_rng(5)
    d, C, F, G = 4, 2, 5, 3
    W1 = np.zeros((F, 2 * d + C))
    b1 = np.array([1.0, -2.0, 0.5, -0.1, 3.0])
    W2 = rng.standard_normal((G, F))
    b2 = rng.standard_normal(G)
    g = oracle.router_score(W1, b1, W2, b2, rng.standard_normal(d), rng.random(C),
                            rng.standard_normal(d), 0.1, 0.1)
    u = np.array([1.0, 0.0, 0.5, 0.0, 3.0])           # ReLU(b1) by hand
    assert np.max(np.abs(g - (W2 @ u + b2))) < 1e-15


# ---------------------------------------------------------------------------
# Top-K_i selection
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("G", [4, 8])
def test_topk_equals_best_subset_brute_force(oracle, G):
    rng = np.random.default_rng(G)
    for _ in range(50):
        gam = rng.standard_normal(G)
        for k in range(G + 1):
            idx, margin = oracle.topk(gam, k)
            best = max(itertools.combinations(range(G), k), key=lambda s: sum(gam[list(s)]))
            assert tuple(idx) == tuple(sorted(best))
            assert list(idx) == sorted(idx) and len(set(idx)) == k
            srt = np.sort(gam)[::-1]
            if 0 < k < G:
                assert margin == srt[k - 1] - srt[k]
            else:
                assert margin == math.inf


def test_topk_near_ties(oracle):
    # exact ties: the lower group index wins
    idx, m = oracle.topk(np.zeros(16), 4)
    assert list(idx) == [0, 1, 2, 3] and m == 0.0
    g = np.array([0.5, 0.5 + 5e-5, 0.3, 0.5 + 2e-4, 0.5 + 5e-5, -1.0])
    idx, m = oracle.topk(g, 1)
    assert list(idx) == [3] and m == pytest.approx(1.5e-4, abs=1e-15)
    idx, m = oracle.topk(g, 2)            # tie between 1 and 4 -> 1
    assert list(idx) == [1, 3] and m == 0.0
    idx, m = oracle.topk(g, 3)
    assert list(idx) == [1, 3, 4] and m == pytest.approx(5e-5, abs=1e-15)


# ---------------------------------------------------------------------------
# Rotation (Sec. 3.2)
# ---------------------------------------------------------------------------

def test_rotate_is_transpose_product(oracle):
    dh = 8
    R = np.zeros((dh, dh))
    for m in range(dh):
        R[m, (m + 1) % dh] = 1.0          # a cyclic permutation (not symmetric)
    v = np.arange(dh, dtype=float) + 1
    # z = R^T v: z_n = v_{n-1}
    assert np.array_equal(oracle.rotate(R, v), np.roll(v, 1))


def test_rotate_preserves_norm(oracle):
    rng = np.random.default_rng(6)
    dh, G = 64, 8
    R = haar(rng, dh)
    v = rng.standard_normal(dh)
    z = oracle.rotate(R, v)
    assert abs(np.linalg.norm(z) - np.linalg.norm(v)) < 1e-12
    groups = z.reshape(G, -1)
    assert abs(np.sum(groups ** 2) - v @ v) < 1e-11
    assert np.max(np.abs(R @ z - v)) < 1e-12        # lossless round trip


# ---------------------------------------------------------------------------
# Whole path invariants
# ---------------------------------------------------------------------------

def test_all_groups_kept_equals_dense_attention(oracle):
    rng = np.random.default_rng(7)
    G = 4
    p = rnd_problem(rng, n_tok=((5, 3, 0, 0), (2, 4, 1, 0)), k=((G,) * 4, (G,) * 4), n_q=(4, 3))
    _, c, o = run(oracle, p)
    assert rel_err(o, dense_attention(p), p["dh"]) <= 1e-10


def test_no_groups_kept_gives_zero(oracle):
    rng = np.random.default_rng(8)
    p = rnd_problem(rng, n_tok=((5, 3, 0, 0),), k=((0, 0, 0, 0),), n_q=(4,))
    _, c, o = run(oracle, p)
    assert c["packed"].size == 0 and np.array_equal(o, np.zeros_like(o))


def _vtil(p, idx_of_token):
    """v~_j = R_h M_j R_h^T v_j materialised per token (numpy)."""
    dh, G = p["dh"], p["G"]
    ds = dh // G

    def fn(e, h, r0, r1):
        out = []
        Rh = p["R"][h]
        for r in range(r0, r1):
            m = np.zeros(dh)
            for g in idx_of_token[r]:
                m[g * ds:(g + 1) * ds] = 1.0
            out.append(Rh @ np.diag(m) @ Rh.T @ p["v"][r, h * dh:(h + 1) * dh])
        return np.array(out)
    return fn


def test_every_mask_on_tiny_input_equals_dense_over_routed_values(oracle):
    rng = np.random.default_rng(9)
    G = 4
    for k in range(G + 1):
        p = rnd_problem(rng, H=2, dh=8, G=G, n_tok=((3, 0, 0, 0),), k=((k, G, G, G),), n_q=(2,))
        subsets = list(itertools.combinations(range(G), k))
        for masks in itertools.product(subsets, repeat=3):
            fx = np.array([g for m in masks for g in m], np.uint8)
            _, c, o = run(oracle, p, idx_force=fx)
            ref = dense_attention(p, _vtil(p, {r: masks[r] for r in range(3)}))
            assert np.max(np.abs(o - ref)) <= 1e-12, (k, masks)


def test_complement_masks_sum_to_dense(oracle):
    rng = np.random.default_rng(10)
    G, n = 8, 6
    base = rnd_problem(rng, H=2, dh=16, G=G, n_tok=((n, 0, 0, 0),), n_q=(3,))
    for k in (1, 3, 5):
        sel = [np.sort(rng.choice(G, k, replace=False)) for _ in range(n)]
        comp = [np.setdiff1d(np.arange(G), s) for s in sel]
        p1 = dict(base, k=np.array([[k, G, G, G]]))
        p2 = dict(base, k=np.array([[G - k, G, G, G]]))
        _, _, o1 = run(oracle, p1, idx_force=np.concatenate(sel).astype(np.uint8))
        _, _, o2 = run(oracle, p2, idx_force=np.concatenate(comp).astype(np.uint8))
        assert rel_err(o1 + o2, dense_attention(base), 16) <= 1e-12
    # sum over single-group outputs
    acc = 0
    for g in range(G):
        pg = dict(base, k=np.array([[1, G, G, G]]))
        _, _, og = run(oracle, pg, idx_force=np.full(n, g, np.uint8))
        acc = acc + og
    assert rel_err(acc, dense_attention(base), 16) <= 1e-12


def test_identity_rotation_zeroes_unkept_value_columns(oracle):
    # the paper's "plain" control: R = I, no role term
    rng = np.random.default_rng(11)
    H, dh, G = 2, 16, 4
    ds = dh // G
    p = rnd_problem(rng, H=H, dh=dh, G=G, n_tok=((6, 2, 0, 0),), k=((2, 3, G, G),), n_q=(3,),
                    R=np.stack([np.eye(dh)] * H))
    spec, c, o = run(oracle, p, alpha_role=0.0)
    lay = spec.lay
    kept = {}
    for m in range(2):
        n, k = p["n_tok"][0][m], p["k"][0][m]
        r0 = lay["row_off"][m]
        for i in range(n):
            kept[r0 + i] = c["idx"][lay["idx_off"][m] + i * k: lay["idx_off"][m] + (i + 1) * k]

    def fn(e, h, r0, r1):
        V = p["v"][r0:r1, h * dh:(h + 1) * dh].copy()
        for r in range(r0, r1):
            mask = np.zeros(dh, bool)
            for g in kept[r]:
                mask[g * ds:(g + 1) * ds] = True
            V[r - r0, ~mask] = 0.0
        return V
    assert np.max(np.abs(o - dense_attention(p, fn))) <= 1e-12


def test_attention_weights_are_softmax_of_scaled_scores(oracle):
    # R = I, all kept, v_j = e_j: output column j is p_j
    rng = np.random.default_rng(12)
    H, dh, G, n = 1, 16, 4, 10
    p = rnd_problem(rng, H=H, dh=dh, G=G, n_tok=((n, 0, 0, 0),), k=((G,) * 4,), n_q=(5,),
                    R=np.eye(dh)[None])
    p["v"] = np.eye(dh)[:n]
    for scale in (0.0, 0.37):
        _, _, o = run(oracle, p, scale=scale)
        s = p["q"] @ p["K"].T * (1 / math.sqrt(dh) if scale == 0.0 else scale)
        P = scipy.special.softmax(s, axis=1)
        assert np.max(np.abs(o[:, :n] - P)) < 1e-15
        assert np.max(np.abs(o[:, n:])) == 0.0


def test_token_permutation_invariance(oracle):
    rng = np.random.default_rng(13)
    G = 4
    p = rnd_problem(rng, H=2, dh=16, G=G, n_tok=((7, 3, 0, 0),), k=((2, 1, G, G),), n_q=(4,))
    _, _, o = run(oracle, p)
    perm = np.concatenate([rng.permutation(7), 7 + rng.permutation(3)])
    p2 = dict(p, h=p["h"][perm], v=p["v"][perm], K=p["K"][perm])
    _, _, o2 = run(oracle, p2)
    assert np.max(np.abs(o - o2)) < 1e-12


def test_group_permutation_equivariance(oracle):
    rng = np.random.default_rng(14)
    G, dh, H = 4, 16, 2
    ds = dh // G
    p = rnd_problem(rng, H=H, dh=dh, G=G, n_tok=((7, 3, 0, 0),), k=((2, 1, G, G),), n_q=(4,))
    spec, c, o = run(oracle, p)
    pi = np.array([2, 0, 3, 1])           # new group s holds old group pi[s]
    cols = np.concatenate([np.arange(pi[s] * ds, (pi[s] + 1) * ds) for s in range(G)])
    p2 = dict(p, R=p["R"][:, :, cols], W2=p["W2"][pi], b2=p["b2"][pi])
    _, c2, o2 = run(oracle, p2)
    assert np.max(np.abs(o - o2)) < 1e-12
    # the kept set is relabelled: new group s kept <=> old group pi[s] kept
    lay = spec.lay
    for m in range(2):
        n, k = p["n_tok"][0][m], p["k"][0][m]
        for i in range(n):
            a = c["idx"][lay["idx_off"][m] + i * k: lay["idx_off"][m] + (i + 1) * k]
            b = c2["idx"][lay["idx_off"][m] + i * k: lay["idx_off"][m] + (i + 1) * k]
            assert sorted(pi[b]) == sorted(a)


def test_compress_scores_use_episode_language_mean_only(oracle):
    rng = np.random.default_rng(15)
    G = 8
    p = rnd_problem(rng, H=2, dh=16, G=G, C=3, F=8, n_tok=((4, 3, 0, 0), (2, 5, 0, 0)),
                    k=((3, 2, G, G), (1, 4, G, G)), n_q=(2, 2))
    spec, c, _ = run(oracle, p, alpha_role=0.3, alpha_lang=0.6)
    d = spec.d
    for e in range(2):
        r0 = spec.ep_row[e]
        nv, nl = p["n_tok"][e][0], p["n_tok"][e][1]
        cl = p["h"][r0 + nv:r0 + nv + nl].mean(0)
        for r in range(r0, r0 + nv + nl):
            a = scipy.special.softmax(p["W_re"] @ p["h"][r] + p["b_re"])
            x = np.concatenate([p["h"][r], 0.3 * a, 0.6 * cl])
            g = p["W2"] @ np.maximum(p["W1"] @ x + p["b1"], 0) + p["b2"]
            assert np.max(np.abs(c["gamma"][r] - g)) < 1e-12
    # language-only score of an episode with no language tokens: c = 0
    p0 = rnd_problem(rng, H=2, dh=16, G=G, n_tok=((4, 0, 0, 0),), k=((3, G, G, G),), n_q=(1,))
    _, c0, _ = run(oracle, p0, alpha_role=0.3, alpha_lang=0.6)
    r = 1
    a = scipy.special.softmax(p0["W_re"] @ p0["h"][r] + p0["b_re"])
    x = np.concatenate([p0["h"][r], 0.3 * a, np.zeros(d)])
    g = p0["W2"] @ np.maximum(p0["W1"] @ x + p0["b1"], 0) + p0["b2"]
    assert np.max(np.abs(c0["gamma"][r] - g)) < 1e-12


def test_packed_values_are_rotated_groups(oracle):
    rng = np.random.default_rng(16)
    G, dh, H = 4, 16, 2
    ds = dh // G
    p = rnd_problem(rng, H=H, dh=dh, G=G, n_tok=((5, 2, 0, 0),), k=((2, G, G, G),), n_q=(1,))
    spec, c, _ = run(oracle, p)
    lay = spec.lay
    n, k = 5, 2
    for i in range(n):
        sel = c["idx"][i * k:(i + 1) * k]
        for h in range(H):
            z = p["R"][h].T @ p["v"][i, h * dh:(h + 1) * dh]
            got = c["packed"][((h * n + i) * k) * ds:((h * n + i) * k + k) * ds]
            want = np.concatenate([z[g * ds:(g + 1) * ds] for g in sel])
            assert np.max(np.abs(got - want)) < 1e-12
    # the language segment keeps every group, indices 0..G-1
    assert list(c["idx"][lay["idx_off"][1]:lay["idx_off"][1] + G]) == list(range(G))


def test_empty_cache_gives_zero_output(oracle):
    rng = np.random.default_rng(17)
    p = rnd_problem(rng, n_tok=((0, 0, 0, 0), (3, 1, 0, 0)), k=((2, 2, 4, 4), (2, 2, 4, 4)), n_q=(3, 2))
    _, _, o = run(oracle, p)
    assert np.array_equal(o[:3], np.zeros_like(o[:3]))
    assert np.any(o[3:] != 0)


def test_bad_forced_indices_rejected(oracle):
    rng = np.random.default_rng(18)
    p = rnd_problem(rng, n_tok=((2, 0, 0, 0),), k=((2, 4, 4, 4),), n_q=(1,))
    with pytest.raises(ValueError):
        run(oracle, p, idx_force=np.array([0, 4, 1, 2], np.uint8))   # 4 >= G
    with pytest.raises(ValueError):
        run(oracle, p, idx_force=np.array([1, 1, 1, 2], np.uint8))   # not ascending


# ---------------------------------------------------------------------------
# Additive router (Eq. routingscore as printed, linear scoring heads)
# ---------------------------------------------------------------------------

def test_additive_router_parameter_count_matches_paper():
    # two linear S x d heads with biases (f_v, f_lang) and the S x C role
    # projection, per layer, 32 layers, S = 16, d = 4096, C = 6: the paper
    # reports about 4.20M routing-head parameters (Sec. 4, implementation)
    S, d, C, L = 16, 4096, 6, 32
    per_layer = 2 * (S * d + S) + S * C
    assert round(per_layer * L / 1e6, 2) == 4.20


def _selectors(rng, G, d):
    perm = rng.permutation(d)[:G]
    W = np.zeros((G, d))
    W[np.arange(G), perm] = 1.0
    return W, perm


def test_additive_router_token_term_alone(oracle):
    rng = np.random.default_rng(30)
    d, G, C = 10, 4, 3
    W_v, perm = _selectors(rng, G, d)
    b_v = rng.standard_normal(G)
    h = rng.standard_normal(d)
    g = oracle.router_score_linear(W_v, b_v, rng.standard_normal((G, C)), rng.standard_normal((G, d)),
                                   rng.standard_normal(G), h, rng.random(C), rng.standard_normal(d), 0.0, 0.0)
    assert np.array_equal(g, h[perm] + b_v)


def test_additive_router_role_term_alone(oracle):
    rng = np.random.default_rng(31)
    d, G, C = 10, 6, 3
    # row s of W_role picks role s mod C with weight w_s
    w = rng.standard_normal(G)
    W_role = np.zeros((G, C))
    W_role[np.arange(G), np.arange(G) % C] = w
    a = rng.random(C)
    g = oracle.router_score_linear(np.zeros((G, d)), np.zeros(G), W_role, np.zeros((G, d)), np.zeros(G),
                                   rng.standard_normal(d), a, rng.standard_normal(d), 0.25, 0.7)
    assert np.max(np.abs(g - 0.25 * w * a[np.arange(G) % C])) < 1e-16


def test_additive_router_language_term_alone(oracle):
    rng = np.random.default_rng(32)
    d, G, C = 10, 4, 3
    W_l, perm = _selectors(rng, G, d)
    b_l = rng.standard_normal(G)
    h_lang = rng.standard_normal((5, d))
    c = oracle.lang_pool(h_lang)
    g = oracle.router_score_linear(np.zeros((G, d)), np.zeros(G), rng.standard_normal((G, C)), W_l, b_l,
                                   rng.standard_normal(d), rng.random(C), c, 0.0, 0.125)
    # the language weight scales the head's bias too: alpha_lang * (W_l c + b_l)
    assert np.max(np.abs(g - 0.125 * (h_lang.mean(0)[perm] + b_l))) < 1e-15


def test_additive_router_terms_add(oracle):
    rng = np.random.default_rng(33)
    d, G, C = 12, 4, 3
    W_v, pv = _selectors(rng, G, d)
    W_l, pl = _selectors(rng, G, d)
    w = rng.standard_normal(G)
    W_role = np.zeros((G, C))
    W_role[np.arange(G), np.arange(G) % C] = w
    b_v, b_l = rng.standard_normal(G), rng.standard_normal(G)
    h, c, a = rng.standard_normal(d), rng.standard_normal(d), rng.random(C)
    g = oracle.router_score_linear(W_v, b_v, W_role, W_l, b_l, h, a, c, -0.3, 0.6)
    want = (h[pv] + b_v) - 0.3 * w * a[np.arange(G) % C] + 0.6 * (c[pl] + b_l)
    assert np.max(np.abs(g - want)) < 1e-15


def test_additive_router_compress_keeps_best_subset_and_packs_rotated_groups(oracle):
    rng = np.random.default_rng(34)
    H, dh, G, C = 2, 8, 4, 3
    d = H * dh
    n_tok, k = ((6, 3, 0, 0),), ((2, 1, G, G),)
    p = rnd_problem(rng, H=H, dh=dh, G=G, C=C, F=4, n_tok=n_tok, k=k, n_q=(1,))
    spec = oracle.Spec(H, dh, G, C, 4, p["n_tok"], p["k"], p["n_q"])
    W_v, pv = _selectors(rng, G, d)
    W_role = rng.standard_normal((G, C))
    W_l, pl = _selectors(rng, G, d)
    b_v, b_l = rng.standard_normal(G), rng.standard_normal(G)
    out = oracle.compress_layer_linear(spec, p["h"], p["v"], p["R"], p["W_re"], p["b_re"], W_v, b_v, W_role,
                                       W_l, b_l, 0.2, 0.4)
    cl = p["h"][6:9].mean(0)
    lay = spec.lay
    ds = dh // G
    for r in range(9):
        kk = 2 if r < 6 else 1
        a = scipy.special.softmax(p["W_re"] @ p["h"][r] + p["b_re"])
        gam = (p["h"][r][pv] + b_v) + 0.2 * (W_role @ a) + 0.4 * (cl[pl] + b_l)
        assert np.max(np.abs(out["gamma"][r] - gam)) < 1e-12
        best = max(itertools.combinations(range(G), kk), key=lambda s: sum(gam[list(s)]))
        m, i = (0, r) if r < 6 else (1, r - 6)
        sel = out["idx"][lay["idx_off"][m] + i * kk:lay["idx_off"][m] + (i + 1) * kk]
        assert tuple(sel) == tuple(sorted(best))
        n = 6 if r < 6 else 3
        for hh in range(H):
            z = p["R"][hh].T @ p["v"][r, hh * dh:(hh + 1) * dh]
            base = lay["packed_off"][m] + ((hh * n + i) * kk) * ds
            want = np.concatenate([z[g * ds:(g + 1) * ds] for g in sel])
            assert np.max(np.abs(out["packed"][base:base + kk * ds] - want)) < 1e-12


# ---------------------------------------------------------------------------
# Per-token budgets (Sec. 3.5). The allocator's formula is this build's
# reading (rank-linear weights, water-filled at S, largest remainders); the
# paper fixes its constraints, pinned here with independent computations.
# ---------------------------------------------------------------------------

def _waterfill(n, B, S):
    """Real shares x_r = min(S, lam * (n - r)) with sum x = B, by bisection
    on lam (independent of the oracle's integer closed form)."""
    w = np.arange(n, 0, -1, dtype=np.float64)
    if B == n * S:
        return np.full(n, float(S))
    lo, hi = 0.0, float(S)
    for _ in range(200):
        lam = 0.5 * (lo + hi)
        if np.minimum(S, lam * w).sum() < B:
            lo = lam
        else:
            hi = lam
    return np.minimum(S, hi * w)


@pytest.mark.parametrize("n,B,S,want", [
    (4, 8, 16, [3, 2, 2, 1]),      # x = 3.2 2.4 1.6 0.8 -> floors 3 2 1 0, two left to .8, .6
    (3, 6, 16, [3, 2, 1]),         # exact shares
    (2, 7, 4, [4, 3]),             # rank 0 saturates (x would be 4.67 > S)
    (5, 80, 16, [16] * 5),         # K_m = S: everything kept
    (5, 0, 16, [0] * 5),           # K_m = 0: nothing kept
    (1, 9, 16, [9]),               # a single token takes the whole budget
])
def test_budget_shares_hand_computed(oracle, n, B, S, want):
    assert list(oracle.budget_shares(n, B, S)) == want


def test_budget_shares_constraints_and_nearest_integers(oracle):
    rng = np.random.default_rng(40)
    for _ in range(300):
        S = int(rng.choice([4, 8, 16]))
        n = int(rng.integers(1, 70))
        Km = int(rng.integers(0, S + 1))
        B = Km * n
        K = oracle.budget_shares(n, B, S).astype(np.int64)
        x = _waterfill(n, B, S)
        assert K.sum() == B and K.min() >= 0 and K.max() <= S          # Sec. 3.5 constraints
        assert np.all(np.diff(K) <= 0)                                   # better rank, no fewer groups
        assert np.all(np.abs(K - x) < 1.0 + 1e-9)                        # a rounding of the shares
        # largest remainders: every rank rounded up has a fractional part no
        # smaller than every rank rounded down
        fr = x - np.floor(x + 1e-12)
        up = K > np.floor(x + 1e-12)
        if up.any() and (~up).any():
            assert fr[up].min() >= fr[~up & (fr > 1e-9)].max(initial=0.0) - 1e-9


def test_budget_shares_minimise_distance_brute_force(oracle):
    # the integer vector with the budget's sum and bounds closest to the real
    # shares (least squares), by enumeration, when that minimiser is unique
    for S in (2, 3, 4):
        for n in range(1, 6):
            for Km in range(S + 1):
                B = Km * n
                x = _waterfill(n, B, S)
                cands = [c for c in itertools.product(range(S + 1), repeat=n) if sum(c) == B]
                dist = [float(np.sum((np.array(c) - x) ** 2)) for c in cands]
                best = min(dist)
                winners = [c for c, dd in zip(cands, dist) if abs(dd - best) < 1e-9]
                K = tuple(int(v) for v in oracle.budget_shares(n, B, S))
                if len(winners) == 1:
                    assert K == winners[0], (S, n, Km, K, winners)
                else:   # tied fractional parts: the better ranks round up
                    assert K in winners and K == max(winners), (S, n, Km, K, winners)


def test_budget_allocate_follows_priority_ranks(oracle):
    rng = np.random.default_rng(41)
    pri = rng.standard_normal(9)
    K = oracle.budget_allocate(pri, 9 * 5, 16)
    byrank = oracle.budget_shares(9, 45, 16)
    order = np.argsort(-pri, kind="stable")
    assert list(K[order]) == list(byrank)
    perm = rng.permutation(9)
    assert list(oracle.budget_allocate(pri[perm], 45, 16)) == list(K[perm])   # token order irrelevant
    # equal priorities: the lower token index ranks first
    assert list(oracle.budget_allocate([0.5, 0.5, 0.5, 0.5], 8, 16)) == [3, 2, 2, 1]


def _budget_problem(rng, n_tok, k, G=4, H=2, dh=8, C=3):
    p = rnd_problem(rng, H=H, dh=dh, G=G, C=C, F=4, n_tok=n_tok, k=k, n_q=tuple(3 for _ in n_tok))
    d = H * dh
    p["W_v"] = 0.3 * rng.standard_normal((G, d))
    p["b_v"] = 0.3 * rng.standard_normal(G)
    p["W_role"] = rng.standard_normal((G, C))
    p["W_l"] = 0.3 * rng.standard_normal((G, d))
    p["b_l"] = 0.3 * rng.standard_normal(G)
    p["u"] = rng.standard_normal(C)
    return p


def _route_budget(oracle, p, k_force=None):
    spec = oracle.Spec(p["H"], p["dh"], p["G"], p["C"], p["F"], p["n_tok"], p["k"], p["n_q"])
    out = oracle.route_layer_budget(spec, p["h"], p["W_re"], p["b_re"], p["W_v"], p["b_v"], p["W_role"], p["W_l"],
                                    p["b_l"], p["u"], 0.1, 0.1, k_force=k_force)
    return spec, out


def test_budget_routing_counts_priorities_and_best_subsets(oracle):
    rng = np.random.default_rng(42)
    G = 4
    p = _budget_problem(rng, n_tok=((7, 4, 0, 0), (3, 2, 2, 0)), k=((2, 1, G, G), (3, 0, 0, G)), G=G)
    spec, out = _route_budget(oracle, p)
    lay = spec.lay
    offs = oracle.budget_idx_offsets(spec, out["ktok"])
    cl = [p["h"][7:11].mean(0), p["h"][14:16].mean(0)]
    nt = p["n_tok"].reshape(-1)
    kt = p["k"].reshape(-1)
    for sgi in range(8):
        e, n, km, r0 = sgi // 4, int(nt[sgi]), int(kt[sgi]), int(lay["row_off"][sgi])
        if n == 0:
            continue
        kk = out["ktok"][r0:r0 + n]
        assert kk.sum() == km * n                                       # B_m = K_m |I_m|
        if km in (0, G):
            assert np.all(kk == km)
            continue
        # priorities pi = u . softmax(W_re h + b_re), computed here with scipy
        a = scipy.special.softmax(p["h"][r0:r0 + n] @ p["W_re"].T + p["b_re"], axis=1)
        pri = a @ p["u"]
        assert np.max(np.abs(out["pri"][r0:r0 + n] - pri)) < 1e-12
        order = np.argsort(-pri, kind="stable")
        assert list(kk[order]) == list(oracle.budget_shares(n, km * n, G))
        for i in range(n):
            r = r0 + i
            gam = (p["W_v"] @ p["h"][r] + p["b_v"]) + 0.1 * (p["W_role"] @ a[i]) + \
                0.1 * (p["W_l"] @ cl[e] + p["b_l"])
            assert np.max(np.abs(out["gamma"][r] - gam)) < 1e-12
            best = max(itertools.combinations(range(G), int(kk[i])), key=lambda s: sum(gam[list(s)]))
            sel = out["idx"][offs[r]:offs[r] + int(kk[i])]
            assert tuple(sel) == tuple(sorted(best))


def test_budget_equal_counts_match_fixed_k_packing(oracle):
    # forcing K_i = K_m for every token must reproduce the fixed-k layout of
    # the C packer exactly (the numpy packer is written independently)
    rng = np.random.default_rng(43)
    G = 4
    p = _budget_problem(rng, n_tok=((5, 3, 0, 0),), k=((2, 1, G, 0),), G=G)
    rows = int(np.sum(p["n_tok"]))
    kf = np.array([2] * 5 + [1] * 3, np.int32)
    spec, out = _route_budget(oracle, p, k_force=kf)
    packed = oracle.pack_layer_budget(spec, p["v"], p["R"], out["idx"], out["ktok"])
    c = oracle.compress_layer(spec, p["h"], p["v"], p["R"], p["W_re"], p["b_re"], np.zeros((1, 2 * spec.d + spec.C)),
                              np.zeros(1), np.zeros((G, 1)), np.zeros(G), 0.1, 0.1, idx_force=out["idx"])
    assert rows == 8
    assert np.max(np.abs(packed - c["packed"])) < 1e-12
    o1 = oracle.attend_layer_budget(spec, p["q"], p["K"], packed, out["idx"], out["ktok"], p["R"])
    o2 = oracle.attend_layer(spec, p["q"], p["K"], c["packed"], c["idx"], p["R"])
    assert np.max(np.abs(o1 - o2)) < 1e-12


def test_budget_every_count_vector_equals_dense_over_routed_values(oracle):
    # every admissible per-token count vector (sum = B_m, 0..S) on a tiny
    # segment, each with the router's best subsets: attention equals dense
    # attention over explicitly built R M_j R^T v_j
    rng = np.random.default_rng(44)
    G = 4
    p = _budget_problem(rng, n_tok=((3, 0, 0, 0),), k=((2, G, G, G),), G=G)
    for kf in itertools.product(range(G + 1), repeat=3):
        if sum(kf) != 6:
            continue
        spec, out = _route_budget(oracle, p, k_force=np.array(kf, np.int32))
        offs = oracle.budget_idx_offsets(spec, out["ktok"])
        packed = oracle.pack_layer_budget(spec, p["v"], p["R"], out["idx"], out["ktok"])
        o = oracle.attend_layer_budget(spec, p["q"], p["K"], packed, out["idx"], out["ktok"], p["R"])
        masks = {r: tuple(out["idx"][offs[r]:offs[r] + kf[r]]) for r in range(3)}
        ref = dense_attention(p, _vtil(p, masks))
        assert np.max(np.abs(o - ref)) <= 1e-12, kf


def test_budget_forced_counts_must_meet_the_budget(oracle):
    rng = np.random.default_rng(45)
    p = _budget_problem(rng, n_tok=((3, 0, 0, 0),), k=((2, 4, 4, 4),))
    with pytest.raises(ValueError):
        _route_budget(oracle, p, k_force=np.array([2, 2, 1], np.int32))   # sums to 5, not 6
    with pytest.raises(ValueError):
        _route_budget(oracle, p, k_force=np.array([5, 1, 0], np.int32))   # 5 > S


# ---------------------------------------------------------------------------
# Token-level reduction (Sec. 3.1, Sec. 4.1)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("ratio,total", [(0.015625, 8), (0.03125, 16), (0.0625, 32)])
def test_select_counts_match_the_papers_visual_budgets(oracle, ratio, total):
    # Sec. 4.1: retention ratios 1/64, 1/32, 1/16 keep 8, 16, 32 of the 512
    # visual tokens, split evenly over the two 256-token camera views
    assert 2 * oracle.select_count(256, ratio) == total
    assert oracle.select_count(512, ratio) == total


def test_select_count_is_a_ceiling(oracle):
    assert oracle.select_count(10, 0.25) == 3       # ceil(2.5)
    assert oracle.select_count(7, 1.0) == 7
    assert oracle.select_count(300, 0.0625) == 19   # ceil(18.75)


def test_select_keeps_the_best_subset_brute_force(oracle):
    rng = np.random.default_rng(50)
    for _ in range(40):
        n = int(rng.integers(1, 9))
        r = float(rng.choice([0.25, 0.5, 0.75, 1.0]))
        s = rng.standard_normal((1, 2, n))
        x = rng.standard_normal((1, 2, n, 3))
        keep, xk = oracle.select_tokens(s, x, r)
        k = math.ceil(r * n)
        for v in range(2):
            best = max(itertools.combinations(range(n), k), key=lambda c: sum(s[0, v, list(c)]))
            assert tuple(keep[0, v]) == tuple(sorted(best))
            assert np.array_equal(xk[0, v], x[0, v, list(sorted(best))])


def test_select_ties_and_nan(oracle):
    s = np.array([[[0.5, 0.5, 0.5, 0.5]], [[np.nan, -np.inf, 0.0, -0.0]]])
    s = s.reshape(2, 1, 4)
    keep, _ = oracle.select_tokens(s, np.zeros((2, 1, 4, 1)), 0.5)
    assert list(keep[0, 0]) == [0, 1]     # equal scores: lower index first
    assert list(keep[1, 0]) == [2, 3]     # 0 and -0 tie above -inf; NaN lowest


# ---------------------------------------------------------------------------
# Dense rotation (one d x d R, S contiguous groups of d / S dims; Sec. 4.1)
# ---------------------------------------------------------------------------

def _dense_run(oracle, p, Rd, idx_force):
    spec = oracle.Spec(p["H"], p["dh"], p["G"], p["C"], p["F"], p["n_tok"], p["k"], p["n_q"])
    packed = oracle.pack_layer_dense(spec, p["v"], Rd, idx_force)
    return spec, packed, oracle.attend_layer_dense(spec, p["q"], p["K"], packed, idx_force, Rd)


def _all_idx(n_rows, G, k):
    return np.tile(np.arange(k, dtype=np.uint8) if k < G else np.arange(G, dtype=np.uint8), n_rows)


def test_dense_all_groups_kept_equals_dense_attention(oracle):
    rng = np.random.default_rng(70)
    H, dh, G = 2, 8, 4
    p = rnd_problem(rng, H=H, dh=dh, G=G, n_tok=((5, 3, 0, 0),), k=((G, G, G, G),), n_q=(4,))
    Rd = haar(rng, H * dh)
    _, _, o = _dense_run(oracle, p, Rd, _all_idx(8, G, G))
    assert rel_err(o, dense_attention(p), dh) < 1e-10      # R M R^T v = v when every group is kept


def test_dense_no_groups_kept_gives_zero(oracle):
    rng = np.random.default_rng(71)
    p = rnd_problem(rng, H=2, dh=8, G=4, n_tok=((5, 3, 0, 0),), k=((0, 0, 4, 4),), n_q=(4,))
    _, _, o = _dense_run(oracle, p, haar(rng, 16), np.zeros(0, np.uint8))
    assert np.all(o == 0)


def test_dense_every_mask_equals_attention_over_explicit_routed_values(oracle):
    rng = np.random.default_rng(72)
    H, dh, G = 2, 4, 4
    d, gw = H * dh, H * dh // G
    for k in (1, 2, 3):
        p = rnd_problem(rng, H=H, dh=dh, G=G, n_tok=((3, 0, 0, 0),), k=((k, G, G, G),), n_q=(2,))
        Rd = haar(rng, d)
        subsets = list(itertools.combinations(range(G), k))
        for masks in itertools.product(subsets, repeat=3):
            fx = np.array([g for m in masks for g in m], np.uint8)
            _, _, o = _dense_run(oracle, p, Rd, fx)
            vt = []
            for r in range(3):
                mvec = np.zeros(d)
                for g in masks[r]:
                    mvec[g * gw:(g + 1) * gw] = 1.0
                vt.append(Rd @ np.diag(mvec) @ Rd.T @ p["v"][r])   # v~ = R M R^T v, all heads at once
            vt = np.array(vt)
            ref = dense_attention(p, lambda e, h, r0, r1: vt[r0:r1, h * dh:(h + 1) * dh])
            assert np.max(np.abs(o - ref)) <= 1e-12, (k, masks)


def test_dense_block_diagonal_rotation_reproduces_the_per_head_oracle(oracle):
    # R = blockdiag(R_1 .. R_H) with the permutation that makes dense group s
    # the s-th group of every head: the dense restatement (numpy) must give
    # the per-head C oracle's values and outputs exactly
    rng = np.random.default_rng(73)
    H, dh, G = 3, 8, 4
    ds, d = dh // G, H * dh
    p = rnd_problem(rng, H=H, dh=dh, G=G, n_tok=((6, 4, 0, 0),), k=((2, 3, G, G),), n_q=(3,))
    spec, c, o_head = run(oracle, p)
    B = np.zeros((d, d))
    for hh in range(H):
        B[hh * dh:(hh + 1) * dh, hh * dh:(hh + 1) * dh] = p["R"][hh]
    perm = np.zeros(d, np.int64)     # dense coordinate -> per-head coordinate
    for s_ in range(G):
        for hh in range(H):
            for t in range(ds):
                perm[s_ * H * ds + hh * ds + t] = hh * dh + s_ * ds + t
    Rd = B[:, perm]
    packed = oracle.pack_layer_dense(spec, p["v"], Rd, c["idx"])
    o_dense = oracle.attend_layer_dense(spec, p["q"], p["K"], packed, c["idx"], Rd)
    assert np.max(np.abs(o_dense - o_head)) < 1e-12
    lay = spec.lay
    for m, (n, k) in enumerate(((6, 2), (4, 3))):
        a = packed[lay["packed_off"][m]: lay["packed_off"][m] + n * k * H * ds].reshape(n, k, H, ds)
        b = c["packed"][lay["packed_off"][m]: lay["packed_off"][m] + H * n * k * ds].reshape(H, n, k, ds)
        assert np.max(np.abs(a - b.transpose(1, 2, 0, 3))) < 1e-12
