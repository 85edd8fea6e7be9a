"""GPU-vs-oracle parity helpers (used by the -m gpu tests and smoke()).

Inputs come from paper_2608_18410_gb300.synth (seeded, shared by both
sides); expected values come only from the fp64 oracle.

Tolerances (stated for the method's outputs): group indices and packed
positions bit-exact wherever the oracle's top-k margin exceeds 1e-4, else
any valid top-k (every kept score >= every dropped score - 1e-4); packed
values and attention outputs within max|err| <= tol * ||row||_2 with
tol = 1e-2 for bf16 storage / fp32 accumulation and 1e-5 for fp32, a row
being one (token, head) vector of z or one (query, head) vector of o; an
all-zero oracle row must come back exactly zero.
"""
from __future__ import annotations

import numpy as np

import oracle
from paper_2608_18410_gb300 import synth

MARGIN = 1e-4
TOL = {"bf16": 1e-2, "f32": 1e-5}


def to_torch(x, dtype, device="cuda"):
    import torch
    if x.dtype == np.uint16:
        return torch.from_numpy(x.view(np.int16)).to(device).view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(x)).to(device)


def from_torch(t, dtype):
    import torch
    t = t.detach().cpu()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    return t.numpy()


def make_rolesub(wl):
    from paper_2608_18410_gb300.rolesub import RoleSub
    return RoleSub(wl.L, wl.H, wl.dh, wl.G, wl.C, wl.F, wl.dtype, wl.n_tok_array(), wl.k_array(),
                   wl.n_query_array())


def run_gpu(wl, inp, rs=None, add=None):
    """compress + attend on the GPU; returns numpy packed, idx, o and the status.

    add: weights of the additive routing score (synth.gen_additive_weights);
    when given, compress runs rolesub_compress_additive instead.
    """
    import torch
    rs = rs or make_rolesub(wl)
    dev = {k: to_torch(v, wl.dtype) for k, v in inp.items()}
    if add is None:
        packed, idx = rs.compress(dev["h"], dev["v"], dev["R"], dev["W_re"], dev["b_re"], dev["W1"],
                                  dev["b1"], dev["W2"], dev["b2"], wl.alpha_role, wl.alpha_lang)
    else:
        da = {k: to_torch(v, wl.dtype) for k, v in add.items()}
        packed, idx = rs.compress_additive(dev["h"], dev["v"], dev["R"], dev["W_re"], dev["b_re"], da["W_v"],
                                           da["b_v"], da["W_role"], da["W_l"], da["b_l"], wl.alpha_role,
                                           wl.alpha_lang)
    o = rs.attend(dev["q"], dev["K"], packed, idx, dev["R"])
    torch.cuda.synchronize()
    status = rs.device_status()
    return {"packed": from_torch(packed, wl.dtype), "idx": from_torch(idx, wl.dtype),
            "o": from_torch(o, wl.dtype), "status": status, "rs": rs}



def check_layer_episode(wl, inp, gpu, layer, e, report=None, add=None):
    """Oracle compress + attend of one (layer, episode); compares with the GPU.

    add: the additive router's weights when the GPU ran that router; the
    oracle then routes with compress_layer_linear.

    Returns a dict of statistics; raises AssertionError on any violation.
    """
    G, H, dh = wl.G, wl.H, wl.dh
    ds = dh // G
    tol = TOL[wl.dtype]
    ep = wl.episodes[e]
    glob = oracle.layout(wl.n_tok_array(), wl.k_array(), H, dh, G)
    n_tok = np.array(ep.n_tok(), np.int32)
    kk = np.array(ep.k(G), np.int32)
    spec = oracle.Spec(H, dh, G, wl.C, wl.F, n_tok[None], kk[None], [ep.n_query])
    loc = spec.lay
    r0 = int(glob["row_off"][4 * e])
    r1 = r0 + ep.n_cache
    q0 = int(sum(x.n_query for x in wl.episodes[:e]))
    W = lambda name: synth.widen(inp[name][layer], wl.dtype)
    h = synth.widen(inp["h"][layer, r0:r1], wl.dtype)
    v = synth.widen(inp["v"][layer, r0:r1], wl.dtype)
    R = W("R")
    args = (R, W("W_re"), inp["b_re"][layer].astype(np.float64), W("W1"),
            inp["b1"][layer].astype(np.float64), W("W2"), inp["b2"][layer].astype(np.float64),
            wl.alpha_role, wl.alpha_lang)
    if add is None:
        ref = oracle.compress_layer(spec, h, v, *args)
    else:
        A = lambda name: synth.widen(add[name][layer], wl.dtype)
        ref = oracle.compress_layer_linear(
            spec, h, v, R, W("W_re"), inp["b_re"][layer].astype(np.float64), A("W_v"),
            add["b_v"][layer].astype(np.float64), A("W_role"), A("W_l"), add["b_l"][layer].astype(np.float64),
            wl.alpha_role, wl.alpha_lang, want_z=False)

    # ---- group indices -------------------------------------------------
    gidx = gpu["idx"][layer]
    gpu_idx_local = np.zeros(max(loc["idx_bytes"], 1), np.uint8)
    n_exact = n_margin = 0
    for m in range(4):
        n, k = int(n_tok[m]), int(kk[m])
        if n == 0 or k == 0:
            continue
        gs = gidx[glob["idx_off"][4 * e + m]: glob["idx_off"][4 * e + m] + n * k].reshape(n, k)
        os_ = ref["idx"][loc["idx_off"][m]: loc["idx_off"][m] + n * k].reshape(n, k)
        gpu_idx_local[loc["idx_off"][m]: loc["idx_off"][m] + n * k] = gs.reshape(-1)
        for i in range(n):
            r = int(loc["row_off"][m]) + i
            if k == G:
                assert np.array_equal(gs[i], np.arange(G)), (layer, e, m, i, gs[i])
                continue
            marg = ref["margin"][r]
            if marg > MARGIN:
                assert np.array_equal(gs[i], os_[i]), (layer, e, m, i, gs[i], os_[i], marg)
                n_exact += 1
            else:
                g = gs[i].astype(int)
                assert len(set(g)) == k and np.all(np.diff(g) > 0) and np.all(g < G), (gs[i],)
                gam = ref["gamma"][r]
                dropped = np.setdiff1d(np.arange(G), g)
                if len(dropped):
                    assert gam[g].min() >= gam[dropped].max() - MARGIN, (gam, g)
                n_margin += 1

    # ---- packed values: oracle z at the GPU's indices --------------------
    forced = oracle.compress_layer(spec, h, v, *args, idx_force=gpu_idx_local)
    zref = forced["z"].reshape(-1, H, dh)
    gp = synth.widen(gpu["packed"][layer], wl.dtype)
    worst_pack = 0.0
    for m in range(4):
        n, k = int(n_tok[m]), int(kk[m])
        if n == 0 or k == 0:
            continue
        a = gp[glob["packed_off"][4 * e + m]: glob["packed_off"][4 * e + m] + H * n * k * ds].reshape(H, n, k, ds)
        b = forced["packed"][loc["packed_off"][m]: loc["packed_off"][m] + H * n * k * ds].reshape(H, n, k, ds)
        nrm = np.linalg.norm(zref[loc["row_off"][m]: loc["row_off"][m] + n], axis=2).T  # [H][n]
        err = np.abs(a - b).max(axis=(2, 3))
        assert np.all(err <= tol * nrm + (nrm == 0) * 0.0), (layer, e, m, float((err / np.maximum(nrm, 1e-30)).max()))
        worst_pack = max(worst_pack, float((err / np.maximum(nrm, 1e-30)).max()))

    # ---- attention over the GPU's routed cache ---------------------------
    worst_o = 0.0
    if ep.n_query:
        qe = synth.widen(inp["q"][layer, q0:q0 + ep.n_query], wl.dtype)
        Ke = synth.widen(inp["K"][layer, r0:r1], wl.dtype)
        o_ref = oracle.attend_layer(spec, qe, Ke, forced["packed"], forced["idx"], R)
        o_gpu = synth.widen(gpu["o"][layer, q0:q0 + ep.n_query], wl.dtype)
        a = o_gpu.reshape(-1, H, dh)
        b = o_ref.reshape(-1, H, dh)
        nrm = np.linalg.norm(b, axis=2)
        err = np.abs(a - b).max(axis=2)
        zero = nrm == 0
        assert np.all(err[zero] == 0), "zero oracle rows must be exactly zero"
        assert np.all(err <= tol * nrm), (layer, e, float((err / np.maximum(nrm, 1e-30)).max()))
        worst_o = float((err[~zero] / nrm[~zero]).max()) if np.any(~zero) else 0.0
    return {"exact_idx": n_exact, "margin_idx": n_margin, "worst_pack": worst_pack, "worst_o": worst_o}


def check_attend_standalone(wl, inp, rs, layer_list=None, episodes=None):
    """Attention alone on synthetic packed values and indices (no router)."""
    import torch
    glob = oracle.layout(wl.n_tok_array(), wl.k_array(), wl.H, wl.dh, wl.G)
    segs = [(int(wl.n_tok_array().reshape(-1)[s]), int(wl.k_array().reshape(-1)[s]),
             int(glob["packed_off"][s]), int(glob["idx_off"][s])) for s in range(4 * wl.E)]
    packed, idx = synth.gen_packed(wl, glob["packed_elems"], glob["idx_bytes"], segs)
    dev_p = to_torch(packed if packed.size else np.zeros((wl.L, 1), packed.dtype), wl.dtype)
    dev_i = to_torch(idx if idx.size else np.zeros((wl.L, 16), np.uint8), wl.dtype)
    q = to_torch(inp["q"], wl.dtype)
    K = to_torch(inp["K"], wl.dtype)
    R = to_torch(inp["R"], wl.dtype)
    o = rs.attend(q, K, dev_p, dev_i, R)
    torch.cuda.synchronize()
    og = synth.widen(from_torch(o, wl.dtype), wl.dtype)
    tol = TOL[wl.dtype]
    worst = 0.0
    spec = oracle.Spec(wl.H, wl.dh, wl.G, wl.C, wl.F, wl.n_tok_array(), wl.k_array(), wl.n_query_array())
    for layer in (layer_list or range(wl.L)):
        ref = oracle.attend_layer(spec, synth.widen(inp["q"][layer], wl.dtype),
                                  synth.widen(inp["K"][layer], wl.dtype),
                                  synth.widen(packed[layer], wl.dtype), idx[layer],
                                  synth.widen(inp["R"][layer], wl.dtype), episodes=episodes)
        a = og[layer].reshape(-1, wl.H, wl.dh)
        b = ref.reshape(-1, wl.H, wl.dh)
        rows = np.concatenate([np.arange(spec.ep_q[e], spec.ep_q[e + 1]) for e in (episodes or range(wl.E))]) \
            if wl.E else np.zeros(0, int)
        a, b = a[rows], b[rows]
        nrm = np.linalg.norm(b, axis=2)
        err = np.abs(a - b).max(axis=2)
        assert np.all(err[nrm == 0] == 0)
        assert np.all(err <= tol * nrm), float((err / np.maximum(nrm, 1e-30)).max())
        if np.any(nrm > 0):
            worst = max(worst, float((err[nrm > 0] / nrm[nrm > 0]).max()))
    return worst
