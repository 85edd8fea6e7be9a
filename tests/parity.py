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


PRI_MARGIN = 1e-4


def run_gpu_budget(wl, inp, add, u, rs=None):
    """compress_budget + attend_budget on the GPU; numpy packed, idx, k_tok, o, status."""
    import torch
    rs = rs or make_rolesub(wl)
    dev = {k: to_torch(v, wl.dtype) for k, v in inp.items()}
    da = {k: to_torch(v, wl.dtype) for k, v in add.items()}
    du = torch.from_numpy(np.ascontiguousarray(u, np.float32)).cuda()
    packed, idx, ktok = rs.compress_budget(dev["h"], dev["v"], dev["R"], dev["W_re"], dev["b_re"], da["W_v"],
                                           da["b_v"], da["W_role"], da["W_l"], da["b_l"], du, wl.alpha_role,
                                           wl.alpha_lang)
    o = rs.attend_budget(dev["q"], dev["K"], packed, idx, ktok, dev["R"])
    torch.cuda.synchronize()
    return {"packed": from_torch(packed, wl.dtype), "idx": from_torch(idx, wl.dtype),
            "ktok": ktok.cpu().numpy(), "o": from_torch(o, wl.dtype), "status": rs.device_status(), "rs": rs}


def check_budget_layer_episode(wl, inp, add, u, gpu, layer, e):
    """Per-token budgets of one (layer, episode) against the oracle.

    Counts: every segment's counts meet its budget and bounds, form the
    allocator's multiset, follow every priority order wider than PRI_MARGIN
    and equal the oracle's wherever a token's priority is that far from all
    others. Indices, packed values and outputs are then checked on the GPU's
    counts (the oracle routes with them forced), with the margin and row-norm
    rules of check_layer_episode.
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
    A = lambda name: synth.widen(add[name][layer], wl.dtype)
    h = synth.widen(inp["h"][layer, r0:r1], wl.dtype)
    v = synth.widen(inp["v"][layer, r0:r1], wl.dtype)
    R = W("R")
    rargs = (W("W_re"), inp["b_re"][layer].astype(np.float64), A("W_v"), add["b_v"][layer].astype(np.float64),
             A("W_role"), A("W_l"), add["b_l"][layer].astype(np.float64), u[layer].astype(np.float64),
             wl.alpha_role, wl.alpha_lang)
    ref = oracle.route_layer_budget(spec, h, *rargs)
    gk = gpu["ktok"][layer, r0:r1].astype(np.int64)
    n_exact_k = 0
    for m in range(4):
        n, km, rs_ = int(n_tok[m]), int(kk[m]), int(loc["row_off"][m])
        if n == 0:
            continue
        g = gk[rs_:rs_ + n]
        o = ref["ktok"][rs_:rs_ + n]
        assert g.sum() == km * n and g.min() >= 0 and g.max() <= G, (layer, e, m, g)
        assert sorted(g) == sorted(o), (layer, e, m)
        if km in (0, G):
            assert np.all(g == km)
            continue
        pri = ref["pri"][rs_:rs_ + n]
        diff = pri[:, None] - pri[None, :]
        clear = diff > PRI_MARGIN
        assert np.all(g[:, None] >= g[None, :] - ~clear * 1000), (layer, e, m)
        sep = np.all((np.abs(diff) > PRI_MARGIN) | np.eye(n, dtype=bool), axis=1)
        assert np.array_equal(g[sep], o[sep]), (layer, e, m)
        n_exact_k += int(sep.sum())

    # ---- indices on the GPU's counts ------------------------------------
    forced = oracle.route_layer_budget(spec, h, *rargs, k_force=gk.astype(np.int32))
    offs_loc = oracle.budget_idx_offsets(spec, gk)
    gidx = gpu["idx"][layer]
    idx_local = np.zeros(max(loc["idx_bytes"], 1), np.uint8)
    n_exact = n_margin = 0
    for m in range(4):
        n, km, rs_ = int(n_tok[m]), int(kk[m]), int(loc["row_off"][m])
        if n == 0 or km == 0:
            continue
        seg = gidx[glob["idx_off"][4 * e + m]: glob["idx_off"][4 * e + m] + n * km]
        idx_local[loc["idx_off"][m]: loc["idx_off"][m] + n * km] = seg
        for i in range(n):
            r = rs_ + i
            k_i = int(gk[r])
            a0 = int(offs_loc[r])
            gs = idx_local[a0:a0 + k_i]
            os_ = forced["idx"][a0:a0 + k_i]
            if km == G:
                assert np.array_equal(gs, np.arange(G)), (layer, e, m, i)
                continue
            if k_i in (0, G) or forced["margin"][r] > MARGIN:
                assert np.array_equal(gs, os_), (layer, e, m, i, gs, os_)
                n_exact += 1
            else:
                sel = gs.astype(int)
                assert len(set(sel)) == k_i and np.all(np.diff(sel) > 0) and np.all(sel < G), (gs,)
                gam = forced["gamma"][r]
                dropped = np.setdiff1d(np.arange(G), sel)
                assert gam[sel].min() >= gam[dropped].max() - MARGIN, (gam, sel)
                n_margin += 1

    # ---- packed values and attention on the GPU's indices and counts -----
    pk = oracle.pack_layer_budget(spec, v, R, idx_local, gk)
    gp = synth.widen(gpu["packed"][layer], wl.dtype)
    zrows = np.stack([v[:, hh * dh:(hh + 1) * dh] @ R[hh] for hh in range(H)], axis=1)   # [rows][H][dh]
    for m in range(4):
        n, km, rs_ = int(n_tok[m]), int(kk[m]), int(loc["row_off"][m])
        if n == 0 or km == 0:
            continue
        B = n * km
        a = gp[glob["packed_off"][4 * e + m]: glob["packed_off"][4 * e + m] + H * B * ds].reshape(H, B, ds)
        b = pk[loc["packed_off"][m]: loc["packed_off"][m] + H * B * ds].reshape(H, B, ds)
        err = np.abs(a - b).max(axis=2)                                   # [H][B]
        owner = np.repeat(np.arange(n), gk[rs_:rs_ + n])                  # token of each stored group
        nrm = np.linalg.norm(zrows[rs_ + owner], axis=2).T                # [H][B]
        assert np.all(err <= tol * nrm), (layer, e, m, float((err / np.maximum(nrm, 1e-30)).max()))
    worst_o = 0.0
    if ep.n_query:
        qe = synth.widen(inp["q"][layer, q0:q0 + ep.n_query], wl.dtype)
        Ke = synth.widen(inp["K"][layer, r0:r1], wl.dtype)
        o_ref = oracle.attend_layer_budget(spec, qe, Ke, pk, idx_local, gk, R)
        o_gpu = synth.widen(gpu["o"][layer, q0:q0 + ep.n_query], wl.dtype)
        a = o_gpu.reshape(-1, H, dh)
        b = o_ref.reshape(-1, H, dh)
        nrm = np.linalg.norm(b, axis=2)
        err = np.abs(a - b).max(axis=2)
        zero = nrm == 0
        assert np.all(err[zero] == 0), "zero oracle rows must be exactly zero"
        assert np.all(err <= tol * nrm), (layer, e, float((err / np.maximum(nrm, 1e-30)).max()))
        worst_o = float((err[~zero] / nrm[~zero]).max()) if np.any(~zero) else 0.0
    return {"exact_k": n_exact_k, "exact_idx": n_exact, "margin_idx": n_margin, "worst_o": worst_o}
