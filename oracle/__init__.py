"""fp64 CPU oracle for RoleSub (test infrastructure).

Only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package. The product path (the CUDA library and
its Python binding) never imports it, and it never imports the product.

The arithmetic lives in ``rolesub_oracle.c`` (plain double-precision loops,
each function citing the passage of the paper it restates); this module only
builds that file with gcc and marshals numpy arrays through ctypes.

Parity status of each function (what pins it, in tests/test_oracle_pins.py):
  layout          -- Tables 1 and 3 KV fractions, hand-computed offsets
  lang_pool       -- closed form (mean), empty-set case
  role            -- scipy.special.softmax, uniform case
  router_score    -- one-block-at-a-time special cases (h / role / language)
  router_score_linear -- the additive form: selector-matrix closed forms for
                     each term, one term at a time and together; parameter
                     count against the paper's 4.20M routing heads
  topk            -- brute-force subset enumeration, hand-built near-ties
  rotate          -- permutation matrices, norm preservation
  budget_shares / budget_allocate -- Sec. 3.5 allocator (reading: rank-linear
                     weights, water-filled at S, largest remainders): hand-
                     computed cases, the budget and bound constraints, an
                     independent bisection water-fill, brute-force nearest
                     integer vector on tiny cases
  route_layer_budget / pack_layer_budget / attend_layer_budget -- per-token
                     K_i: counts from the allocator over pi = u . a (scipy
                     softmax), brute-force top-K_i, equal counts == the
                     fixed-k C path, every mask == dense R M R^T v attention
  select_count / select_tokens -- Sec. 3.1 / 4.1 token reduction: the
                     paper's 8 / 16 / 32 of 512 visual tokens, brute-force
                     best subsets, ties and NaN scores, rows copied exactly
  pack_layer_dense / attend_layer_dense -- one dense d x d R (Sec. 4.1):
                     all kept == dense attention, none kept == 0, every mask
                     == dense attention over explicit R M R^T v, and the
                     per-head C oracle reproduced exactly by the dense R
                     blockdiag(R_h) with the head-interleaving permutation
  compress/attend -- all-kept == dense attention (1e-10), none-kept == 0,
                     every mask on tiny inputs == dense attention over
                     R M R^T v, complement linearity, R = I textbook case,
                     token / group permutation equivariance
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "rolesub_oracle.c")
_LIB = os.path.join(_HERE, "librolesub_oracle.so")
_lock = threading.Lock()
_lib = None

_dp = ctypes.POINTER(ctypes.c_double)
_ip = ctypes.POINTER(ctypes.c_int)
_llp = ctypes.POINTER(ctypes.c_longlong)
_ubp = ctypes.POINTER(ctypes.c_ubyte)


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (no fast-math, no FMA contraction)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off",
                               "-fno-fast-math", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def lib():
    global _lib
    with _lock:
        if _lib is None:
            build()
            L = ctypes.CDLL(_LIB)
            L.oracle_layout.argtypes = [ctypes.c_int] * 4 + [_ip, _ip, _llp, _llp, _llp, _llp]
            L.oracle_layout.restype = ctypes.c_int
            L.oracle_lang_pool.argtypes = [ctypes.c_int, ctypes.c_int, _dp, _dp]
            L.oracle_lang_pool.restype = None
            L.oracle_role.argtypes = [ctypes.c_int, ctypes.c_int, _dp, _dp, _dp, _dp]
            L.oracle_role.restype = None
            L.oracle_router_score.argtypes = [ctypes.c_int] * 4 + [_dp] * 7 + [ctypes.c_double] * 2 + [_dp]
            L.oracle_router_score.restype = None
            L.oracle_router_score_linear.argtypes = [ctypes.c_int] * 3 + [_dp] * 8 + [ctypes.c_double] * 2 + [_dp]
            L.oracle_router_score_linear.restype = None
            L.oracle_route_episode_linear.argtypes = (
                [ctypes.c_int] * 3 + [_ip, _ip, _llp] + [_dp] * 8 + [ctypes.c_double] * 2 + [_ubp, _dp, _dp])
            L.oracle_route_episode_linear.restype = ctypes.c_int
            L.oracle_budget_shares.argtypes = [ctypes.c_int, ctypes.c_longlong, ctypes.c_int, _ip]
            L.oracle_budget_shares.restype = ctypes.c_int
            L.oracle_budget_allocate.argtypes = [ctypes.c_int, ctypes.c_longlong, ctypes.c_int, _dp, _ip]
            L.oracle_budget_allocate.restype = ctypes.c_int
            L.oracle_route_episode_budget.argtypes = (
                [ctypes.c_int] * 3 + [_ip, _ip, _llp] + [_dp] * 9 + [ctypes.c_double] * 2
                + [_ip, _ubp, _ip, _dp, _dp, _dp])
            L.oracle_route_episode_budget.restype = ctypes.c_int
            L.oracle_topk.argtypes = [ctypes.c_int, ctypes.c_int, _dp, _ubp, _dp]
            L.oracle_topk.restype = None
            L.oracle_rotate.argtypes = [ctypes.c_int, _dp, _dp, _dp]
            L.oracle_rotate.restype = None
            L.oracle_compress_episode.argtypes = (
                [ctypes.c_int] * 5 + [_ip, _ip, _llp, _llp] + [_dp] * 9
                + [ctypes.c_double] * 2 + [_ubp, _dp, _ubp, _dp, _dp, _dp])
            L.oracle_compress_episode.restype = ctypes.c_int
            L.oracle_attend_episode.argtypes = (
                [ctypes.c_int] * 3 + [_ip, _ip, _llp, _llp, ctypes.c_int, _dp, _dp, _dp, _ubp, _dp,
                                      ctypes.c_double, ctypes.c_int, ctypes.c_int, _dp])
            L.oracle_attend_episode.restype = ctypes.c_int
            _lib = L
    return _lib


def _d(a):
    a = np.ascontiguousarray(a, dtype=np.float64)
    return a, a.ctypes.data_as(_dp)


def _i(a):
    a = np.ascontiguousarray(a, dtype=np.int32)
    return a, a.ctypes.data_as(_ip)


def _ll(a):
    a = np.ascontiguousarray(a, dtype=np.int64)
    return a, a.ctypes.data_as(_llp)


def _u8(a):
    return a.ctypes.data_as(_ubp)


# ---------------------------------------------------------------------------
# Fine-grained functions (pinned one by one)
# ---------------------------------------------------------------------------

def layout(n_tok, k, H, dh, G):
    """Offsets of every segment of one layer; n_tok, k are [E][4] (vis, lang, prop, act)."""
    n_tok = np.asarray(n_tok, np.int32).reshape(-1, 4)
    k = np.asarray(k, np.int32).reshape(-1, 4)
    E = n_tok.shape[0]
    S = E * 4
    row = np.zeros(S, np.int64)
    pk = np.zeros(S, np.int64)
    ix = np.zeros(S, np.int64)
    tot = np.zeros(3, np.int64)
    n_a, n_p = _i(n_tok)
    k_a, k_p = _i(k)
    rc = lib().oracle_layout(E, H, dh, G, n_p, k_p, row.ctypes.data_as(_llp), pk.ctypes.data_as(_llp),
                             ix.ctypes.data_as(_llp), tot.ctypes.data_as(_llp))
    if rc != 0:
        raise ValueError("oracle_layout: bad arguments")
    return {"row_off": row, "packed_off": pk, "idx_off": ix, "rows": int(tot[0]),
            "packed_elems": int(tot[1]), "idx_bytes": int(tot[2])}


def lang_pool(h_lang):
    h_lang = np.asarray(h_lang, np.float64)
    n, d = h_lang.shape if h_lang.size else (0, h_lang.shape[-1])
    c = np.zeros(d)
    ha, hp = _d(h_lang if n else np.zeros((1, d)))
    lib().oracle_lang_pool(d, n, hp, c.ctypes.data_as(_dp))
    return c


def role(W_re, b_re, h):
    W_re, wp = _d(W_re)
    b_re, bp = _d(b_re)
    h, hp = _d(h)
    C, d = W_re.shape
    a = np.zeros(C)
    lib().oracle_role(d, C, wp, bp, hp, a.ctypes.data_as(_dp))
    return a


def router_score(W1, b1, W2, b2, h, a, c, alpha_role, alpha_lang):
    W1, w1 = _d(W1)
    b1, bb1 = _d(b1)
    W2, w2 = _d(W2)
    b2, bb2 = _d(b2)
    h, hp = _d(h)
    a, ap = _d(a)
    c, cp = _d(c)
    F = W1.shape[0]
    G = W2.shape[0]
    d = h.shape[0]
    C = a.shape[0]
    assert W1.shape[1] == 2 * d + C and W2.shape[1] == F
    g = np.zeros(G)
    lib().oracle_router_score(d, C, F, G, w1, bb1, w2, bb2, hp, ap, cp, float(alpha_role),
                              float(alpha_lang), g.ctypes.data_as(_dp))
    return g


def router_score_linear(W_v, b_v, W_role, W_l, b_l, h, a, c, alpha_role, alpha_lang):
    """Additive router (Eq. routingscore as printed) for one token."""
    W_v, wv = _d(W_v)
    b_v, bv = _d(b_v)
    W_role, wr = _d(W_role)
    W_l, wl = _d(W_l)
    b_l, bl = _d(b_l)
    h, hp = _d(h)
    a, ap = _d(a)
    c, cp = _d(c)
    G, d = W_v.shape
    C = a.shape[0]
    assert W_l.shape == (G, d) and W_role.shape == (G, C) and h.shape[0] == d
    g = np.zeros(G)
    lib().oracle_router_score_linear(d, C, G, wv, bv, wr, wl, bl, hp, ap, cp, float(alpha_role),
                                     float(alpha_lang), g.ctypes.data_as(_dp))
    return g


def topk(gamma, k):
    gamma, gp = _d(gamma)
    G = gamma.shape[0]
    idx = np.zeros(max(k, 1), np.uint8)
    m = np.zeros(1)
    lib().oracle_topk(G, k, gp, _u8(idx), m.ctypes.data_as(_dp))
    return idx[:k].copy(), float(m[0])


def rotate(R, v):
    R, rp = _d(R)
    v, vp = _d(v)
    z = np.zeros(R.shape[0])
    lib().oracle_rotate(R.shape[0], rp, vp, z.ctypes.data_as(_dp))
    return z


# ---------------------------------------------------------------------------
# Whole-path helpers (per layer, per episode)
# ---------------------------------------------------------------------------

class Spec:
    """Geometry of one cache: per-episode token counts and kept groups."""

    def __init__(self, H, dh, G, C, F, n_tok, k, n_q):
        self.H, self.dh, self.G, self.C, self.F = H, dh, G, C, F
        self.n_tok = np.asarray(n_tok, np.int32).reshape(-1, 4)
        self.k = np.asarray(k, np.int32).reshape(-1, 4)
        self.n_q = np.asarray(n_q, np.int32).reshape(-1)
        self.E = self.n_tok.shape[0]
        self.d = H * dh
        self.lay = layout(self.n_tok, self.k, H, dh, G)
        self.ep_row = np.concatenate([[0], np.cumsum(self.n_tok.sum(1))]).astype(np.int64)
        self.ep_q = np.concatenate([[0], np.cumsum(self.n_q)]).astype(np.int64)


def compress_layer(spec: Spec, h, v, R, W_re, b_re, W1, b1, W2, b2, alpha_role, alpha_lang,
                   episodes=None, idx_force=None, packed=None, idx=None, want_z=True):
    """Compress one layer (all episodes, or the listed ones).

    h, v: [rows][d] float64 (widened inputs). Returns dict with packed
    [packed_elems] float64, idx [idx_bytes] uint8, gamma [rows][G], margin [rows],
    z [rows][d] (rows of episodes not processed stay NaN / zero).
    """
    s = spec
    lay = s.lay
    if packed is None:
        packed = np.zeros(lay["packed_elems"], np.float64)
    if idx is None:
        idx = np.zeros(max(lay["idx_bytes"], 1), np.uint8)
    gamma = np.full((lay["rows"], s.G), np.nan)
    margin = np.full(lay["rows"], np.nan)
    z = np.zeros((lay["rows"], s.d)) if want_z else None
    Rd, Rp = _d(R)
    Wre, Wrep = _d(W_re)
    bre, brep = _d(b_re)
    W1d, W1p = _d(W1)
    b1d, b1p = _d(b1)
    W2d, W2p = _d(W2)
    b2d, b2p = _d(b2)
    fx = None
    if idx_force is not None:
        fx = np.ascontiguousarray(idx_force, np.uint8)
    eps = range(s.E) if episodes is None else episodes
    for e in eps:
        r0, r1 = int(s.ep_row[e]), int(s.ep_row[e + 1])
        he, hp = _d(h[r0:r1] if r1 > r0 else np.zeros((1, s.d)))
        ve, vp = _d(v[r0:r1] if r1 > r0 else np.zeros((1, s.d)))
        nt, ntp = _i(s.n_tok[e])
        kk, kp = _i(s.k[e])
        po, pop = _ll(lay["packed_off"][4 * e:4 * e + 4])
        io, iop = _ll(lay["idx_off"][4 * e:4 * e + 4])
        g_e = np.full((max(r1 - r0, 1), s.G), np.nan)
        m_e = np.full(max(r1 - r0, 1), np.nan)
        z_e = np.zeros((max(r1 - r0, 1), s.d))
        rc = lib().oracle_compress_episode(
            s.H, s.dh, s.G, s.C, s.F, ntp, kp, pop, iop, hp, vp, Rp, Wrep, brep, W1p, b1p, W2p, b2p,
            float(alpha_role), float(alpha_lang), None if fx is None else _u8(fx),
            packed.ctypes.data_as(_dp), _u8(idx), g_e.ctypes.data_as(_dp), m_e.ctypes.data_as(_dp),
            z_e.ctypes.data_as(_dp))
        if rc != 0:
            raise ValueError("oracle_compress_episode: bad arguments or indices")
        gamma[r0:r1] = g_e[:r1 - r0]
        margin[r0:r1] = m_e[:r1 - r0]
        if want_z:
            z[r0:r1] = z_e[:r1 - r0]
    return {"packed": packed, "idx": idx[:lay["idx_bytes"]], "gamma": gamma, "margin": margin, "z": z}


def compress_layer_linear(spec: Spec, h, v, R, W_re, b_re, W_v, b_v, W_role, W_l, b_l, alpha_role, alpha_lang,
                          episodes=None, want_z=True):
    """Compress one layer with the additive router: route every (listed)
    episode, then rotate and pack with those indices (compress_layer with
    idx_force). Same return dict as compress_layer."""
    s = spec
    lay = s.lay
    idx = np.zeros(max(lay["idx_bytes"], 1), np.uint8)
    gamma = np.full((lay["rows"], s.G), np.nan)
    margin = np.full(lay["rows"], np.nan)
    Wre, Wrep = _d(W_re)
    bre, brep = _d(b_re)
    Wv, Wvp = _d(W_v)
    bv, bvp = _d(b_v)
    Wr, Wrp = _d(W_role)
    Wl, Wlp = _d(W_l)
    bl, blp = _d(b_l)
    eps = list(range(s.E)) if episodes is None else list(episodes)
    for e in eps:
        r0, r1 = int(s.ep_row[e]), int(s.ep_row[e + 1])
        he, hp = _d(h[r0:r1] if r1 > r0 else np.zeros((1, s.d)))
        nt, ntp = _i(s.n_tok[e])
        kk, kp = _i(s.k[e])
        io, iop = _ll(lay["idx_off"][4 * e:4 * e + 4])
        g_e = np.full((max(r1 - r0, 1), s.G), np.nan)
        m_e = np.full(max(r1 - r0, 1), np.nan)
        rc = lib().oracle_route_episode_linear(
            s.d, s.G, s.C, ntp, kp, iop, hp, Wrep, brep, Wvp, bvp, Wrp, Wlp, blp,
            float(alpha_role), float(alpha_lang), _u8(idx), g_e.ctypes.data_as(_dp), m_e.ctypes.data_as(_dp))
        if rc != 0:
            raise ValueError("oracle_route_episode_linear: bad arguments")
        gamma[r0:r1] = g_e[:r1 - r0]
        margin[r0:r1] = m_e[:r1 - r0]
    # rotation and packing with the routed indices (router weights unused there)
    zF = np.zeros((1, 2 * s.d + s.C))
    out = compress_layer(spec, h, v, R, W_re, b_re, zF, np.zeros(1), np.zeros((s.G, 1)), np.zeros(s.G),
                         alpha_role, alpha_lang, episodes=eps, idx_force=idx, want_z=want_z)
    out["gamma"] = gamma
    out["margin"] = margin
    return out


def attend_layer(spec: Spec, q, K, packed, idx, R, scale=0.0, episodes=None, heads=None, out=None):
    """Attention of every (listed) episode's queries over its routed cache.

    q: [q_rows][d], K: [rows][d], packed: [packed_elems] float64, idx uint8.
    Returns o [q_rows][d] float64 (unprocessed entries stay zero).
    """
    s = spec
    lay = s.lay
    o = np.zeros((int(s.ep_q[-1]), s.d)) if out is None else out
    pk, pkp = _d(packed if packed.size else np.zeros(1))
    ix = np.ascontiguousarray(idx if idx.size else np.zeros(1, np.uint8), np.uint8)
    Rd, Rp = _d(R)
    h0, h1 = (0, s.H) if heads is None else heads
    eps = range(s.E) if episodes is None else episodes
    for e in eps:
        r0, r1 = int(s.ep_row[e]), int(s.ep_row[e + 1])
        q0, q1 = int(s.ep_q[e]), int(s.ep_q[e + 1])
        if q1 == q0:
            continue
        qe, qp = _d(q[q0:q1])
        ke, kp_ = _d(K[r0:r1] if r1 > r0 else np.zeros((1, s.d)))
        nt, ntp = _i(s.n_tok[e])
        kk, kp = _i(s.k[e])
        po, pop = _ll(lay["packed_off"][4 * e:4 * e + 4])
        io, iop = _ll(lay["idx_off"][4 * e:4 * e + 4])
        oe = np.zeros((q1 - q0, s.d))
        rc = lib().oracle_attend_episode(s.H, s.dh, s.G, ntp, kp, pop, iop, q1 - q0, qp, kp_, pkp,
                                         _u8(ix), Rp, float(scale), h0, h1, oe.ctypes.data_as(_dp))
        if rc != 0:
            raise ValueError("oracle_attend_episode: bad arguments or indices")
        o[q0:q1, :] = np.where(np.isin(np.arange(s.d) // s.dh, np.arange(h0, h1))[None, :], oe, o[q0:q1])
    return o


# ---------------------------------------------------------------------------
# Per-token budgets (Sec. 3.5)
# ---------------------------------------------------------------------------

def budget_shares(n, B, S):
    """Counts by priority rank (rank 0 = highest) of the allocator reading."""
    out = np.zeros(max(n, 1), np.int32)
    if lib().oracle_budget_shares(int(n), int(B), int(S), out.ctypes.data_as(_ip)) != 0:
        raise ValueError("oracle_budget_shares: bad arguments")
    return out[:n]


def budget_allocate(pri, B, S):
    """Per-token counts for priorities pri (ties: lower index ranks higher)."""
    pri, pp = _d(np.asarray(pri, np.float64).reshape(-1))
    n = pri.size
    out = np.zeros(max(n, 1), np.int32)
    if lib().oracle_budget_allocate(n, int(B), int(S), pp if n else None, out.ctypes.data_as(_ip)) != 0:
        raise ValueError("oracle_budget_allocate: bad arguments")
    return out[:n]


def budget_idx_offsets(spec: Spec, ktok_layer):
    """Where each routed token's indices start: per segment, idx_off + the
    prefix sum of the counts of the tokens before it (Sec. 3.5 packing)."""
    lay = spec.lay
    nt = spec.n_tok.reshape(-1)
    out = np.zeros(int(spec.ep_row[-1]), np.int64)
    for sgi in range(nt.size):
        r0, n = int(lay["row_off"][sgi]), int(nt[sgi])
        if n:
            kk = np.asarray(ktok_layer[r0:r0 + n], np.int64)
            out[r0:r0 + n] = lay["idx_off"][sgi] + np.concatenate([[0], np.cumsum(kk)[:-1]])
    return out


def route_layer_budget(spec: Spec, h, W_re, b_re, W_v, b_v, W_role, W_l, b_l, u, alpha_role, alpha_lang,
                       episodes=None, k_force=None):
    """Additive-router scores, priorities pi = u . a and per-token budgets for
    every (listed) episode of one layer; returns idx [idx_bytes] uint8,
    ktok [rows] int32, gamma [rows][G], pri [rows], margin [rows]."""
    s = spec
    lay = s.lay
    rows = int(s.ep_row[-1])
    idx = np.zeros(max(lay["idx_bytes"], 1), np.uint8)
    ktok = np.zeros(max(rows, 1), np.int32)
    gamma = np.full((max(rows, 1), s.G), np.nan)
    pri = np.full(max(rows, 1), np.nan)
    margin = np.full(max(rows, 1), np.nan)
    Wre, Wrep = _d(W_re)
    bre, brep = _d(b_re)
    Wv, Wvp = _d(W_v)
    bv, bvp = _d(b_v)
    Wr, Wrp = _d(W_role)
    Wl, Wlp = _d(W_l)
    bl, blp = _d(b_l)
    uu, up = _d(u)
    kf = None if k_force is None else np.ascontiguousarray(k_force, np.int32)
    for e in (range(s.E) if episodes is None else episodes):
        r0, r1 = int(s.ep_row[e]), int(s.ep_row[e + 1])
        n = max(r1 - r0, 1)
        he, hp = _d(h[r0:r1] if r1 > r0 else np.zeros((1, s.d)))
        nt, ntp = _i(s.n_tok[e])
        kk, kp = _i(s.k[e])
        io, iop = _ll(lay["idx_off"][4 * e:4 * e + 4])
        kt = np.zeros(n, np.int32)
        g_e = np.full((n, s.G), np.nan)
        p_e = np.full(n, np.nan)
        m_e = np.full(n, np.nan)
        kfe = None if kf is None else np.ascontiguousarray(
            kf[r0:r1] if r1 > r0 else np.zeros(1, np.int32), np.int32)
        rc = lib().oracle_route_episode_budget(
            s.d, s.G, s.C, ntp, kp, iop, hp, Wrep, brep, Wvp, bvp, Wrp, Wlp, blp, up, float(alpha_role),
            float(alpha_lang), None if kfe is None else kfe.ctypes.data_as(_ip), _u8(idx),
            kt.ctypes.data_as(_ip), g_e.ctypes.data_as(_dp), p_e.ctypes.data_as(_dp), m_e.ctypes.data_as(_dp))
        if rc != 0:
            raise ValueError("oracle_route_episode_budget: bad arguments or forced counts")
        ktok[r0:r1] = kt[:r1 - r0]
        gamma[r0:r1] = g_e[:r1 - r0]
        pri[r0:r1] = p_e[:r1 - r0]
        margin[r0:r1] = m_e[:r1 - r0]
    return {"idx": idx[:lay["idx_bytes"]], "ktok": ktok[:rows], "gamma": gamma[:rows], "pri": pri[:rows],
            "margin": margin[:rows]}


def pack_layer_budget(spec: Spec, v, R, idx, ktok, episodes=None):
    """Sec. 3.2 with per-token counts: z = R_h^T v_{i,h}; segment of n tokens
    holds [H][sum_i K_i][d_s] values, token i's kept groups at the prefix
    sum of the counts before it, in its index order. Returns packed
    [packed_elems] float64 (unlisted episodes stay zero)."""
    s = spec
    lay = s.lay
    ds = s.dh // s.G
    packed = np.zeros(max(lay["packed_elems"], 1))
    nt = s.n_tok.reshape(-1)
    R = np.asarray(R, np.float64)
    eps = range(s.E) if episodes is None else episodes
    for e in eps:
        for m in range(4):
            sgi = 4 * e + m
            n, r0 = int(nt[sgi]), int(lay["row_off"][sgi])
            if n == 0:
                continue
            kk = np.asarray(ktok[r0:r0 + n], np.int64)
            tot = int(kk.sum())
            pref = np.concatenate([[0], np.cumsum(kk)[:-1]])
            io, po = int(lay["idx_off"][sgi]), int(lay["packed_off"][sgi])
            for hh in range(s.H):
                z = np.asarray(v[r0:r0 + n, hh * s.dh:(hh + 1) * s.dh], np.float64) @ R[hh]   # rows: z = R^T v
                for i in range(n):
                    for j in range(int(kk[i])):
                        g = int(idx[io + pref[i] + j])
                        dst = po + (hh * tot + pref[i] + j) * ds
                        packed[dst:dst + ds] = z[i, g * ds:(g + 1) * ds]
    return packed[:lay["packed_elems"]]


def attend_layer_budget(spec: Spec, q, K, packed, idx, ktok, R, scale=0.0, episodes=None):
    """Attention over a cache packed with per-token counts (Sec. 3):
    p = softmax_j(q . k_j * scale) over the episode's cache tokens,
    y = sum_j p_j M_j z_j (zeros outside the kept groups), o = R_h y.
    Returns o [q_rows][d] float64."""
    s = spec
    lay = s.lay
    ds = s.dh // s.G
    sc = scale if scale > 0 else 1.0 / np.sqrt(s.dh)
    o = np.zeros((int(s.ep_q[-1]), s.d))
    nt = s.n_tok.reshape(-1)
    R = np.asarray(R, np.float64)
    for e in (range(s.E) if episodes is None else episodes):
        r0, r1 = int(s.ep_row[e]), int(s.ep_row[e + 1])
        q0, q1 = int(s.ep_q[e]), int(s.ep_q[e + 1])
        if q1 == q0 or r1 == r0:
            continue
        for hh in range(s.H):
            ztil = np.zeros((r1 - r0, s.dh))
            for m in range(4):
                sgi = 4 * e + m
                n, rs_ = int(nt[sgi]), int(lay["row_off"][sgi])
                if n == 0:
                    continue
                kk = np.asarray(ktok[rs_:rs_ + n], np.int64)
                tot = int(kk.sum())
                pref = np.concatenate([[0], np.cumsum(kk)[:-1]])
                io, po = int(lay["idx_off"][sgi]), int(lay["packed_off"][sgi])
                for i in range(n):
                    for j in range(int(kk[i])):
                        g = int(idx[io + pref[i] + j])
                        src = po + (hh * tot + pref[i] + j) * ds
                        ztil[rs_ - r0 + i, g * ds:(g + 1) * ds] = packed[src:src + ds]
            qh = np.asarray(q[q0:q1, hh * s.dh:(hh + 1) * s.dh], np.float64)
            kh = np.asarray(K[r0:r1, hh * s.dh:(hh + 1) * s.dh], np.float64)
            sco = qh @ kh.T * sc
            sco -= sco.max(axis=1, keepdims=True)
            p = np.exp(sco)
            p /= p.sum(axis=1, keepdims=True)
            o[q0:q1, hh * s.dh:(hh + 1) * s.dh] = (p @ ztil) @ R[hh].T
    return o


# ---------------------------------------------------------------------------
# Token-level reduction (Sec. 3.1)
# ---------------------------------------------------------------------------

def select_count(n_view, ratio):
    """Tokens kept per view: ceil(r * n) (Sec. 3.1), the budget split evenly
    over the camera views (Sec. 4.1)."""
    return int(math.ceil(float(ratio) * int(n_view)))


def select_tokens(scores, x, ratio):
    """scores [E][V][n], x [E][V][n][...]: per (episode, view) the k highest
    scores (ties: lower index; NaN lowest), in token order. Returns
    keep_idx [E][V][k] int32 and x_keep [E][V][k][...]."""
    scores = np.asarray(scores, np.float64)
    E, V, n = scores.shape
    k = select_count(n, ratio)
    keep = np.zeros((E, V, k), np.int32)
    for e in range(E):
        for v in range(V):
            s = scores[e, v]
            # plain selection by the ranking rule, one token at a time
            order = sorted(range(n), key=lambda i: (0 if math.isnan(s[i]) else 1,
                                                    -math.inf if math.isnan(s[i]) else s[i], -i), reverse=True)
            keep[e, v] = np.sort(np.array(order[:k], np.int64)).astype(np.int32)
    xk = np.take_along_axis(np.asarray(x), keep.reshape(E, V, k, *([1] * (np.asarray(x).ndim - 3))), axis=2)
    return keep, xk


# ---------------------------------------------------------------------------
# Dense rotation (Sec. 4.1 geometry: one d x d orthonormal R per layer, S
# contiguous groups of d / S rotated dimensions)
# ---------------------------------------------------------------------------

def pack_layer_dense(spec: Spec, v, Rd, idx, episodes=None):
    """Sec. 3.2 with one dense R: z_i = R^T v_i over all d = H d_h dims, split
    into S contiguous groups of g = d / S; segment (n tokens, k) holds
    [n][k][g] values (the kept groups in index order). Returns packed
    [packed_elems] float64."""
    s = spec
    lay = s.lay
    g = s.d // s.G
    packed = np.zeros(max(lay["packed_elems"], 1))
    nt = s.n_tok.reshape(-1)
    kt = s.k.reshape(-1)
    Rd = np.asarray(Rd, np.float64)
    for e in (range(s.E) if episodes is None else episodes):
        for m in range(4):
            sgi = 4 * e + m
            n, k, r0 = int(nt[sgi]), int(kt[sgi]), int(lay["row_off"][sgi])
            if n == 0 or k == 0:
                continue
            io, po = int(lay["idx_off"][sgi]), int(lay["packed_off"][sgi])
            z = np.asarray(v[r0:r0 + n], np.float64) @ Rd          # rows: z = R^T v
            for i in range(n):
                for j in range(k):
                    grp = int(idx[io + i * k + j])
                    dst = po + (i * k + j) * g
                    packed[dst:dst + g] = z[i, grp * g:(grp + 1) * g]
    return packed[:lay["packed_elems"]]


def attend_layer_dense(spec: Spec, q, K, packed, idx, Rd, scale=0.0, episodes=None):
    """Attention over a dense-R cache (Sec. 3): per head h,
    p = softmax_j(q_h . k_{j,h} * scale), y = sum_j p_j M_j z_j (all d rotated
    dims, zeros outside the kept groups), o_h = R[rows of head h] y.
    Returns o [q_rows][d] float64."""
    s = spec
    lay = s.lay
    g = s.d // s.G
    sc = scale if scale > 0 else 1.0 / np.sqrt(s.dh)
    o = np.zeros((int(s.ep_q[-1]), s.d))
    nt = s.n_tok.reshape(-1)
    kt = s.k.reshape(-1)
    Rd = np.asarray(Rd, np.float64)
    for e in (range(s.E) if episodes is None else episodes):
        r0, r1 = int(s.ep_row[e]), int(s.ep_row[e + 1])
        q0, q1 = int(s.ep_q[e]), int(s.ep_q[e + 1])
        if q1 == q0 or r1 == r0:
            continue
        zm = np.zeros((r1 - r0, s.d))          # M_j z_j of every cache token
        for m in range(4):
            sgi = 4 * e + m
            n, k, rs_ = int(nt[sgi]), int(kt[sgi]), int(lay["row_off"][sgi])
            io, po = int(lay["idx_off"][sgi]), int(lay["packed_off"][sgi])
            for i in range(n):
                for j in range(k):
                    grp = int(idx[io + i * k + j])
                    src = po + (i * k + j) * g
                    zm[rs_ - r0 + i, grp * g:(grp + 1) * g] = packed[src:src + g]
        for hh in range(s.H):
            qh = np.asarray(q[q0:q1, hh * s.dh:(hh + 1) * s.dh], np.float64)
            kh = np.asarray(K[r0:r1, hh * s.dh:(hh + 1) * s.dh], np.float64)
            sco = qh @ kh.T * sc
            sco -= sco.max(axis=1, keepdims=True)
            p = np.exp(sco)
            p /= p.sum(axis=1, keepdims=True)
            o[q0:q1, hh * s.dh:(hh + 1) * s.dh] = (p @ zm) @ Rd[hh * s.dh:(hh + 1) * s.dh, :].T
    return o
