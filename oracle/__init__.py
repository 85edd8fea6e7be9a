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
  compress/attend -- all-kept == dense attention (1e-10), none-kept == 0,
                     every mask on tiny inputs == dense attention over
                     R M R^T v, complement linearity, R = I textbook case,
                     token / group permutation equivariance
"""
from __future__ import annotations

import ctypes
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
