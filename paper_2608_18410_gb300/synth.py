"""Seeded synthetic inputs for the RoleSub hot path.

This module only draws numbers; it holds none of the method's arithmetic, so
both the CUDA path and the fp64 oracle can be fed from it.

Shapes follow OpenVLA-OFT-7B (Llama-2-7B backbone: 32 heads x 128) as used in
the paper's setup (Sec. 4.1, "Model" and "RoleSub configuration"); weights are
random (no trained checkpoints exist here).

Recipe (one numpy PCG64 stream per tensor block):
  stream = PCG64(SeedSequence([seed, layer, episode, tensor_id]))
  activations h, v, q, K   ~ N(0, 1)      drawn in float32
  weights W_re, W1, W2     ~ N(0, 0.02)   drawn in float32, scaled in float32
  biases  b_re, b1, b2     ~ N(0, 0.02)   float32 (biases are always fp32)
  additive router (gen_additive_weights):
    W_v, W_l ~ N(0, 0.02), W_role ~ N(0, 1), b_v, b_l ~ N(0, 0.02) (fp32)
  per-token budgets (gen_priority): u ~ N(0, 1) (fp32), one C-vector per layer
  dense rotation (gen_dense_rotation): one d x d orthonormal R per layer, Haar
    from the QR of an fp64 Gaussian for d <= 1024, else kron(Q1, Q2) of two
    Haar factors (64 x 64 each at d = 4096): dense and orthonormal
  R_h: Haar-random orthogonal d_h x d_h, from the QR factorisation of an
       fp64 N(0, 1) matrix with column signs fixed by sign(diag(R_qr)).
bf16 tensors are rounded float32 -> bf16 with round-to-nearest-even and are
returned as uint16 bit patterns; `widen()` turns them back into exact float64.

Row order of the cache (per layer): episode-major, then kind-minor
(vis, lang, prop, act); query rows are episode-major.
"""
from __future__ import annotations

import dataclasses
from concurrent.futures import ThreadPoolExecutor

import numpy as np

KINDS = ("vis", "lang", "prop", "act")

TID = {"h": 1, "v": 2, "q": 3, "K": 4, "R": 5, "W_re": 6, "b_re": 7,
       "W1": 8, "b1": 9, "W2": 10, "b2": 11, "episodes": 12, "near_tie": 13,
       "packed": 14, "idx": 15, "W_v": 16, "b_v": 17, "W_role": 18, "W_l": 19, "b_l": 20,
       "u": 21, "R_dense": 22}


@dataclasses.dataclass(frozen=True)
class Episode:
    """One policy episode's retained cache: token counts and kept groups."""
    n_vis: int
    n_lang: int
    n_query: int
    k_vis: int
    k_lang: int
    n_prop: int = 0
    n_act: int = 0
    k_prop: int = -1   # -1: same as num_groups (uncompressed)
    k_act: int = -1

    def n_tok(self):
        return (self.n_vis, self.n_lang, self.n_prop, self.n_act)

    def k(self, G):
        kp = G if self.k_prop < 0 else self.k_prop
        ka = G if self.k_act < 0 else self.k_act
        return (self.k_vis, self.k_lang, kp, ka)

    @property
    def n_cache(self):
        return self.n_vis + self.n_lang + self.n_prop + self.n_act


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    dtype: str            # "f32" or "bf16"
    L: int                # layers
    H: int                # heads
    dh: int               # head dim
    G: int                # value groups per head
    C: int                # latent role dim
    F: int                # router hidden width
    episodes: tuple
    seed: int
    alpha_role: float = 0.1
    alpha_lang: float = 0.1
    near_tie: bool = False
    describe: str = ""

    @property
    def d(self):
        return self.H * self.dh

    @property
    def rows(self):
        return sum(e.n_cache for e in self.episodes)

    @property
    def q_rows(self):
        return sum(e.n_query for e in self.episodes)

    @property
    def E(self):
        return len(self.episodes)

    def n_tok_array(self):
        return np.array([e.n_tok() for e in self.episodes], dtype=np.int32)

    def k_array(self):
        return np.array([e.k(self.G) for e in self.episodes], dtype=np.int32)

    def n_query_array(self):
        return np.array([e.n_query for e in self.episodes], dtype=np.int32)

    def with_layers(self, L):
        return dataclasses.replace(self, L=L)

    def with_dtype(self, dtype):
        return dataclasses.replace(self, dtype=dtype)


# ---------------------------------------------------------------------------
# The five workloads: tiny fp32, one OpenVLA-OFT layer, the 32-layer sweep,
# aggressive near-tie compression, batched ragged serving.
# ---------------------------------------------------------------------------

def c0():
    return Workload("c0_tiny_f32", "f32", L=1, H=8, dh=64, G=8, C=16, F=64,
                    episodes=(Episode(64, 16, 8, 4, 4),), seed=0,
                    describe="1 layer, 8x64 heads, 64 vis + 16 lang cache tokens, 8 queries, G=8 k=4, fp32")


def c1():
    return Workload("c1_oft_layer_bf16", "bf16", L=1, H=32, dh=128, G=16, C=64, F=256,
                    episodes=(Episode(128, 48, 64, 4, 16),), seed=1,
                    describe="1 OpenVLA-OFT layer: 32x128 heads, 128 vis (k=4/16) + 48 lang (k=16/16), 64 queries, bf16")


C2_POINTS = [(nv, kv) for nv in (256, 128, 64) for kv in (8, 4, 2)]


def c2(n_vis=128, k_vis=4):
    return Workload(f"c2_stack_nv{n_vis}_k{k_vis}", "bf16", L=32, H=32, dh=128, G=16, C=64, F=256,
                    episodes=(Episode(n_vis, 48, 64, k_vis, 16),), seed=2,
                    describe=f"32-layer stack, {n_vis} vis (k={k_vis}/16) + 48 lang (k=16), 64 queries, bf16")


def c3():
    return Workload("c3_aggressive_near_tie", "bf16", L=32, H=32, dh=128, G=16, C=64, F=256,
                    episodes=(Episode(64, 48, 64, 2, 4),), seed=3, near_tie=True,
                    describe="32 layers, 64 vis (k=2/16) + 48 lang (k=4/16), 64 queries, router near-ties, bf16")


def c4(num_episodes=64):
    rng = _rng(4, 0, 0, TID["episodes"])
    eps = []
    for _ in range(num_episodes):
        nv = int(rng.integers(32, 257))
        nl = int(rng.integers(16, 65))
        kv = int(rng.choice([2, 4, 8]))
        kl = int(rng.choice([2, 4, 8]))
        eps.append(Episode(nv, nl, 64, kv, kl))
    return Workload(f"c4_batched_ragged_b{num_episodes}", "bf16", L=32, H=32, dh=128, G=16, C=64, F=256,
                    episodes=tuple(eps), seed=4,
                    describe=f"batch {num_episodes} ragged episodes (vis U[32,256], lang U[16,64], k in {{2,4,8}}), 32 layers, 64 queries each, bf16")


WORKLOADS = {"c0": c0, "c1": c1, "c2": c2, "c3": c3, "c4": c4}


# ---------------------------------------------------------------------------
# Drawing
# ---------------------------------------------------------------------------

def _rng(seed, layer, episode, tid):
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, layer, episode, tid])))


def f32_to_bf16_bits(x):
    """float32 -> bf16 bit patterns, round-to-nearest-even (finite inputs)."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    r = (b + np.uint32(0x7FFF) + ((b >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)
    return r.astype(np.uint16)


def bf16_bits_to_f32(b):
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def widen(x, dtype):
    """Exact float64 copy of a stored tensor (bf16 bits or float32)."""
    if dtype == "bf16":
        return bf16_bits_to_f32(x).astype(np.float64)
    return np.asarray(x, dtype=np.float32).astype(np.float64)


def _store(x32, dtype):
    return f32_to_bf16_bits(x32) if dtype == "bf16" else np.ascontiguousarray(x32, dtype=np.float32)


def _normal(seed, layer, ep, tid, shape, scale=1.0):
    x = _rng(seed, layer, ep, tid).standard_normal(size=shape, dtype=np.float32)
    if scale != 1.0:
        x *= np.float32(scale)
    return x


def haar_orthogonal(rng, n):
    a = rng.standard_normal(size=(n, n))
    qm, rm = np.linalg.qr(a)
    s = np.sign(np.diag(rm))
    s[s == 0] = 1.0
    return qm * s[None, :]


def storage_dtype(dtype):
    return np.uint16 if dtype == "bf16" else np.float32


def alloc_inputs(wl: Workload):
    """Empty host arrays (numpy) for every input of compress + attend."""
    sd = storage_dtype(wl.dtype)
    L, d, rows, qr = wl.L, wl.d, wl.rows, wl.q_rows
    return {
        "h": np.empty((L, rows, d), sd),
        "v": np.empty((L, rows, d), sd),
        "K": np.empty((L, rows, d), sd),
        "q": np.empty((L, qr, d), sd),
        "R": np.empty((L, wl.H, wl.dh, wl.dh), sd),
        "W_re": np.empty((L, wl.C, d), sd),
        "b_re": np.empty((L, wl.C), np.float32),
        "W1": np.empty((L, wl.F, 2 * d + wl.C), sd),
        "b1": np.empty((L, wl.F), np.float32),
        "W2": np.empty((L, wl.G, wl.F), sd),
        "b2": np.empty((L, wl.G), np.float32),
    }


def _fill_layer_weights(wl, out, layer, slot=None):
    slot = layer if slot is None else slot
    s, d = wl.seed, wl.d
    R = np.empty((wl.H, wl.dh, wl.dh), np.float64)
    rng = _rng(s, layer, 0, TID["R"])
    for hh in range(wl.H):
        R[hh] = haar_orthogonal(rng, wl.dh)
    out["R"][slot] = _store(R.astype(np.float32), wl.dtype)
    out["W_re"][slot] = _store(_normal(s, layer, 0, TID["W_re"], (wl.C, d), 0.02), wl.dtype)
    out["b_re"][slot] = _normal(s, layer, 0, TID["b_re"], (wl.C,), 0.02)
    out["W1"][slot] = _store(_normal(s, layer, 0, TID["W1"], (wl.F, 2 * d + wl.C), 0.02), wl.dtype)
    out["b1"][slot] = _normal(s, layer, 0, TID["b1"], (wl.F,), 0.02)
    W2 = _normal(s, layer, 0, TID["W2"], (wl.G, wl.F), 0.02)
    b2 = _normal(s, layer, 0, TID["b2"], (wl.G,), 0.02)
    if wl.near_tie:
        W2, b2 = _near_tie_rows(wl, layer, W2, b2)
    out["W2"][slot] = _store(W2, wl.dtype)
    out["b2"][slot] = b2


def _near_tie_rows(wl, layer, W2, b2):
    """Router output rows built to make near-tied group scores.

    The G rows split into clusters of 4. Rows inside a cluster are identical,
    so their scores differ only by their fp32 biases: cluster 0 has identical
    biases (exact ties), the others add offsets drawn uniformly in [0, 1e-3).
    """
    rng = _rng(wl.seed, layer, 0, TID["near_tie"])
    W2 = W2.copy()
    b2 = b2.copy()
    for c0_ in range(0, wl.G, 4):
        base = c0_
        for j in range(c0_, min(c0_ + 4, wl.G)):
            W2[j] = W2[base]
            off = 0.0 if c0_ == 0 else float(rng.uniform(0.0, 1e-3))
            b2[j] = np.float32(b2[base] + np.float32(off))
    return W2, b2


def _fill_layer_acts(wl, out, layer):
    s, d = wl.seed, wl.d
    r = 0
    qrow = 0
    for e, ep in enumerate(wl.episodes):
        n = ep.n_cache
        if n:
            out["h"][layer, r:r + n] = _store(_normal(s, layer, e, TID["h"], (n, d)), wl.dtype)
            out["v"][layer, r:r + n] = _store(_normal(s, layer, e, TID["v"], (n, d)), wl.dtype)
            out["K"][layer, r:r + n] = _store(_normal(s, layer, e, TID["K"], (n, d)), wl.dtype)
        if ep.n_query:
            out["q"][layer, qrow:qrow + ep.n_query] = _store(
                _normal(s, layer, e, TID["q"], (ep.n_query, d)), wl.dtype)
        r += n
        qrow += ep.n_query


def gen_layer_weights(wl: Workload, layer: int):
    """The weights of one layer, the same draws as gen_inputs makes for it."""
    sd = storage_dtype(wl.dtype)
    d = wl.d
    out = {"R": np.empty((1, wl.H, wl.dh, wl.dh), sd), "W_re": np.empty((1, wl.C, d), sd),
           "b_re": np.empty((1, wl.C), np.float32), "W1": np.empty((1, wl.F, 2 * d + wl.C), sd),
           "b1": np.empty((1, wl.F), np.float32), "W2": np.empty((1, wl.G, wl.F), sd),
           "b2": np.empty((1, wl.G), np.float32)}
    _fill_layer_weights(wl, out, layer, slot=0)
    return {k: v[0] for k, v in out.items()}


def gen_episode_acts(wl: Workload, layer: int, e: int):
    """h, v, K [n_cache][d] and q [n_query][d] of one episode of one layer,
    the same draws as gen_inputs makes for it."""
    s, d = wl.seed, wl.d
    ep = wl.episodes[e]
    out = {}
    for name in ("h", "v", "K"):
        out[name] = _store(_normal(s, layer, e, TID[name], (ep.n_cache, d)), wl.dtype) if ep.n_cache else \
            np.empty((0, d), storage_dtype(wl.dtype))
    out["q"] = _store(_normal(s, layer, e, TID["q"], (ep.n_query, d)), wl.dtype) if ep.n_query else \
        np.empty((0, d), storage_dtype(wl.dtype))
    return out


def gen_inputs(wl: Workload, threads: int = 8):
    """All inputs of every layer, as host numpy arrays."""
    out = alloc_inputs(wl)
    jobs = []
    with ThreadPoolExecutor(max_workers=max(1, threads)) as ex:
        for layer in range(wl.L):
            jobs.append(ex.submit(_fill_layer_weights, wl, out, layer))
            jobs.append(ex.submit(_fill_layer_acts, wl, out, layer))
        for j in jobs:
            j.result()
    return out


def gen_additive_weights(wl: Workload):
    """Token, role and language heads of the additive routing score, every layer.

    W_v, W_l [L][G][d] and W_role [L][G][C] in the workload's storage dtype;
    b_v, b_l [L][G] float32. W_role is drawn at unit scale: it maps a
    probability vector, so its term is comparable to the others at
    alpha_role = 0.1. With wl.near_tie, groups form clusters of 4 with
    identical rows of W_v, W_role, W_l and b_l, and b_v as in the
    concatenation router's near-tie recipe (cluster 0 tied exactly, the others
    offset by uniform [0, 1e-3)).
    """
    s, d, G, C, L = wl.seed, wl.d, wl.G, wl.C, wl.L
    sd = storage_dtype(wl.dtype)
    out = {"W_v": np.empty((L, G, d), sd), "b_v": np.empty((L, G), np.float32),
           "W_role": np.empty((L, G, C), sd), "W_l": np.empty((L, G, d), sd),
           "b_l": np.empty((L, G), np.float32)}
    for layer in range(L):
        Wv = _normal(s, layer, 0, TID["W_v"], (G, d), 0.02)
        bv = _normal(s, layer, 0, TID["b_v"], (G,), 0.02)
        Wr = _normal(s, layer, 0, TID["W_role"], (G, C))
        Wl = _normal(s, layer, 0, TID["W_l"], (G, d), 0.02)
        bl = _normal(s, layer, 0, TID["b_l"], (G,), 0.02)
        if wl.near_tie:
            rng = _rng(s, layer, 0, TID["near_tie"])
            for c0_ in range(0, G, 4):
                for j in range(c0_, min(c0_ + 4, G)):
                    Wv[j], Wr[j], Wl[j], bl[j] = Wv[c0_], Wr[c0_], Wl[c0_], bl[c0_]
                    off = 0.0 if c0_ == 0 else float(rng.uniform(0.0, 1e-3))
                    bv[j] = np.float32(bv[c0_] + np.float32(off))
        out["W_v"][layer] = _store(Wv, wl.dtype)
        out["b_v"][layer] = bv
        out["W_role"][layer] = _store(Wr, wl.dtype)
        out["W_l"][layer] = _store(Wl, wl.dtype)
        out["b_l"][layer] = bl
    return out


def gen_priority(wl: Workload):
    """Priority vectors u [L][C] float32 of the per-token budget allocator."""
    return np.stack([_normal(wl.seed, layer, 0, TID["u"], (wl.C,)) for layer in range(wl.L)]).astype(np.float32)


def gen_dense_rotation(wl: Workload):
    """One d x d orthonormal R per layer (storage dtype), [L][d][d]."""
    d = wl.d
    out = np.empty((wl.L, d, d), storage_dtype(wl.dtype))
    for layer in range(wl.L):
        rng = _rng(wl.seed, layer, 0, TID["R_dense"])
        if d <= 1024:
            R = haar_orthogonal(rng, d)
        else:
            a = 1 << (int(np.log2(d)) // 2)
            R = np.kron(haar_orthogonal(rng, a), haar_orthogonal(rng, d // a))
        out[layer] = _store(R.astype(np.float32), wl.dtype)
    return out


def gen_packed(wl: Workload, packed_elems_per_layer: int, idx_bytes_per_layer: int, seg_table):
    """Synthetic packed values and group indices for testing attention alone.

    seg_table: iterable of (n_tokens, k, packed_off, idx_off) per segment.
    Indices are k distinct ascending groups per token drawn uniformly.
    """
    sd = storage_dtype(wl.dtype)
    packed = np.zeros((wl.L, packed_elems_per_layer), sd)
    idx = np.zeros((wl.L, idx_bytes_per_layer), np.uint8)
    for layer in range(wl.L):
        rng = _rng(wl.seed, layer, 0, TID["idx"])
        x = _normal(wl.seed, layer, 0, TID["packed"], (packed_elems_per_layer,))
        packed[layer] = _store(x, wl.dtype)
        for (n, k, _poff, ioff) in seg_table:
            for i in range(n):
                sel = np.sort(rng.choice(wl.G, size=k, replace=False)) if k < wl.G else np.arange(wl.G)
                idx[layer, ioff + i * k: ioff + (i + 1) * k] = sel.astype(np.uint8)
    return packed, idx
