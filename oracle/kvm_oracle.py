"""fp64 CPU oracle for true-tail incremental memory maintenance.

TEST INFRASTRUCTURE ONLY.  The test suite, the smoke check and the CPU-baseline
leg of the benchmark may import this module; the library's product path never
does, and this module imports nothing from the library.

What it computes (Xu, "Long-Lived Characters, Local Inference: Incremental
Memory Maintenance for Game NPCs", §4):
  * A character context is a state (A_t, R_t, p_t): per attention layer the
    live KV cache A, per gated-delta-rule layer the recurrent state S (the
    part of R this path carries), and the next position id p (§4.1).
  * A maintenance round first removes the KV of superseded records from every
    attention layer, A_bar = A \\ A[D_t] (Eq. 2), then runs the replacement
    tokens U_t forward at the true tail, (A', R', p') = F(U_t; A_bar, R, p)
    (Eq. 3): new keys are rotated at their actual positions p, p+1, ...,
    stored keys are never re-rotated, removed positions become holes and the
    cursor only moves forward (§4.2); the recurrent state continues from its
    previous value and is not rolled back by a removal (§4.1).
  * Attention layers are causal GQA softmax attention with rotary position
    embedding on the first R dims of each head (RoFormer, cited in §4.2).
  * Gated-delta-rule layers follow Gated DeltaNet (Yang et al. 2025, the
    recurrent layer family named in §4.1 and §5.1):
        S_t = alpha_t S_{t-1} (I - beta_t k_t k_t^T) + beta_t v_t k_t^T,
        o_t = S_t q_t.
Everything is plain fp64 numpy, written in the order the definitions state it:
token by token for the recurrence, one query row at a time over an explicit
key list for attention, an explicit keep mask for removal.  `gdn_chunked` is a
second, independent formulation (chunked WY/UT form) used only to pin the
chunk algebra the GPU kernel relies on.

Readings where the paper is silent (each also listed in the design notes):
  - recurrence gate placement as above; o_t = S_t q_t with no output scaling
  - attention scale 1/sqrt(head_dim)
  - RoPE pairs (d, d + R/2) for d < R/2 (half-split), frequency
    theta^(-2d/R) with the exponent over the R rotary dims; dims >= R pass
  - GQA: query head h reads KV head h // (Hq / Hkv)
  - spans are half-open [begin, end) live-index ranges on the current
    compacted cache; removal happens before the tail forward
  - an empty cache is allowed: the tail then attends to itself only
"""
from __future__ import annotations

import math
import numpy as np


# ----------------------------------------------------------------------------
# input widening (bf16 / fp32 bytes -> fp64)
# ----------------------------------------------------------------------------
def bf16_to_f64(u16) -> np.ndarray:
    """bf16 bit patterns (uint16) -> fp64 values."""
    u = np.asarray(u16, dtype=np.uint16).astype(np.uint32) << 16
    return u.view(np.float32).astype(np.float64)


def f32_to_f64(x) -> np.ndarray:
    return np.asarray(x, dtype=np.float32).astype(np.float64)


# ----------------------------------------------------------------------------
# Removal of superseded KV (Eq. 2; §4.2 span verification)
# ----------------------------------------------------------------------------
class SpanError(ValueError):
    """A deletion range that does not describe live entries (§4.2: the runtime
    verifies deletion ranges against live spans)."""


def validate_spans(L: int, begins, ends) -> None:
    """Spans must be non-empty, inside [0, L), sorted and pairwise disjoint."""
    begins = [int(x) for x in begins]
    ends = [int(x) for x in ends]
    if len(begins) != len(ends):
        raise SpanError("begin/end count mismatch")
    prev_end = 0
    for i, (b, e) in enumerate(zip(begins, ends)):
        if not (0 <= b < e <= L):
            raise SpanError(f"span {i} [{b},{e}) empty or outside [0,{L})")
        if i > 0 and b < prev_end:
            raise SpanError(f"span {i} overlaps or precedes span {i-1}")
        prev_end = e


def keep_mask(L: int, begins, ends) -> np.ndarray:
    """keep[i] is False exactly when live index i lies in a removed span."""
    validate_spans(L, begins, ends)
    keep = np.ones(L, dtype=bool)
    for b, e in zip(begins, ends):
        keep[int(b):int(e)] = False
    return keep


def kv_compact(K, V, pos, begins, ends):
    """A_bar = A \\ A[D_t] (Eq. 2) for one attention layer of one character.

    K, V: [Hkv][L][D] (any dtype: bytes are carried, not converted);
    pos: [L] position ids.  Survivors keep their values and positions and
    their relative order; nothing is re-rotated (§4.2).
    Returns (K', V', pos', gather) with gather[j] = old live index of new j.
    """
    L = pos.shape[0]
    keep = keep_mask(L, begins, ends)
    gather = np.nonzero(keep)[0]
    return K[:, keep, :], V[:, keep, :], pos[keep], gather.astype(np.int64)


# ----------------------------------------------------------------------------
# Rotary position embedding at absolute positions (§4.2, RoFormer)
# ----------------------------------------------------------------------------
def rope_frequencies(R: int, theta: float) -> np.ndarray:
    """omega_d = theta^(-2d/R), d = 0 .. R/2-1."""
    d = np.arange(R // 2, dtype=np.float64)
    return np.power(float(theta), -2.0 * d / R)


def rope(x: np.ndarray, positions, R: int, theta: float) -> np.ndarray:
    """Rotate the first R dims of each head of x [n][H][D] at positions [n].

    Pair (d, d+R/2) is rotated by angle positions * omega_d:
        x'_d       = x_d cos - x_{d+R/2} sin
        x'_{d+R/2} = x_{d+R/2} cos + x_d sin
    Dims >= R are returned unchanged.
    """
    x = np.asarray(x, dtype=np.float64)
    out = x.copy()
    if R == 0:
        return out
    h = R // 2
    ang = np.asarray(positions, dtype=np.float64)[:, None] * rope_frequencies(R, theta)[None, :]
    c = np.cos(ang)[:, None, :]
    s = np.sin(ang)[:, None, :]
    lo = x[:, :, :h]
    hi = x[:, :, h:R]
    out[:, :, :h] = lo * c - hi * s
    out[:, :, h:R] = hi * c + lo * s
    return out


# ----------------------------------------------------------------------------
# Tail attention (Eq. 3 for a full-attention layer)
# ----------------------------------------------------------------------------
def attend_row(q_row: np.ndarray, keys: np.ndarray, values: np.ndarray) -> np.ndarray:
    """softmax(q . k_j / sqrt(D)) weighted sum of v_j over an explicit key list.

    q_row [D], keys [n][D], values [n][D]; n >= 1."""
    D = q_row.shape[0]
    s = keys @ q_row / math.sqrt(D)
    w = np.exp(s - s.max())
    return (w[:, None] * values).sum(axis=0) / w.sum()


def tail_attention(q_rot, K_all, V_all, L_prev: int) -> np.ndarray:
    """Causal GQA attention of M tail queries over L_prev surviving entries
    plus the tail's own keys.

    q_rot [M][Hq][D] (already rotated), K_all/V_all [Hkv][L_prev+M][D] with
    the tail's keys at indices L_prev .. L_prev+M-1.  Tail token i sees every
    survivor and tail keys j <= i (every survivor precedes the tail in
    position, so this order rule is the position mask pos_j <= pos_i).
    Query head h reads KV head h // (Hq/Hkv).  Returns [M][Hq][D] fp64."""
    M, Hq, D = q_rot.shape
    Hkv = K_all.shape[0]
    g = Hq // Hkv
    out = np.zeros((M, Hq, D))
    for i in range(M):
        n_vis = L_prev + i + 1
        for h in range(Hq):
            kv = h // g
            out[i, h] = attend_row(q_rot[i, h], K_all[kv, :n_vis], V_all[kv, :n_vis])
    return out


# ----------------------------------------------------------------------------
# Attention-probe diagnostics (§5.3; Appendix C)
# ----------------------------------------------------------------------------
def probe_distributions(cache: AttnCache, q_raw) -> np.ndarray:
    """Per probe query and head, the attention distribution over the live
    entries.  The probe queries are those of the last n_q live entries:
    q_raw [n_q][Hq][D] unrotated; query i sits at live index L - n_q + i,
    is rotated at that entry's position by the caller-supplied rotation
    (rotate_probe_queries) and sees entries 0 .. L - n_q + i.  Removed
    records left no entries, so the softmax denominator runs over live
    tokens only.  Returns [n_q][Hq][L], zero past each query's limit."""
    q = np.asarray(q_raw, np.float64)
    n_q, Hq, D = q.shape
    Hkv = cache.K.shape[0]
    g = Hq // Hkv
    L = cache.live
    out = np.zeros((n_q, Hq, L))
    for i in range(n_q):
        n_vis = L - n_q + i + 1
        for h in range(Hq):
            s = cache.K[h // g, :n_vis] @ q[i, h] / math.sqrt(D)
            w = np.exp(s - s.max())
            out[i, h, :n_vis] = w / w.sum()
    return out


def rotate_probe_queries(cache: AttnCache, q_raw, R: int, theta: float) -> np.ndarray:
    """Rotate probe query i at the position of live entry L - n_q + i."""
    n_q = np.asarray(q_raw).shape[0]
    return rope(q_raw, cache.pos[cache.live - n_q:], R, theta)


def attention_probe(cache: AttnCache, q_raw, R: int, theta: float) -> np.ndarray:
    """The probe distribution over the live entries [L]: the per query and
    head distributions averaged over the n_q queries and every head."""
    d = probe_distributions(cache, rotate_probe_queries(cache, q_raw, R, theta))
    return d.mean(axis=(0, 1))


def group_mass(a, group_of, n_groups: int) -> np.ndarray:
    """Summed probability of each group; entries with group -1 count for none."""
    m = np.zeros(n_groups)
    for x, gid in zip(np.asarray(a, np.float64), np.asarray(group_of)):
        if gid >= 0:
            m[int(gid)] += x
    return m


def effective_group_count(mass) -> float:
    """exp(-sum_i a_i log a_i) for the group probabilities a_i = mass_i /
    sum(mass) (0 log 0 = 0), the dispersion measure of §5.3."""
    m = np.asarray(mass, np.float64)
    a = m / m.sum()
    nz = a[a > 0]
    return float(np.exp(-(nz * np.log(nz)).sum()))


def total_variation(p, q) -> float:
    """Total variation distance 0.5 * sum |p_i - q_i| (§6.3)."""
    return float(0.5 * np.abs(np.asarray(p, np.float64) - np.asarray(q, np.float64)).sum())


# ----------------------------------------------------------------------------
# Gated delta rule (§4.1, Gated DeltaNet)
# ----------------------------------------------------------------------------
def gdn_recurrent(q, k, v, alpha, beta, S0):
    """Token-by-token recurrence from the carried state S0.

    q, k [M][H][d_k], v [M][H][d_v], alpha, beta [M][H], S0 [H][d_v][d_k].
        S_t = alpha_t S_{t-1} (I - beta_t k_t k_t^T) + beta_t v_t k_t^T
        o_t = S_t q_t
    Returns (o [M][H][d_v], S_M [H][d_v][d_k])."""
    q = np.asarray(q, np.float64)
    k = np.asarray(k, np.float64)
    v = np.asarray(v, np.float64)
    alpha = np.asarray(alpha, np.float64)
    beta = np.asarray(beta, np.float64)
    S = np.array(S0, dtype=np.float64, copy=True)
    M, H, dk = k.shape
    dv = v.shape[2]
    eye = np.eye(dk)
    o = np.zeros((M, H, dv))
    for t in range(M):
        for h in range(H):
            kt = k[t, h][:, None]                       # column vector
            vt = v[t, h][:, None]
            S[h] = alpha[t, h] * S[h] @ (eye - beta[t, h] * (kt @ kt.T)) \
                + beta[t, h] * (vt @ kt.T)
            o[t, h] = S[h] @ q[t, h]
    return o, S


def gdn_chunked(q, k, v, alpha, beta, S0, C: int = 64):
    """Same result as `gdn_recurrent`, computed chunk by chunk (WY/UT form).

    Within a chunk of c tokens starting from state S0, with g_t = sum_{u<=t}
    log alpha_u and Gamma_t = exp(g_t):
      L[t,j]  = exp(g_t - g_j) beta_j (k_t . k_j)   for j < t, else 0
      T       = (I + L)^-1                          (unit lower triangular)
      E       = T V - T diag(Gamma) K S0^T          (E_j = u_j / beta_j, the
                                                     pre-gate delta values)
      O       = diag(Gamma) Q S0^T + ((Q K^T) * Dec * beta_j) E,
                Dec[t,j] = exp(g_t - g_j) for j <= t, else 0
      S_next  = Gamma_c S0 + E^T diag(beta_j exp(g_c - g_j)) K
    Chunks start at the first tail token; the last chunk may be short."""
    q = np.asarray(q, np.float64)
    k = np.asarray(k, np.float64)
    v = np.asarray(v, np.float64)
    alpha = np.asarray(alpha, np.float64)
    beta = np.asarray(beta, np.float64)
    S = np.array(S0, dtype=np.float64, copy=True)
    M, H, dk = k.shape
    dv = v.shape[2]
    o = np.zeros((M, H, dv))
    for c0 in range(0, M, C):
        c1 = min(M, c0 + C)
        for h in range(H):
            Q = q[c0:c1, h]
            K = k[c0:c1, h]
            V = v[c0:c1, h]
            b = beta[c0:c1, h]
            g = np.cumsum(np.log(alpha[c0:c1, h]))
            n = c1 - c0
            dec = np.exp(g[:, None] - g[None, :])
            Lm = np.tril(dec * (K @ K.T) * b[None, :], -1)
            T = np.linalg.inv(np.eye(n) + Lm)
            E = T @ V - T @ (np.exp(g)[:, None] * K) @ S[h].T
            A = np.tril((Q @ K.T) * dec * b[None, :])
            o[c0:c1, h] = np.exp(g)[:, None] * (Q @ S[h].T) + A @ E
            S[h] = np.exp(g[-1]) * S[h] + E.T @ ((b * np.exp(g[-1] - g))[:, None] * K)
    return o, S


# ----------------------------------------------------------------------------
# Short convolution of a gated-delta-rule layer (§4.1: R_t holds the
# recurrent and the convolution states, and both continue without rollback)
# ----------------------------------------------------------------------------
def silu(x):
    """x * sigmoid(x)."""
    x = np.asarray(x, np.float64)
    return x / (1.0 + np.exp(-x))


def short_conv(x, state, w):
    """Causal depthwise convolution of width 4 over a tail, continuing from
    the carried state.

    x [M][C] pre-convolution inputs of the tail; state [3][C] the last three
    inputs before it (oldest first; zeros for a fresh context); w [C][4].
    With xx = [state; x], output t is y_t[c] = sum_{i=0..3} w[c][i] xx[t+i][c]
    (tap 3 is the current token).  Returns (y [M][C] before the activation,
    the new state: the last three rows of xx)."""
    x = np.asarray(x, np.float64)
    w = np.asarray(w, np.float64)
    xx = np.concatenate([np.asarray(state, np.float64), x], axis=0)
    M = x.shape[0]
    y = np.zeros_like(x)
    for t in range(M):
        for i in range(4):
            y[t] += w[:, i] * xx[t + i]
    return y, xx[-3:].copy()


def gdn_conv_inputs(q, k, v, conv_state, w):
    """Delta-rule inputs of a layer with short convolution: the channels of
    q [M][H][d_k], k [M][H][d_k], v [M][H][d_v] (in that order) go through
    short_conv and SiLU, then each head's k is scaled to unit L2 norm.
    Returns (q', k', v', new conv state)."""
    q = np.asarray(q, np.float64)
    k = np.asarray(k, np.float64)
    v = np.asarray(v, np.float64)
    M, H, dk = q.shape
    dv = v.shape[2]
    x = np.concatenate([q.reshape(M, H * dk), k.reshape(M, H * dk), v.reshape(M, H * dv)], axis=1)
    y, new_state = short_conv(x, conv_state, w)
    y = silu(y)
    q2 = y[:, :H * dk].reshape(M, H, dk)
    k2 = y[:, H * dk:2 * H * dk].reshape(M, H, dk)
    v2 = y[:, 2 * H * dk:].reshape(M, H, dv)
    k2 = k2 / np.linalg.norm(k2, axis=-1, keepdims=True)
    return q2, k2, v2, new_state


# ----------------------------------------------------------------------------
# Character state and one maintenance round (Eqs. 2-3)
# ----------------------------------------------------------------------------
class AttnCache:
    """Live KV of one attention layer: K, V [Hkv][L][D] fp64, pos [L] int64."""

    def __init__(self, K, V, pos):
        self.K = np.asarray(K, np.float64)
        self.V = np.asarray(V, np.float64)
        self.pos = np.asarray(pos, np.int64)

    @property
    def live(self) -> int:
        return int(self.pos.shape[0])

    def copy(self):
        return AttnCache(self.K.copy(), self.V.copy(), self.pos.copy())


class CharacterState:
    """(A_t, R_t, p_t) of one character (§4.1): caches[layer] for attention
    layers, states[layer] = S [H][d_v][d_k] for delta-rule layers, cursor p;
    conv[layer] = the short-convolution state [3][C] of delta-rule layers
    that have one (empty otherwise)."""

    def __init__(self, caches: dict, states: dict, cursor: int, conv: dict | None = None):
        self.caches = caches
        self.states = states
        self.cursor = int(cursor)
        self.conv = dict(conv) if conv else {}

    @classmethod
    def empty(cls, layer_kind, Hkv, D, H, dk, dv):
        caches, states = {}, {}
        for l, kind in enumerate(layer_kind):
            if kind == 1:
                caches[l] = AttnCache(np.zeros((Hkv, 0, D)), np.zeros((Hkv, 0, D)),
                                      np.zeros(0, np.int64))
            else:
                states[l] = np.zeros((H, dv, dk))
        return cls(caches, states, 0)

    def copy(self):
        return CharacterState({l: c.copy() for l, c in self.caches.items()},
                              {l: s.copy() for l, s in self.states.items()},
                              self.cursor, {l: c.copy() for l, c in self.conv.items()})


def tail_attn_prefill(cache: AttnCache, q, k_new, v_new, p: int, R: int, theta: float, positions=None):
    """Append the tail's rotated keys and values at the true tail and attend.

    q [M][Hq][D], k_new/v_new [M][Hkv][D] (unrotated, fp64); tail token i has
    position p + i, or positions[i] when given (the placement variants of
    §5.2: gapped or slot-preserving position ids).  Attention is causal in
    processing order either way (every survivor and tail keys j <= i).
    Returns (out [M][Hq][D], new cache)."""
    M = q.shape[0]
    if positions is None:
        positions = p + np.arange(M, dtype=np.int64)
    positions = np.asarray(positions, dtype=np.int64)
    q_rot = rope(q, positions, R, theta)
    k_rot = rope(k_new, positions, R, theta)
    L_prev = cache.live
    K_all = np.concatenate([cache.K, np.transpose(k_rot, (1, 0, 2))], axis=1)
    V_all = np.concatenate([cache.V, np.transpose(np.asarray(v_new, np.float64), (1, 0, 2))], axis=1)
    out = tail_attention(q_rot, K_all, V_all, L_prev)
    return out, AttnCache(K_all, V_all, np.concatenate([cache.pos, positions]))


def rerotate_keys(cache: AttnCache, begin: int, end: int, new_pos, R: int, theta: float) -> AttnCache:
    """Tail-and-relocate (§5.2): the stored keys of live entries [begin, end)
    were rotated at cache.pos; turn them to new_pos.  A key rotated at p and
    then by the angle of (q - p) is the key rotated at q, so each entry is
    rotated by its (new - old) difference; values are untouched.  Returns a
    new cache with the keys and positions replaced."""
    out = cache.copy()
    new_pos = np.asarray(new_pos, dtype=np.int64)
    delta = new_pos - cache.pos[begin:end]
    ks = np.transpose(cache.K[:, begin:end], (1, 0, 2))          # [n][Hkv][D]
    out.K[:, begin:end] = np.transpose(rope(ks, delta, R, theta), (1, 0, 2))
    out.pos[begin:end] = new_pos
    return out


def maintenance_round(state: CharacterState, layer_kind, begins, ends,
                      inputs: dict, R: int, theta: float, positions=None, delimiters=None,
                      conv_weights: dict | None = None):
    """One round for one character: Eq. 2 on every attention layer, then
    Eq. 3 layer by layer in model order, then p += M.

    inputs[layer] = dict(q, k, v[, alpha, beta]) as fp64 arrays (tail only).
    positions: optional [M] position ids of the tail (placement variants,
    §5.2); the cursor then moves to max(p, largest id + 1).
    delimiters: optional (begins, ends), half-open tail-index ranges of
    maintenance delimiters (§4.2): processed with the tail, then their
    direct KV are removed from every attention layer; their effect on the
    recurrent states and on later tail tokens remains, and their position
    ids stay consumed.
    conv_weights: optional {layer: w [C][4]} of delta-rule layers with short
    convolution; their q/k/v inputs are then pre-convolution projections,
    convolved from state.conv[layer] (zeros if absent) by gdn_conv_inputs.
    Returns (outputs {layer: [M][heads][dim]}, new state).  `state` is not
    modified."""
    new = state.copy()
    for l, kind in enumerate(layer_kind):
        if kind == 1:
            c = new.caches[l]
            K, V, pos, _ = kv_compact(c.K, c.V, c.pos, begins, ends)
            new.caches[l] = AttnCache(K, V, pos)
    M = None
    outs = {}
    for l, kind in enumerate(layer_kind):
        x = inputs[l]
        M = x["q"].shape[0]
        if kind == 1:
            outs[l], new.caches[l] = tail_attn_prefill(new.caches[l], x["q"], x["k"], x["v"],
                                                       new.cursor, R, theta, positions)
        else:
            q, k, v = x["q"], x["k"], x["v"]
            if conv_weights is not None and l in conv_weights:
                w = np.asarray(conv_weights[l], np.float64)
                st0 = new.conv.get(l, np.zeros((3, w.shape[0])))
                q, k, v, new.conv[l] = gdn_conv_inputs(q, k, v, st0, w)
            outs[l], new.states[l] = gdn_recurrent(q, k, v, x["alpha"], x["beta"], new.states[l])
    if M is not None:
        if positions is None:
            new.cursor += M
        elif M > 0:
            new.cursor = max(new.cursor, int(np.max(positions)) + 1)
    if delimiters is not None and len(delimiters[0]) > 0:
        for l, kind in enumerate(layer_kind):
            if kind == 1:
                c = new.caches[l]
                L_prev = c.live - M
                db = [L_prev + int(x) for x in delimiters[0]]
                de = [L_prev + int(x) for x in delimiters[1]]
                K, V, pos, _ = kv_compact(c.K, c.V, c.pos, db, de)
                new.caches[l] = AttnCache(K, V, pos)
    return outs, new


def refill(layer_kind, inputs: dict, Hkv, D, H, dk, dv, R, theta, conv_weights=None):
    """Dense refill: the whole token sequence read from an empty state at
    positions 0 .. n-1 (the reference construction of §5.2)."""
    empty = CharacterState.empty(layer_kind, Hkv, D, H, dk, dv)
    return maintenance_round(empty, layer_kind, [], [], inputs, R, theta, conv_weights=conv_weights)
