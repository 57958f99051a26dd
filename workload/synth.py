"""Seeded synthetic inputs for true-tail memory maintenance workloads.

This module only draws numbers: token tensors, gates, removal spans and
workload shapes.  It holds none of the maintenance arithmetic (no RoPE, no
attention, no delta rule, no compaction), so the fp64 oracle and the CUDA
library can both consume its output without sharing any of the method.

Every array is produced from ``numpy.random.default_rng(seed_tuple)`` (PCG64 +
SeedSequence), which yields the same stream on x86_64 and aarch64.  bf16
tensors are returned as ``uint16`` bit patterns (round-to-nearest-even from
fp64), fp32 tensors as ``float32``; both sides read the same bytes.

Distributions (the value recipe of the workloads):
  q, v        ~ N(0, 1) per element
  k           ~ N(0, 1), then scaled to unit L2 norm per (token, head)
  alpha       = sigmoid(x), x ~ N(3, 0.5)      (per token, per head, fp32)
  beta        = sigmoid(y), y ~ N(0, 1)        (per token, per head, fp32)
  prefix keys = unit-norm isotropic Gaussian per (slot, head).  A rotation
                of an isotropic vector is isotropic, so these have the same
                distribution as keys rotated at their prefix positions.
  prefix S    ~ N(0, 0.2^2) per element (for prefixes too long to refill on
                the CPU; short prefixes are refilled by the caller instead)
Removal spans: a total of round(frac * L) live entries split into s >= 1
parts by a uniform random composition, interleaved with s + 1 random gaps
(interior gaps >= 1) that cover the survivors.
"""
from __future__ import annotations

from dataclasses import dataclass, field
import numpy as np

GDN = 0
ATTN = 1


# ----------------------------------------------------------------------------
# bit-level helpers (format conversion only)
# ----------------------------------------------------------------------------
def f64_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp64 values to bf16 (8 significant bits, round half to even).

    Returns the bf16 bit patterns as uint16.  Inputs here are finite and of
    normal magnitude; zeros map to +0/-0.
    """
    x = np.asarray(x, dtype=np.float64)
    m, e = np.frexp(x)                       # x = m * 2**e, 0.5 <= |m| < 1
    y = np.ldexp(np.rint(m * 256.0), e - 8)  # np.rint rounds half to even
    y32 = y.astype(np.float32)               # exact: y has 8 significant bits
    return (y32.view(np.uint32) >> 16).astype(np.uint16)


def bf16_bits_to_f32(u: np.ndarray) -> np.ndarray:
    u = np.asarray(u, dtype=np.uint16)
    return (u.astype(np.uint32) << 16).view(np.float32)


def _rng(*seed: int) -> np.random.Generator:
    return np.random.default_rng([int(s) for s in seed])


def _sigmoid(x: np.ndarray) -> np.ndarray:
    return 1.0 / (1.0 + np.exp(-x))


# ----------------------------------------------------------------------------
# token tensors
# ----------------------------------------------------------------------------
def normal_bf16(seed: tuple, shape, unit_last: bool = False,
                scale: float = 1.0) -> np.ndarray:
    """N(0, scale^2) values rounded to bf16; optionally unit-normalised along
    the last axis in fp64 before rounding."""
    x = _rng(*seed).standard_normal(shape) * scale
    if unit_last:
        x = x / np.linalg.norm(x, axis=-1, keepdims=True)
    return f64_to_bf16_bits(x)


def gates(seed: tuple, n: int, heads: int):
    """alpha = sigmoid(N(3, 0.5)), beta = sigmoid(N(0, 1)), fp32 [n][heads]."""
    r = _rng(*seed)
    a = _sigmoid(r.normal(3.0, 0.5, size=(n, heads))).astype(np.float32)
    b = _sigmoid(r.standard_normal((n, heads))).astype(np.float32)
    return a, b


def conv_weights(seed: tuple, channels: int, std: float = 0.5) -> np.ndarray:
    """Short-convolution taps of a delta-rule layer, fp32 [channels][4],
    N(0, std^2) (four taps of std 0.5 keep the pre-activation near unit
    scale for unit-scale inputs)."""
    return (_rng(*seed).standard_normal((channels, 4)) * std).astype(np.float32)


def state_f32(seed: tuple, shape, std: float = 0.2) -> np.ndarray:
    return (_rng(*seed).standard_normal(shape) * std).astype(np.float32)


def removal_spans(seed: tuple, L: int, total: int, n_spans: int):
    """Random disjoint, sorted live-index spans [begin, end) removing `total`
    entries of a cache of `L` live entries in `n_spans` runs.

    Returns (begins, ends) as int32 arrays.  `total` may be 0 (no spans).
    """
    if total <= 0 or n_spans <= 0:
        return np.zeros(0, np.int32), np.zeros(0, np.int32)
    n_spans = min(n_spans, total)
    survivors = L - total
    if survivors < n_spans - 1:
        raise ValueError("not enough survivors to separate the spans")
    r = _rng(*seed)
    # composition of `total` into n_spans positive parts
    cuts = np.sort(r.choice(np.arange(1, total), size=n_spans - 1, replace=False)) \
        if n_spans > 1 else np.zeros(0, np.int64)
    parts = np.diff(np.concatenate([[0], cuts, [total]]))
    # survivors split into n_spans + 1 gaps, interior gaps >= 1
    free = survivors - (n_spans - 1)
    cuts_g = np.sort(r.integers(0, free + 1, size=n_spans))
    gaps = np.diff(np.concatenate([[0], cuts_g, [free]]))
    gaps[1:-1] += 1
    begins, ends = [], []
    at = 0
    for s in range(n_spans):
        at += int(gaps[s])
        begins.append(at)
        at += int(parts[s])
        ends.append(at)
    assert at + int(gaps[-1]) == L
    return np.asarray(begins, np.int32), np.asarray(ends, np.int32)


# ----------------------------------------------------------------------------
# workload shapes
# ----------------------------------------------------------------------------
@dataclass
class ModelShape:
    layer_kind: list            # GDN / ATTN per layer, model order
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    rotary_dim: int
    rope_theta: float
    n_gdn_heads: int
    d_k: int
    d_v: int

    @property
    def attn_layers(self):
        return [i for i, t in enumerate(self.layer_kind) if t == ATTN]

    @property
    def gdn_layers(self):
        return [i for i, t in enumerate(self.layer_kind) if t == GDN]


def pattern_3to1(n_layers: int) -> list:
    """Three delta-rule layers, then one full-attention layer, repeating."""
    return [ATTN if (i % 4) == 3 else GDN for i in range(n_layers)]


TINY = ModelShape([GDN, ATTN], 8, 2, 64, 64, 1.0e4, 8, 64, 64)


def npc_shape(n_layers: int) -> ModelShape:
    return ModelShape(pattern_3to1(n_layers), 16, 2, 256, 64, 1.0e4, 16, 128, 128)


@dataclass
class Workload:
    name: str
    index: int                  # seed base: index * 1000 + round
    shape: ModelShape
    prefix_len: list            # N_b per character
    rounds: int
    # per round, per character: (removal fraction, number of spans, tail M)
    plan: list = field(default_factory=list)
    refill_compare: bool = False
    # population index of each character (its seeds); None: 0 .. n_chars-1.
    # A rank's share of a partitioned population keeps its characters' ids,
    # so they draw the same numbers as in the whole population.
    char_ids: list | None = None

    @property
    def n_chars(self):
        return len(self.prefix_len)

    def gid(self, b: int) -> int:
        return b if self.char_ids is None else int(self.char_ids[b])

    def subset(self, chars) -> "Workload":
        """The workload restricted to characters `chars` (population indices
        in order), with their plans and seeds."""
        chars = [int(b) for b in chars]
        sub = Workload(self.name, self.index, self.shape, [self.prefix_len[b] for b in chars], self.rounds,
                       [[row[b] for b in chars] for row in self.plan], self.refill_compare,
                       [self.gid(b) for b in chars])
        return sub

    def capacity(self, align: int = 128) -> list:
        """Slots per character that hold the prefix plus every tail of the
        run (live length never exceeds the prefix plus the tails added)."""
        caps = []
        for b, n in enumerate(self.prefix_len):
            live, peak = n, n
            for r in range(self.rounds):
                frac, _, m = self.plan[r][b]
                live = live - int(round(frac * live)) + m
                peak = max(peak, live)
            caps.append(-(-peak // align) * align)
        return caps


def make_workload(name: str, n_layers: int | None = None) -> Workload:
    """The five synthetic workloads:
      tiny   : 1 delta-rule + 1 attention layer (8 heads, d 64), prefix 512,
               remove 64 in 2 spans, tail 64, one round
      npc    : 4 layers 3:1, prefix 8192, 8 chained rounds, 1-4 spans ~5%,
               tail 256
      long   : 48 layers 3:1, prefix 32768, 1 round, 10 spans = 3%, tail 1024
      pop    : 32 characters, prefix U[2048,16384], 2-8% in 1-6 spans,
               tail U[64,512], 12 layers 3:1
      refill : npc stack, no removals, prefix 16384 + tail 512, compared with
               a from-scratch prefill of 16896 tokens
    `n_layers` overrides the layer count (tests use shallower stacks)."""
    if name == "tiny":
        w = Workload("tiny", 0, TINY, [512], 1)
        w.plan = [[(64 / 512, 2, 64)]]
    elif name == "npc":
        w = Workload("npc", 1, npc_shape(n_layers or 4), [8192], 8)
        r = _rng(1, 999)
        w.plan = [[(0.05, int(r.integers(1, 5)), 256)] for _ in range(8)]
    elif name == "long":
        w = Workload("long", 2, npc_shape(n_layers or 48), [32768], 1)
        w.plan = [[(0.03, 10, 1024)]]
    elif name == "pop":
        r = _rng(3, 999)
        n = [int(x) for x in r.integers(2048, 16385, size=32)]
        w = Workload("pop", 3, npc_shape(n_layers or 12), n, 1)
        w.plan = [[(float(r.uniform(0.02, 0.08)), int(r.integers(1, 7)),
                    int(r.integers(64, 513))) for _ in range(32)]]
    elif name == "refill":
        w = Workload("refill", 4, npc_shape(n_layers or 4), [16384], 1,
                     refill_compare=True)
        w.plan = [[(0.0, 0, 512)]]
    else:
        raise KeyError(name)
    return w


# ----------------------------------------------------------------------------
# per-round and prefix inputs
# ----------------------------------------------------------------------------
def tail_inputs(w: Workload, rnd: int, tails: list, layers=None) -> dict:
    """Inputs of one maintenance round, packed over characters.

    tails[b] = M_b.  Returns {layer: dict(q, k, v[, alpha, beta])} with
    q/k/v as bf16 bits [sum M][heads][dim]; alpha/beta fp32 [sum M][heads].
    `layers` restricts the draw to some layers (each layer has its own seeds,
    so a layer's values do not depend on which others are drawn).
    """
    s = w.shape
    base = w.index * 1000 + rnd
    out = {}
    for layer, kind in enumerate(s.layer_kind):
        if layers is not None and layer not in layers:
            continue
        parts = {"q": [], "k": [], "v": [], "alpha": [], "beta": []}
        for b, m in enumerate(tails):
            sd = (base, w.gid(b), layer)
            if kind == ATTN:
                parts["q"].append(normal_bf16(sd + (0,), (m, s.n_q_heads, s.head_dim)))
                parts["k"].append(normal_bf16(sd + (1,), (m, s.n_kv_heads, s.head_dim), unit_last=True))
                parts["v"].append(normal_bf16(sd + (2,), (m, s.n_kv_heads, s.head_dim)))
            else:
                parts["q"].append(normal_bf16(sd + (0,), (m, s.n_gdn_heads, s.d_k)))
                parts["k"].append(normal_bf16(sd + (1,), (m, s.n_gdn_heads, s.d_k), unit_last=True))
                parts["v"].append(normal_bf16(sd + (2,), (m, s.n_gdn_heads, s.d_v)))
                a, bt = gates(sd + (3,), m, s.n_gdn_heads)
                parts["alpha"].append(a)
                parts["beta"].append(bt)
        out[layer] = {k: np.concatenate(v) for k, v in parts.items() if v}
    return out


def round_plan(w: Workload, rnd: int, live: list):
    """Spans and tail lengths of round `rnd` given live lengths `live[b]`.

    Returns (span_cu [B+1], begins, ends, tails [B]) with spans packed over
    characters in character order."""
    cu, bs, es, tails = [0], [], [], []
    for b, L in enumerate(live):
        frac, n_sp, m = w.plan[rnd][b]
        total = int(round(frac * L))
        bb, ee = removal_spans((w.index * 1000 + rnd, w.gid(b), 7777), L, total, n_sp)
        bs.append(bb)
        es.append(ee)
        cu.append(cu[-1] + len(bb))
        tails.append(m)
    cat = lambda xs: np.concatenate(xs).astype(np.int32) if xs else np.zeros(0, np.int32)
    return np.asarray(cu, np.int32), cat(bs), cat(es), tails


def prefix_tokens(w: Workload, b: int, layer: int, n: int) -> dict:
    """Raw (unrotated) prefix tokens of character b for a refill."""
    s = w.shape
    sd = (w.index * 1000 + 999, w.gid(b), layer)
    if s.layer_kind[layer] == ATTN:
        return {"q": normal_bf16(sd + (0,), (n, s.n_q_heads, s.head_dim)),
                "k": normal_bf16(sd + (1,), (n, s.n_kv_heads, s.head_dim), unit_last=True),
                "v": normal_bf16(sd + (2,), (n, s.n_kv_heads, s.head_dim))}
    a, bt = gates(sd + (3,), n, s.n_gdn_heads)
    return {"q": normal_bf16(sd + (0,), (n, s.n_gdn_heads, s.d_k)),
            "k": normal_bf16(sd + (1,), (n, s.n_gdn_heads, s.d_k), unit_last=True),
            "v": normal_bf16(sd + (2,), (n, s.n_gdn_heads, s.d_v)),
            "alpha": a, "beta": bt}


def prefix_cache(w: Workload, b: int, layer: int, n: int):
    """Stored prefix KV of one attention layer: keys as unit-norm isotropic
    bf16 vectors (already in stored, rotated form), values N(0,1) bf16,
    positions 0..n-1.  Shapes K,V [Hkv][n][D]."""
    s = w.shape
    sd = (w.index * 1000 + 998, w.gid(b), layer)
    K = normal_bf16(sd + (0,), (s.n_kv_heads, n, s.head_dim), unit_last=True)
    V = normal_bf16(sd + (1,), (s.n_kv_heads, n, s.head_dim))
    return K, V, np.arange(n, dtype=np.int32)


def prefix_state(w: Workload, b: int, layer: int) -> np.ndarray:
    s = w.shape
    return state_f32((w.index * 1000 + 997, w.gid(b), layer), (s.n_gdn_heads, s.d_v, s.d_k))


# ----------------------------------------------------------------------------
# device-side draws (benchmark inputs too large to draw on the CPU quickly)
# ----------------------------------------------------------------------------
def device_round_inputs(w: Workload, seed: int, tails: list, device="cuda") -> dict:
    """Same distributions as `tail_inputs`, drawn on the GPU with a seeded
    torch generator (not bit-identical to the numpy draws).  Returns
    {layer: dict of torch tensors} packed over characters."""
    import torch
    s = w.shape
    total = int(sum(tails))
    g = torch.Generator(device=device)
    out = {}
    for layer, kind in enumerate(s.layer_kind):
        g.manual_seed(int(seed) * 1009 + layer)
        if kind == ATTN:
            q = torch.randn((total, s.n_q_heads, s.head_dim), generator=g, device=device)
            k = torch.randn((total, s.n_kv_heads, s.head_dim), generator=g, device=device)
            v = torch.randn((total, s.n_kv_heads, s.head_dim), generator=g, device=device)
            d = {}
        else:
            q = torch.randn((total, s.n_gdn_heads, s.d_k), generator=g, device=device)
            k = torch.randn((total, s.n_gdn_heads, s.d_k), generator=g, device=device)
            v = torch.randn((total, s.n_gdn_heads, s.d_v), generator=g, device=device)
            a = torch.sigmoid(3.0 + 0.5 * torch.randn((total, s.n_gdn_heads), generator=g, device=device))
            bt = torch.sigmoid(torch.randn((total, s.n_gdn_heads), generator=g, device=device))
            d = {"alpha": a.float().contiguous(), "beta": bt.float().contiguous()}
        k = k / k.norm(dim=-1, keepdim=True)
        d.update({"q": q.bfloat16().contiguous(), "k": k.bfloat16().contiguous(),
                  "v": v.bfloat16().contiguous()})
        out[layer] = d
    return out


def simulate_plan(w: Workload):
    """Spans and tails of every round of `w`, following live lengths from the
    prefix: list of (span_cu, begins, ends, tails)."""
    live = list(w.prefix_len)
    plan = []
    for r in range(w.rounds):
        cu, bs, es, tails = round_plan(w, r, live)
        plan.append((cu, bs, es, tails))
        for b in range(w.n_chars):
            removed = int((es[cu[b]:cu[b + 1]] - bs[cu[b]:cu[b + 1]]).sum())
            live[b] = live[b] - removed + tails[b]
    return plan
