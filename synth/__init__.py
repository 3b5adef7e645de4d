"""Seeded synthetic inputs for the split-VFL training step.

This module produces the *inputs* of a training run -- feature matrices, labels,
initial parameters and the workload presets -- and nothing else.  It holds none
of the training method's arithmetic: both the CPU oracle (``oracle/``) and the
GPU path (``paper_2510_12494_gb300``) receive these arrays as plain inputs, so the
two sides never share computation code.

Randomness comes from Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel
random numbers: as easy as 1, 2, 3", SC'11), used as a counter-based stream:
key = (seed lo32, seed hi32), counter = (block lo32, block hi32, sub, tag), four
32-bit words per block.  Every element of every matrix is addressed by its flat
index, so any row range can be generated independently and identically.

The paper's datasets (Energy, Blog, Bank, Credit, its scikit-learn synthetic
set) are not available; the five presets below only take their *shapes and
value distributions* (the paper's Table 6 and Sec. 5.1 give the shapes), never
their records.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

__all__ = [
    "philox4x32_10", "u32_stream", "uniform_stream", "normal_stream",
    "VflPreset", "PRESETS", "preset", "layer_shapes", "make_dataset", "init_params",
    "TAG_X", "TAG_LABEL", "TAG_TEACHER", "TAG_INIT",
]

# Philox4x32 round multipliers and key-schedule (Weyl) increments, SC'11 Sec. 5.
_M0 = 0xD2511F53
_M1 = 0xCD9E8D57
_W0 = 0x9E3779B9
_W1 = 0xBB67AE85
_MASK = 0xFFFFFFFF

# Stream tags (counter word 3): one per kind of draw.
TAG_X = 0x58        # feature matrices
TAG_LABEL = 0x4C    # label noise (Bernoulli draws)
TAG_TEACHER = 0x54  # teacher-model parameters
TAG_INIT = 0x49     # initial model parameters


def philox4x32_10(c0, c1, c2, c3, k0: int, k1: int):
    """Ten Philox4x32 rounds on uint64 arrays that hold 32-bit values.

    Round r uses key (k0 + r*W0, k1 + r*W1) mod 2^32; each round multiplies
    words 0 and 2 by M0 and M1 into 64-bit products and recombines the high and
    low halves with the other two words and the key.
    """
    c0 = np.asarray(c0, dtype=np.uint64)
    c1 = np.asarray(c1, dtype=np.uint64)
    c2 = np.asarray(c2, dtype=np.uint64)
    c3 = np.asarray(c3, dtype=np.uint64)
    k0 &= _MASK
    k1 &= _MASK
    m0 = np.uint64(_M0)
    m1 = np.uint64(_M1)
    lo = np.uint64(_MASK)
    s32 = np.uint64(32)
    for r in range(10):
        if r:
            k0 = (k0 + _W0) & _MASK
            k1 = (k1 + _W1) & _MASK
        p0 = c0 * m0
        p1 = c2 * m1
        c0, c1, c2, c3 = ((p1 >> s32) ^ c1 ^ np.uint64(k0), p1 & lo,
                          (p0 >> s32) ^ c3 ^ np.uint64(k1), p0 & lo)
    return c0, c1, c2, c3


def u32_stream(seed: int, tag: int, sub: int, start: int, count: int) -> np.ndarray:
    """Words [start, start+count) of the stream (seed, tag, sub) as uint64 values < 2^32."""
    if count <= 0:
        return np.zeros(0, dtype=np.uint64)
    b0 = start // 4
    b1 = (start + count - 1) // 4 + 1
    words = np.empty((b1 - b0, 4), dtype=np.uint64)
    step = 1 << 15            # blocks per pass: keeps the temporaries cache-resident
    for a in range(b0, b1, step):
        blk = np.arange(a, min(b1, a + step), dtype=np.uint64)
        x = philox4x32_10(blk & np.uint64(_MASK), blk >> np.uint64(32),
                          np.full(blk.shape, sub & _MASK, np.uint64),
                          np.full(blk.shape, tag & _MASK, np.uint64),
                          seed & _MASK, (seed >> 32) & _MASK)
        for j in range(4):
            words[a - b0:a - b0 + blk.size, j] = x[j]
    off = start - 4 * b0
    return words.reshape(-1)[off:off + count]


def uniform_stream(seed: int, tag: int, sub: int, start: int, count: int) -> np.ndarray:
    """Uniform [0, 1) doubles: word * 2^-32."""
    return u32_stream(seed, tag, sub, start, count).astype(np.float64) * 2.0 ** -32


def normal_stream(seed: int, tag: int, sub: int, start: int, count: int) -> np.ndarray:
    """Standard normals by Box-Muller on word pairs (2i, 2i+1); element i is the
    cosine (even i) or sine (odd i) branch of pair i//2."""
    if count <= 0:
        return np.zeros(0, dtype=np.float64)
    p0 = start // 2
    p1 = (start + count - 1) // 2 + 1
    w = u32_stream(seed, tag, sub, 2 * p0, 2 * (p1 - p0)).astype(np.float64)
    a = (w[0::2] + 1.0) * 2.0 ** -32          # (0, 1]
    b = w[1::2] * 2.0 ** -32                  # [0, 1)
    r = np.sqrt(-2.0 * np.log(a))
    t = 2.0 * np.pi * b
    z = np.stack([r * np.cos(t), r * np.sin(t)], axis=1).reshape(-1)
    off = start - 2 * p0
    return z[off:off + count]


# --------------------------------------------------------------------------
# Workload presets: the five synthetic tabular workloads (shapes only).
# --------------------------------------------------------------------------
@dataclass(frozen=True)
class VflPreset:
    cid: int
    name: str
    n_rows: int
    d_passive: int
    d_active: int
    passive: tuple          # output width of each passive bottom Linear layer
    active: tuple           # output width of each active bottom Linear layer
    top: tuple              # output width of each top Linear layer (last = n_out)
    loss: str               # "bce" | "ce"
    batch: int
    epochs: int
    lr: float
    staleness: int
    schedule: str           # "sync" | "seeded"
    dtype: str              # "fp32" | "bf16"
    workers: int            # worker streams per party
    dp_clip: float = 0.0    # > 0 enables DP on the exchanged tensor named by dp_target
    dp_sigma: float = 0.0
    seed: int = 0
    dp_target: str = "grad" # "grad": the published embedding gradient; "emb": the published embedding
    ps_dt0: int = 0         # > 0: per-worker replicas averaged after the epochs Eq. 5 selects (Delta T_0)

    @property
    def n_out(self) -> int:
        return self.top[-1]

    @property
    def e_passive(self) -> int:
        return self.passive[-1]

    @property
    def e_active(self) -> int:
        return self.active[-1]

    @property
    def steps_per_epoch(self) -> int:
        return -(-self.n_rows // self.batch)

    def with_(self, **kw) -> "VflPreset":
        d = {f: getattr(self, f) for f in self.__dataclass_fields__}
        d.update(kw)
        return VflPreset(**d)


PRESETS = {
    1: VflPreset(1, "tiny-sync", 4096, 10, 10, (32, 16), (32, 16), (32, 1), "bce",
                 256, 1, 0.01, 0, "sync", "fp32", 1),
    2: VflPreset(2, "credit-shaped", 30000, 12, 11, (128, 64), (128, 64), (64, 1), "bce",
                 1024, 5, 0.01, 2, "seeded", "fp32", 2),
    3: VflPreset(3, "multiclass", 500000, 27, 27, (256, 256, 128), (256, 256, 128), (256, 7), "ce",
                 4096, 1, 0.01, 2, "seeded", "bf16", 1),
    4: VflPreset(4, "wide-dp", 1000000, 1000, 1000, (512, 256), (512, 256), (256, 1), "bce",
                 8192, 1, 0.01, 4, "seeded", "bf16", 1, dp_clip=1.0, dp_sigma=1.0),
    5: VflPreset(5, "hetero", 200000, 2560, 512, (1024, 1024, 1024, 256), (128, 256), (256, 10), "ce",
                 2048, 1, 0.01, 4, "seeded", "bf16", 8),
}


def preset(cid: int, **overrides) -> VflPreset:
    p = PRESETS[cid]
    return p.with_(**overrides) if overrides else p


def layer_shapes(p: VflPreset):
    """[(party, layer, out, in)] for party 0 = passive bottom, 1 = active bottom, 2 = top."""
    out = []
    for party, d_in, widths in ((0, p.d_passive, p.passive), (1, p.d_active, p.active),
                                (2, p.e_active + p.e_passive, p.top)):
        for l, w in enumerate(widths):
            out.append((party, l, w, d_in))
            d_in = w
    return out


# --------------------------------------------------------------------------
# Datasets.  Columns [0, d_passive) belong to the passive party, the rest to
# the active party.  Returns fp32 features and int32 labels for rows [r0, r1).
# --------------------------------------------------------------------------
def _normal_matrix(seed, sub, r0, r1, d):
    return normal_stream(seed, TAG_X, sub, r0 * d, (r1 - r0) * d).reshape(r1 - r0, d)


def _uniform_matrix(seed, sub, r0, r1, d):
    return uniform_stream(seed, TAG_X, sub, r0 * d, (r1 - r0) * d).reshape(r1 - r0, d)


def _sigmoid(x):
    return 0.5 * (1.0 + np.tanh(0.5 * x))


def _bernoulli(seed, sub, r0, r1, prob):
    u = uniform_stream(seed, TAG_LABEL, sub, r0, r1 - r0)
    return (u < prob).astype(np.int32)


def _teacher_normal(seed, sub, shape, std):
    n = int(np.prod(shape))
    return normal_stream(seed, TAG_TEACHER, sub, 0, n).reshape(shape) * std


def _features_cfg1(seed, r0, r1):
    return _normal_matrix(seed, 1, r0, r1, 20)


def _label_cfg1(seed, x, r0, r1):
    w = _teacher_normal(seed, 1, (20,), math.sqrt(1.0 / 20))
    return _bernoulli(seed, 1, r0, r1, _sigmoid(x @ w))


def _features_cfg2(seed, r0, r1):
    cont = _normal_matrix(seed, 2, r0, r1, 14)
    cat = np.floor(7.0 * _uniform_matrix(seed, 3, r0, r1, 9))      # {0..6}
    # passive: 7 continuous + 5 categorical; active: 7 continuous + 4 categorical
    return np.concatenate([cont[:, :7], cat[:, :5], cont[:, 7:], cat[:, 5:]], axis=1)


def _score_cfg2(seed, x):
    w1 = _teacher_normal(seed, 2, (16, 23), math.sqrt(1.0 / 23))
    w2 = _teacher_normal(seed, 3, (16,), math.sqrt(1.0 / 16))
    return np.maximum(x @ w1.T, 0.0) @ w2


def _features_cfg3(seed, r0, r1):
    n = r1 - r0
    cont = _normal_matrix(seed, 4, r0, r1, 10)
    g = u32_stream(seed, TAG_X, 5, 2 * r0, 2 * n).reshape(n, 2)
    h4 = (g[:, 0] * np.uint64(4)) >> np.uint64(32)
    h40 = (g[:, 1] * np.uint64(40)) >> np.uint64(32)
    oh4 = np.zeros((n, 4))
    oh4[np.arange(n), h4.astype(np.int64)] = 1.0
    oh40 = np.zeros((n, 40))
    oh40[np.arange(n), h40.astype(np.int64)] = 1.0
    return np.concatenate([cont, oh4, oh40], axis=1)


def _label_cfg3(seed, x):
    w1 = _teacher_normal(seed, 4, (64, 54), math.sqrt(1.0 / 54))
    w2 = _teacher_normal(seed, 5, (7, 64), math.sqrt(1.0 / 64))
    return np.argmax(np.maximum(x @ w1.T, 0.0) @ w2.T, axis=1).astype(np.int32)


def _features_cfg4(seed, r0, r1):
    # Bernoulli(0.05): word * 2^-32 < 0.05  <=>  word < 214748365 (same test, in integers)
    w = u32_stream(seed, TAG_X, 6, r0 * 2000, (r1 - r0) * 2000).reshape(r1 - r0, 2000)
    return (w < np.uint64(214748365)).astype(np.float32)


def _teacher_cfg4(seed):
    # 100 distinct coordinates by a partial Fisher-Yates shuffle, N(0,1) values.
    perm = np.arange(2000)
    u = u32_stream(seed, TAG_TEACHER, 6, 0, 100)
    for i in range(100):
        j = i + int((int(u[i]) * (2000 - i)) >> 32)
        perm[i], perm[j] = perm[j], perm[i]
    w = np.zeros(2000)
    w[perm[:100]] = normal_stream(seed, TAG_TEACHER, 7, 0, 100)
    return w


def _label_cfg4(seed, x, r0, r1):
    w = _teacher_cfg4(seed)
    return _bernoulli(seed, 4, r0, r1, _sigmoid(x @ w - 0.05 * w.sum()))


def _features_cfg5(seed, r0, r1):
    u = _uniform_matrix(seed, 7, r0, r1, 3072)
    U = _normal_matrix(seed, 8, r0, r1, 16)
    V = _teacher_normal(seed, 8, (16, 3072), 1.0)
    return 0.5 * u + 0.5 * _sigmoid(U @ V / 4.0)


def _label_cfg5(seed, x):
    # the teacher sees centred features so that no class dominates through the offset
    w = _teacher_normal(seed, 9, (10, 3072), math.sqrt(12.0 / 3072))
    return np.argmax((x - 0.5) @ w.T, axis=1).astype(np.int32)


def _features_custom(seed, r0, r1, d):
    return _normal_matrix(seed, 20, r0, r1, d)


def _label_custom(seed, x, r0, r1, n_out, loss):
    # a linear teacher over all columns: Bernoulli(sigmoid) for BCE, argmax over n_out classes for CE
    d = x.shape[1]
    if loss == "bce":
        w = _teacher_normal(seed, 20, (d,), math.sqrt(1.0 / d))
        return _bernoulli(seed, 20, r0, r1, _sigmoid(x @ w))
    w = _teacher_normal(seed, 21, (n_out, d), math.sqrt(1.0 / d))
    return np.argmax(x @ w.T, axis=1).astype(np.int32)


def make_dataset(p: VflPreset, rows=None, chunk: int | None = None):
    """(x_passive fp32 [n, d_p], x_active fp32 [n, d_a], y int32 [n]) for rows
    [r0, r1) of preset ``p`` (all rows by default).  cid 0 is a model of any
    shape: N(0, 1) features and labels from a seeded linear teacher."""
    r0, r1 = (0, p.n_rows) if rows is None else rows
    if not (0 <= r0 <= r1 <= p.n_rows):
        raise ValueError(f"row range {rows} outside [0, {p.n_rows}]")
    seed = p.seed
    if chunk is None:           # about 4M elements per pass
        chunk = max(1024, (1 << 22) // (p.d_passive + p.d_active))
    xs, ys = [], []
    if p.cid == 2:
        # the label threshold is the empirical 78th percentile over all rows
        allx = _features_cfg2(seed, 0, p.n_rows)
        s = _score_cfg2(seed, allx)
        thr = np.sort(s)[int(0.78 * p.n_rows)]
        x = allx[r0:r1]
        xs.append(x)
        ys.append((s[r0:r1] > thr).astype(np.int32))
    else:
        for a in range(r0, r1, chunk):
            b = min(r1, a + chunk)
            if p.cid == 0:
                x = _features_custom(seed, a, b, p.d_passive + p.d_active)
                y = _label_custom(seed, x, a, b, p.n_out, p.loss)
            elif p.cid == 1:
                x = _features_cfg1(seed, a, b); y = _label_cfg1(seed, x, a, b)
            elif p.cid == 3:
                x = _features_cfg3(seed, a, b); y = _label_cfg3(seed, x)
            elif p.cid == 4:
                x = _features_cfg4(seed, a, b); y = _label_cfg4(seed, x, a, b)
            elif p.cid == 5:
                x = _features_cfg5(seed, a, b); y = _label_cfg5(seed, x)
            else:
                raise ValueError(f"no data recipe for preset {p.cid}")
            xs.append(x)
            ys.append(y)
    x = np.concatenate(xs, axis=0) if xs else np.zeros((0, p.d_passive + p.d_active))
    y = np.concatenate(ys) if ys else np.zeros(0, np.int32)
    if x.shape[1] != p.d_passive + p.d_active:
        raise ValueError(f"preset {p.cid}'s recipe makes {x.shape[1]} columns, "
                         f"not d_passive + d_active = {p.d_passive + p.d_active}")
    xp = np.ascontiguousarray(x[:, :p.d_passive], dtype=np.float32)
    xa = np.ascontiguousarray(x[:, p.d_passive:], dtype=np.float32)
    return xp, xa, np.ascontiguousarray(y, dtype=np.int32)


def init_params(p: VflPreset, seed: int | None = None):
    """{(party, layer): (W [out,in] fp32, b [out] fp32)} with every entry drawn
    from U(-1/sqrt(in), 1/sqrt(in))."""
    seed = p.seed if seed is None else seed
    params = {}
    for party, l, out, fin in layer_shapes(p):
        n = out * fin + out
        u = uniform_stream(seed, TAG_INIT, (party << 8) | l, 0, n)
        v = (2.0 * u - 1.0) / math.sqrt(fin)
        W = v[:out * fin].reshape(out, fin).astype(np.float32)
        b = v[out * fin:].astype(np.float32)
        params[(party, l)] = (W, b)
    return params
