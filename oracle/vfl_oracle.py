"""CPU oracle of the PubSub-VFL split-learning training step (arxiv 2510.12494).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this module.  It shares no code with
the CUDA path: it has its own Philox generator, its own schedule code and its
own bf16 rounding, and it computes everything in float64 with numpy.

What it computes, in the paper's order (Algorithm 1, Sec. 3, App. C, App. D):

* Sec. 3: the passive party P_p holds x^p and bottom model f_p (parameters
  theta_2); the active party P_a holds x^a, the labels, bottom model f_a and the
  top model g (together theta_1).  Forward: z^p = f_p(x^p), z^a = f_a(x^a),
  y_hat = g(z^a, z^p).  Loss: binary cross-entropy (Eq. 1) or, for multiclass
  presets, softmax cross-entropy, averaged over the batch.  Backward: P_a
  computes grad wrt theta_1 and wrt z^p, sends the latter back, P_p computes the
  grad wrt theta_2.  Both apply gradient descent (Eq. 2).
* Algorithm 1: publisher phase (passive forward, optional Gaussian noise,
  publish to the embedding channel of batch B_j), subscriber phase (fetch,
  active forward, loss, gradients, publish grad wrt z^p to the gradient
  channel), backward phase (fetch, passive gradient, update theta_2).
* App. D (Assumption 4 and the theorem): with bounded staleness the gradient
  applied at iteration t was evaluated at theta_{t - tau(t)}, tau(t) <= Delta T,
  and the update is theta_{t+1} = theta_t - eta * (g_{t - tau(t)} + xi_dp).
* App. C / Assumption 5: Gaussian noise on the exchanged tensor.

Readings where the paper is silent:

* Two lags per step: tau_p(k) is the age of the passive weights that produced
  the embedding of step k; tau_a(k) the age of the active + top weights that
  produced its gradient.  The passive backward of step k re-uses the same
  passive version and the saved activations of its forward.  Updates are
  applied to the current parameters in step order.
* Batches: step k is epoch k // nb, batch j = k mod nb (identity order), rows
  [j B, min(n, (j+1) B)); the last, partial batch is a real batch (the paper
  keeps ceil(n/B) channels, Sec. 4.1).
* BCE in the stable logit form (equal to Eq. 1 on probabilities); softmax CE.
* ReLU after every bottom layer, including the cut layer; none after the top's
  last layer; ReLU'(0) = 0.  Concatenation order [z^a | z^p].
* DP variant on the published embedding gradient: per row g_i = B_k dZ_i is
  clipped to L2 norm C and N(0, (sigma C)^2 I) noise is added, then divided by
  B_k again.  Noise: Philox4x32-10 with key (seed lo, seed hi) and counter
  (col // 4, row in batch, k, 0x4450); Box-Muller on 24-bit uniforms.
* DP variant on the published embedding (App. C, the paper's own target): per
  row c_i = min(1, C/||z_i||) (1 for a zero row) and the published embedding is
  c_i z_i + sigma C xi_i, xi from the same generator with counter word 3 =
  0x4445.  The backward is straight-through: the passive party scales the
  received gradient by c_i (the Jacobian of c_i and of the noise are ignored)
  before its own ReLU mask on the clean z.  sigma for a target mu-GDP level
  follows Eq. 25 with the O(.)'s constant taken as 1.
* Intra-party semi-asynchronous parameter server (Sec. 4.1, Eq. 5, Algorithm
  1), when cfg.ps_dt0 > 0: each party keeps one replica of its parameters per
  worker (cfg.workers of them); step k is served by worker pair k mod W, whose
  replicas it reads (the latest: no staleness within a replica's chain) and
  updates.  After epoch t (1-based) each party's replicas are averaged (sum over
  the workers in order, divided by W) and every replica takes the average when
  t mod Delta T_t == 0, Delta T_t = ceil(Delta T_0 / 2 tanh(2 t / Delta T_0 - 2)
  + Delta T_0 / 2) (Eq. 5).
* Waiting deadline and buffer overflow (Sec. 4.1, Algorithm 1's subscriber
  branch): a step whose embedding the subscriber does not get (deadline passed,
  or dropped oldest-first from a full buffer) is dropped: its publisher's work
  is discarded, nothing else runs, no loss is recorded and neither party's
  parameters change (version k+1 = version k), and its batch is reassigned to
  the next step.  Step k therefore trains batch j = (k - D(k)) mod nb, D(k) the
  drops before k; an epoch ends with the step that completes batch nb - 1.
  Drops come in as a per-step 0/1 input; make_drops draws them: step k drops
  when word 0 of Philox(key=(seed lo, seed hi), ctr=(k lo, k hi, 2, 0x4452)) is
  below floor(rate 2^32).
* bf16 presets round to bf16 (round-to-nearest-even, via fp32) at: the inputs,
  each weight version's compute copy (biases stay fp32), every stored hidden
  activation and embedding, and every activation gradient handed from one layer
  to the next (including both published cut-layer gradients, the noisy
  published embedding and the scaled gradient the passive backward starts
  from).  Logits, loss and
  d(logits) stay unrounded; master weights and weight gradients are never
  rounded.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

# ---------------------------------------------------------------------------
# Philox4x32-10 (Salmon et al., SC'11): constants and rounds from the paper.
# ---------------------------------------------------------------------------
PHILOX_M = (0xD2511F53, 0xCD9E8D57)
PHILOX_W = (0x9E3779B9, 0xBB67AE85)
_U32 = 0xFFFFFFFF
TAG_SCHED = 0x5343      # counter word 3 of the staleness-schedule draws
TAG_DP = 0x4450         # counter word 3 of the DP noise draws on the published gradient
TAG_DPE = 0x4445        # counter word 3 of the DP noise draws on the published embedding
TAG_DROP = 0x4452       # counter word 3 of the waiting-deadline drop draws


def philox(ctr, key):
    """Philox4x32-10 of counters ctr = (c0, c1, c2, c3) (uint64 arrays of
    32-bit values, broadcastable) under key = (k0, k1) python ints."""
    c = [np.asarray(v, dtype=np.uint64) & np.uint64(_U32) for v in ctr]
    c = np.broadcast_arrays(*c)
    k0, k1 = key[0] & _U32, key[1] & _U32
    for r in range(10):
        prod0 = c[0] * np.uint64(PHILOX_M[0])
        prod1 = c[2] * np.uint64(PHILOX_M[1])
        hi0, lo0 = prod0 >> np.uint64(32), prod0 & np.uint64(_U32)
        hi1, lo1 = prod1 >> np.uint64(32), prod1 & np.uint64(_U32)
        c = [hi1 ^ c[1] ^ np.uint64(k0), lo1, hi0 ^ c[3] ^ np.uint64(k1), lo0]
        k0 = (k0 + PHILOX_W[0]) & _U32
        k1 = (k1 + PHILOX_W[1]) & _U32
    return c


# ---------------------------------------------------------------------------
# Staleness schedule (seeded, realisable: versions never go backwards).
# ---------------------------------------------------------------------------
SCHED_SYNC, SCHED_MAX, SCHED_SEEDED = 0, 1, 2


def make_schedule(seed: int, S: int, kind: int, n_steps: int):
    """(tau_p, tau_a) int32 arrays of length n_steps.

    SYNC: tau = 0.  MAX: tau(k) = min(k, S).  SEEDED: tau(0) = 0 and
    tau(k) = min(k, S, tau(k-1) + 1, u_k mod (S+1)) with u_k word 0 of
    Philox(key=(seed lo, seed hi), ctr=(k lo, k hi, party, TAG_SCHED)); party
    0 = passive, 1 = active.  The tau(k-1)+1 cap keeps k - tau(k) non-decreasing
    (Assumption 4 only asks tau(t) <= Delta T).
    """
    if S < 0 or n_steps < 0:
        raise ValueError("S and n_steps must be >= 0")
    out = []
    k = np.arange(n_steps, dtype=np.uint64)
    for party in (0, 1):
        tau = np.zeros(n_steps, dtype=np.int32)
        if kind == SCHED_MAX:
            tau[:] = np.minimum(np.arange(n_steps), S)
        elif kind == SCHED_SEEDED:
            u = philox((k & np.uint64(_U32), k >> np.uint64(32), np.uint64(party), np.uint64(TAG_SCHED)),
                       (seed & _U32, (seed >> 32) & _U32))[0]
            prev = 0
            for i in range(n_steps):
                t = 0 if i == 0 else min(i, S, prev + 1, int(u[i]) % (S + 1))
                tau[i] = t
                prev = t
        elif kind != SCHED_SYNC:
            raise ValueError(f"unknown schedule kind {kind}")
        out.append(tau)
    return out[0], out[1]


# ---------------------------------------------------------------------------
# bf16 rounding (round to nearest even on the fp32 value, NaN kept quiet).
# ---------------------------------------------------------------------------
def bf16_round(x):
    f = np.asarray(x, dtype=np.float64).astype(np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    r = ((u + np.uint64(0x7FFF) + ((u >> np.uint64(16)) & np.uint64(1))) & np.uint64(0xFFFF0000))
    out = r.astype(np.uint32).view(np.float32).copy()
    nan = np.isnan(f)
    if nan.any():
        out[nan] = np.float32(np.nan)
    return out.astype(np.float64)


def _store(x, dtype):
    """A tensor as the GPU stores it: unchanged for fp32, bf16-rounded for bf16."""
    return bf16_round(x) if dtype == "bf16" else np.asarray(x, dtype=np.float64)


# ---------------------------------------------------------------------------
# Model pieces (Sec. 3).
# ---------------------------------------------------------------------------
def mlp_forward(layers, x, relu_last: bool, dtype: str):
    """Activations [x, h_1, ..., h_L] of Linear(+ReLU) layers; h_l = relu(h_{l-1} W_l^T + b_l).
    ``layers`` holds (W compute copy, b).  A last layer without ReLU returns
    unrounded pre-activations (the logits)."""
    hs = [x]
    for i, (W, b) in enumerate(layers):
        pre = hs[-1] @ W.T + b
        if i == len(layers) - 1 and not relu_last:
            hs.append(pre)
        else:
            hs.append(_store(np.maximum(pre, 0.0), dtype))
    return hs


def mlp_backward(layers, hs, g_out, relu_last: bool, dtype: str, need_dx: bool, round_dx: bool = True):
    """Gradients of Linear(+ReLU) layers by the chain rule.

    g_out is dLoss/d(h_L).  For a ReLU layer dpre = g * [h > 0]; then
    dW = dpre^T h_{l-1}, db = sum_rows dpre, and g_{l-1} = dpre W (stored,
    i.e. bf16-rounded for bf16, except the input gradient when round_dx is
    False).  Returns ([(dW, db)], dLoss/dx or None)."""
    L = len(layers)
    grads = [None] * L
    g = g_out
    dx = None
    for i in reversed(range(L)):
        W, _ = layers[i]
        relu = relu_last or i < L - 1
        dpre = g * (hs[i + 1] > 0) if relu else g
        grads[i] = (dpre.T @ hs[i], dpre.sum(axis=0))
        if i > 0:
            g = _store(dpre @ W, dtype)
        elif need_dx:
            dx = dpre @ W
            if round_dx:
                dx = _store(dx, dtype)
    return grads, dx


def loss_and_dlogits(s, y, loss: str):
    """Per-batch mean loss and d(mean loss)/d(logits).

    BCE (Eq. 1) in logit form: l_i = max(s,0) - s y + log(1 + exp(-|s|)),
    dl/ds = sigmoid(s) - y.  Softmax CE: l_i = logsumexp(s_i) - s_{i,y_i},
    dl/ds = softmax(s_i) - onehot(y_i).  Both averaged over the B_k rows."""
    B = s.shape[0]
    if loss == "bce":
        s1 = s[:, 0]
        yf = y.astype(np.float64)
        li = np.maximum(s1, 0.0) - s1 * yf + np.log1p(np.exp(-np.abs(s1)))
        sig = 1.0 / (1.0 + np.exp(-s1))
        ds = ((sig - yf) / B)[:, None]
    elif loss == "ce":
        m = s.max(axis=1, keepdims=True)
        e = np.exp(s - m)
        z = e.sum(axis=1, keepdims=True)
        li = (np.log(z) + m)[:, 0] - s[np.arange(B), y]
        p = e / z
        p[np.arange(B), y] -= 1.0
        ds = p / B
    else:
        raise ValueError(f"unknown loss {loss!r}")
    return li.mean(), ds, li


def dp_normals(seed: int, k: int, rows: int, cols: int, tag: int = TAG_DP):
    """N(0,1) draws xi[i, c] for the DP noise of step k (App. C, Assumption 5):
    Philox4x32-10, key (seed lo, seed hi), counter (c // 4, i, k, tag); the
    block's words (x0, x1) give columns 4q, 4q+1 and (x2, x3) columns 4q+2,
    4q+3 by Box-Muller with u1 = ((x >> 8) + 1) 2^-24, u2 = (y >> 8) 2^-24."""
    nq = (cols + 3) // 4
    q = np.arange(nq, dtype=np.uint64)[None, :]
    i = np.arange(rows, dtype=np.uint64)[:, None]
    x = philox((q, i, np.uint64(k & _U32), np.uint64(tag)), (seed & _U32, (seed >> 32) & _U32))
    out = np.empty((rows, nq, 4))
    for pair in (0, 1):
        a, b = x[2 * pair], x[2 * pair + 1]
        u1 = ((a >> np.uint64(8)).astype(np.float64) + 1.0) * 2.0 ** -24
        u2 = (b >> np.uint64(8)).astype(np.float64) * 2.0 ** -24
        r = np.sqrt(-2.0 * np.log(u1))
        out[:, :, 2 * pair] = r * np.cos(2.0 * np.pi * u2)
        out[:, :, 2 * pair + 1] = r * np.sin(2.0 * np.pi * u2)
    return out.reshape(rows, 4 * nq)[:, :cols]


def dp_clip_noise(dz, k: int, clip: float, sigma: float, seed: int):
    """Per-row clipping + Gaussian noise on the published gradient (readings in
    the module docstring): g_i = B dz_i, g_i <- g_i min(1, C/||g_i||) + sigma C xi_i,
    dz_i <- g_i / B."""
    B = dz.shape[0]
    g = dz * B
    norm = np.sqrt((g * g).sum(axis=1, keepdims=True))
    with np.errstate(divide="ignore", invalid="ignore"):
        factor = np.where(norm > clip, clip / norm, 1.0)
    g = g * factor
    if sigma != 0.0:
        g = g + sigma * clip * dp_normals(seed, k, B, dz.shape[1])
    return g / B


def dp_embed(z, k: int, clip: float, sigma: float, seed: int):
    """Gaussian mechanism on the published embedding (App. C): per row
    c_i = min(1, C/||z_i||) (1 for a zero row), z~_i = c_i z_i + sigma C xi_i.
    Returns (z~, c)."""
    norm = np.sqrt((z * z).sum(axis=1))
    with np.errstate(divide="ignore", invalid="ignore"):
        c = np.where(norm > clip, clip / norm, 1.0)
    out = z * c[:, None]
    if sigma != 0.0:
        out = out + sigma * clip * dp_normals(seed, k, z.shape[0], z.shape[1], TAG_DPE)
    return out, c


def make_drops(seed: int, rate: float, n_steps: int):
    """uint8 [n_steps]: 1 where the step is dropped (waiting deadline), drawn as
    word 0 of Philox(key=(seed lo, seed hi), ctr=(k lo, k hi, 2, TAG_DROP)) below
    floor(rate * 2^32), rate in [0, 1]."""
    if not (0.0 <= rate <= 1.0) or n_steps < 0:
        raise ValueError("rate must be in [0, 1] and n_steps >= 0")
    k = np.arange(n_steps, dtype=np.uint64)
    u = philox((k & np.uint64(_U32), k >> np.uint64(32), np.uint64(2), np.uint64(TAG_DROP)),
               (seed & _U32, (seed >> 32) & _U32))[0]
    thr = min(1 << 32, int(math.floor(rate * 4294967296.0)))
    return (u.astype(np.uint64) < np.uint64(thr)).astype(np.uint8) if thr < (1 << 32) else np.ones(n_steps, np.uint8)


def ps_interval(t: int, dt0: int) -> int:
    """Synchronization interval Delta T_t of the intra-party parameter server
    after epoch t (Eq. 5)."""
    return math.ceil(dt0 / 2.0 * math.tanh(2.0 * t / dt0 - 2.0) + dt0 / 2.0)


def ps_aggregates_after(t: int, dt0: int) -> bool:
    """Whether the replicas are averaged at the end of epoch t (1-based): t mod Delta T_t == 0."""
    return t % ps_interval(t, dt0) == 0


def gdp_sigma(mu: float, batch: int, n: int, queries: int) -> float:
    """Noise multiplier for mu-GDP on the published embedding, Eq. 25 with the
    O(.)'s constant taken as 1: sigma = N_m sqrt(K) / (mu N), N_m the minibatch
    size, N the whole dataset, K the number of batches the worker processes."""
    return batch * math.sqrt(queries) / (mu * n)


# ---------------------------------------------------------------------------
# Training (Algorithm 1 with the delayed update of App. D).
# ---------------------------------------------------------------------------
def _copy_params(ps):
    return [(W.copy(), b.copy()) for W, b in ps]


@dataclass
class StepRecord:
    k: int
    batch: int
    rows: tuple
    tau_p: int
    tau_a: int
    version_p: int
    version_a: int
    loss: float
    zp: np.ndarray = None        # published embedding  [B_k, e_p]
    za: np.ndarray = None        # active embedding     [B_k, e_a]
    logits: np.ndarray = None    # [B_k, n_out]
    ds: np.ndarray = None        # d(mean loss)/d(logits) [B_k, n_out]
    dzp: np.ndarray = None       # published gradient   [B_k, e_p]
    dza: np.ndarray = None       # [B_k, e_a]
    grads: dict = None           # (party, layer) -> (dW, db)
    params: dict = None          # (party, layer) -> (W, b) after this step
    dropped: bool = False        # waiting deadline: nothing trained, batch reassigned to the next step


@dataclass
class Oracle:
    """One training run.  ``cfg`` needs: d_passive, d_active, passive, active,
    top, loss, batch, lr, staleness, dtype, dp_clip, dp_sigma, seed.
    ``params`` maps (party, layer) -> (W [out,in], b [out]); party 0 = passive
    bottom (theta_2), 1 = active bottom and 2 = top (together theta_1)."""
    cfg: object
    xp: np.ndarray
    xa: np.ndarray
    y: np.ndarray
    params: dict
    dp_seed: int = 0
    k: int = 0
    versions_p: dict = field(default_factory=dict)
    versions_a: dict = field(default_factory=dict)
    channel_e: dict = field(default_factory=dict)
    channel_g: dict = field(default_factory=dict)
    emb_scale: dict = field(default_factory=dict)   # step -> per-row clip factors of its published embedding
    replicas: list = None                            # parameter-server mode: [(P, A, T)] per worker
    n_done: int = 0                                  # batches trained (steps not dropped)

    def __post_init__(self):
        c = self.cfg
        self.n = self.xp.shape[0]
        self.nb = -(-self.n // c.batch)
        self.dtype = c.dtype
        self.xp_c = _store(self.xp, self.dtype)
        self.xa_c = _store(self.xa, self.dtype)
        lp = len(c.passive)
        la = len(c.active)
        lt = len(c.top)
        P = [tuple(np.asarray(v, np.float64) for v in self.params[(0, l)]) for l in range(lp)]
        A = [tuple(np.asarray(v, np.float64) for v in self.params[(1, l)]) for l in range(la)]
        T = [tuple(np.asarray(v, np.float64) for v in self.params[(2, l)]) for l in range(lt)]
        self.versions_p = {0: P}
        self.versions_a = {0: (A, T)}
        self.ps = getattr(c, "ps_dt0", 0) > 0
        if self.ps:
            if c.staleness != 0:
                raise ValueError("the parameter-server mode reads each replica's latest version (staleness 0)")
            self.replicas = [(_copy_params(P), _copy_params(A), _copy_params(T)) for _ in range(c.workers)]

    # compute copies of a stored version (bf16 presets round W, never b)
    def _compute(self, layers):
        return [(_store(W, self.dtype), b) for W, b in layers]

    def batch_rows(self, k: int = None):
        """Batch id and rows of the next step (the batch after the last one trained;
        without drops, step k's batch is k mod nb)."""
        j = self.n_done % self.nb if k is None or k == self.k else k % self.nb
        r0 = j * self.cfg.batch
        return j, r0, min(self.n, r0 + self.cfg.batch)

    def step(self, tau_p: int, tau_a: int, record: bool = False, drop: bool = False) -> StepRecord:
        c = self.cfg
        k = self.k
        if not (0 <= tau_p <= min(k, c.staleness) and 0 <= tau_a <= min(k, c.staleness)):
            raise ValueError(f"step {k}: staleness ({tau_p}, {tau_a}) outside [0, min(k, S={c.staleness})]")
        j, r0, r1 = self.batch_rows()
        if drop:
            # the subscriber gave up on the embedding: no loss, no update, the batch goes to step k+1
            self.versions_p[k + 1] = self.versions_p[k]
            self.versions_a[k + 1] = self.versions_a[k]
            for d in (self.versions_p, self.versions_a):
                for v in [v for v in d if v < k + 1 - c.staleness]:
                    del d[v]
            self.k = k + 1
            rec = StepRecord(k, j, (r0, r1), tau_p, tau_a, k - tau_p, k - tau_a, float("nan"), dropped=True)
            if record and self.ps:
                rec.params = self.replica_params(k % c.workers)
            elif record:
                rec.params = self.current_params()
            return rec
        Bk = r1 - r0
        vp, va = k - tau_p, k - tau_a
        if self.ps:   # worker pair k mod W serves the step with its own replicas
            w = k % c.workers
            self.versions_p[vp] = self.replicas[w][0]
            self.versions_a[va] = (self.replicas[w][1], self.replicas[w][2])

        # Publisher phase (passive): z^p = f_p(x^p; theta_2^(k - tau_p)), publish to C_e[B_j].
        P = self._compute(self.versions_p[vp])
        hp = mlp_forward(P, self.xp_c[r0:r1], True, self.dtype)
        emb_dp = c.dp_clip > 0.0 and getattr(c, "dp_target", "grad") == "emb"
        if emb_dp:   # App. C: Gaussian noise on the published embedding
            zpub, self.emb_scale[k] = dp_embed(hp[-1], k, c.dp_clip, c.dp_sigma, self.dp_seed)
            zpub = _store(zpub, self.dtype)
        else:
            zpub = hp[-1]
        self.channel_e[k] = (zpub, j, vp)

        # Subscriber phase (active): fetch z^p, z^a = f_a(x^a), y_hat = g(z^a, z^p),
        # loss, grads wrt theta_1 and z^p; publish grad to C_g[B_j].
        zp, j_e, _ = self.channel_e.pop(k)
        assert j_e == j
        A_m, T_m = self.versions_a[va]
        A, T = self._compute(A_m), self._compute(T_m)
        ha = mlp_forward(A, self.xa_c[r0:r1], True, self.dtype)
        ht = mlp_forward(T, np.concatenate([ha[-1], zp], axis=1), False, self.dtype)
        logits = ht[-1]
        loss, ds, _ = loss_and_dlogits(logits, self.y[r0:r1], c.loss)
        gT, dtop = mlp_backward(T, ht, ds, False, self.dtype, need_dx=True, round_dx=False)
        ea = ha[-1].shape[1]
        dza = _store(dtop[:, :ea], self.dtype)
        dzp = dtop[:, ea:]
        if c.dp_clip > 0.0 and not emb_dp:
            dzp = dp_clip_noise(dzp, k, c.dp_clip, c.dp_sigma, self.dp_seed)
        dzp = _store(dzp, self.dtype)
        gA, _ = mlp_backward(A, ha, dza, True, self.dtype, need_dx=False)
        self.channel_g[k] = (dzp, j, va)

        # Backward phase (passive): fetch the gradient, backprop through the same
        # passive version with the saved activations.
        dzp_f, j_g, _ = self.channel_g.pop(k)
        assert j_g == j
        # straight-through backward of the embedding mechanism: scale by c_i, ignore its Jacobian
        dzp_in = _store(self.emb_scale.pop(k)[:, None] * dzp_f, self.dtype) if emb_dp else dzp_f
        gP, _ = mlp_backward(P, hp, dzp_in, True, self.dtype, need_dx=False)

        # Gradient descent (Eq. 2) in the delayed form of App. D:
        # theta^(k+1) = theta^(k) - eta * g evaluated at theta^(k - tau).
        lr = c.lr
        curP = self.versions_p[k]
        curA, curT = self.versions_a[k]
        newP = [(W - lr * dW, b - lr * db) for (W, b), (dW, db) in zip(curP, gP)]
        newA = [(W - lr * dW, b - lr * db) for (W, b), (dW, db) in zip(curA, gA)]
        newT = [(W - lr * dW, b - lr * db) for (W, b), (dW, db) in zip(curT, gT)]
        if self.ps:
            self.replicas[k % c.workers] = (newP, newA, newT)
            if j == self.nb - 1 and ps_aggregates_after((self.n_done + 1) // self.nb, c.ps_dt0):
                self._ps_average()
            newP, newA, newT = self.replicas[0]      # the stored version: replica 0 (see current_params)
        self.versions_p[k + 1] = newP
        self.versions_a[k + 1] = (newA, newT)
        # only the last S+1 versions can ever be read again
        for d in (self.versions_p, self.versions_a):
            for v in [v for v in d if v < k + 1 - c.staleness]:
                del d[v]
        self.k = k + 1
        self.n_done += 1

        rec = StepRecord(k, j, (r0, r1), tau_p, tau_a, vp, va, float(loss))
        if record:
            rec.zp, rec.za, rec.logits, rec.dzp, rec.dza = zp, ha[-1], logits, dzp_f, dza
            rec.ds = ds
            rec.grads = {}
            for party, g in ((0, gP), (1, gA), (2, gT)):
                for l, gl in enumerate(g):
                    rec.grads[(party, l)] = gl
            rec.params = self.replica_params(k % c.workers) if self.ps else self.current_params()
        return rec

    def _ps_average(self):
        """Every party's replicas take their mean (sum over the workers in order, divided by W)."""
        W = len(self.replicas)
        avg = []
        for part in range(3):
            layers = []
            for l in range(len(self.replicas[0][part])):
                Ws = sum(self.replicas[w][part][l][0] for w in range(W)) / W
                bs = sum(self.replicas[w][part][l][1] for w in range(W)) / W
                layers.append((Ws, bs))
            avg.append(layers)
        self.replicas = [tuple(_copy_params(p) for p in avg) for _ in range(W)]

    def replica_params(self, w: int):
        """Parameter-server mode: replica w's parameters {(party, layer): (W, b)}."""
        out = {}
        for party, layers in enumerate(self.replicas[w]):
            for l, (W, b) in enumerate(layers):
                out[(party, l)] = (W.copy(), b.copy())
        return out

    def current_params(self):
        """The parameters after the last step (parameter-server mode: replica 0's)."""
        if self.ps:
            return self.replica_params(0)
        out = {}
        P = self.versions_p[self.k]
        A, T = self.versions_a[self.k]
        for party, layers in ((0, P), (1, A), (2, T)):
            for l, (W, b) in enumerate(layers):
                out[(party, l)] = (W.copy(), b.copy())
        return out

    def run(self, tau_p, tau_a, n_steps: int, record_steps=(), drops=None):
        """n_steps steps from the current k; returns (per-step mean losses, NaN for a
        dropped step; records)."""
        losses, recs = [], {}
        rs = set(record_steps)
        for _ in range(n_steps):
            k = self.k
            r = self.step(int(tau_p[k]), int(tau_a[k]), record=k in rs, drop=drops is not None and bool(drops[k]))
            losses.append(r.loss)
            if k in rs:
                recs[k] = r
        return np.array(losses), recs

    def epoch_loss(self, losses, k0: int):
        """Mean per-sample loss over the steps k0 .. k0+len(losses)-1 (each step's
        mean weighted by its row count)."""
        tot, n = 0.0, 0
        for i, l in enumerate(losses):
            _, r0, r1 = self.batch_rows(k0 + i)
            tot += l * (r1 - r0)
            n += r1 - r0
        return tot / n

    def full_loss(self):
        """Loss of the current parameters over all rows (no training)."""
        P = self._compute(self.versions_p[self.k])
        A_m, T_m = self.versions_a[self.k]
        A, T = self._compute(A_m), self._compute(T_m)
        zp = mlp_forward(P, self.xp_c, True, self.dtype)[-1]
        za = mlp_forward(A, self.xa_c, True, self.dtype)[-1]
        s = mlp_forward(T, np.concatenate([za, zp], axis=1), False, self.dtype)[-1]
        return loss_and_dlogits(s, self.y, self.cfg.loss)[0]
