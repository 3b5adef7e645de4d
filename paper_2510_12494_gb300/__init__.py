"""Python binding of libvfl, the GB300 split-VFL training step (PubSub-VFL,
arxiv 2510.12494).  Argument marshalling only: every step of the training
path runs in the library's CUDA kernels.  PyTorch provides the device
workspace and the CUDA streams.

There is no CPU fallback: if libvfl.so is missing, importing the library
raises; build it with ``paper_2510_12494_gb300.build.build()``.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libvfl.so")

VFL_OK, VFL_E_INVAL, VFL_E_OOM, VFL_E_CUDA, VFL_E_STATE, VFL_E_VERSION, VFL_E_TIMEOUT = range(7)
MAX_LAYERS = 8
LOSS_BCE, LOSS_CE = 0, 1
FP32, BF16 = 0, 1
DP_GRAD, DP_EMB = 0, 1
SCHED_SYNC, SCHED_MAX, SCHED_SEEDED = 0, 1, 2
TAP_EMB, TAP_GRAD, TAP_LOGITS, TAP_ZA, TAP_DZA = range(5)


def TAP_ACT(party: int, layer: int) -> int:
    """Tap code of the output of Linear+ReLU layer `layer` of `party` (0 passive, 1 active, 2 top hidden)."""
    return 16 + 16 * party + layer
PASSIVE, ACTIVE, TOP = 0, 1, 2
KERNEL_CLASSES = 20

STATUS_NAMES = {0: "VFL_OK", 1: "VFL_E_INVAL", 2: "VFL_E_OOM", 3: "VFL_E_CUDA", 4: "VFL_E_STATE",
                5: "VFL_E_VERSION", 6: "VFL_E_TIMEOUT"}


class VflError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


class VflConfig(ctypes.Structure):
    _fields_ = [
        ("d_passive", ctypes.c_int32), ("d_active", ctypes.c_int32),
        ("n_passive", ctypes.c_int32), ("n_active", ctypes.c_int32), ("n_top", ctypes.c_int32),
        ("passive_out", ctypes.c_int32 * MAX_LAYERS), ("active_out", ctypes.c_int32 * MAX_LAYERS),
        ("top_out", ctypes.c_int32 * MAX_LAYERS),
        ("loss", ctypes.c_int32), ("dtype", ctypes.c_int32), ("batch", ctypes.c_int32),
        ("lr", ctypes.c_float), ("staleness", ctypes.c_int32), ("workers", ctypes.c_int32),
        ("dp_clip", ctypes.c_float), ("dp_sigma", ctypes.c_float), ("dp_seed", ctypes.c_uint64),
        ("dp_target", ctypes.c_int32), ("ps_dt0", ctypes.c_int32),
    ]


class VflPlanModel(ctypes.Structure):
    """vfl_plan_model: the delay, communication and memory constants of Eq. 7-15."""
    _fields_ = [(f, ctypes.c_double) for f in (
        "lambda_a", "gamma_a", "phi_a", "beta_a", "lambda_top", "gamma_top", "phi_top", "beta_top",
        "lambda_p", "gamma_p", "phi_p", "beta_p", "C_a", "C_p", "bytes_per_row", "bandwidth",
        "M_A0", "rho_A", "M_A_max", "M_P0", "rho_P", "M_P_max", "chi")]


EXPORTS = {
    # name: (restype, argtypes)
    "vfl_workspace_bytes": (ctypes.c_int32, [ctypes.POINTER(VflConfig), ctypes.c_int64, ctypes.POINTER(ctypes.c_uint64)]),
    "vfl_create": (ctypes.c_int32, [ctypes.POINTER(VflConfig), ctypes.c_int64, ctypes.c_void_p, ctypes.c_uint64,
                                    ctypes.POINTER(ctypes.c_void_p)]),
    "vfl_destroy": (ctypes.c_int32, [ctypes.c_void_p]),
    "vfl_set_streams": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_int32, ctypes.POINTER(ctypes.c_void_p)]),
    "vfl_load_data": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p]),
    "vfl_bind_host_data": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                                            ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p]),
    "vfl_bind_host_data_bf16": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                                                 ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p]),
    "vfl_bind_host_data_bits": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                                                 ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p]),
    "vfl_set_params": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_int32, ctypes.c_int32, ctypes.c_void_p,
                                        ctypes.c_void_p]),
    "vfl_get_params": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_int32, ctypes.c_int32, ctypes.c_void_p,
                                        ctypes.c_void_p]),
    "vfl_get_grads": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                                       ctypes.c_void_p, ctypes.c_void_p]),
    "vfl_step_cursor": (ctypes.c_int32, [ctypes.c_void_p, ctypes.POINTER(ctypes.c_int64)]),
    "vfl_get_version": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_int32, ctypes.c_int32, ctypes.c_int64,
                                         ctypes.c_void_p, ctypes.c_void_p]),
    "vfl_set_cursor": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_int64]),
    "vfl_set_version": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_int32, ctypes.c_int32, ctypes.c_int64,
                                         ctypes.c_void_p, ctypes.c_void_p]),
    "vfl_get_replica": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                                         ctypes.c_void_p, ctypes.c_void_p]),
    "vfl_set_replica": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                                         ctypes.c_void_p, ctypes.c_void_p]),
    "vfl_ps_interval": (ctypes.c_int32, [ctypes.c_int64, ctypes.c_int32, ctypes.POINTER(ctypes.c_int64)]),
    "vfl_plan_bmax": (ctypes.c_int32, [ctypes.POINTER(VflPlanModel), ctypes.POINTER(ctypes.c_double)]),
    "vfl_plan_delay": (ctypes.c_int32, [ctypes.POINTER(VflPlanModel), ctypes.c_int32, ctypes.c_int32, ctypes.c_double,
                                        ctypes.POINTER(ctypes.c_double)]),
    "vfl_plan": (ctypes.c_int32, [ctypes.POINTER(VflPlanModel), ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                                  ctypes.c_int32, ctypes.c_void_p, ctypes.c_int32, ctypes.POINTER(ctypes.c_int32),
                                  ctypes.POINTER(ctypes.c_int32), ctypes.POINTER(ctypes.c_int32),
                                  ctypes.POINTER(ctypes.c_double)]),
    "vfl_fit_power": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int32, ctypes.POINTER(ctypes.c_double),
                                       ctypes.POINTER(ctypes.c_double)]),
    "vfl_gdp_sigma": (ctypes.c_int32, [ctypes.c_double, ctypes.c_int64, ctypes.c_int64, ctypes.c_int64,
                                       ctypes.POINTER(ctypes.c_double)]),
    "vfl_make_schedule": (ctypes.c_int32, [ctypes.c_uint64, ctypes.c_int32, ctypes.c_int32, ctypes.c_int64,
                                           ctypes.c_void_p, ctypes.c_void_p]),
    "vfl_passive_forward": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32]),
    "vfl_active_step": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32]),
    "vfl_passive_backward": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_int64]),
    "vfl_train_steps": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int64, ctypes.c_void_p,
                                         ctypes.c_void_p, ctypes.c_void_p]),
    "vfl_graph_capture": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int64, ctypes.c_void_p,
                                           ctypes.c_void_p, ctypes.c_void_p, ctypes.POINTER(ctypes.c_void_p)]),
    "vfl_drop_step": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_int64]),
    "vfl_graph_update": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64, ctypes.c_int64,
                                          ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p]),
    "vfl_set_order": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_int32]),
    "vfl_init_params": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_uint64]),
    "vfl_train_epoch": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p, ctypes.c_void_p,
                                         ctypes.c_void_p, ctypes.POINTER(ctypes.c_float)]),
    "vfl_get_drops": (ctypes.c_int32, [ctypes.c_void_p, ctypes.POINTER(ctypes.c_int64)]),
    "vfl_set_drops": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_int64]),
    "vfl_make_drops": (ctypes.c_int32, [ctypes.c_uint64, ctypes.c_double, ctypes.c_int64, ctypes.c_void_p]),
    "vfl_graph_launch": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_void_p]),
    "vfl_graph_destroy": (ctypes.c_int32, [ctypes.c_void_p]),
    "vfl_synchronize": (ctypes.c_int32, [ctypes.c_void_p]),
    "vfl_read_losses": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int64, ctypes.c_void_p]),
    "vfl_tap": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_void_p, ctypes.c_int64]),
    "vfl_step_rows": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_int64, ctypes.POINTER(ctypes.c_int64),
                                       ctypes.POINTER(ctypes.c_int32)]),
    "vfl_fetch_loss": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p]),
    "vfl_wait_channel": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_int64]),
    "vfl_check_channel": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64]),
    "vfl_kernel_launches": (ctypes.c_int64, [ctypes.c_void_p]),
    "vfl_exchange_bytes": (ctypes.c_int32, [ctypes.c_void_p, ctypes.POINTER(ctypes.c_int64),
                                            ctypes.POINTER(ctypes.c_int64)]),
    "vfl_profile": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_int32]),
    "vfl_profile_get": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_int32, ctypes.POINTER(ctypes.c_int64),
                                         ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_double),
                                         ctypes.POINTER(ctypes.c_double)]),
    "vfl_kernel_class_name": (ctypes.c_char_p, [ctypes.c_int32]),
    "vfl_weight_grad_noalloc": (ctypes.c_int32, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int32, ctypes.c_int32,
                                                 ctypes.c_int32, ctypes.c_int32, ctypes.c_void_p, ctypes.c_void_p,
                                                 ctypes.c_void_p]),
    "vfl_measure_peak": (ctypes.c_int32, [ctypes.c_int32, ctypes.c_int64, ctypes.POINTER(ctypes.c_double),
                                          ctypes.POINTER(ctypes.c_float)]),
    "vfl_last_error": (ctypes.c_char_p, [ctypes.c_void_p]),
}
PEAK_FFMA, PEAK_TF32_MMA = 0, 1

_lib = None


def lib():
    """The loaded libvfl.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"{LIB_PATH} is missing: build it with paper_2510_12494_gb300.build.build() "
                              "(there is no CPU fallback)")
        L = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in EXPORTS.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _check(st: int, ctx=None):
    if st != VFL_OK:
        msg = lib().vfl_last_error(ctx)
        raise VflError(st, msg.decode() if msg else "")


def make_config(p) -> VflConfig:
    """VflConfig from an object with the preset fields (d_passive, d_active,
    passive, active, top, loss, dtype, batch, lr, staleness, workers, dp_clip,
    dp_sigma, seed)."""
    c = VflConfig()
    c.d_passive, c.d_active = p.d_passive, p.d_active
    c.n_passive, c.n_active, c.n_top = len(p.passive), len(p.active), len(p.top)
    for arr, vals in ((c.passive_out, p.passive), (c.active_out, p.active), (c.top_out, p.top)):
        for i, v in enumerate(vals):
            arr[i] = v
    c.loss = LOSS_BCE if p.loss == "bce" else LOSS_CE
    c.dtype = FP32 if p.dtype == "fp32" else BF16
    c.batch = p.batch
    c.lr = p.lr
    c.staleness = p.staleness
    c.workers = p.workers
    c.dp_clip = p.dp_clip
    c.dp_sigma = p.dp_sigma
    c.dp_seed = getattr(p, "dp_seed", getattr(p, "seed", 0))
    c.dp_target = DP_EMB if getattr(p, "dp_target", "grad") == "emb" else DP_GRAD
    c.ps_dt0 = getattr(p, "ps_dt0", 0)
    return c


def ps_interval(t: int, dt0: int) -> int:
    """Delta T_t of Eq. 5 as the runtime computes it (see vfl_ps_interval)."""
    out = ctypes.c_int64()
    _check(lib().vfl_ps_interval(t, dt0, ctypes.byref(out)))
    return out.value


def gdp_sigma(mu: float, batch: int, n_rows: int, queries: int) -> float:
    """Noise multiplier for mu-GDP on the published embedding (Eq. 25, see vfl_gdp_sigma)."""
    out = ctypes.c_double()
    _check(lib().vfl_gdp_sigma(mu, batch, n_rows, queries, ctypes.byref(out)))
    return out.value


def make_schedule(seed: int, S: int, kind: int, n_steps: int):
    """(tau_p, tau_a) int32 arrays from the library's host-side schedule."""
    tp = np.zeros(max(n_steps, 1), np.int32)
    ta = np.zeros(max(n_steps, 1), np.int32)
    _check(lib().vfl_make_schedule(seed, S, kind, n_steps, _ptr(tp), _ptr(ta)))
    return tp[:n_steps], ta[:n_steps]


def plan_model(**kw) -> VflPlanModel:
    """A vfl_plan_model from keyword constants (unnamed ones 0; C_a, C_p, bandwidth and chi default 1)."""
    m = VflPlanModel()
    m.C_a = m.C_p = m.bandwidth = m.chi = 1.0
    for k, v in kw.items():
        setattr(m, k, float(v))
    return m


def plan_bmax(m: VflPlanModel) -> float:
    out = ctypes.c_double()
    _check(lib().vfl_plan_bmax(ctypes.byref(m), ctypes.byref(out)))
    return out.value


def plan_delay(m: VflPlanModel, w_a: int, w_p: int, batch: float) -> float:
    out = ctypes.c_double()
    _check(lib().vfl_plan_delay(ctypes.byref(m), w_a, w_p, batch, ctypes.byref(out)))
    return out.value


def plan(m: VflPlanModel, wa_range, wp_range, batches):
    """Algorithm 2 (vfl_plan): (w_a, w_p, B, O)."""
    b = np.ascontiguousarray(batches, np.int32)
    wa, wp, bb, o = ctypes.c_int32(), ctypes.c_int32(), ctypes.c_int32(), ctypes.c_double()
    _check(lib().vfl_plan(ctypes.byref(m), wa_range[0], wa_range[1], wp_range[0], wp_range[1], _ptr(b), len(b),
                          ctypes.byref(wa), ctypes.byref(wp), ctypes.byref(bb), ctypes.byref(o)))
    return wa.value, wp.value, bb.value, o.value


def fit_power(x, t):
    """(coef, expo) of t = coef * x^expo (vfl_fit_power)."""
    x = np.ascontiguousarray(x, np.float64)
    t = np.ascontiguousarray(t, np.float64)
    c, e = ctypes.c_double(), ctypes.c_double()
    _check(lib().vfl_fit_power(_ptr(x), _ptr(t), len(x), ctypes.byref(c), ctypes.byref(e)))
    return c.value, e.value


def measure_peak(kind: int, iters: int):
    """(flop, ms) of one timed throughput launch (vfl_measure_peak) on the current device."""
    f, ms = ctypes.c_double(), ctypes.c_float()
    _check(lib().vfl_measure_peak(kind, iters, ctypes.byref(f), ctypes.byref(ms)))
    return f.value, float(ms.value)


def make_drops(seed: int, rate: float, n_steps: int):
    """uint8 drop marks from the library's seeded draws (see vfl_make_drops)."""
    out = np.zeros(max(n_steps, 1), np.uint8)
    _check(lib().vfl_make_drops(seed, rate, n_steps, _ptr(out)))
    return out[:n_steps]


def _drops_ptr(drops, end):
    if drops is None:
        return None, None
    d = np.ascontiguousarray(drops, np.uint8)
    assert len(d) >= end
    return d, _ptr(d)


def weight_grad_noalloc(dpre, x, dW, db, dtype: int, stream=None):
    """dW = dpre^T x and db = column sums of dpre on device tensors (dpre [rows,
    out], x [rows, in], dW [out, in] fp32, db [out] fp32), using the library's
    fixed scratch instead of any allocation.  Enqueued on ``stream`` (a
    torch.cuda.Stream; default: the current stream)."""
    import torch
    if dtype not in (FP32, BF16):
        raise ValueError(f"dtype must be FP32 or BF16, got {dtype}")
    if dpre.dim() != 2 or x.dim() != 2 or dW.dim() != 2 or db.dim() != 1:
        raise ValueError("dpre, x and dW must be matrices and db a vector")
    rows, out = dpre.shape
    if x.shape[0] != rows or tuple(dW.shape) != (out, x.shape[1]) or tuple(db.shape) != (out,):
        raise ValueError(f"shapes disagree: dpre {tuple(dpre.shape)}, x {tuple(x.shape)}, dW {tuple(dW.shape)}, "
                         f"db {tuple(db.shape)}")
    # the kernel reads and writes raw row-major buffers of these element types: anything else would be
    # read or written past its end
    want = torch.float32 if dtype == FP32 else torch.bfloat16
    for name, t, dt in (("dpre", dpre, want), ("x", x, want), ("dW", dW, torch.float32), ("db", db, torch.float32)):
        if t.dtype != dt:
            raise ValueError(f"{name} must be {dt}, got {t.dtype}")
        if not t.is_contiguous():
            raise ValueError(f"{name} must be contiguous (row-major)")
    s = stream if stream is not None else torch.cuda.current_stream()
    for name, t in (("dpre", dpre), ("x", x), ("dW", dW), ("db", db)):
        if t.device.type != "cuda" or t.device.index != s.device.index:
            raise ValueError(f"{name} must be on {s.device}, the stream's device (got {t.device})")
    _check(lib().vfl_weight_grad_noalloc(ctypes.c_void_p(dpre.data_ptr()), ctypes.c_void_p(x.data_ptr()), rows, out,
                                         x.shape[1], dtype, ctypes.c_void_p(dW.data_ptr()),
                                         ctypes.c_void_p(db.data_ptr()), ctypes.c_void_p(s.cuda_stream)))


def pack_bits(x: np.ndarray) -> np.ndarray:
    """Binary features [n, d] (every value 0 or 1) as the [n, ceil(d / 32)] int32 words
    vfl_bind_host_data_bits reads: feature c of a row in bit c mod 32 of word c // 32."""
    x = np.asarray(x)
    if not ((x == 0) | (x == 1)).all():
        raise ValueError("pack_bits: features must be 0 or 1")
    n, d = x.shape
    w = (d + 31) // 32
    b = np.zeros((n, 4 * w), np.uint8)
    b[:, : (d + 7) // 8] = np.packbits(x.astype(np.uint8, copy=False), axis=1, bitorder="little")
    return b.view("<u4").view(np.int32).reshape(n, w)


def workspace_bytes(p, n_rows: int) -> int:
    cfg = make_config(p)
    out = ctypes.c_uint64()
    _check(lib().vfl_workspace_bytes(ctypes.byref(cfg), n_rows, ctypes.byref(out)))
    return out.value


class Context:
    """One training context on the current CUDA device."""

    def __init__(self, p, n_rows: int, streams=None):
        import torch
        self.p = p
        self.cfg = make_config(p)
        self.n_rows = n_rows
        L = lib()
        nbytes = workspace_bytes(p, n_rows)
        self.workspace = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
        handle = ctypes.c_void_p()
        _check(L.vfl_create(ctypes.byref(self.cfg), n_rows, ctypes.c_void_p(self.workspace.data_ptr()),
                            nbytes, ctypes.byref(handle)))
        self.h = handle
        # the parties' worker streams one priority level above the I/O stream of the host-data bindings, so
        # that the SMs go to a step's kernels before the staging of steps further ahead
        self.streams = streams if streams is not None else [torch.cuda.Stream(priority=-1)
                                                            for _ in range(2 * p.workers)]
        arr = (ctypes.c_void_p * len(self.streams))(*[s.cuda_stream for s in self.streams])
        self._call(L.vfl_set_streams, len(self.streams), arr)
        self.nb = -(-n_rows // p.batch)

    def _call(self, f, *args):
        st = f(self.h, *args)
        if st != VFL_OK:
            msg = lib().vfl_last_error(self.h)
            raise VflError(st, msg.decode() if msg else "")

    def close(self):
        if getattr(self, "h", None):
            for g in getattr(self, "_graphs", []):
                lib().vfl_graph_destroy(g)
            self._graphs = []
            lib().vfl_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # data / parameters -----------------------------------------------------
    def load_data(self, xp, xa, y):
        xp = np.ascontiguousarray(xp, np.float32)
        xa = np.ascontiguousarray(xa, np.float32)
        y = np.ascontiguousarray(y, np.int32)
        assert xp.shape == (self.n_rows, self.p.d_passive) and xa.shape == (self.n_rows, self.p.d_active)
        self._call(lib().vfl_load_data, _ptr(xp), _ptr(xa), _ptr(y))

    def bind_host_data(self, xp, xa, y, loss_out=None):
        """Every later step reads its rows from these host tensors (pinned torch
        tensors [n_rows, d_p] / [n_rows, d_a] fp32, or bf16 for a bf16 context
        (vfl_bind_host_data_bf16), and [n_rows] int32) on an I/O
        stream of the context, and writes its mean loss into loss_out[k % len(loss_out)]
        (a pinned fp32 tensor, optional); see vfl_bind_host_data.
        bind_host_data(None, None, None) unbinds.  The tensors stay referenced while bound."""
        import torch
        if xp is None:
            self._call(lib().vfl_bind_host_data, None, None, None, None, 0, None)
            self._host_data = None
            return
        assert tuple(xp.shape) == (self.n_rows, self.p.d_passive) and tuple(xa.shape) == (self.n_rows, self.p.d_active)
        assert tuple(y.shape) == (self.n_rows,)
        assert xp.dtype == xa.dtype and xp.dtype in (torch.float32, torch.bfloat16) and y.dtype == torch.int32
        assert xp.is_contiguous() and xa.is_contiguous() and y.is_contiguous()
        if not hasattr(self, "_io_stream"):
            self._io_stream = torch.cuda.Stream()
        lp = ctypes.c_void_p(loss_out.data_ptr()) if loss_out is not None else None
        cap = len(loss_out) if loss_out is not None else 0
        fn = lib().vfl_bind_host_data_bf16 if xp.dtype == torch.bfloat16 else lib().vfl_bind_host_data
        self._call(fn, ctypes.c_void_p(xp.data_ptr()), ctypes.c_void_p(xa.data_ptr()),
                   ctypes.c_void_p(y.data_ptr()), lp, cap, ctypes.c_void_p(self._io_stream.cuda_stream))
        self._host_data = (xp, xa, y, loss_out)

    def bind_host_bits(self, xp_bits, xa_bits, y, loss_out=None):
        """bind_host_data for binary features held bit-packed (vfl_bind_host_data_bits): pinned int32
        tensors [n_rows, ceil(d_p / 32)] / [n_rows, ceil(d_a / 32)] of 32-bit words (pack_bits), the
        labels and the loss ring as in bind_host_data.  bind_host_data(None, None, None) unbinds."""
        import torch
        assert tuple(xp_bits.shape) == (self.n_rows, (self.p.d_passive + 31) // 32)
        assert tuple(xa_bits.shape) == (self.n_rows, (self.p.d_active + 31) // 32)
        assert tuple(y.shape) == (self.n_rows,)
        assert xp_bits.dtype == xa_bits.dtype == torch.int32 and y.dtype == torch.int32
        assert xp_bits.is_contiguous() and xa_bits.is_contiguous() and y.is_contiguous()
        if not hasattr(self, "_io_stream"):
            self._io_stream = torch.cuda.Stream()
        lp = ctypes.c_void_p(loss_out.data_ptr()) if loss_out is not None else None
        cap = len(loss_out) if loss_out is not None else 0
        self._call(lib().vfl_bind_host_data_bits, ctypes.c_void_p(xp_bits.data_ptr()),
                   ctypes.c_void_p(xa_bits.data_ptr()), ctypes.c_void_p(y.data_ptr()), lp, cap,
                   ctypes.c_void_p(self._io_stream.cuda_stream))
        self._host_data = (xp_bits, xa_bits, y, loss_out)

    def set_params(self, params: dict):
        for (party, l), (W, b) in params.items():
            W = np.ascontiguousarray(W, np.float32)
            b = np.ascontiguousarray(b, np.float32)
            self._call(lib().vfl_set_params, party, l, _ptr(W), _ptr(b))

    def _shape(self, party, l):
        widths = (self.p.passive, self.p.active, self.p.top)[party]
        fin = (self.p.d_passive, self.p.d_active, self.p.e_active + self.p.e_passive)[party] if l == 0 else widths[l - 1]
        return widths[l], fin

    def get_params(self):
        out = {}
        for party, widths in ((0, self.p.passive), (1, self.p.active), (2, self.p.top)):
            for l in range(len(widths)):
                o, i = self._shape(party, l)
                W = np.zeros((o, i), np.float32)
                b = np.zeros(o, np.float32)
                self._call(lib().vfl_get_params, party, l, _ptr(W), _ptr(b))
                out[(party, l)] = (W, b)
        return out

    def get_grads(self, worker: int = 0, parties=(0, 1, 2)):
        out = {}
        for party in parties:
            widths = (self.p.passive, self.p.active, self.p.top)[party]
            for l in range(len(widths)):
                o, i = self._shape(party, l)
                dW = np.zeros((o, i), np.float32)
                db = np.zeros(o, np.float32)
                self._call(lib().vfl_get_grads, party, l, worker, _ptr(dW), _ptr(db))
                out[(party, l)] = (dW, db)
        return out

    # checkpoint / restore --------------------------------------------------
    def cursor(self) -> int:
        k = ctypes.c_int64()
        self._call(lib().vfl_step_cursor, ctypes.byref(k))
        return k.value

    def get_version(self, v: int):
        """{(party, layer): (W, b)} of stored weight version v (compute copy, as fp32)."""
        out = {}
        for party, widths in ((0, self.p.passive), (1, self.p.active), (2, self.p.top)):
            for l in range(len(widths)):
                o, i = self._shape(party, l)
                W = np.zeros((o, i), np.float32)
                b = np.zeros(o, np.float32)
                self._call(lib().vfl_get_version, party, l, v, _ptr(W), _ptr(b))
                out[(party, l)] = (W, b)
        return out

    def get_replica(self, w: int):
        """Parameter-server mode: {(party, layer): (W, b)} of worker w's replica (fp32 masters)."""
        out = {}
        for party, widths in ((0, self.p.passive), (1, self.p.active), (2, self.p.top)):
            for l in range(len(widths)):
                o, i = self._shape(party, l)
                W = np.zeros((o, i), np.float32)
                b = np.zeros(o, np.float32)
                self._call(lib().vfl_get_replica, w, party, l, _ptr(W), _ptr(b))
                out[(party, l)] = (W, b)
        return out

    def set_replica(self, w: int, params: dict):
        for (party, l), (W, b) in params.items():
            W = np.ascontiguousarray(W, np.float32)
            b = np.ascontiguousarray(b, np.float32)
            self._call(lib().vfl_set_replica, w, party, l, _ptr(W), _ptr(b))

    def set_cursor(self, k: int):
        self._call(lib().vfl_set_cursor, k)

    def set_version(self, v: int, params: dict, parties=(0, 1, 2)):
        for (party, l), (W, b) in params.items():
            if party not in parties:
                continue
            W = np.ascontiguousarray(W, np.float32)
            b = np.ascontiguousarray(b, np.float32)
            self._call(lib().vfl_set_version, party, l, v, _ptr(W), _ptr(b))

    @property
    def ps(self) -> bool:
        return self.cfg.ps_dt0 > 0

    def checkpoint(self):
        """(k, {version: params}, fp32 masters of version k, dropped steps so far); in
        the parameter-server mode (k, {worker: replica}, None, dropped steps)."""
        k = self.cursor()
        if self.ps:
            return k, {w: self.get_replica(w) for w in range(self.p.workers)}, None, self.drops()
        vers = {v: self.get_version(v) for v in range(max(0, k - self.p.staleness), k + 1)}
        return k, vers, self.get_params(), self.drops()

    def restore(self, ckpt):
        k, vers, master, drops = ckpt
        self.set_cursor(k)
        self.set_drops(drops)
        if self.ps:
            for w, params in vers.items():
                self.set_replica(w, params)
            return
        for v, params in vers.items():
            self.set_version(v, master if v == k else params)

    # the three phases and the whole DAG ------------------------------------
    def passive_forward(self, k, tau_p):
        self._call(lib().vfl_passive_forward, k, tau_p)

    def active_step(self, k, tau_a):
        self._call(lib().vfl_active_step, k, tau_a)

    def passive_backward(self, k):
        self._call(lib().vfl_passive_backward, k)

    def init_params(self, seed: int):
        """Seeded initial parameters (vfl_init_params; the recipe of synth.init_params)."""
        self._call(lib().vfl_init_params, seed)

    def train_epoch(self, epoch, tau_p, tau_a, drops=None, mean_loss=True):
        """Steps of one epoch (vfl_train_epoch); returns the epoch's mean loss per sample (or None)."""
        tau_p = np.ascontiguousarray(tau_p, np.int32)
        tau_a = np.ascontiguousarray(tau_a, np.int32)
        end = (epoch + 1) * self.nb
        assert len(tau_p) >= end and len(tau_a) >= end
        d, dp = _drops_ptr(drops, end)
        out = ctypes.c_float()
        self._call(lib().vfl_train_epoch, epoch, _ptr(tau_p), _ptr(tau_a), dp, ctypes.byref(out) if mean_loss else None)
        return out.value if mean_loss else None

    def drop_step(self, k):
        """The subscriber of step k gives up on its embedding (see vfl_drop_step)."""
        self._call(lib().vfl_drop_step, k)

    def drops(self) -> int:
        n = ctypes.c_int64()
        self._call(lib().vfl_get_drops, ctypes.byref(n))
        return n.value

    def set_drops(self, n: int):
        self._call(lib().vfl_set_drops, n)

    def train_steps(self, k0, n, tau_p, tau_a, drops=None):
        tau_p = np.ascontiguousarray(tau_p, np.int32)
        tau_a = np.ascontiguousarray(tau_a, np.int32)
        assert len(tau_p) >= k0 + n and len(tau_a) >= k0 + n
        d, dp = _drops_ptr(drops, k0 + n)
        self._call(lib().vfl_train_steps, k0, n, _ptr(tau_p), _ptr(tau_a), dp)

    def capture(self, k0, n, tau_p, tau_a, drops=None):
        """A CUDA graph of steps [k0, k0+n) (see vfl_graph_capture); replay with launch_graph."""
        tau_p = np.ascontiguousarray(tau_p, np.int32)
        tau_a = np.ascontiguousarray(tau_a, np.int32)
        assert len(tau_p) >= k0 + n and len(tau_a) >= k0 + n
        d, dp = _drops_ptr(drops, k0 + n)
        g = ctypes.c_void_p()
        self._call(lib().vfl_graph_capture, k0, n, _ptr(tau_p), _ptr(tau_a), dp, ctypes.byref(g))
        self._graphs = getattr(self, "_graphs", []) + [g]
        return g

    def update_graph(self, g, k0, n, tau_p, tau_a, drops=None) -> bool:
        """Re-record g for steps [k0, k0+n) in place (vfl_graph_update); False when the shape differs."""
        tau_p = np.ascontiguousarray(tau_p, np.int32)
        tau_a = np.ascontiguousarray(tau_a, np.int32)
        assert len(tau_p) >= k0 + n and len(tau_a) >= k0 + n
        d, dp = _drops_ptr(drops, k0 + n)
        st = lib().vfl_graph_update(self.h, g, k0, n, _ptr(tau_p), _ptr(tau_a), dp)
        if st == VFL_E_STATE:
            return False
        _check(st, self.h)
        return True

    def set_order(self, uniform: bool):
        """VFL_ORDER_UNIFORM (True) or VFL_ORDER_OVERLAP (False), see vfl_set_order."""
        self._call(lib().vfl_set_order, 1 if uniform else 0)

    def launch_graph(self, g):
        self._call(lib().vfl_graph_launch, g)

    def synchronize(self):
        self._call(lib().vfl_synchronize)

    def read_losses(self, k0, n):
        out = np.zeros(max(n, 1), np.float32)
        self._call(lib().vfl_read_losses, k0, n, _ptr(out))
        return out[:n]

    def fetch_loss(self, k, host_ptr: int):
        """Asynchronous device->host copy of step k's mean loss to host address host_ptr."""
        self._call(lib().vfl_fetch_loss, k, ctypes.c_void_p(host_ptr))

    def batch_rows(self, k):
        """(first row, end row) of the batch step k trains, as the library assigns it."""
        r0 = ctypes.c_int64()
        n = ctypes.c_int32()
        self._call(lib().vfl_step_rows, k, ctypes.byref(r0), ctypes.byref(n))
        return r0.value, r0.value + n.value

    def tap(self, k, what):
        r0, r1 = self.batch_rows(k)
        if what >= 16:
            party, layer = divmod(what - 16, 16)
            cols = (self.p.passive, self.p.active, self.p.top)[party][layer]
        else:
            cols = {TAP_EMB: self.p.e_passive, TAP_GRAD: self.p.e_passive, TAP_LOGITS: self.p.n_out,
                    TAP_ZA: self.p.e_active, TAP_DZA: self.p.e_active}[what]
        out = np.zeros((r1 - r0, cols), np.float32)
        self._call(lib().vfl_tap, k, what, _ptr(out), out.size)
        return out

    def wait_channel(self, which, k, max_iters):
        self._call(lib().vfl_wait_channel, which, k, max_iters)

    def check_channel(self, which, k):
        self._call(lib().vfl_check_channel, which, k)

    @property
    def launches(self) -> int:
        return lib().vfl_kernel_launches(self.h)

    def exchange_bytes(self):
        """(embedding, gradient) payload bytes published so far (vfl_exchange_bytes)."""
        e, g = ctypes.c_int64(), ctypes.c_int64()
        _check(lib().vfl_exchange_bytes(self.h, ctypes.byref(e), ctypes.byref(g)), self.h)
        return e.value, g.value

    def profile(self, enable: bool):
        self._call(lib().vfl_profile, 1 if enable else 0)

    def profile_summary(self):
        """{class name: (launches, ms, flops, bytes)} of the last profiled region."""
        out = {}
        for c in range(KERNEL_CLASSES):
            n, ms, fl, by = ctypes.c_int64(), ctypes.c_double(), ctypes.c_double(), ctypes.c_double()
            _check(lib().vfl_profile_get(self.h, c, ctypes.byref(n), ctypes.byref(ms), ctypes.byref(fl),
                                         ctypes.byref(by)), self.h)
            if n.value:
                out[lib().vfl_kernel_class_name(c).decode()] = (n.value, ms.value, fl.value, by.value)
        return out
