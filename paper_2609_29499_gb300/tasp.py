"""Thin Python binding of the TASP C ABI (include/tasp.h).

Argument marshalling only: every step of the path runs in the CUDA library
``libtasp.so`` built in-tree by ``paper_2609_29499_gb300.build``. There is no
fallback: if the library is missing or cannot be loaded, ``load()`` raises.
PyTorch supplies device buffers and streams (``tensor.data_ptr()``,
``torch.cuda.current_stream().cuda_stream``).
"""
from __future__ import annotations

import ctypes
import os
from ctypes import POINTER, c_double, c_float, c_int32, c_int64, c_size_t, c_uint32, c_uint64, c_void_p

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libtasp.so")

OK, EINVAL, EMASK, ECAP, ENOMEM, EBUSY, ECUDA, EUNSUP = 0, -1, -2, -3, -4, -5, -6, -7
MASK_ALL_KEEP, MASK_GREEDY, MASK_EXPLICIT, MASK_GREEDY_QHEADS, MASK_EXPLICIT_QHEADS = 0, 1, 2, 3, 4
PANELS_COMPACT, PANELS_ROW_INDEXED = 0, 1
(EXPORT_KEEP_GROUPS, EXPORT_KEEP_CHANS, EXPORT_QKV_W, EXPORT_QKV_S, EXPORT_O_W, EXPORT_O_S, EXPORT_GU_W,
 EXPORT_GU_S, EXPORT_DOWN_W, EXPORT_DOWN_S, EXPORT_KEEP_QHEADS, EXPORT_QKV_G, EXPORT_O_G, EXPORT_GU_G,
 EXPORT_DOWN_G) = range(15)
KERNEL_KINDS = 7
KERNEL_NAMES = ("qkv", "attention", "o_proj", "gate_up", "down", "lm_head", "other")

# Symbols declared in include/tasp.h (the CPU test checks they are all exported).
EXPORTED = ("tasp_compile_mask", "tasp_prefill", "tasp_decode_step", "tasp_release", "tasp_session_create",
            "tasp_session_fill_synthetic", "tasp_session_position", "tasp_session_status", "tasp_decode_step_host", "tasp_mask_select",
            "tasp_mask_select_qheads", "tasp_set_memory_limit", "tasp_memory_in_use", "tasp_dispatch",
            "tasp_plan_layer_qheads", "tasp_plan_layout",
            "tasp_plan_info_get", "tasp_plan_layer_dims", "tasp_plan_export", "tasp_layer_step",
            "tasp_profile_step", "tasp_step_launches", "tasp_decode_step_static", "tasp_session_kv_export",
            "tasp_session_prefill", "tasp_decode_step_union", "tasp_union_status",
            "tasp_test_set_wait_limit", "tasp_test_skip_gemv_copies", "tasp_spectral_layer",
            "tasp_last_error",
            "tasp_version")


class ModelDesc(ctypes.Structure):
    _fields_ = [("L", c_int32), ("d", c_int32), ("Hq", c_int32), ("Hkv", c_int32), ("dh", c_int32),
                ("df", c_int32), ("vocab", c_int32), ("chan_unit", c_int32), ("rms_eps", c_float),
                ("rope_theta", c_float), ("seed", c_uint64), ("quant_group", c_int32)]


class MaskDesc(ctypes.Structure):
    _fields_ = [("kind", c_int32), ("panel_mode", c_int32), ("flop_budget", c_double), ("r_lo", c_double),
                ("r_hi", c_double), ("scores", POINTER(c_uint32)), ("target_u24", POINTER(c_uint32)),
                ("keep_groups", POINTER(c_int32)), ("n_groups", POINTER(c_int32)),
                ("keep_units", POINTER(c_int32)), ("n_units", POINTER(c_int32)),
                ("keep_qheads", POINTER(c_int32)), ("n_qheads", POINTER(c_int32))]


class PlanInfo(ctypes.Structure):
    _fields_ = [("L", c_int32), ("panel_bytes", c_int64), ("store_bytes", c_int64),
                ("weight_bytes_per_token", c_int64), ("flops_retained", c_int64), ("flops_dense", c_int64),
                ("launched_flops", c_int64)]


class TaspError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__(f"tasp error {code}: {msg}")
        self.code = code


_lib = None


def load(path: str = LIB_PATH):
    """Load libtasp.so (raises if it is missing: there is no CPU fallback)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with paper_2609_29499_gb300.build.build()")
    try:  # make the CUDA runtime that PyTorch ships visible first, when torch is installed
        import torch  # noqa: F401
    except Exception:
        pass
    lib = ctypes.CDLL(path)
    P = c_void_p
    sig = {
        "tasp_compile_mask": (c_int32, [POINTER(ModelDesc), POINTER(MaskDesc), POINTER(P)]),
        "tasp_prefill": (c_int32, [P, P, c_int32, c_int32, P, POINTER(P), P]),
        "tasp_decode_step": (c_int32, [POINTER(P), c_int32, P, P, P, P]),
        "tasp_release": (c_int32, [P]),
        "tasp_session_create": (c_int32, [P, c_int32, POINTER(P)]),
        "tasp_session_fill_synthetic": (c_int32, [P, c_int32, c_uint64, P]),
        "tasp_session_position": (c_int32, [P, POINTER(c_int32)]),
        "tasp_session_status": (c_int32, [P, c_int32, POINTER(c_int32)]),
        "tasp_decode_step_host": (c_int32, [POINTER(P), c_int32, P, P, P, P]),
        "tasp_mask_select": (c_int32, [POINTER(ModelDesc), POINTER(MaskDesc), P, P, P, P, P]),
        "tasp_mask_select_qheads": (c_int32, [POINTER(ModelDesc), POINTER(MaskDesc), P, P, P, P, P, P, P]),
        "tasp_set_memory_limit": (c_int32, [c_int64]),
        "tasp_test_set_wait_limit": (c_int32, [c_int64]),
        "tasp_spectral_layer": (c_int32, [P, c_int32, P, P, P, P]),
        "tasp_test_skip_gemv_copies": (c_int32, [c_int32]),
        "tasp_dispatch": (c_int32, [P, c_int32, c_float, POINTER(c_int32)]),
        "tasp_plan_layer_qheads": (c_int32, [P, c_int32, POINTER(c_int32)]),
        "tasp_plan_layout": (c_int32, [POINTER(ModelDesc), POINTER(MaskDesc), c_int32, P, P, P, P, P, P]),
        "tasp_memory_in_use": (c_int32, [POINTER(c_int64)]),
        "tasp_plan_info_get": (c_int32, [P, POINTER(PlanInfo)]),
        "tasp_plan_layer_dims": (c_int32, [P, c_int32, P]),
        "tasp_plan_export": (c_int32, [P, c_int32, c_int32, P, c_size_t]),
        "tasp_layer_step": (c_int32, [P, c_int32, P, P, P]),
        "tasp_profile_step": (c_int32, [POINTER(P), c_int32, P, P, P, P, P]),
        "tasp_step_launches": (c_int32, [POINTER(P), c_int32, c_int32, POINTER(c_int32)]),
        "tasp_decode_step_static": (c_int32, [P, P, P, P, P]),
        "tasp_session_kv_export": (c_int32, [P, c_int32, c_int32, P, c_size_t]),
        "tasp_session_prefill": (c_int32, [P, P, c_int32, P, P]),
        "tasp_decode_step_union": (c_int32, [POINTER(P), c_int32, P, P, P, P]),
        "tasp_union_status": (c_int32, [POINTER(P), c_int32, POINTER(c_int32), POINTER(c_int32)]),
        "tasp_last_error": (ctypes.c_char_p, []),
        "tasp_version": (ctypes.c_char_p, []),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    _lib = lib
    return lib


def _check(rc):
    if rc != OK:
        raise TaspError(rc, load().tasp_last_error().decode())


def model_desc(shape) -> ModelDesc:
    """ModelDesc from any object with L, d, Hq, Hkv, dh, df, vocab, chan_unit, eps, rope_theta, seed."""
    return ModelDesc(shape.L, shape.d, shape.Hq, shape.Hkv, shape.dh, shape.df, shape.vocab, shape.chan_unit,
                     shape.eps, shape.rope_theta, shape.seed, getattr(shape, "quant_group", 0))


class _MaskArgs:
    """Owns the numpy buffers a MaskDesc points to."""

    def __init__(self, kind, panel_mode=PANELS_COMPACT, budget=0.57, r_lo=0.35, r_hi=0.85, scores=None,
                 target_u24=None, groups=None, units=None, qheads=None):
        self.keep = []
        d = MaskDesc()
        d.kind, d.panel_mode, d.flop_budget, d.r_lo, d.r_hi = kind, panel_mode, budget, r_lo, r_hi
        if scores is not None:
            s = np.ascontiguousarray(scores, dtype=np.uint32)
            t = np.ascontiguousarray(target_u24, dtype=np.uint32)
            self.keep += [s, t]
            d.scores = s.ctypes.data_as(POINTER(c_uint32))
            d.target_u24 = t.ctypes.data_as(POINTER(c_uint32))
        if groups is not None:
            kg = np.ascontiguousarray(np.concatenate([np.asarray(g, np.int32) for g in groups] + [np.zeros(0, np.int32)]))
            ng = np.ascontiguousarray([len(g) for g in groups], dtype=np.int32)
            ku = np.ascontiguousarray(np.concatenate([np.asarray(u, np.int32) for u in units] + [np.zeros(0, np.int32)]))
            nu = np.ascontiguousarray([len(u) for u in units], dtype=np.int32)
            self.keep += [kg, ng, ku, nu]
            d.keep_groups = kg.ctypes.data_as(POINTER(c_int32))
            d.n_groups = ng.ctypes.data_as(POINTER(c_int32))
            d.keep_units = ku.ctypes.data_as(POINTER(c_int32))
            d.n_units = nu.ctypes.data_as(POINTER(c_int32))
        if qheads is not None:
            kq = np.ascontiguousarray(np.concatenate([np.asarray(h, np.int32) for h in qheads] + [np.zeros(0, np.int32)]))
            nq = np.ascontiguousarray([len(h) for h in qheads], dtype=np.int32)
            self.keep += [kq, nq]
            d.keep_qheads = kq.ctypes.data_as(POINTER(c_int32))
            d.n_qheads = nq.ctypes.data_as(POINTER(c_int32))
        self.desc = d


def greedy_mask(scores, target_u24, budget=0.57, r_lo=0.35, r_hi=0.85, panel_mode=PANELS_COMPACT):
    return _MaskArgs(MASK_GREEDY, panel_mode, budget, r_lo, r_hi, scores=scores, target_u24=target_u24)


def explicit_mask(groups, units, panel_mode=PANELS_COMPACT):
    return _MaskArgs(MASK_EXPLICIT, panel_mode, groups=groups, units=units)


def greedy_qhead_mask(scores, target_u24, budget=0.57, r_lo=0.35, r_hi=0.85, panel_mode=PANELS_COMPACT):
    """Greedy over query-head candidates; ``scores`` [L, Hq + df/chan_unit] (heads first)."""
    return _MaskArgs(MASK_GREEDY_QHEADS, panel_mode, budget, r_lo, r_hi, scores=scores, target_u24=target_u24)


def explicit_qhead_mask(qheads, units, panel_mode=PANELS_COMPACT):
    """Retained query heads and channel units per layer; the closure adds their KV heads."""
    m = _MaskArgs(MASK_EXPLICIT_QHEADS, panel_mode, qheads=qheads)
    ku = np.ascontiguousarray(np.concatenate([np.asarray(u, np.int32) for u in units] + [np.zeros(0, np.int32)]))
    nu = np.ascontiguousarray([len(u) for u in units], dtype=np.int32)
    m.keep += [ku, nu]
    m.desc.keep_units = ku.ctypes.data_as(POINTER(c_int32))
    m.desc.n_units = nu.ctypes.data_as(POINTER(c_int32))
    return m


def all_keep_mask():
    return _MaskArgs(MASK_ALL_KEEP)


def mask_select(shape, mask: _MaskArgs):
    """Host-only mask compilation: (groups per layer, channel units per layer, flops array)."""
    lib = load()
    L, G, U = shape.L, shape.Hkv, shape.df // shape.chan_unit
    kg = np.zeros(L * G, np.int32)
    ng = np.zeros(L, np.int32)
    ku = np.zeros(L * U, np.int32)
    nu = np.zeros(L, np.int32)
    fl = np.zeros(L + 3, np.int64)
    md = model_desc(shape)
    _check(lib.tasp_mask_select(ctypes.byref(md), ctypes.byref(mask.desc), kg.ctypes.data, ng.ctypes.data,
                                ku.ctypes.data, nu.ctypes.data, fl.ctypes.data))
    groups, units, og, ou = [], [], 0, 0
    for layer in range(L):
        groups.append(kg[og:og + ng[layer]].tolist())
        units.append(ku[ou:ou + nu[layer]].tolist())
        og += ng[layer]
        ou += nu[layer]
    return groups, units, fl


def mask_select_qheads(shape, mask: _MaskArgs):
    """Host-only mask compilation with the retained query heads:
    (query heads per layer, KV heads per layer, channel units per layer, flops array)."""
    lib = load()
    L, U = shape.L, shape.df // shape.chan_unit
    kq = np.zeros(L * shape.Hq, np.int32)
    nq = np.zeros(L, np.int32)
    kg = np.zeros(L * shape.Hkv, np.int32)
    ng = np.zeros(L, np.int32)
    ku = np.zeros(L * U, np.int32)
    nu = np.zeros(L, np.int32)
    fl = np.zeros(L + 3, np.int64)
    md = model_desc(shape)
    _check(lib.tasp_mask_select_qheads(ctypes.byref(md), ctypes.byref(mask.desc), kq.ctypes.data, nq.ctypes.data,
                                       kg.ctypes.data, ng.ctypes.data, ku.ctypes.data, nu.ctypes.data,
                                       fl.ctypes.data))
    out = []
    for flat, counts in ((kq, nq), (kg, ng), (ku, nu)):
        lists, o = [], 0
        for layer in range(L):
            lists.append(flat[o:o + counts[layer]].tolist())
            o += counts[layer]
        out.append(lists)
    return out[0], out[1], out[2], fl


def dispatch(probs, tau: float = 0.85) -> int:
    """Plan index for a turn: the most probable task's mask if its probability reaches tau, else
    len(probs), the dense plan."""
    p = np.ascontiguousarray(probs, dtype=np.float32)
    v = c_int32()
    _check(load().tasp_dispatch(p.ctypes.data, len(p), tau, ctypes.byref(v)))
    return v.value


def set_memory_limit(nbytes: int):
    """Cap the device memory of the library's arenas (0 = no cap)."""
    _check(load().tasp_set_memory_limit(int(nbytes)))


SPECTRAL_FEATURES = ("alpha", "r_eff", "spectral_norm", "setol", "lambda_min", "ks")


def spectral_layer(shape, layer: int, stream=None, phase_ms=None):
    """Spectral descriptors of every candidate unit of one layer on the device: (features
    [H_q + df / chan_unit][6] in SPECTRAL_FEATURES order, eigenvalues per block, descending).
    ``phase_ms`` (a float64 array of 4) receives the device time of the block generation,
    Gram matrices, eigensolver and statistics steps."""
    nh, nc = 4 * shape.dh, 3 * shape.chan_unit
    nu = shape.df // shape.chan_unit
    feat = np.zeros((shape.Hq + nu, len(SPECTRAL_FEATURES)), np.float64)
    lam = np.zeros(shape.Hq * nh + nu * nc, np.float64)
    md = model_desc(shape)
    ph = phase_ms.ctypes.data if phase_ms is not None else None
    _check(load().tasp_spectral_layer(ctypes.byref(md), layer, feat.ctypes.data, lam.ctypes.data, ph,
                                      _stream_ptr(stream)))
    blocks, o = [], 0
    for i in range(shape.Hq + nu):
        n = nh if i < shape.Hq else nc
        blocks.append(lam[o:o + n])
        o += n
    return feat, blocks


def test_set_wait_limit(cycles: int):
    """Failure-detection test hook: clock-cycle limit of the one-session GEMVs' bounded waits
    (0 = the default)."""
    _check(load().tasp_test_set_wait_limit(int(cycles)))


def test_skip_gemv_copies(launches: int):
    """Failure-detection test hook: the next `launches` one-session GEMV launches issue no
    weight copies (their first wait runs out)."""
    _check(load().tasp_test_skip_gemv_copies(int(launches)))


def memory_in_use() -> int:
    v = c_int64()
    _check(load().tasp_memory_in_use(ctypes.byref(v)))
    return v.value


def plan_layout(shape, mask: _MaskArgs, layer: int) -> dict:
    """Host-only: the qkv row sources, O column sources and partial-group tables of one layer."""
    lib = load()
    cnt = np.zeros(5, np.int32)
    md = model_desc(shape)
    _check(lib.tasp_plan_layout(ctypes.byref(md), ctypes.byref(mask.desc), layer, None, None, None, None, None,
                                cnt.ctypes.data))
    out = {k: np.zeros(int(n), dt) for k, n, dt in zip(("qkv_src", "o_src", "role", "slot", "blk_of"), cnt,
                                                      (np.int32, np.int32, np.int16, np.int16, np.int16))}
    _check(lib.tasp_plan_layout(ctypes.byref(md), ctypes.byref(mask.desc), layer, out["qkv_src"].ctypes.data,
                                out["o_src"].ctypes.data, out["role"].ctypes.data, out["slot"].ctypes.data,
                                out["blk_of"].ctypes.data, cnt.ctypes.data))
    return out


def _stream_ptr(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return int(stream)


class Plan:
    def __init__(self, shape, mask: _MaskArgs):
        lib = load()
        self.shape = shape
        self.handle = c_void_p()
        md = model_desc(shape)
        _check(lib.tasp_compile_mask(ctypes.byref(md), ctypes.byref(mask.desc), ctypes.byref(self.handle)))

    def info(self) -> dict:
        pi = PlanInfo()
        _check(load().tasp_plan_info_get(self.handle, ctypes.byref(pi)))
        return {name: getattr(pi, name) for name, _ in PlanInfo._fields_}

    def layer_dims(self, layer):
        out = np.zeros(2, np.int32)
        _check(load().tasp_plan_layer_dims(self.handle, layer, out.ctypes.data))
        return int(out[0]), int(out[1])

    def layer_qheads(self, layer) -> int:
        v = c_int32()
        _check(load().tasp_plan_layer_qheads(self.handle, layer, ctypes.byref(v)))
        return v.value

    def export(self, layer, item):
        sh = self.shape
        m_kv, c = self.layer_dims(layer)
        m_q = self.layer_qheads(layer)
        spec = {
            EXPORT_KEEP_GROUPS: (np.int32, (m_kv,)),
            EXPORT_KEEP_QHEADS: (np.int32, (m_q,)),
            EXPORT_QKV_G: (np.uint16, ((m_q + 2 * m_kv) * sh.dh, sh.d // max(1, getattr(sh, "quant_group", 0)))),
            EXPORT_O_G: (np.uint16, (sh.d, m_q * sh.dh // max(1, getattr(sh, "quant_group", 0)))),
            EXPORT_GU_G: (np.uint16, (2 * c, sh.d // max(1, getattr(sh, "quant_group", 0)))),
            EXPORT_DOWN_G: (np.uint16, (sh.d, c // max(1, getattr(sh, "quant_group", 0)))),
            EXPORT_KEEP_CHANS: (np.int32, (c,)),
            EXPORT_QKV_W: (np.int8, ((m_q + 2 * m_kv) * sh.dh, sh.d)),
            EXPORT_QKV_S: (np.float32, ((m_q + 2 * m_kv) * sh.dh,)),
            EXPORT_O_W: (np.int8, (sh.d, m_q * sh.dh)),
            EXPORT_O_S: (np.float32, (sh.d,)),
            EXPORT_GU_W: (np.int8, (2 * c, sh.d)),
            EXPORT_GU_S: (np.float32, (2 * c,)),
            EXPORT_DOWN_W: (np.int8, (sh.d, c)),
            EXPORT_DOWN_S: (np.float32, (sh.d,)),
        }[item]
        out = np.zeros(spec[1], dtype=spec[0])
        _check(load().tasp_plan_export(self.handle, layer, item, out.ctypes.data, out.nbytes))
        return out

    def release(self):
        if self.handle:
            _check(load().tasp_release(self.handle))
            self.handle = c_void_p()


class Session:
    def __init__(self, plan: Plan, max_tokens: int, handle=None):
        self.plan = plan
        self.handle = c_void_p() if handle is None else handle
        if handle is None:
            _check(load().tasp_session_create(plan.handle, max_tokens, ctypes.byref(self.handle)))

    def fill_synthetic(self, t_prior: int, kv_seed: int, stream=None):
        _check(load().tasp_session_fill_synthetic(self.handle, t_prior, kv_seed, _stream_ptr(stream)))

    @property
    def position(self) -> int:
        v = c_int32()
        _check(load().tasp_session_position(self.handle, ctypes.byref(v)))
        return v.value

    @classmethod
    def prefill(cls, plan: "Plan", embeds_bf16, max_new_tokens: int, logits=None, stream=None) -> "Session":
        """Prefill a prompt (CUDA bfloat16 tensor [T, d]) into a new session bound to `plan`."""
        _check_prompt(plan.shape, embeds_bf16, logits)
        h = c_void_p()
        _check(load().tasp_prefill(plan.handle, embeds_bf16.data_ptr(), int(embeds_bf16.shape[0]), max_new_tokens,
                                   _stream_ptr(stream), ctypes.byref(h),
                                   logits.data_ptr() if logits is not None else None))
        return cls(plan, 0, handle=h)

    def prefill_into(self, embeds_bf16, logits=None, stream=None):
        """Prefill a prompt into this (existing) session from position 0."""
        _check_prompt(self.plan.shape, embeds_bf16, logits)
        _check(load().tasp_session_prefill(self.handle, embeds_bf16.data_ptr(), int(embeds_bf16.shape[0]),
                                           _stream_ptr(stream), logits.data_ptr() if logits is not None else None))

    def kv(self, layer: int, which: int) -> np.ndarray:
        """Cached keys (which=0) or values (1) of a layer: BF16 bits [m_kv, position, dh]."""
        m_kv, _ = self.plan.layer_dims(layer)
        pos = self.position
        out = np.zeros((m_kv, pos, self.plan.shape.dh), np.uint16)
        _check(load().tasp_session_kv_export(self.handle, layer, which, out.ctypes.data, out.nbytes))
        return out

    def device_error(self, clear=True) -> int:
        """Device error word of this session's kernels (0 = none); synchronizes."""
        v = c_int32()
        _check(load().tasp_session_status(self.handle, int(clear), ctypes.byref(v)))
        return v.value

    def layer_step(self, layer, x_in, x_out, stream=None):
        import torch
        for t in (x_in, x_out):
            _need(t, self.plan.shape.d, torch.float32, True, "layer residual")
        _check(load().tasp_layer_step(self.handle, layer, x_in.data_ptr(), x_out.data_ptr(), _stream_ptr(stream)))

    def release(self):
        if self.handle:
            _check(load().tasp_release(self.handle))
            self.handle = c_void_p()


def _handles(sessions):
    arr = (c_void_p * len(sessions))(*[s.handle.value for s in sessions])
    return ctypes.cast(arr, POINTER(c_void_p)), arr


def _need(t, want, dt, device, what="buffer"):
    """Raise unless t holds at least `want` contiguous elements of dtype dt on the GPU (device=True)
    or the host; the library takes raw pointers and cannot check them itself."""
    if t.dtype != dt or not t.is_contiguous() or t.numel() < want or t.is_cuda != device:
        raise ValueError(f"{what} needs {want} contiguous {dt} elements on the {'GPU' if device else 'host'}")


def _check_buffers(sessions, x, hidden, logits, device):
    """Sizes, dtypes and placement of the caller buffers of an n-session step."""
    import torch
    if not sessions:
        raise ValueError("need at least one session")
    sh = sessions[0].plan.shape
    n = len(sessions)
    for t, want, dt in ((x, n * sh.d, torch.bfloat16), (hidden, n * sh.d, torch.float32),
                        (logits, n * sh.vocab, torch.float32)):
        if t is not None:
            _need(t, want, dt, device)


def _check_prompt(shape, embeds, logits):
    import torch
    if embeds.dim() != 2 or embeds.shape[1] != shape.d or embeds.shape[0] < 1:
        raise ValueError(f"prompt embeddings must be [T >= 1, {shape.d}]")
    _need(embeds, embeds.shape[0] * shape.d, torch.bfloat16, True, "prompt")
    if logits is not None:
        _need(logits, shape.vocab, torch.float32, True, "logits")


def decode_step(sessions, x_bf16, hidden=None, logits=None, stream=None):
    """One decode step; x_bf16 is a CUDA bfloat16 tensor [n, d]; hidden / logits float32 CUDA tensors or None.
    Sessions are grouped by up to 4 per weight pass."""
    _check_buffers(sessions, x_bf16, hidden, logits, True)
    p, keep = _handles(sessions)
    _check(load().tasp_decode_step(p, len(sessions), x_bf16.data_ptr(),
                                   hidden.data_ptr() if hidden is not None else None,
                                   logits.data_ptr() if logits is not None else None, _stream_ptr(stream)))


def decode_step_union(sessions, x_bf16, hidden=None, logits=None, stream=None):
    """Union-of-masks decode step: up to 16 sessions whose plans may differ (one shared store), every
    weight row read once for all of them; buffers as in decode_step."""
    _check_buffers(sessions, x_bf16, hidden, logits, True)
    p, keep = _handles(sessions)
    _check(load().tasp_decode_step_union(p, len(sessions), x_bf16.data_ptr(),
                                         hidden.data_ptr() if hidden is not None else None,
                                         logits.data_ptr() if logits is not None else None, _stream_ptr(stream)))


def union_status(sessions):
    """(device error word, graph launches) of the union workspace of these sessions."""
    p, keep = _handles(sessions)
    err, nl = c_int32(0), c_int32(0)
    _check(load().tasp_union_status(p, len(sessions), ctypes.byref(err), ctypes.byref(nl)))
    return err.value, nl.value


def decode_step_static(session, x_bf16, hidden=None, logits=None, stream=None):
    """Allocation-free decode step of one session (static attention scratch, no CUDA graph)."""
    _check_buffers([session], x_bf16, hidden, logits, True)
    _check(load().tasp_decode_step_static(session.handle, x_bf16.data_ptr(),
                                          hidden.data_ptr() if hidden is not None else None,
                                          logits.data_ptr() if logits is not None else None, _stream_ptr(stream)))


def decode_step_host(sessions, x_bf16_host, hidden_host=None, logits_host=None, stream=None):
    """Decode step with host buffers (torch CPU tensors, ideally pinned); synchronizes the stream."""
    _check_buffers(sessions, x_bf16_host, hidden_host, logits_host, False)
    p, keep = _handles(sessions)
    _check(load().tasp_decode_step_host(p, len(sessions), x_bf16_host.data_ptr(),
                                        hidden_host.data_ptr() if hidden_host is not None else None,
                                        logits_host.data_ptr() if logits_host is not None else None,
                                        _stream_ptr(stream)))


def profile_step(sessions, x_bf16, logits=None, stream=None):
    """Eager step with CUDA events around each kernel: {kind: (ms, launches)}."""
    _check_buffers(sessions, x_bf16, None, logits, True)
    p, keep = _handles(sessions)
    ms = np.zeros(KERNEL_KINDS, np.float32)
    cnt = np.zeros(KERNEL_KINDS, np.int32)
    _check(load().tasp_profile_step(p, len(sessions), x_bf16.data_ptr(),
                                    logits.data_ptr() if logits is not None else None, _stream_ptr(stream),
                                    ms.ctypes.data, cnt.ctypes.data))
    return {KERNEL_NAMES[k]: (float(ms[k]), int(cnt[k])) for k in range(KERNEL_KINDS)}


def step_launches(sessions, with_logits=True) -> int:
    p, keep = _handles(sessions)
    v = c_int32()
    _check(load().tasp_step_launches(p, len(sessions), int(with_logits), ctypes.byref(v)))
    return v.value


def version() -> str:
    return load().tasp_version().decode()
