"""ctypes binding of librc (include/rc.h): argument marshalling only.

Every computation runs in librc's CUDA kernels. The binding never falls back
to another implementation: if librc.so is missing it raises, and CUDA
failures surface as :class:`RcError` with the library's message.

PyTorch is used only for device memory and streams: tensors are passed by
``data_ptr()`` and the stream by ``torch.cuda.current_stream().cuda_stream``.
"""
from __future__ import annotations

import ctypes as C
import math
import os
from typing import Iterable, Sequence

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "librc.so")

# ------------------------------------------------------------------ enums --
OK, ERR_INVALID_ARG, ERR_UNSUPPORTED_OP, ERR_ILLEGAL_SCHEDULE, ERR_DUPLICATE, ERR_CUDA, \
    ERR_DEVICE_TIMEOUT, ERR_TIMEOUT, ERR_PARITY, ERR_OOM, ERR_EXHAUSTED = range(11)
STATUS_NAMES = {0: "OK", 1: "INVALID_ARG", 2: "UNSUPPORTED_OP", 3: "ILLEGAL_SCHEDULE", 4: "DUPLICATE",
                5: "CUDA", 6: "DEVICE_TIMEOUT", 7: "TIMEOUT", 8: "PARITY", 9: "OOM", 10: "EXHAUSTED"}

OP_GEMM_F32, OP_LINEAR, OP_SWIGLU, OP_MLP, OP_ATTENTION, OP_CONV2D, OP_MOE_ROUTE, OP_MOE, OP_DECODER_LAYER = range(9)
EPI_BIAS, EPI_RELU, EPI_SILU = 1, 2, 4
BOUND_NAMES = {0: "tensor", 1: "hbm", 2: "fp32_simt"}

T_TILE_SIZE, T_PARALLEL, T_COMPUTE_LOCATION, T_UNROLL, T_LOOP_ORDER, T_FUSE, T_LAYOUT, T_VECTORIZE, \
    T_PIPELINE_STAGES, T_SPLIT_K = range(10)
T_NAMES = ["TileSize", "Parallel", "ComputeLocation", "Unroll", "LoopOrder", "Fuse", "Layout", "Vectorize",
           "PipelineStages", "SplitK"]
MAX_TENSORS = 10
MAX_STAGES = 6


class OpDesc(C.Structure):
    _fields_ = [("kind", C.c_int32), ("flags", C.c_int32),
                ("m", C.c_int64), ("n", C.c_int64), ("k", C.c_int64),
                ("batch", C.c_int64), ("seq", C.c_int64), ("heads_q", C.c_int64), ("heads_kv", C.c_int64),
                ("head_dim", C.c_int64), ("causal", C.c_int32), ("scale", C.c_double),
                ("img_n", C.c_int64), ("img_h", C.c_int64), ("img_w", C.c_int64), ("c_in", C.c_int64),
                ("c_out", C.c_int64), ("kr", C.c_int64), ("ks", C.c_int64), ("stride", C.c_int64),
                ("pad", C.c_int64),
                ("tokens", C.c_int64), ("hidden", C.c_int64), ("experts", C.c_int64), ("inter", C.c_int64),
                ("top_k", C.c_int64), ("logits_fp32", C.c_int32), ("renorm", C.c_int32),
                ("rope_theta", C.c_double), ("norm_eps", C.c_double)]


class OpInfo(C.Structure):
    _fields_ = [("flops", C.c_double), ("bytes", C.c_double), ("bound", C.c_int32), ("n_tensors", C.c_int32),
                ("workspace_bytes", C.c_int64)]


class Transform(C.Structure):
    _fields_ = [("kind", C.c_int32), ("axis", C.c_int32), ("stage", C.c_int32), ("reserved", C.c_int32),
                ("value", C.c_int64 * 4)]

    def __repr__(self):
        v = f"{self.value[0]}" + (f"/{self.value[1]}" if self.kind == T_LOOP_ORDER else "")
        ax = f"[{'MNK'[self.axis]}]" if self.kind == T_TILE_SIZE else ""
        return f"{T_NAMES[self.kind]}{ax}@{self.stage}={v}"


class Knobs(C.Structure):
    _fields_ = [(n, C.c_int32) for n in ("tile_m", "tile_n", "tile_k", "unroll", "stages", "split_k", "raster",
                                         "group", "persistent", "fuse", "layout", "vec", "location")]

    def as_dict(self):
        return {n: getattr(self, n) for n, _ in self._fields_}


class Tensors(C.Structure):
    _fields_ = [("p", C.c_void_p * MAX_TENSORS)]


class MeasureOpts(C.Structure):
    _fields_ = [("warmup", C.c_int32), ("repeats", C.c_int32), ("flush_l2", C.c_int32), ("budget_s", C.c_double)]


class Measurement(C.Structure):
    _fields_ = [("status", C.c_int32), ("ms_median", C.c_double), ("ms_min", C.c_double), ("ms_mean", C.c_double),
                ("tflops", C.c_double), ("gbps", C.c_double), ("sched_hash", C.c_uint64), ("n_stages", C.c_int32),
                ("stage_ms", C.c_double * MAX_STAGES)]

    def as_dict(self):
        d = {n: getattr(self, n) for n, _ in self._fields_ if n != "stage_ms"}
        d["stage_ms"] = [self.stage_ms[i] for i in range(self.n_stages)]
        return d


class SearchOpts(C.Structure):
    _fields_ = [("seed", C.c_uint64), ("c", C.c_double), ("branching", C.c_int32), ("horizon", C.c_int32),
                ("rollout", C.c_int32), ("max_tries", C.c_int32), ("surrogate", C.c_int32), ("screen", C.c_int32),
                ("stage_mask", C.c_uint32), ("root", C.c_void_p)]


class SearchStats(C.Structure):
    _fields_ = [("nodes", C.c_int64), ("samples", C.c_int64), ("iterations", C.c_int64),
                ("best_reward", C.c_double), ("model_samples", C.c_int64), ("model_features", C.c_int64),
                ("predicted", C.c_int64)]


class RcError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"rc {STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


_lib = None

# name -> (restype, argtypes)
_P = C.c_void_p
_PROTOS = {
    "rc_op_describe": (C.c_int, [C.POINTER(OpDesc), C.POINTER(_P)]),
    "rc_op_info": (C.c_int, [_P, C.POINTER(OpInfo)]),
    "rc_op_destroy": (None, [_P]),
    "rc_schedule_apply": (C.c_int, [_P, _P, C.POINTER(Transform), C.c_size_t, C.POINTER(_P)]),
    "rc_schedule_knobs": (C.c_int, [_P, C.c_int32, C.POINTER(Knobs)]),
    "rc_schedule_num_stages": (C.c_int32, [_P]),
    "rc_schedule_hash": (C.c_uint64, [_P]),
    "rc_schedule_to_string": (C.c_int, [_P, C.c_char_p, C.c_size_t, C.POINTER(C.c_size_t)]),
    "rc_schedule_clone": (C.c_int, [_P, C.POINTER(_P)]),
    "rc_schedule_destroy": (None, [_P]),
    "rc_transform_space": (C.c_int, [_P, C.POINTER(Transform), C.c_size_t, C.POINTER(C.c_size_t)]),
    "rc_run": (C.c_int, [_P, _P, C.POINTER(Tensors), _P]),
    "rc_run_host": (C.c_int, [_P, _P, C.POINTER(Tensors), _P]),
    "rc_run_profiled": (C.c_int, [_P, _P, C.POINTER(Tensors), _P, C.POINTER(C.c_double), C.c_size_t,
                                  C.POINTER(C.c_size_t)]),
    "rc_op_check": (C.c_int, [_P, _P]),
    "rc_candidate_measure": (C.c_int, [_P, C.POINTER(_P), C.c_size_t, C.POINTER(Tensors), _P,
                                       C.POINTER(MeasureOpts), C.POINTER(Measurement)]),
    "rc_search_create": (C.c_int, [_P, C.POINTER(SearchOpts), C.POINTER(_P)]),
    "rc_search_step": (C.c_int, [_P, C.POINTER(Measurement), C.c_size_t, C.POINTER(_P), C.c_size_t,
                                 C.POINTER(C.c_size_t)]),
    "rc_search_best": (C.c_int, [_P, C.POINTER(_P), C.POINTER(Measurement)]),
    "rc_search_get_stats": (C.c_int, [_P, C.POINTER(SearchStats)]),
    "rc_search_predict": (C.c_int, [_P, _P, C.POINTER(C.c_double)]),
    "rc_search_node": (C.c_int, [_P, C.c_int64, C.POINTER(C.c_int64), C.POINTER(C.c_double),
                                 C.POINTER(C.c_int64), C.POINTER(C.c_uint64)]),
    "rc_search_destroy": (None, [_P]),
    "rc_moe_route_noalloc": (C.c_int, [_P, C.c_int32, C.c_int64, C.c_int64, C.c_int64, C.c_int32, _P, _P, _P, _P,
                                       _P]),
    "rc_selftest_bounded_wait": (C.c_int, [C.c_double, _P]),
    "rc_last_error": (C.c_char_p, []),
    "rc_version": (C.c_char_p, []),
}


def lib():
    """Load librc.so (raises if it has not been built: there is no fallback)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"librc.so is not built ({LIB_PATH}); run paper_2506_01374_gb300.build.build()")
        L = C.CDLL(LIB_PATH)
        for name, (res, args) in _PROTOS.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def _check(st: int, what: str = ""):
    if st != OK:
        msg = lib().rc_last_error().decode(errors="replace")
        raise RcError(st, f"{what}: {msg}" if what else msg)


def T(kind: int, value: int, axis: int = 0, stage: int = 0, group: int = 0) -> Transform:
    """Build one transformation (rc_transform)."""
    t = Transform()
    t.kind, t.axis, t.stage, t.reserved = kind, axis, stage, 0
    t.value[0] = value
    t.value[1] = group
    return t


def _ptr(x) -> int | None:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    if hasattr(x, "ctypes"):
        return x.ctypes.data
    raise TypeError(f"cannot take a pointer of {type(x)}")


def _tensors(ts: Sequence) -> Tensors:
    if len(ts) > MAX_TENSORS:
        raise ValueError("too many tensor slots")
    t = Tensors()
    for i, x in enumerate(ts):
        t.p[i] = _ptr(x)
    return t


def _stream(stream) -> int | None:
    if stream is None:
        try:
            import torch
            if torch.cuda.is_available():
                return torch.cuda.current_stream().cuda_stream
        except ImportError:
            pass
        return None
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


class Schedule:
    """An owned or borrowed rc_schedule handle."""

    def __init__(self, handle: int, owned: bool = True):
        self.h = handle
        self.owned = owned

    def __del__(self):
        if getattr(self, "owned", False) and self.h and _lib is not None:
            _lib.rc_schedule_destroy(self.h)
            self.h = None

    @property
    def num_stages(self) -> int:
        return lib().rc_schedule_num_stages(self.h)

    def knobs(self, stage: int = 0) -> dict:
        k = Knobs()
        _check(lib().rc_schedule_knobs(self.h, stage, C.byref(k)), "rc_schedule_knobs")
        return k.as_dict()

    @property
    def hash(self) -> int:
        return lib().rc_schedule_hash(self.h)

    def clone(self) -> "Schedule":
        """An owned copy (outlives the search or op call that produced this handle)."""
        c = _P()
        _check(lib().rc_schedule_clone(self.h, C.byref(c)), "rc_schedule_clone")
        return Schedule(c.value)

    def __str__(self):
        need = C.c_size_t(0)
        _check(lib().rc_schedule_to_string(self.h, None, 0, C.byref(need)))
        buf = C.create_string_buffer(need.value)
        _check(lib().rc_schedule_to_string(self.h, buf, need.value, C.byref(need)))
        return buf.value.decode()

    __repr__ = __str__


class Op:
    """An operator (program P0) described through rc_op_describe."""

    def __init__(self, kind: int, **fields):
        d = OpDesc()
        d.kind = kind
        d.renorm = 1
        for k, v in fields.items():
            setattr(d, k, v)
        h = _P()
        _check(lib().rc_op_describe(C.byref(d), C.byref(h)), "rc_op_describe")
        self.h = h.value
        self.desc = d

    def __del__(self):
        if getattr(self, "h", None) and _lib is not None:
            _lib.rc_op_destroy(self.h)
            self.h = None

    @property
    def info(self) -> dict:
        i = OpInfo()
        _check(lib().rc_op_info(self.h, C.byref(i)))
        return {"flops": i.flops, "bytes": i.bytes, "bound": BOUND_NAMES[i.bound], "n_tensors": i.n_tensors,
                "workspace_bytes": i.workspace_bytes}

    def schedule(self, *transforms: Transform, base: Schedule | None = None) -> Schedule:
        arr = (Transform * max(1, len(transforms)))(*transforms)
        h = _P()
        _check(lib().rc_schedule_apply(self.h, base.h if base else None, arr, len(transforms), C.byref(h)),
               "rc_schedule_apply")
        return Schedule(h.value)

    def transform_space(self) -> list:
        n = C.c_size_t(0)
        _check(lib().rc_transform_space(self.h, None, 0, C.byref(n)))
        arr = (Transform * max(1, n.value))()
        _check(lib().rc_transform_space(self.h, arr, n.value, C.byref(n)))
        return list(arr[: n.value])

    def run(self, sched: Schedule, tensors: Sequence, stream=None):
        t = _tensors(tensors)
        _check(lib().rc_run(self.h, sched.h, C.byref(t), _stream(stream)), "rc_run")

    def run_profiled(self, sched: Schedule, tensors: Sequence, stream=None) -> list:
        """Run once with events between stages; returns per-stage device ms (synchronises)."""
        t = _tensors(tensors)
        out = (C.c_double * MAX_STAGES)()
        n = C.c_size_t(0)
        _check(lib().rc_run_profiled(self.h, sched.h, C.byref(t), _stream(stream), out, MAX_STAGES, C.byref(n)),
               "rc_run_profiled")
        return [out[i] for i in range(n.value)]

    def run_host(self, sched: Schedule, arrays: Sequence, stream=None):
        t = _tensors(arrays)
        _check(lib().rc_run_host(self.h, sched.h, C.byref(t), _stream(stream)), "rc_run_host")

    def check(self, stream=None):
        _check(lib().rc_op_check(self.h, _stream(stream)), "rc_op_check")

    def measure(self, scheds: Iterable[Schedule], tensors: Sequence, stream=None, warmup: int = 5,
                repeats: int = 20, flush_l2: bool = True, budget_s: float = 0.0) -> list:
        scheds = list(scheds)
        hs = (_P * max(1, len(scheds)))(*[s.h for s in scheds])
        out = (Measurement * max(1, len(scheds)))()
        o = MeasureOpts(warmup, repeats, int(flush_l2), budget_s)
        t = _tensors(tensors)
        st = lib().rc_candidate_measure(self.h, hs, len(scheds), C.byref(t), _stream(stream), C.byref(o), out)
        if st not in (OK, ERR_TIMEOUT):
            _check(st, "rc_candidate_measure")
        return [out[i] for i in range(len(scheds))]


class Search:
    """LLM-free MCTS over an op's schedule space (rc_search_*)."""

    def __init__(self, op: Op, seed: int = 0, c: float = math.sqrt(2.0), branching: int = 2, horizon: int = 8,
                 rollout: int = 2, max_tries: int = 64, surrogate: bool = False, screen: int = 1,
                 stages: Sequence[int] | None = None, root: Schedule | None = None):
        """stages: tune only these stages of a composite op (objective = their summed time);
        root: start from this schedule instead of P0 (rewards are speedups over it)."""
        self.op = op
        mask = 0 if not stages else sum(1 << int(g) for g in set(stages))
        o = SearchOpts(seed, c, branching, horizon, rollout, max_tries, int(surrogate), screen, mask,
                       root.h if root is not None else None)
        h = _P()
        _check(lib().rc_search_create(op.h, C.byref(o), C.byref(h)), "rc_search_create")
        self.h = h.value
        self._cap = 64

    def __del__(self):
        if getattr(self, "h", None) and _lib is not None:
            _lib.rc_search_destroy(self.h)
            self.h = None

    def step(self, results: Sequence[Measurement] = ()) -> list:
        """Feed the previous batch's measurements; get the next batch ([] when exhausted)."""
        res = (Measurement * max(1, len(results)))(*results)
        nxt = (_P * self._cap)()
        n = C.c_size_t(0)
        st = lib().rc_search_step(self.h, res, len(results), nxt, self._cap, C.byref(n))
        if st == ERR_EXHAUSTED:
            return []
        _check(st, "rc_search_step")
        return [Schedule(nxt[i], owned=False) for i in range(n.value)]

    def best(self):
        """Best measured schedule (an owned copy, valid after the search is gone) and its measurement."""
        h = _P()
        m = Measurement()
        _check(lib().rc_search_best(self.h, C.byref(h), C.byref(m)), "rc_search_best")
        c = _P()
        _check(lib().rc_schedule_clone(h.value, C.byref(c)), "rc_schedule_clone")
        return Schedule(c.value), m

    def stats(self) -> dict:
        s = SearchStats()
        _check(lib().rc_search_get_stats(self.h, C.byref(s)))
        return {n: getattr(s, n) for n, _ in SearchStats._fields_}

    def predict(self, sched: Schedule) -> float:
        """The learned surrogate's predicted device time (ms) of sched (rc_search_predict)."""
        ms = C.c_double()
        _check(lib().rc_search_predict(self.h, sched.h, C.byref(ms)), "rc_search_predict")
        return ms.value

    def node(self, i: int) -> dict:
        p, q, n, h = C.c_int64(), C.c_double(), C.c_int64(), C.c_uint64()
        _check(lib().rc_search_node(self.h, i, C.byref(p), C.byref(q), C.byref(n), C.byref(h)))
        return {"parent": p.value, "Q": q.value, "N": n.value, "hash": h.value}


def moe_route_noalloc(logits, tokens: int, experts: int, top_k: int, ids, weights, offsets, perm,
                      renorm: bool = True, logits_fp32: bool = False, stream=None):
    """rc_moe_route_noalloc: routing without any device allocation (fixed library scratch)."""
    _check(lib().rc_moe_route_noalloc(_ptr(logits), int(logits_fp32), tokens, experts, top_k, int(renorm), _ptr(ids),
                                      _ptr(weights), _ptr(offsets), _ptr(perm), _stream(stream)),
           "rc_moe_route_noalloc")


def selftest_bounded_wait(wait_ms: float = 50.0, stream=None) -> int:
    """Run the bounded-wait self-test; returns its status (ERR_DEVICE_TIMEOUT means it worked)."""
    return lib().rc_selftest_bounded_wait(wait_ms, _stream(stream))


def version() -> str:
    return lib().rc_version().decode()
