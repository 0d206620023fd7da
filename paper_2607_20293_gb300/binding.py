"""ctypes binding of the C ABI in include/evo.h (argument marshalling only).

Every computation happens in libevo.so.  torch is used for device memory and
streams: device arguments are torch CUDA tensors (their data pointers are
passed through), host lattices are numpy uint8 arrays.  load() raises if the
library has not been built; there is no other implementation to fall back to.
"""
from __future__ import annotations

import ctypes
import os
import weakref

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libevo.so")
LIB_PATH_DEBUG = os.path.join(HERE, "libevo_debug.so")

OK, ERR_ARG, ERR_SHAPE, ERR_SCHEDULE, ERR_CUDA, ERR_TIMEOUT, ERR_OOM, ERR_UNSUPPORTED, ERR_CORRUPT = range(9)
SAMPLERS = {"ddpm": 0, "ddim": 1}
DTYPES = {"fp32": 0, "bf16": 1}
EMPTY = {"zero": 0, "force": 1}

_FIELDS = ["n_layer", "n_emb", "n_head", "horizon", "action_dim", "n_obs", "obs_dim", "n_steps",
           "train_steps", "sampler", "dtype", "empty_cache", "cluster", "job_samples", "debug_sync", "wide_rows"]


class EvoConfig(ctypes.Structure):
    _fields_ = [(f, ctypes.c_int32) for f in _FIELDS]


class SearchConfig(ctypes.Structure):
    _fields_ = [("n_units", ctypes.c_int32), ("n_steps", ctypes.c_int32), ("budget", ctypes.c_int32),
                ("block_wise", ctypes.c_int32), ("population", ctypes.c_int32), ("elites", ctypes.c_int32),
                ("generations", ctypes.c_int32), ("tournament", ctypes.c_int32), ("guided", ctypes.c_int32),
                ("gamma", ctypes.c_int32), ("eps", ctypes.c_float), ("pad_", ctypes.c_float),
                ("crossover_rate", ctypes.c_double), ("mutation_rate", ctypes.c_double),
                ("early_stop", ctypes.c_int32), ("pad2_", ctypes.c_int32), ("q_base", ctypes.c_double),
                ("delta_acc", ctypes.c_double), ("seed", ctypes.c_uint64)]


class SearchResult(ctypes.Structure):
    _fields_ = [("best_fitness", ctypes.c_double), ("generations", ctypes.c_int32), ("evaluations", ctypes.c_int32),
                ("formal_evaluations", ctypes.c_int32), ("memo_hits", ctypes.c_int32),
                ("stopped_early", ctypes.c_int32), ("pad_", ctypes.c_int32)]


FITNESS_FN = ctypes.CFUNCTYPE(ctypes.c_int32, ctypes.c_void_p, ctypes.POINTER(ctypes.c_uint8), ctypes.c_int32,
                              ctypes.c_int32, ctypes.c_int32, ctypes.POINTER(ctypes.c_double))


class EvoError(RuntimeError):
    def __init__(self, code: int, what: str):
        self.code = code
        detail = ""
        if code == ERR_CUDA and _lib is not None:
            detail = f", CUDA error {_lib.evo_last_cuda_error()}"
        super().__init__(f"{what}: {status_string(code)} ({code}{detail})")


_lib = None
_lib_debug = None
# handles alive in this process (their guard bands can be checked after a test)
_live: "weakref.WeakSet[Evo]" = weakref.WeakSet()
# guard failures found when a handle was closed
guard_failures: list[str] = []


def load(debug: bool = False) -> ctypes.CDLL:
    """The library (debug=True: the build with device-side index checks)."""
    global _lib, _lib_debug
    if (_lib_debug if debug else _lib) is not None:
        return _lib_debug if debug else _lib
    path = LIB_PATH_DEBUG if debug else LIB_PATH
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with paper_2607_20293_gb300.build.build("
                           f"{'debug=True' if debug else ''})")
    lib = ctypes.CDLL(path)
    P, I32, I64, SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t
    cfgp = ctypes.POINTER(EvoConfig)
    sig = {
        "evo_weight_count": (SZ, [cfgp]),
        "evo_create": (I32, [P, SZ, cfgp, I32, ctypes.POINTER(P)]),
        "evo_destroy": (I32, [P]),
        "evo_denoise": (I32, [P, P, P, P, I32, I32, P, P]),
        "evo_denoise_trace": (I32, [P, P, P, P, I32, I32, P, P, P]),
        "evo_denoise_noalloc": (I32, [P, P, P, P, I32, I32, P, P]),
        "evo_test_wait_timeout": (I32, [P, I32, ctypes.c_int64, P]),
        "evo_check_guards": (I32, [P]),
        "evo_test_gelu": (I32, [P, P, ctypes.c_int64, I32, P]),
        "evo_denoise_population": (I32, [P, P, P, P, I32, I32, I32, P, P, P]),
        "evo_flops": (I32, [P, P, I32, ctypes.POINTER(I64)]),
        "evo_flops_cfg": (I32, [cfgp, P, I32, ctypes.POINTER(I64)]),
        "evo_schedule_from_positions": (I32, [P, I32, I32, I32, P]),
        "evo_schedule_fixed_interval": (I32, [I32, I32, I32, P]),
        "evo_get_status": (I32, [P]),
        "evo_set_profile_events": (I32, [P, P, P]),
        "evo_get_launch_info": (I32, [P, ctypes.POINTER(I32), ctypes.POINTER(I32), ctypes.POINTER(I32),
                                      ctypes.POINTER(I32)]),
        "evo_get_last_call": (I32, [P, ctypes.POINTER(I32), ctypes.POINTER(I64)]),
        "evo_last_cuda_error": (I32, []),
        "evo_search": (I32, [ctypes.POINTER(SearchConfig), P, FITNESS_FN, FITNESS_FN, P, P, ctypes.POINTER(SearchResult)]),
        "evo_redundancy_scratch_bytes": (SZ, [I32, I32, I32, I32, I32]),
        "evo_redundancy_map": (I32, [P, I32, I32, I32, I32, I32, P, P, P]),
        "evo_guided_schedules": (I32, [P, I32, I32, I32, ctypes.c_float, I32, P, I32, P, P]),
        "evo_status_string": (ctypes.c_char_p, [I32]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    if debug:
        _lib_debug = lib
    else:
        _lib = lib
    return lib


def status_string(code: int) -> str:
    return load().evo_status_string(code).decode()


def _check(code: int, what: str):
    if code != OK:
        raise EvoError(code, what)


def make_config(cfg: dict, cluster: int = 0, job_samples: int = 0, empty: str = "zero",
                debug_sync: bool = False, wide_rows: int = 0) -> EvoConfig:
    return EvoConfig(cfg["n_layer"], cfg["n_emb"], cfg["n_head"], cfg["horizon"], cfg["action_dim"],
                     cfg["n_obs"], cfg["obs_dim"], cfg["n_steps"], cfg["train_steps"],
                     SAMPLERS[cfg["sampler"]], DTYPES[cfg["dtype"]], EMPTY[empty], cluster, job_samples,
                     int(debug_sync), wide_rows)


def weight_names(cfg: dict) -> list[str]:
    names = ["obs_w", "obs_b", "cond_pos", "cm_w1", "cm_b1", "cm_w2", "cm_b2", "in_w", "in_b", "pos"]
    per = ["ln1_g", "ln1_b", "sa_wqkv", "sa_bqkv", "sa_wo", "sa_bo", "ln2_g", "ln2_b", "ca_wq", "ca_bq",
           "ca_wkv", "ca_bkv", "ca_wo", "ca_bo", "ln3_g", "ln3_b", "ff_w1", "ff_b1", "ff_w2", "ff_b2"]
    for l in range(cfg["n_layer"]):
        names += [f"l{l}.{n}" for n in per]
    return names + ["lnf_g", "lnf_b", "head_w", "head_b"]


def pack_blob(cfg: dict, weights: dict) -> np.ndarray:
    """Concatenate named float32 tensors in the blob order of evo_weight_count."""
    blob = np.concatenate([np.ascontiguousarray(weights[n], dtype=np.float32).ravel() for n in weight_names(cfg)])
    want = load().evo_weight_count(ctypes.byref(make_config(cfg)))
    if blob.size != want:
        raise ValueError(f"weight blob has {blob.size} floats, the library expects {want}")
    return blob


def _ptr(x) -> int | None:
    if x is None:
        return None
    if isinstance(x, np.ndarray):
        if not x.flags["C_CONTIGUOUS"]:
            raise ValueError("arrays passed to the C ABI must be C-contiguous")
        return x.ctypes.data
    if not x.is_contiguous():
        raise ValueError("tensors passed to the C ABI must be contiguous")
    return x.data_ptr()


def _lattice(S):
    """numpy lattices are passed as host memory (C-contiguous uint8); torch uint8
    tensors on the GPU as device memory."""
    if isinstance(S, np.ndarray):
        S = np.ascontiguousarray(S, dtype=np.uint8)
    return S


def _stream(stream) -> int | None:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return stream if isinstance(stream, int) else stream.cuda_stream


def flops_cfg(cfg: dict, S, empty: str = "zero") -> int:
    S = np.ascontiguousarray(S, dtype=np.uint8)
    out = ctypes.c_int64()
    c = make_config(cfg, empty=empty)
    _check(load().evo_flops_cfg(ctypes.byref(c), S.ctypes.data, S.shape[0], ctypes.byref(out)), "evo_flops")
    return out.value


def schedule_from_positions(positions, n_units: int, T: int) -> np.ndarray:
    bt = np.ascontiguousarray(np.asarray(positions, dtype=np.int16).reshape(-1, 2))
    out = np.zeros((n_units, T), dtype=np.uint8)
    _check(load().evo_schedule_from_positions(bt.ctypes.data if bt.size else None, bt.shape[0], n_units, T,
                                              out.ctypes.data), "evo_schedule_from_positions")
    return out


def schedule_fixed_interval(n_units: int, T: int, M: int) -> np.ndarray:
    """Fixed-interval baseline lattice [n_units][T]: every unit at t = floor(i T / M), i < M."""
    out = np.zeros((n_units, T), dtype=np.uint8)
    _check(load().evo_schedule_fixed_interval(n_units, T, M, out.ctypes.data), "evo_schedule_fixed_interval")
    return out


class Evo:
    """One evo_handle: packed weights, caches and workspace on the current GPU."""

    def __init__(self, cfg: dict, weights: dict, max_batch: int, cluster: int = 0, job_samples: int = 0,
                 empty: str = "zero", debug_sync: bool = False, wide_rows: int = 0, debug_lib: bool = False):
        lib = self._lib = load(debug_lib)
        self.cfg = dict(cfg)
        self._c = make_config(cfg, cluster, job_samples, empty, debug_sync, wide_rows)
        self._blob = pack_blob(cfg, weights)
        h = ctypes.c_void_p()
        _check(lib.evo_create(self._blob.ctypes.data, self._blob.size, ctypes.byref(self._c), max_batch,
                              ctypes.byref(h)), "evo_create")
        self._h = h
        self.max_batch = max_batch
        _live.add(self)

    def close(self):
        if getattr(self, "_h", None) and self._h.value:
            rc = self._lib.evo_check_guards(self._h)
            if rc != OK:
                guard_failures.append(f"handle {self.cfg.get('n_emb')}x{self.cfg.get('n_layer')}: "
                                      f"{status_string(rc)}")
            self._lib.evo_destroy(self._h)
            self._h = ctypes.c_void_p()
            _live.discard(self)

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def launch_info(self) -> dict:
        v = [ctypes.c_int32() for _ in range(4)]
        _check(self._lib.evo_get_launch_info(self._h, *[ctypes.byref(x) for x in v]), "evo_get_launch_info")
        return dict(cluster=v[0].value, job_samples=v[1].value, max_clusters=v[2].value, smem_bytes=v[3].value)

    def last_call(self) -> dict:
        """path of the last call ("cluster" or "wide") and the kernels it launched"""
        path, k = ctypes.c_int32(), ctypes.c_int64()
        _check(self._lib.evo_get_last_call(self._h, ctypes.byref(path), ctypes.byref(k)), "evo_get_last_call")
        return dict(path="wide" if path.value == 1 else "cluster", kernels=k.value)

    def denoise(self, obs, noise, S, out=None, stream=None, trace=None):
        import torch
        N = obs.shape[0]
        if out is None:
            out = torch.empty((N, self.cfg["horizon"], self.cfg["action_dim"]), dtype=torch.float32,
                              device=obs.device)
        S = _lattice(S)
        if trace is None:
            rc = self._lib.evo_denoise(self._h, _ptr(obs), _ptr(noise), _ptr(S), S.shape[0], N, _ptr(out),
                                    _stream(stream))
        else:
            rc = self._lib.evo_denoise_trace(self._h, _ptr(obs), _ptr(noise), _ptr(S), S.shape[0], N, _ptr(out),
                                          _ptr(trace), _stream(stream))
        _check(rc, "evo_denoise")
        return out

    def denoise_noalloc(self, obs, noise, S, out, stream=None):
        """evo_denoise with its per-call scratch in the library's static device
        array (no device allocation); `out` must be provided."""
        S = _lattice(S)
        rc = self._lib.evo_denoise_noalloc(self._h, _ptr(obs), _ptr(noise), _ptr(S), S.shape[0], obs.shape[0],
                                        _ptr(out), _stream(stream))
        _check(rc, "evo_denoise_noalloc")
        return out

    def population(self, obs, noise, S_pop, out=None, dev=None, stream=None, want_actions=True):
        import torch
        N_obs = obs.shape[0]
        S_pop = _lattice(S_pop)
        P = S_pop.shape[0]
        if out is None and want_actions:
            out = torch.empty((P, N_obs, self.cfg["horizon"], self.cfg["action_dim"]), dtype=torch.float32,
                              device=obs.device)
        if dev is None:
            dev = torch.empty((P,), dtype=torch.float32, device=obs.device)
        rc = self._lib.evo_denoise_population(self._h, _ptr(obs), _ptr(noise), _ptr(S_pop), P, S_pop.shape[1], N_obs,
                                           _ptr(out), _ptr(dev), _stream(stream))
        _check(rc, "evo_denoise_population")
        return out, dev

    def flops(self, S) -> int:
        S = np.ascontiguousarray(S, dtype=np.uint8)
        out = ctypes.c_int64()
        _check(self._lib.evo_flops(self._h, S.ctypes.data, S.shape[0], ctypes.byref(out)), "evo_flops")
        return out.value

    def set_profile_events(self, start=None, stop=None):
        """Bracket every denoising-loop kernel launch with these torch.cuda.Events
        (they must have been recorded once, so that their CUDA events exist)."""
        sp = start.cuda_event if start is not None else None
        ep = stop.cuda_event if stop is not None else None
        _check(self._lib.evo_set_profile_events(self._h, sp, ep), "evo_set_profile_events")

    def status(self) -> int:
        return self._lib.evo_get_status(self._h)

    def check_guards(self) -> int:
        """evo_check_guards: OK, or ERR_CORRUPT if a kernel wrote past an activation buffer."""
        return self._lib.evo_check_guards(self._h)

    def test_wait_timeout(self, helper: int, limit: int, stream=None):
        """Run the bounded-wait helper of the loop kernel (0) or the tensor-core
        kernels (1) on a barrier nothing arrives at, so that it gives up."""
        _check(self._lib.evo_test_wait_timeout(self._h, helper, limit, _stream(stream)), "evo_test_wait_timeout")


METRICS = {"cosine": 0, "mse": 1, "l1": 2, "w1": 3}


def redundancy_map(trace, metric: str = "cosine", stream=None):
    """Eq. 6 map d [U][T] from a device trace [T][U][N][H][E] (evo_denoise_trace
    with the all-refresh lattice)."""
    import torch
    T, U, N = trace.shape[:3]
    n = int(np.prod(trace.shape[3:]))
    m = METRICS[metric]
    lib = load()
    nb = lib.evo_redundancy_scratch_bytes(T, U, N, n, m)
    if nb == 0:
        raise EvoError(ERR_SHAPE, "evo_redundancy_scratch_bytes")
    scratch = torch.empty(nb, dtype=torch.uint8, device=trace.device)
    d = torch.empty((U, T), dtype=torch.float32, device=trace.device)
    _check(lib.evo_redundancy_map(_ptr(trace), T, U, N, n, m, _ptr(d), _ptr(scratch), _stream(stream)),
           "evo_redundancy_map")
    return d


def test_gelu(x, packed: bool = False, stream=None):
    """evo_test_gelu: the feed-forward units' device GELU (scalar form, or the
    packed pair form of the GEMM epilogue) applied to a contiguous fp32 CUDA
    tensor (a new tensor of the same shape)."""
    import torch
    y = torch.empty_like(x)
    _check(load().evo_test_gelu(_ptr(x), _ptr(y), x.numel(), int(packed), _stream(stream)), "evo_test_gelu")
    return y


def guided_schedules(d, K: int, rnd, eps: float = 0.05, gamma: int = 2, stream=None):
    """P lattices [P][U][T] of K cells each by Eq. 7 from the device map d [U][T];
    rnd: device uint64 tensor [P][K] (torch has no uint64: pass int64 with the same bits)."""
    import torch
    U, T = d.shape
    P = rnd.shape[0]
    S = torch.empty((P, U, T), dtype=torch.uint8, device=d.device)
    _check(load().evo_guided_schedules(_ptr(d), U, T, K, float(eps), int(gamma), _ptr(rnd), P, _ptr(S),
                                       _stream(stream)), "evo_guided_schedules")
    return S


def search(n_units: int, n_steps: int, budget: int, quick, formal=None, d_map=None, block_wise: bool = False,
           population: int = 30, elites: int = 10, generations: int = 30, tournament: int = 3, guided: int = 0,
           crossover_rate: float = 0.9, mutation_rate: float = 0.02, eps: float = 0.05, gamma: int = 2,
           early_stop: bool = False, q_base: float = 0.0, delta_acc: float = 0.0, seed: int = 0):
    """evo_search with Python fitness callables: f(S [P][n_units][T] uint8) -> [P] floats.
    Returns (best lattice, best fitness, stats dict)."""
    cfg = SearchConfig(n_units, n_steps, budget, int(block_wise), population, elites, generations, tournament,
                       guided, gamma, eps, 0.0, crossover_rate, mutation_rate, int(early_stop), 0, q_base,
                       delta_acc, seed & ((1 << 64) - 1))
    errors = []

    def wrap(f):
        if f is None:
            return ctypes.cast(None, FITNESS_FN)

        def cb(user, S, P, U, T, out):
            try:
                arr = np.ctypeslib.as_array(S, shape=(P, U, T)).copy()
                vals = f(arr)
                for i in range(P):
                    out[i] = float(vals[i])
                return 0
            except Exception as e:          # reported after the call returns
                errors.append(e)
                return 1
        return FITNESS_FN(cb)

    qf, ff = wrap(quick), wrap(formal)
    dm = None if d_map is None else np.ascontiguousarray(d_map, dtype=np.float32)
    best = np.zeros((n_units, n_steps), dtype=np.uint8)
    res = SearchResult()
    rc = load().evo_search(ctypes.byref(cfg), None if dm is None else dm.ctypes.data, qf, ff, None,
                           best.ctypes.data, ctypes.byref(res))
    if errors:
        raise errors[0]
    _check(rc, "evo_search")
    stats = dict(generations=res.generations, evaluations=res.evaluations,
                 formal_evaluations=res.formal_evaluations, memo_hits=res.memo_hits,
                 stopped_early=res.stopped_early)
    return best, res.best_fitness, stats
