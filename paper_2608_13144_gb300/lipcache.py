"""Python binding of the certified cache lookup (argument marshalling only).

Every step of the lookup runs in the CUDA kernels of liblipcache.so, called
through the C ABI of include/lipcache.h. PyTorch provides device memory and
the current stream; tensors are passed by pointer.
"""
from __future__ import annotations

import ctypes as C

import numpy as np
import torch

from . import _lib
from ._lib import Info, check

RADIUS_MODES = {"conservative": _lib.RADIUS_CONSERVATIVE, "tight": _lib.RADIUS_TIGHT}
PROBE_PATHS = {"auto": _lib.PROBE_AUTO, "tensor": _lib.PROBE_TENSOR, "exact": _lib.PROBE_EXACT,
               "tensor_single": _lib.PROBE_TENSOR_SINGLE, "tensor_pair": _lib.PROBE_TENSOR_PAIR}
RADIUS_POLICIES = {"certified": 0, "global": 1, "interclass": 2}
SELECT_STRATEGIES = {"all": 0, "radius_dedup": 1, "kcenter": 2}


def _stream(device: torch.device):
    return C.c_void_p(torch.cuda.current_stream(device).cuda_stream)


def _ptr(t):
    return C.c_void_p(t.data_ptr()) if t is not None else None


class LipCache:
    """Feature cache C = {(z_i, y~_i, r_i)} on one GPU (Sec. 3.3-3.4)."""

    def __init__(self, d: int, C_classes: int, capacity: int, radius_mode: str = "conservative",
                 device: int | torch.device | None = None):
        self.L = _lib.load()
        self.device = torch.device("cuda", torch.cuda.current_device() if device is None else
                                   torch.device("cuda", device).index if isinstance(device, int) else device.index)
        self.d, self.C = int(d), int(C_classes)
        h = C.c_void_p()
        with torch.cuda.device(self.device):
            check(self.L.lipcache_create(self.d, self.C, int(capacity), RADIUS_MODES[radius_mode], C.byref(h)))
        self._h = h

    # -- lifecycle
    def close(self):
        if getattr(self, "_h", None):
            self.L.lipcache_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    def _dev(self, t: torch.Tensor, dtype: torch.dtype, name: str) -> torch.Tensor:
        if t.device != self.device or t.dtype != dtype:
            raise ValueError(f"{name} must be a {dtype} tensor on {self.device}")
        return t.contiguous()

    # -- Algorithm 1
    def set_head(self, W: torch.Tensor, b: torch.Tensor) -> float:
        W = self._dev(W, torch.float32, "W")
        b = self._dev(b, torch.float32, "b")
        if tuple(W.shape) != (self.C, self.d) or tuple(b.shape) != (self.C,):
            raise ValueError("W must be C x d and b must have C entries")
        sigma = C.c_double()
        check(self.L.lipcache_set_head(self._h, _ptr(W), _ptr(b), C.byref(sigma), _stream(self.device)))
        return sigma.value

    def insert(self, H: torch.Tensor, payload: torch.Tensor | None = None, require_consistency: bool = False,
               wait: bool = True):
        """Certify and append rows of H. Returns (index, radius, n_accepted):
        index[i] is the cache index of row i or -1 if it was skipped. With
        wait=False the call does not synchronise (n_accepted is None; index
        and radius are filled in stream order; `size` settles later)."""
        H = self._dev(H, torch.float32, "H")
        n = H.shape[0]
        if H.dim() != 2 or (n and H.shape[1] != self.d):
            raise ValueError("H must be n x d")
        if payload is not None:
            payload = self._dev(payload, torch.int32, "payload")
        index = torch.empty(n, dtype=torch.int64, device=self.device)
        radius = torch.empty(n, dtype=torch.float32, device=self.device)
        acc = C.c_int64()
        check(self.L.lipcache_insert(self._h, _ptr(H), n, _ptr(payload), int(bool(require_consistency)),
                                     _ptr(index), _ptr(radius), C.byref(acc) if wait else None,
                                     _stream(self.device)))
        return index, radius, (acc.value if wait else None)

    def insert_select(self, H: torch.Tensor, payload: torch.Tensor | None = None, require_consistency: bool = False,
                      strategy: str = "radius_dedup", budget_total: int = 0, budget_per_class: int = 0):
        """Algorithm 1 with a selection strategy S ("radius_dedup": radius-
        prioritised de-duplication; "kcenter": K-center per class; "all":
        insert). Returns (index, radius, n_selected); index[i] is the cache
        index of row i or -1."""
        H = self._dev(H, torch.float32, "H")
        n = H.shape[0]
        if H.dim() != 2 or (n and H.shape[1] != self.d):
            raise ValueError("H must be n x d")
        if payload is not None:
            payload = self._dev(payload, torch.int32, "payload")
        index = torch.empty(n, dtype=torch.int64, device=self.device)
        radius = torch.empty(n, dtype=torch.float32, device=self.device)
        got = C.c_int64()
        check(self.L.lipcache_insert_select(self._h, _ptr(H), n, _ptr(payload), int(bool(require_consistency)),
                                            SELECT_STRATEGIES[strategy], int(budget_total), int(budget_per_class),
                                            _ptr(index), _ptr(radius), C.byref(got), _stream(self.device)))
        return index, radius, got.value

    # -- Algorithm 2
    def probe(self, Q: torch.Tensor, out=None):
        """Nearest certified hit per query: (index, label, dist); -1/-1/inf on a miss."""
        Q = self._dev(Q, torch.float32, "Q")
        B = Q.shape[0]
        if Q.dim() != 2 or (B and Q.shape[1] != self.d):
            raise ValueError("Q must be B x d")
        if out is None:
            out = (torch.empty(B, dtype=torch.int64, device=self.device),
                   torch.empty(B, dtype=torch.int32, device=self.device),
                   torch.empty(B, dtype=torch.float32, device=self.device))
        idx, lab, dist = out
        check(self.L.lipcache_probe(self._h, _ptr(Q), B, _ptr(idx), _ptr(lab), _ptr(dist), _stream(self.device)))
        return idx, lab, dist

    def probe_writeback(self, Q: torch.Tensor, payload: torch.Tensor | None = None,
                        require_consistency: bool = False):
        """Probe, then certify and append the missed queries (Algorithm 2 with
        write-back). The batch is probed against the cache as it was before
        the call. Returns (index, label, dist, inserted, n_inserted);
        inserted[k] is the new cache index of query k or -1."""
        Q = self._dev(Q, torch.float32, "Q")
        B = Q.shape[0]
        if Q.dim() != 2 or (B and Q.shape[1] != self.d):
            raise ValueError("Q must be B x d")
        if payload is not None:
            payload = self._dev(payload, torch.int32, "payload")
        idx = torch.empty(B, dtype=torch.int64, device=self.device)
        lab = torch.empty(B, dtype=torch.int32, device=self.device)
        dist = torch.empty(B, dtype=torch.float32, device=self.device)
        ins = torch.empty(B, dtype=torch.int64, device=self.device)
        n = C.c_int64()
        check(self.L.lipcache_probe_writeback(self._h, _ptr(Q), B, _ptr(payload), int(bool(require_consistency)),
                                              _ptr(idx), _ptr(lab), _ptr(dist), _ptr(ins), C.byref(n),
                                              _stream(self.device)))
        return idx, lab, dist, ins, n.value

    def consistency(self, Q: torch.Tensor, hit_index: torch.Tensor):
        """Certified-consistency check of hits: (per-query int8 1/0/-1,
        n_hits, n_consistent)."""
        Q = self._dev(Q, torch.float32, "Q")
        hit_index = self._dev(hit_index, torch.int64, "hit_index")
        B = Q.shape[0]
        if Q.dim() != 2 or (B and Q.shape[1] != self.d) or hit_index.shape != (B,):
            raise ValueError("Q must be B x d and hit_index must have B entries")
        out = torch.empty(B, dtype=torch.int8, device=self.device)
        nh, nc = C.c_int64(), C.c_int64()
        check(self.L.lipcache_consistency(self._h, _ptr(Q), B, _ptr(hit_index), _ptr(out), C.byref(nh),
                                          C.byref(nc), _stream(self.device)))
        return out, nh.value, nc.value

    def probe_noalloc(self, Q: torch.Tensor, out):
        """probe() without any device allocation, for callers that cannot
        allocate while they run: the scratch is a fixed array inside the
        library (see lipcache_probe_noalloc). `out` must be preallocated;
        overlapping calls on one device race on the shared array."""
        Q = self._dev(Q, torch.float32, "Q")
        idx, lab, dist = out
        check(self.L.lipcache_probe_noalloc(self._h, _ptr(Q), Q.shape[0], _ptr(idx), _ptr(lab), _ptr(dist),
                                            _stream(self.device)))
        return idx, lab, dist

    def probe_host(self, Q, out=None):
        """Probe from host memory (pinned tensors give asynchronous copies)."""
        Q = Q.contiguous()
        if Q.device.type != "cpu" or Q.dtype != torch.float32:
            raise ValueError("Q must be a float32 CPU tensor")
        B = Q.shape[0]
        if out is None:
            out = (torch.empty(B, dtype=torch.int64), torch.empty(B, dtype=torch.int32),
                   torch.empty(B, dtype=torch.float32))
        idx, lab, dist = out
        check(self.L.lipcache_probe_host(self._h, _ptr(Q), B, _ptr(idx), _ptr(lab), _ptr(dist),
                                         _stream(self.device)))
        return idx, lab, dist

    # -- options / introspection
    def set_probe_path(self, path: str):
        check(self.L.lipcache_set_probe_path(self._h, PROBE_PATHS[path]))

    def set_radius_policy(self, policy: str, param: float = 0.0):
        """Switch the probe to the certified radius or to an empirical
        boundary ("global": one threshold tau = param; "interclass": beta =
        param times half the distance between class centroids). Returns the
        C per-class radii as a numpy array."""
        rho = np.zeros(self.C, dtype=np.float64)
        check(self.L.lipcache_set_radius_policy(self._h, RADIUS_POLICIES[policy], float(param),
                                                rho.ctypes.data, _stream(self.device)))
        return rho

    def entries(self, first: int = 0, n: int | None = None) -> dict:
        """Cache entries [first, first + n) as numpy arrays: keys (n x d),
        radius, label (payload) and yG, in insertion order."""
        size = self.size
        n = size - first if n is None else n
        keys = np.empty((n, self.d), dtype=np.float32)
        radius = np.empty(n, dtype=np.float32)
        label = np.empty(n, dtype=np.int32)
        yG = np.empty(n, dtype=np.int32)
        check(self.L.lipcache_read_entries(self._h, int(first), int(n), keys.ctypes.data, radius.ctypes.data,
                                           label.ctypes.data, yG.ctypes.data, _stream(self.device)))
        return {"keys": keys, "radius": radius, "label": label, "yG": yG}

    def head(self) -> tuple[np.ndarray, np.ndarray]:
        """The head (W, b) set by set_head, as numpy arrays."""
        W = np.empty((self.C, self.d), dtype=np.float32)
        b = np.empty(self.C, dtype=np.float32)
        check(self.L.lipcache_read_head(self._h, W.ctypes.data, b.ctypes.data, _stream(self.device)))
        return W, b

    def save(self, path: str):
        """Checkpoint: the configuration, the head and the entries' keys and
        labels (numpy .npz). LipCache.load re-certifies the keys under the
        head, which gives the same radii; radii are stored only to check it."""
        inf = self.info()
        W, b = self.head()
        e = self.entries()
        mode = {v: k for k, v in RADIUS_MODES.items()}[inf["radius_mode"]]
        path_name = {v: k for k, v in PROBE_PATHS.items()}.get(inf["probe_path"], "auto")
        policy = {v: k for k, v in RADIUS_POLICIES.items()}[inf["radius_policy"]]
        np.savez(path, d=self.d, C=self.C, capacity=inf["capacity"], radius_mode=mode,
                 radius_scale=inf["radius_scale"], probe_path=path_name, radius_policy=policy,
                 policy_param=inf["policy_param"], sigma=inf["sigma"], W=W, b=b, keys=e["keys"],
                 label=e["label"], radius=e["radius"])

    @classmethod
    def load(cls, path: str, device: int | torch.device | None = None, batch: int = 65536) -> "LipCache":
        """Restore a checkpoint written by save: create, set_head, re-insert
        the keys with their labels as payload (Algorithm 1 again), restore
        the probe path and radius policy. Raises if sigma or a radius
        differs from the saved one."""
        z = np.load(path if str(path).endswith(".npz") else str(path) + ".npz")
        c = cls(int(z["d"]), int(z["C"]), int(z["capacity"]), str(z["radius_mode"]), device=device)
        c.set_radius_scale(float(z["radius_scale"]))
        sigma = c.set_head(torch.from_numpy(z["W"]).to(c.device), torch.from_numpy(z["b"]).to(c.device))
        if sigma != float(z["sigma"]):
            raise ValueError(f"sigma of the restored head {sigma!r} differs from the saved {float(z['sigma'])!r}")
        keys, label = z["keys"], z["label"]
        for s in range(0, len(keys), batch):
            idx, _, n = c.insert(torch.from_numpy(keys[s:s + batch]).to(c.device),
                                 torch.from_numpy(label[s:s + batch]).to(c.device))
            if n != len(keys[s:s + batch]):
                raise ValueError("a saved entry was not re-certified")
        if not np.array_equal(c.entries()["radius"].view(np.uint32), z["radius"].view(np.uint32)):
            raise ValueError("re-certified radii differ from the saved ones")
        c.set_probe_path(str(z["probe_path"]))
        if str(z["radius_policy"]) != "certified":
            c.set_radius_policy(str(z["radius_policy"]), float(z["policy_param"]))
        return c

    def set_debug(self, flags: int):
        """Failure-detection test hooks (LIPCACHE_DEBUG_*; 0 = off)."""
        check(self.L.lipcache_set_debug(self._h, int(flags)))

    def set_radius_scale(self, kappa: float):
        check(self.L.lipcache_set_radius_scale(self._h, float(kappa)))

    def set_spectral_options(self, squarings: int, max_iter: int):
        check(self.L.lipcache_set_spectral_options(self._h, int(squarings), int(max_iter)))

    def reserve(self, max_batch: int):
        check(self.L.lipcache_reserve(self._h, int(max_batch)))

    def enable_timing(self, on: bool = True):
        check(self.L.lipcache_enable_timing(self._h, int(bool(on))))

    def reset_stats(self):
        check(self.L.lipcache_reset_stats(self._h))

    def info(self) -> dict:
        inf = Info()
        check(self.L.lipcache_get_info(self._h, C.byref(inf)))
        return {name: getattr(inf, name) for name, _ in Info._fields_}

    @property
    def size(self) -> int:
        return int(self.L.lipcache_size(self._h))

    def __len__(self):
        return self.size
