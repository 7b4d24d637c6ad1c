"""Python face of the GB300 embedding key-value store (MLKV interface, Section 3.1).

    store = EmbeddingStore(dim=128, capacity=..., max_batch=..., lr=0.01)
    rows = store.get(keys)            # Get(keys)  -> values
    store.put(keys, values)           # Put(keys, values), upsert
    store.apply_grad(keys, grads)     # per-key Rmw with Adagrad
    store.lookahead(next_keys)        # Lookahead(keys, dest = store buffer)

Keys are int64 CUDA tensors; rows, values and gradients float32 [n, dim] CUDA
tensors.  Every call is enqueued on the current torch stream of the store's
device and runs in the CUDA library; this class only checks tensor types and
passes pointers.

staleness_bound (Open's third argument, Section 3.3.1): 0 runs every call in
order; s >= 1 lets a Get issued on one stream run beside the last s gradient
applies issued on another; STALENESS_ASYNC (INT64_MAX) lets it run beside any.
"""
import ctypes

import torch

from . import _lib as L


class MLKVError(RuntimeError):
    def __init__(self, code: int, message: str):
        super().__init__(f"mlkv status {code}: {message}")
        self.code = code


def _stream(device) -> int:
    return torch.cuda.current_stream(device).cuda_stream


class EmbeddingStore:
    def __init__(self, dim: int, capacity: int, max_batch: int, lr: float = 0.01, eps: float = 1e-8,
                 state_init: float = 0.0, init_lo: float = -0.01, init_hi: float = 0.01, seed: int = 1,
                 insert_on_miss: bool = True, staleness_bound: int = 0, hbm_cache_rows: int = 0,
                 flags: int = 0, device=None):
        self.lib = L.load()
        self.device = torch.device("cuda", torch.cuda.current_device() if device is None
                                   else torch.device(device).index or 0)
        self.dim = int(dim)
        self.max_batch = int(max_batch)
        cfg = L.Config(dim=self.dim, insert_on_miss=int(bool(insert_on_miss)), capacity=int(capacity),
                       max_batch=self.max_batch, lr=lr, eps=eps, state_init=state_init, init_lo=init_lo,
                       init_hi=init_hi, seed=seed & (2**64 - 1), staleness_bound=staleness_bound,
                       hbm_cache_rows=hbm_cache_rows, flags=flags, reserved=0)
        self.config = cfg
        h = ctypes.c_void_p()
        with torch.cuda.device(self.device):
            rc = self.lib.mlkv_open(ctypes.byref(cfg), ctypes.byref(h))
        if rc != L.OK:
            raise MLKVError(rc, self.lib.mlkv_status_string(rc).decode())
        self.h = h

    # -- plumbing ---------------------------------------------------------------
    def _check(self, rc: int):
        if rc != L.OK:
            raise MLKVError(rc, self.lib.mlkv_last_error(self.h).decode() or
                            self.lib.mlkv_status_string(rc).decode())

    def _keys(self, keys: torch.Tensor) -> torch.Tensor:
        if keys.dtype != torch.int64 or keys.device != self.device or keys.dim() != 1:
            raise TypeError("keys must be a 1-d int64 tensor on the store's device")
        return keys.contiguous()

    def _rows(self, x: torch.Tensor, n: int, device=None) -> torch.Tensor:
        device = device or self.device
        if x.dtype != torch.float32 or x.device != device or tuple(x.shape) != (n, self.dim):
            raise TypeError(f"expected float32 [{n}, {self.dim}] on {device}")
        return x.contiguous()

    def _check_out(self, out: torch.Tensor, n: int, device=None) -> torch.Tensor:
        """An output buffer is written in place, so it must be contiguous already."""
        if not out.is_contiguous():
            raise TypeError("output buffer must be contiguous (it is written in place)")
        return self._rows(out, n, device)

    @staticmethod
    def _host_keys(keys: torch.Tensor) -> torch.Tensor:
        if keys.dtype != torch.int64 or keys.device.type != "cpu" or keys.dim() != 1:
            raise TypeError("keys must be a 1-d int64 host tensor")
        return keys.contiguous()

    def close(self):
        if getattr(self, "h", None):
            self.lib.mlkv_close(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # -- the MLKV interface ----------------------------------------------------
    def get(self, keys: torch.Tensor, out: torch.Tensor | None = None) -> torch.Tensor:
        """Get: the row of every key ([n, dim], into `out` when given).  Absent keys
        are inserted with the init row (insert_on_miss), else NaN and NOT_FOUND."""
        keys = self._keys(keys)
        n = keys.numel()
        if out is None:
            out = torch.empty((n, self.dim), dtype=torch.float32, device=self.device)
        out = self._check_out(out, n)
        self._check(self.lib.mlkv_get(self.h, keys.data_ptr(), n, out.data_ptr(), _stream(self.device)))
        return out

    def put(self, keys: torch.Tensor, values: torch.Tensor):
        """Put (upsert): row of each key = its value; the last duplicate wins; a new
        key starts with state_init, a present one keeps its state."""
        keys = self._keys(keys)
        values = self._rows(values, keys.numel())
        self._check(self.lib.mlkv_put(self.h, keys.data_ptr(), keys.numel(), values.data_ptr(),
                                      _stream(self.device)))

    def insert(self, keys: torch.Tensor):
        """Inserts the absent keys with the init row (row ids in first-occurrence order)."""
        keys = self._keys(keys)
        self._check(self.lib.mlkv_insert(self.h, keys.data_ptr(), keys.numel(), _stream(self.device)))

    def apply_grad(self, keys: torch.Tensor, grads: torch.Tensor):
        """The per-key Rmw: each distinct key's gradients summed, then one Adagrad step
        on its row and state."""
        keys = self._keys(keys)
        grads = self._rows(grads, keys.numel())
        self._check(self.lib.mlkv_apply_grad(self.h, keys.data_ptr(), keys.numel(), grads.data_ptr(),
                                             _stream(self.device)))

    def lookahead(self, keys: torch.Tensor):
        """Lookahead: brings the rows of the next batch's keys into the HBM cache on
        the table's side stream (a no-op for an HBM-resident table)."""
        keys = self._keys(keys)
        self._check(self.lib.mlkv_lookahead(self.h, keys.data_ptr(), keys.numel(), _stream(self.device)))

    def find(self, keys: torch.Tensor) -> torch.Tensor:
        keys = self._keys(keys)
        rows = torch.empty(keys.numel(), dtype=torch.int64, device=self.device)
        self._check(self.lib.mlkv_find(self.h, keys.data_ptr(), keys.numel(), rows.data_ptr(),
                                       _stream(self.device)))
        return rows

    def export(self, keys: torch.Tensor):
        keys = self._keys(keys)
        n = keys.numel()
        w = torch.empty((n, self.dim), dtype=torch.float32, device=self.device)
        G = torch.empty((n, self.dim), dtype=torch.float32, device=self.device)
        self._check(self.lib.mlkv_export(self.h, keys.data_ptr(), n, w.data_ptr(), G.data_ptr(),
                                         _stream(self.device)))
        return w, G

    def dedup(self, keys: torch.Tensor):
        keys = self._keys(keys)
        n = keys.numel()
        uniq = torch.empty(max(n, 1), dtype=torch.int64, device=self.device)
        counts = torch.empty(max(n, 1), dtype=torch.int32, device=self.device)
        num = torch.zeros(1, dtype=torch.int64, device=self.device)
        self._check(self.lib.mlkv_dedup(self.h, keys.data_ptr(), n, uniq.data_ptr(), counts.data_ptr(),
                                        num.data_ptr(), _stream(self.device)))
        u = int(num.item())
        return uniq[:u], counts[:u]

    # -- checkpoints (keys in row order, rows, state) -----------------------------
    def import_(self, keys: torch.Tensor, rows: torch.Tensor, state: torch.Tensor | None = None):
        """Upsert rows (and state, when given) of keys; the later duplicate wins."""
        keys = self._keys(keys)
        rows = self._rows(rows, keys.numel())
        st = None if state is None else self._rows(state, keys.numel())
        self._check(self.lib.mlkv_import(self.h, keys.data_ptr(), keys.numel(), rows.data_ptr(),
                                         None if st is None else st.data_ptr(), _stream(self.device)))

    def keys(self) -> torch.Tensor:
        """Every key of the table, in row order."""
        n = self.size()
        out = torch.empty(n, dtype=torch.int64, device=self.device)
        self._check(self.lib.mlkv_dump_keys(self.h, out.data_ptr(), n, _stream(self.device)))
        return out

    def save(self, path: str):
        """Writes a checkpoint (keys in row order, rows, state) to an .npz file."""
        import numpy as np

        keys = self.keys()
        rows, state = [], []
        for s in range(0, keys.numel(), self.max_batch):
            w, G = self.export(keys[s:s + self.max_batch])
            rows.append(w.cpu())
            state.append(G.cpu())
        cat = (lambda xs: torch.cat(xs).numpy()) if rows else (lambda xs: np.zeros((0, self.dim), np.float32))
        np.savez(path, keys=keys.cpu().numpy(), rows=cat(rows), state=cat(state), dim=self.dim)

    def load(self, path: str):
        """Imports a checkpoint written by save() (into an empty table: the same row ids)."""
        import numpy as np

        ck = np.load(path)
        if int(ck["dim"]) != self.dim:
            raise ValueError(f"checkpoint dim {int(ck['dim'])} != table dim {self.dim}")
        keys = torch.from_numpy(ck["keys"]).to(self.device)
        rows = torch.from_numpy(ck["rows"]).to(self.device)
        state = torch.from_numpy(ck["state"]).to(self.device)
        for s in range(0, keys.numel(), self.max_batch):
            e = s + self.max_batch
            self.import_(keys[s:e], rows[s:e].contiguous(), state[s:e].contiguous())

    # -- host-buffer forms (copies inside the call) -----------------------------
    def get_host(self, keys: torch.Tensor, out: torch.Tensor):
        """Get from and into host tensors (pinned for asynchronous copies); `out` is
        valid once the stream has synchronised."""
        keys = self._host_keys(keys)
        out = self._check_out(out, keys.numel(), torch.device("cpu"))
        self._check(self.lib.mlkv_get_host(self.h, keys.data_ptr(), keys.numel(), out.data_ptr(),
                                           _stream(self.device)))

    def apply_grad_host(self, keys: torch.Tensor, grads: torch.Tensor):
        """apply_grad from host tensors (copied to the device inside the call)."""
        keys = self._host_keys(keys)
        grads = self._rows(grads, keys.numel(), torch.device("cpu"))
        self._check(self.lib.mlkv_apply_grad_host(self.h, keys.data_ptr(), keys.numel(),
                                                  grads.data_ptr(), _stream(self.device)))

    # -- status and counters ------------------------------------------------------
    def sync(self) -> int:
        return self.lib.mlkv_sync(self.h)

    def clear_status(self):
        self._check(self.lib.mlkv_clear_status(self.h))

    def size(self) -> int:
        return int(self.lib.mlkv_size(self.h))

    def last_unique(self) -> int:
        return int(self.lib.mlkv_last_unique(self.h))

    def tier_stats(self):
        """(rows fetched host -> HBM, rows written back, cache lines swept for victims)
        since open; zeros when not tiered."""
        f, w, c = ctypes.c_int64(), ctypes.c_int64(), ctypes.c_int64()
        self._check(self.lib.mlkv_tier_stats(self.h, ctypes.byref(f), ctypes.byref(w), ctypes.byref(c)))
        return f.value, w.value, c.value

    def launch_count(self) -> int:
        return int(self.lib.mlkv_launch_count(self.h))

    def time_kernel(self, kernel_id: int):
        self._check(self.lib.mlkv_time_kernel(self.h, kernel_id))

    def kernel_time(self):
        ms = ctypes.c_double()
        n = ctypes.c_int64()
        self._check(self.lib.mlkv_kernel_time(self.h, ctypes.byref(ms), ctypes.byref(n)))
        return ms.value, n.value
