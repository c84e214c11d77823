"""Thin Python binding of the C ABI in ``include/gmgsim.h``.

Argument marshalling only: every step of the simulation runs in the CUDA
kernels of ``libgmgsim.so``.  PyTorch provides device memory and streams.
If the library is missing the calls raise; there is no fallback path.

Names follow the C ABI: ``gmg_create``, ``sim_batch``, ``base_create``,
``sim_incremental``, ``select_best`` (plus the sizing helpers).
"""
from __future__ import annotations

import ctypes as C
import functools
import os
from dataclasses import dataclass
from typing import Optional

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libgmgsim.so")

GMG_OK, GMG_EINVAL, GMG_ENOTTOPO, GMG_ERANGE, GMG_EWS, GMG_ECUDA, GMG_ENOMEM = 0, -1, -2, -3, -4, -5, -6
GMG_TRANSFER_LATENCY, GMG_TRANSFER_ARBITRATED = 0, 1
SIM_OK, SIM_BADDEV, SIM_MOVE_RANGE, SIM_MOVE_DUP, SIM_BADBASE, SIM_QUEUE, SIM_LOOP = range(7)

EXPORTED = ("gmg_workspace_bytes", "gmg_create", "gmg_destroy", "gmg_get_info", "sim_scratch_bytes",
            "sim_batch", "sim_batch_noalloc", "base_workspace_bytes", "base_create", "base_destroy", "inc_scratch_bytes",
            "sim_incremental", "select_best_tmp_bytes", "select_best", "gmg_strerror",
            "gmg_ceil_div_host", "est_state_bytes", "est_reset", "est_update_tmp_bytes", "est_update",
            "est_coefficients",
            "est_predict_durations", "est_links", "round_scratch_bytes", "round_select", "round_candidates",
            "round_commit")


# NVTX ranges around the public calls (for nsys / ncu range filters), when
# the environment sets GMGSIM_NVTX=1; nothing is pushed otherwise.
NVTX = os.environ.get("GMGSIM_NVTX", "") not in ("", "0")


def _traced(name: str):
    def wrap(fn):
        @functools.wraps(fn)
        def call(*a, **kw):
            if not NVTX:
                return fn(*a, **kw)
            import torch
            torch.cuda.nvtx.range_push("gmgsim." + name)
            try:
                return fn(*a, **kw)
            finally:
                torch.cuda.nvtx.range_pop()
        return call
    return wrap


class GmgError(RuntimeError):
    def __init__(self, code: int, what: str):
        super().__init__("%s failed: %s (%d)" % (what, strerror(code), code))
        self.code = code


class _Desc(C.Structure):
    _fields_ = [("n_ops", C.c_int32), ("n_edges", C.c_int32), ("n_dev", C.c_int32),
                ("n_req", C.c_int32)] + [(n, C.c_void_p) for n in (
                    "pred_off", "pred_idx", "cons_off", "cons_idx", "dur_us", "out_bytes",
                    "release_us", "req_id", "scored", "deadline_us", "cap_bytes", "base_bytes",
                    "avail0_us", "bw_B_per_us", "lat_us")] + [
        ("n_types", C.c_int32), ("dev_type", C.c_void_p), ("dur_by_type", C.c_void_p),
        ("link_id", C.c_void_p)]


class _Opts(C.Structure):
    _fields_ = [("score_mode", C.c_int32), ("n_trace", C.c_int32), ("d_trace_k", C.c_void_p),
                ("queue_cap", C.c_int32), ("warps_per_block", C.c_int32),
                ("transfer_mode", C.c_int32), ("gmg_staging", C.c_int32), ("reserved", C.c_int32 * 2)]


class _Out(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in (
        "makespan", "score", "status", "viol_flag", "viol_op", "viol_dev", "viol_time", "peak",
        "sla_miss", "events", "req_done", "trace_start", "trace_finish")]


class _Info(C.Structure):
    _fields_ = [("n_ops", C.c_int32), ("n_edges", C.c_int32), ("n_dev", C.c_int32),
                ("n_req", C.c_int32), ("n_roots", C.c_int32), ("id_bits", C.c_int32),
                ("time_bits", C.c_int32), ("uniform_links", C.c_int32),
                ("time_bound", C.c_int64), ("default_queue_cap", C.c_int64),
                ("batched_sweep", C.c_int32), ("t32", C.c_int32), ("stageable", C.c_int32),
                ("reserved_", C.c_int32)]


_LIB = None


def lib():
    """Load libgmgsim.so (raises if it has not been built)."""
    global _LIB
    if _LIB is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError("libgmgsim.so is not built; run `python -m paper_2608_15762_gb300.build`")
        L = C.CDLL(LIB_PATH)
        vp, i32, i64, sz = C.c_void_p, C.c_int32, C.c_int64, C.c_size_t
        sig = {
            "gmg_workspace_bytes": ([vp], sz),
            "gmg_create": ([vp, vp, sz, vp, vp], C.c_int),
            "gmg_destroy": ([vp], None),
            "gmg_get_info": ([vp, vp], C.c_int),
            "sim_scratch_bytes": ([vp, i32, vp], sz),
            "sim_batch": ([vp, vp, i32, i32, vp, vp, vp, sz, vp], C.c_int),
            "sim_batch_noalloc": ([vp, vp, i32, i32, vp, vp, vp], C.c_int),
            "base_workspace_bytes": ([vp, vp], sz),
            "base_create": ([vp, vp, vp, vp, sz, vp, vp], C.c_int),
            "base_destroy": ([vp], None),
            "inc_scratch_bytes": ([vp, i32, vp], sz),
            "sim_incremental": ([vp, vp, vp, vp, vp, i32, vp, vp, vp, sz, vp], C.c_int),
            "select_best_tmp_bytes": ([i32], sz),
            "select_best": ([vp, i32, i32, vp, vp, sz, vp], C.c_int),
            "gmg_strerror": ([C.c_int], C.c_char_p),
            "gmg_ceil_div_host": ([i64, i64], i64),
            "est_state_bytes": ([i32, i32], sz),
            "est_reset": ([vp, i32, i32, vp], C.c_int),
            "est_update_tmp_bytes": ([i32, i32, i64], sz),
            "est_update": ([vp, i32, i32, vp, vp, vp, i64, vp, sz, vp], C.c_int),
            "est_coefficients": ([vp, i32, i32, vp, vp, vp], C.c_int),
            "est_predict_durations": ([vp, i32, i32, i32, i32, vp, vp, vp, vp, vp], C.c_int),
            "est_links": ([vp, i32, vp, vp, vp, vp, vp], C.c_int),
            "round_scratch_bytes": ([vp], sz),
            "round_select": ([vp, vp, vp, i32, i32, C.c_uint32, vp, sz, vp, vp, vp], C.c_int),
            "round_candidates": ([vp, vp, i32, vp, i32, vp, i32, vp, vp, vp, vp, vp, i32, vp, vp], C.c_int),
            "round_commit": ([vp, i32, vp, vp, vp, i32, vp, vp, vp], C.c_int),
        }
        for name, (args, res) in sig.items():
            f = getattr(L, name)
            f.argtypes = args
            f.restype = res
        _LIB = L
    return _LIB


def strerror(code: int) -> str:
    return lib().gmg_strerror(int(code)).decode()


def _stream_handle(stream) -> Optional[int]:
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    return int(s.cuda_stream) or None


def _np_ptr(a):
    return None if a is None else a.ctypes.data


class _DescHolder:
    def __init__(self, desc):
        d = desc.normalized()
        self.d = d
        self.c = _Desc(d.n_ops, d.n_edges, d.n_dev, d.n_req, _np_ptr(d.pred_off), _np_ptr(d.pred_idx),
                       _np_ptr(d.cons_off), _np_ptr(d.cons_idx), _np_ptr(d.dur), _np_ptr(d.out_bytes),
                       _np_ptr(d.release), _np_ptr(d.req_id), _np_ptr(d.scored), _np_ptr(d.deadline),
                       _np_ptr(d.cap), _np_ptr(d.base), _np_ptr(d.avail0), _np_ptr(d.bw), _np_ptr(d.lat),
                       d.n_types, _np_ptr(d.dev_type), _np_ptr(d.dur_by_type), _np_ptr(d.link_id))


def gmg_workspace_bytes(desc) -> int:
    h = _DescHolder(desc)
    return int(lib().gmg_workspace_bytes(C.addressof(h.c)))


GMG_STAGING_DEFAULT, GMG_STAGING_SHARED, GMG_STAGING_L1 = 0, 1, 2


def _opts(score_mode=0, trace_k=None, queue_cap=0, warps_per_block=0, arbitrated=False,
          gmg_staging=GMG_STAGING_DEFAULT) -> _Opts:
    o = _Opts()
    o.transfer_mode = GMG_TRANSFER_ARBITRATED if arbitrated else GMG_TRANSFER_LATENCY
    o.gmg_staging = int(gmg_staging)
    o.score_mode = score_mode
    o.n_trace = 0 if trace_k is None else int(trace_k.numel())
    o.d_trace_k = None if trace_k is None else trace_k.data_ptr()
    o.queue_cap = queue_cap
    o.warps_per_block = warps_per_block
    return o


def _aligned_empty(nbytes: int, device, align: int = 256):
    """A uint8 device tensor view whose data pointer is `align`-aligned."""
    import torch
    buf = torch.empty(max(int(nbytes), 1) + align, dtype=torch.uint8, device=device)
    off = (-buf.data_ptr()) % align
    return buf[off:off + max(int(nbytes), 1)]


class Gmg:
    """A created GMG: host handle + the device workspace it borrows."""

    def __init__(self, desc, device="cuda", stream=None):
        import torch
        self.desc = desc.normalized()
        self._h = _DescHolder(self.desc)
        nbytes = lib().gmg_workspace_bytes(C.addressof(self._h.c))
        if nbytes == 0:
            # let gmg_create report the reason
            nbytes = 256
        self.device = torch.device(device)
        self.ws = _aligned_empty(nbytes, self.device)
        handle = C.c_void_p()
        rc = lib().gmg_create(C.addressof(self._h.c), self.ws.data_ptr(), self.ws.numel(),
                              _stream_handle(stream), C.addressof(handle))
        if rc != GMG_OK:
            raise GmgError(rc, "gmg_create")
        self.handle = handle

    @property
    def info(self) -> dict:
        i = _Info()
        rc = lib().gmg_get_info(self.handle, C.addressof(i))
        if rc:
            raise GmgError(rc, "gmg_get_info")
        return {n: getattr(i, n) for n, _ in _Info._fields_}

    @property
    def n_ops(self):
        return self.desc.n_ops

    @property
    def n_dev(self):
        return self.desc.n_dev

    @property
    def n_req(self):
        return self.desc.n_req

    def close(self):
        if getattr(self, "handle", None):
            lib().gmg_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


@_traced("gmg_create")
def gmg_create(desc, device="cuda", stream=None) -> Gmg:
    return Gmg(desc, device, stream)


@dataclass
class SimOut:
    """Device output tensors for K candidates (fields of sim_out_t)."""
    makespan: "object"
    score: "object"
    status: "object"
    viol_flag: "object"
    viol_op: "object"
    viol_dev: "object"
    viol_time: "object"
    peak: "object"
    sla_miss: "object"
    events: "object"
    req_done: "object" = None
    trace_start: "object" = None
    trace_finish: "object" = None

    @staticmethod
    def empty(K: int, n_dev: int, n_req: int, device, req_done=False, n_trace=0, n_ops=0) -> "SimOut":
        import torch
        i64, i32 = torch.int64, torch.int32
        return SimOut(
            makespan=torch.empty(K, dtype=i64, device=device),
            score=torch.empty(K, dtype=i64, device=device),
            status=torch.empty(K, dtype=i32, device=device),
            viol_flag=torch.empty(K, dtype=i32, device=device),
            viol_op=torch.empty(K, dtype=i32, device=device),
            viol_dev=torch.empty(K, dtype=i32, device=device),
            viol_time=torch.empty(K, dtype=i64, device=device),
            peak=torch.empty((K, n_dev), dtype=i64, device=device),
            sla_miss=torch.empty(K, dtype=i32, device=device),
            events=torch.empty(K, dtype=i64, device=device),
            req_done=torch.empty((K, n_req), dtype=i64, device=device) if req_done else None,
            trace_start=torch.empty((n_trace, n_ops), dtype=i64, device=device) if n_trace else None,
            trace_finish=torch.empty((n_trace, n_ops), dtype=i64, device=device) if n_trace else None)

    def _c(self) -> _Out:
        def p(t):
            return None if t is None else t.data_ptr()
        return _Out(p(self.makespan), p(self.score), p(self.status), p(self.viol_flag), p(self.viol_op),
                    p(self.viol_dev), p(self.viol_time), p(self.peak), p(self.sla_miss), p(self.events),
                    p(self.req_done), p(self.trace_start), p(self.trace_finish))

    def to_numpy(self) -> dict:
        return {k: (None if v is None else v.cpu().numpy()) for k, v in self.__dict__.items()}


def sim_scratch_bytes(g: Gmg, K: int, **opt) -> int:
    o = _opts(**opt)
    return int(lib().sim_scratch_bytes(g.handle, K, C.addressof(o)))


def inc_scratch_bytes(g: Gmg, K: int, **opt) -> int:
    o = _opts(**opt)
    return int(lib().inc_scratch_bytes(g.handle, K, C.addressof(o)))


class Scratch:
    """A reusable aligned device scratch buffer, grown on demand."""

    def __init__(self, device):
        self.device = device
        self.buf = None

    def get(self, nbytes: int):
        if self.buf is None or self.buf.numel() < nbytes:
            self.buf = _aligned_empty(nbytes, self.device)
        return self.buf


@_traced("sim_batch")
def sim_batch(g: Gmg, place, out: Optional[SimOut] = None, scratch: Optional[Scratch] = None,
              req_done=False, trace_k=None, queue_cap=0, warps_per_block=0, stream=None,
              arbitrated=False, gmg_staging=GMG_STAGING_DEFAULT) -> SimOut:
    """Simulate every row of ``place`` (CUDA uint8 [K, ld], ld % 16 == 0);
    ``arbitrated``: transfers go through the arbiter of Sec. 3.5.2;
    ``gmg_staging``: GMG_STAGING_SHARED stages the GMG's hot fields in every
    CTA's shared memory, GMG_STAGING_L1 reads them through the L1 path."""
    import torch
    assert place.dtype == torch.uint8 and place.dim() == 2 and place.is_contiguous()
    K, ld = place.shape
    n_trace = 0 if trace_k is None else int(trace_k.numel())
    if out is None:
        out = SimOut.empty(K, g.n_dev, g.n_req, place.device, req_done, n_trace, g.n_ops)
    o = _opts(0, trace_k, queue_cap, warps_per_block, arbitrated, gmg_staging)
    need = lib().sim_scratch_bytes(g.handle, K, C.addressof(o))
    scratch = scratch or Scratch(place.device)
    buf = scratch.get(need)
    co = out._c()
    rc = lib().sim_batch(g.handle, place.data_ptr(), K, ld, C.addressof(o), C.addressof(co),
                         buf.data_ptr(), buf.numel(), _stream_handle(stream))
    if rc != GMG_OK:
        raise GmgError(rc, "sim_batch")
    return out


@_traced("sim_batch_noalloc")
def sim_batch_noalloc(g: Gmg, place, out: Optional[SimOut] = None, req_done=False, trace_k=None,
                      stream=None, arbitrated=False) -> SimOut:
    """Like sim_batch, but the library supplies the scratch from its own fixed
    device buffer (for callers that cannot allocate device memory)."""
    import torch
    assert place.dtype == torch.uint8 and place.dim() == 2 and place.is_contiguous()
    K, ld = place.shape
    n_trace = 0 if trace_k is None else int(trace_k.numel())
    if out is None:
        out = SimOut.empty(K, g.n_dev, g.n_req, place.device, req_done, n_trace, g.n_ops)
    o = _opts(0, trace_k, arbitrated=arbitrated)
    co = out._c()
    rc = lib().sim_batch_noalloc(g.handle, place.data_ptr(), K, ld, C.addressof(o), C.addressof(co),
                                 _stream_handle(stream))
    if rc != GMG_OK:
        raise GmgError(rc, "sim_batch_noalloc")
    return out


class Base:
    """A recorded base schedule (base_create) and the workspace it borrows.
    ``arbitrated``: the base placement simulated with arbitrated transfers
    (Sec. 3.5.2), with the arbiter's state at every resume point; such a base
    serves arbitrated candidates only, which it resumes instead of
    re-simulating (at most 32 accelerators)."""

    def __init__(self, g: Gmg, base_place, queue_cap=0, stream=None, arbitrated=False):
        import torch
        assert base_place.dtype == torch.uint8 and base_place.is_contiguous()
        ld = (g.n_ops + 15) // 16 * 16
        row = torch.zeros(max(ld, 16), dtype=torch.uint8, device=base_place.device)
        row[:base_place.numel()] = base_place[:ld].reshape(-1)
        self.row = row
        self.g = g
        o = _opts(0, None, queue_cap, arbitrated=arbitrated)
        self.arbitrated = bool(arbitrated)
        nbytes = lib().base_workspace_bytes(g.handle, C.addressof(o))
        self.ws = _aligned_empty(nbytes, base_place.device)
        h = C.c_void_p()
        rc = lib().base_create(g.handle, row.data_ptr(), C.addressof(o), self.ws.data_ptr(),
                               self.ws.numel(), _stream_handle(stream), C.addressof(h))
        if rc != GMG_OK:
            raise GmgError(rc, "base_create")
        self.handle = h

    def close(self):
        if getattr(self, "handle", None):
            lib().base_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


@_traced("base_create")
def base_create(g: Gmg, base_place, queue_cap=0, stream=None, arbitrated=False) -> Base:
    return Base(g, base_place, queue_cap, stream, arbitrated)


@_traced("sim_incremental")
def sim_incremental(g: Gmg, base: Base, move_off, move_op, move_dev, out: Optional[SimOut] = None,
                    scratch: Optional[Scratch] = None, req_done=False, trace_k=None, queue_cap=0,
                    warps_per_block=0, stream=None, arbitrated=False) -> SimOut:
    """K move lists (CUDA int32 off[K+1], int32 op[M], uint8 dev[M]) against ``base``;
    ``arbitrated``: transfers go through the arbiter of Sec. 3.5.2 -- resumed
    from an arbitrated base, else each moved placement simulated in full."""
    K = int(move_off.numel()) - 1
    n_trace = 0 if trace_k is None else int(trace_k.numel())
    if out is None:
        out = SimOut.empty(K, g.n_dev, g.n_req, move_off.device, req_done, n_trace, g.n_ops)
    o = _opts(0, trace_k, queue_cap, warps_per_block, arbitrated)
    need = lib().inc_scratch_bytes(g.handle, K, C.addressof(o))
    scratch = scratch or Scratch(move_off.device)
    buf = scratch.get(need)
    co = out._c()
    rc = lib().sim_incremental(g.handle, base.handle, move_off.data_ptr(),
                               move_op.data_ptr() if move_op.numel() else None,
                               move_dev.data_ptr() if move_dev.numel() else None, K, C.addressof(o),
                               C.addressof(co), buf.data_ptr(), buf.numel(), _stream_handle(stream))
    if rc != GMG_OK:
        raise GmgError(rc, "sim_incremental")
    return out


@_traced("select_best")
def select_best(out: SimOut, K: Optional[int] = None, score_mode: int = 0, best=None, tmp=None,
                stream=None):
    """Device int64[2] = (best candidate or -1, its score)."""
    import torch
    K = int(out.score.numel()) if K is None else K
    dev = out.score.device
    if best is None:
        best = torch.empty(2, dtype=torch.int64, device=dev)
    need = lib().select_best_tmp_bytes(K)
    if tmp is None or tmp.numel() < need:
        tmp = _aligned_empty(need, dev)
    co = out._c()
    rc = lib().select_best(C.addressof(co), K, score_mode, best.data_ptr(), tmp.data_ptr(), tmp.numel(),
                           _stream_handle(stream))
    if rc != GMG_OK:
        raise GmgError(rc, "select_best")
    return best


def shard_block(rank: int, world: int, total: int) -> range:
    """The contiguous block of ``total`` independent candidates that ``rank``
    of ``world`` simulates (block sizes differ by at most one; no exchange on
    the data path)."""
    return range(total * rank // world, total * (rank + 1) // world)


def select_best_across_ranks(best, to_global, group=None):
    """Combine the ranks' select_best results into the best over all ranks'
    candidates (lowest global index on ties; (-1, INT64_MAX) if none).

    best: int64[2] (local index or -1, score) on this rank's device;
    to_global: maps this rank's local candidate index to its global index.
    One all_gather of 16 bytes per rank; call outside any timed region."""
    import torch
    import torch.distributed as dist
    loc = best.detach().to(torch.int64).reshape(2).cpu().clone()
    if int(loc[0]) >= 0:
        loc[0] = int(to_global(int(loc[0])))
    loc = loc.to(best.device)
    world = dist.get_world_size(group)
    bufs = [torch.empty_like(loc) for _ in range(world)]
    dist.all_gather(bufs, loc, group=group)
    cands = [(int(b[1]), int(b[0])) for b in bufs if int(b[0]) >= 0]
    if not cands:
        return -1, int(np.iinfo(np.int64).max)
    sc, k = min(cands)
    return k, sc


def two_half_index(n_full_local: int, full_lo: int, n_full_total: int, inc_lo: int):
    """Local-to-global candidate index of a rank that simulates full
    placements [full_lo, full_lo + n_full_local) and incremental candidates
    [inc_lo, ...) of a workload whose K candidates list all full placements
    first, then all incremental ones."""
    def f(k: int) -> int:
        return full_lo + k if k < n_full_local else n_full_total + inc_lo + (k - n_full_local)
    return f


def ceil_div_host(n: int, d: int) -> int:
    return int(lib().gmg_ceil_div_host(n, d))


def moves_to_device(moves, device):
    import torch
    return (torch.from_numpy(np.ascontiguousarray(moves.off, np.int32)).to(device),
            torch.from_numpy(np.ascontiguousarray(moves.op, np.int32)).to(device),
            torch.from_numpy(np.ascontiguousarray(moves.dev, np.uint8)).to(device))


# ---------------------------------------------------------------------------
# Online linear estimators (include/gmgest.h)
# ---------------------------------------------------------------------------

def _check(rc: int, what: str) -> None:
    if rc != GMG_OK:
        raise GmgError(rc, what)


class Estimators:
    """Device state of n_est linear estimators with n_feat features (running
    least-squares statistics and fitted coefficients, Sec. 3.3.1)."""

    def __init__(self, n_est: int, n_feat: int, device="cuda", stream=None):
        nbytes = lib().est_state_bytes(int(n_est), int(n_feat))
        if nbytes == 0:
            raise GmgError(GMG_EINVAL, "est_state_bytes")
        self.n_est, self.n_feat = int(n_est), int(n_feat)
        self.state = _aligned_empty(nbytes, device)
        _check(lib().est_reset(self.state.data_ptr(), self.n_est, self.n_feat, _stream_handle(stream)),
               "est_reset")

    @_traced("est_update")
    def update(self, off, x, y, tmp=None, stream=None):
        """Add samples (CSR by estimator: off int32 [n_est+1], x float64
        [S, n_feat], y float64 [S], device tensors) and refit.  tmp: an
        optional reusable buffer from tmp_for(S)."""
        S = int(y.numel())
        if tmp is None:
            tmp = self.tmp_for(S)
        _check(lib().est_update(self.state.data_ptr(), self.n_est, self.n_feat, off.data_ptr(),
                                x.data_ptr() if S else None, y.data_ptr() if S else None, S, tmp.data_ptr(),
                                tmp.numel(), _stream_handle(stream)), "est_update")

    def tmp_for(self, n_samples: int):
        return _aligned_empty(lib().est_update_tmp_bytes(self.n_est, self.n_feat, int(n_samples)),
                              self.state.device)

    def coefficients(self, stream=None):
        import torch
        beta = torch.empty((self.n_est, self.n_feat), dtype=torch.float64, device=self.state.device)
        fitted = torch.empty(self.n_est, dtype=torch.int32, device=self.state.device)
        _check(lib().est_coefficients(self.state.data_ptr(), self.n_est, self.n_feat, beta.data_ptr(),
                                      fitted.data_ptr(), _stream_handle(stream)), "est_coefficients")
        return beta, fitted

    @_traced("est_predict_durations")
    def predict_durations(self, est_of, x, dflt, out=None, stream=None):
        """dur_by_type [n_ops, n_types] int64 from est_of int32 [n_ops, n_types],
        op features x float64 [n_ops, n_feat] and fallback durations dflt
        int64 [n_ops]."""
        import torch
        n_ops, n_types = int(est_of.shape[0]), int(est_of.shape[1])
        if out is None:
            out = torch.empty((n_ops, n_types), dtype=torch.int64, device=self.state.device)
        _check(lib().est_predict_durations(self.state.data_ptr(), self.n_est, self.n_feat, n_ops, n_types,
                                           est_of.data_ptr(), x.data_ptr(), dflt.data_ptr(), out.data_ptr(),
                                           _stream_handle(stream)), "est_predict_durations")
        return out

    @_traced("est_links")
    def links(self, n_dev, bw_dflt, lat_dflt, stream=None):
        """(bw, lat) int64 [n_dev*n_dev] from the transfer estimators
        (n_est = n_dev^2, n_feat = 2)."""
        import torch
        bw = torch.empty(n_dev * n_dev, dtype=torch.int64, device=self.state.device)
        lat = torch.empty_like(bw)
        _check(lib().est_links(self.state.data_ptr(), int(n_dev), bw_dflt.data_ptr(), lat_dflt.data_ptr(),
                               bw.data_ptr(), lat.data_ptr(), _stream_handle(stream)), "est_links")
        return bw, lat


# ---------------------------------------------------------------------------
# A scheduling round of Algorithm 1 (include/gmground.h)
# ---------------------------------------------------------------------------

ROUND_BATCH, ROUND_BUDGET, ROUND_EMPTY, ROUND_NO_FEASIBLE = 0, 1, 2, 3


class Round:
    """Device state of the rounds on one GMG: op states, placement row,
    priorities, templates / roles, partitions and the fixed per-template
    mappings.  step() runs one round entirely on the device: round_select,
    round_candidates, sim_batch over the partition rows, select_best,
    round_commit; the caller reads `info` when it needs to."""

    def __init__(self, g: Gmg, state, place, prio, tmpl, role, part_off, part_dev, mapping, n_roles: int,
                 budget: int, max_batch: int, score_mode: int = 0):
        import torch
        self.g, self.state, self.place, self.prio = g, state, place, prio
        self.tmpl, self.role, self.part_off, self.part_dev, self.map = tmpl, role, part_off, part_dev, mapping
        self.n_roles, self.budget, self.max_batch, self.score_mode = int(n_roles), int(budget), int(max_batch), score_mode
        self.n_part = int(part_off.numel() - 1)
        dev = place.device
        self.ld = int(place.numel())
        self.scratch = _aligned_empty(lib().round_scratch_bytes(g.handle), dev)
        self.scratch.zero_()
        self.epoch = 0
        self.batch = torch.empty(self.max_batch, dtype=torch.int32, device=dev)
        self.info = torch.zeros(8, dtype=torch.int64, device=dev)
        self.rows = _aligned_empty(self.n_part * self.ld, dev, 16).view(self.n_part, self.ld)
        self.out = SimOut.empty(self.n_part, g.desc.n_dev, g.desc.n_req, dev)
        self.sim_scratch = Scratch(dev)
        self.best = torch.empty(2, dtype=torch.int64, device=dev)

    @_traced("round_step")
    def step(self, stream=None):
        h = _stream_handle(stream)
        self.epoch += 1
        _check(lib().round_select(self.g.handle, self.state.data_ptr(), self.prio.data_ptr(), self.budget,
                                  self.max_batch, self.epoch, self.scratch.data_ptr(), self.scratch.numel(),
                                  self.batch.data_ptr(), self.info.data_ptr(), h), "round_select")
        _check(lib().round_candidates(self.g.handle, self.place.data_ptr(), self.ld, self.batch.data_ptr(),
                                      self.max_batch, self.info.data_ptr(), self.n_part, self.part_off.data_ptr(),
                                      self.part_dev.data_ptr(), self.tmpl.data_ptr(), self.role.data_ptr(),
                                      self.map.data_ptr(), self.n_roles, self.rows.data_ptr(), h), "round_candidates")
        sim_batch(self.g, self.rows, out=self.out, scratch=self.sim_scratch, stream=stream)
        select_best(self.out, self.n_part, score_mode=self.score_mode, best=self.best, stream=stream)
        _check(lib().round_commit(self.batch.data_ptr(), self.max_batch, self.info.data_ptr(), self.best.data_ptr(),
                                  self.rows.data_ptr(), self.ld, self.place.data_ptr(), self.state.data_ptr(), h),
               "round_commit")

