"""Thin Python binding of the kvq C ABI (``include/kvq.h``).

Argument marshalling only: every step of the decode path runs in the CUDA
kernels of ``libkvq.so``.  PyTorch supplies device memory and the current CUDA
stream.  The library must have been built (``paper_2607_16248_gb300.build``);
a missing library or a non-CUDA tensor raises instead of falling back.
"""

import ctypes
import math
from dataclasses import dataclass
from pathlib import Path

import torch

_LIB_PATH = Path(__file__).resolve().with_name("libkvq.so")
_lib = None

STATUS_NAMES = {0: "KVQ_OK", 1: "KVQ_ERR_ARG", 2: "KVQ_ERR_SHAPE", 3: "KVQ_ERR_UNSUPPORTED",
                4: "KVQ_ERR_CAPACITY", 5: "KVQ_ERR_ALIGN", 6: "KVQ_ERR_CUDA"}
FLAG_OVERFLOW = 1
FLAG_WAIT_TIMEOUT = 2
FLAG_BAD_PAGE = 4

# Every symbol include/kvq.h declares.
EXPORTS = (
    "kvq_last_error", "kvq_version", "kvq_validate_config", "kvq_page_bytes",
    "kvq_cache_layout", "kvq_cache_bind", "kvq_cache_reset", "kvq_pack",
    "kvq_page_pool_bytes", "kvq_paged_cache_layout", "kvq_paged_cache_bind",
    "kvq_attn_workspace_bytes", "kvq_attn_default_splits", "kvq_attn_splits_for_lengths",
    "kvq_workspace_init",
    "kvq_decode_attn", "kvq_decode_attn_f32", "kvq_decode_step", "kvq_decode_step_f32",
    "kvq_decode_attn_noalloc", "dgap_workspace_bytes",
    "dgap_restore", "kvq_drift_max_vocab", "kvq_drift_metrics", "kvq_drift_window",
    "kvq_selftest_wait_timeout",
)
NOALLOC_SCRATCH_BYTES = 4 << 20


class KvqError(RuntimeError):
    def __init__(self, status, message):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {message}")
        self.status = status


class _Config(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "batch", "n_q_heads", "n_kv_heads", "head_dim", "bits_k", "bits_v",
        "group", "residual", "max_len")]


class _Cache(ctypes.Structure):
    _fields_ = [("pages", ctypes.c_void_p), ("k_resid", ctypes.c_void_p),
                ("v_resid", ctypes.c_void_p), ("seq_len", ctypes.c_void_p),
                ("block_table", ctypes.c_void_p), ("n_pages", ctypes.c_int32)]


class _DriftParams(ctypes.Structure):
    _fields_ = [("alpha", ctypes.c_float), ("window", ctypes.c_int32), ("k_max", ctypes.c_int32),
                ("eps", ctypes.c_float), ("rho_c", ctypes.c_float)]


class _DgapParams(ctypes.Structure):
    _fields_ = [("K", ctypes.c_int32), ("hidden", ctypes.c_int32), ("tau", ctypes.c_float)] + [
        (n, ctypes.c_void_p) for n in ("det_w1", "det_b1", "det_w2", "det_b2",
                                       "cor_w1", "cor_b1", "cor_w2", "cor_b2")]


def lib():
    """Load libkvq.so once (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not _LIB_PATH.exists():
            raise RuntimeError(f"{_LIB_PATH} is missing: build it with "
                               "paper_2607_16248_gb300.build.build()")
        L = ctypes.CDLL(str(_LIB_PATH))
        P, I32, SZ, F32 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_size_t, ctypes.c_float
        cfg_p = ctypes.POINTER(_Config)
        cache_p = ctypes.POINTER(_Cache)
        par_p = ctypes.POINTER(_DgapParams)
        sig = {
            "kvq_last_error": (ctypes.c_char_p, []),
            "kvq_version": (I32, []),
            "kvq_validate_config": (I32, [cfg_p]),
            "kvq_page_bytes": (SZ, [cfg_p]),
            "kvq_cache_layout": (I32, [cfg_p, ctypes.POINTER(SZ), ctypes.POINTER(SZ * 4)]),
            "kvq_cache_bind": (I32, [cfg_p, P, cache_p]),
            "kvq_page_pool_bytes": (SZ, [cfg_p, I32]),
            "kvq_paged_cache_layout": (I32, [cfg_p, ctypes.POINTER(SZ),
                                             ctypes.POINTER(SZ * 4)]),
            "kvq_paged_cache_bind": (I32, [cfg_p, P, P, I32, P, cache_p]),
            "kvq_cache_reset": (I32, [cfg_p, cache_p, P]),
            "kvq_pack": (I32, [cfg_p, cache_p, P, P, I32, I32, I32, P]),
            "kvq_attn_workspace_bytes": (SZ, [cfg_p, I32]),
            "kvq_attn_default_splits": (I32, [cfg_p]),
            "kvq_attn_splits_for_lengths": (I32, [cfg_p, ctypes.POINTER(I32)]),
            "kvq_workspace_init": (I32, [P, SZ, P]),
            "kvq_decode_attn": (I32, [cfg_p, cache_p, P, P, F32, I32, P, SZ, P]),
            "kvq_decode_attn_f32": (I32, [cfg_p, cache_p, P, P, F32, I32, P, SZ, P]),
            "kvq_decode_step": (I32, [cfg_p, cache_p, P, P, P, P, F32, I32, P, SZ, P]),
            "kvq_decode_step_f32": (I32, [cfg_p, cache_p, P, P, P, P, F32, I32, P, SZ, P]),
            "kvq_decode_attn_noalloc": (I32, [cfg_p, cache_p, P, P, F32, I32, P]),
            "dgap_workspace_bytes": (SZ, [I32, I32, par_p]),
            "dgap_restore": (I32, [par_p, P, I32, I32, P, P, P, P, P, P, P, SZ, P]),
            "kvq_drift_max_vocab": (I32, []),
            "kvq_selftest_wait_timeout": (I32, [P, P]),
            "kvq_drift_metrics": (I32, [P, P, I32, I32, ctypes.POINTER(_DriftParams),
                                        P, P, P, P, P, P]),
            "kvq_drift_window": (I32, [P, I32, I32, F32, P, P, P]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def last_error():
    return lib().kvq_last_error().decode()


def _check(status):
    if status != 0:
        raise KvqError(status, last_error())


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _dev(t, dtype, name):
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


# ---------------------------------------------------------------------------
# KV cache
# ---------------------------------------------------------------------------


@dataclass(frozen=True)
class CacheConfig:
    """KbVb cache shape (see kvq_config in include/kvq.h)."""
    batch: int
    n_q_heads: int
    n_kv_heads: int
    bits_k: int
    bits_v: int
    max_len: int
    residual: int = 128
    head_dim: int = 128
    group: int = 32

    def c(self):
        return _Config(self.batch, self.n_q_heads, self.n_kv_heads, self.head_dim,
                       self.bits_k, self.bits_v, self.group, self.residual, self.max_len)

    @property
    def ring(self):
        return self.residual + self.group

    @property
    def max_blocks(self):
        return self.max_len // self.group

    @property
    def page_bytes(self):
        return 512 * (self.bits_k + self.bits_v) + 1024

    def validate(self):
        c = self.c()
        _check(lib().kvq_validate_config(ctypes.byref(c)))

    def layout(self):
        c = self.c()
        total = ctypes.c_size_t()
        offs = (ctypes.c_size_t * 4)()
        _check(lib().kvq_cache_layout(ctypes.byref(c), ctypes.byref(total), ctypes.byref(offs)))
        return total.value, tuple(offs)


def packed_len(L, residual=128, group=32):
    """Tokens held in quantized blocks when L tokens are cached."""
    return group * (max(L - residual, 0) // group)


class QuantKVCache:
    """A KbVb cache bound through the C ABI.

    Contiguous (``n_pages=None``): one device buffer from kvq_cache_layout.
    Paged (``n_pages=N``): the fp16 rings and lengths in one buffer
    (kvq_paged_cache_layout), a pool of N page sets and a device block table
    [batch, max_len / 32] of int32 (all -1, i.e. unmapped, at first); the
    caller maps blocks with ``map_blocks`` before a call writes or reads them.
    """

    def __init__(self, cfg: CacheConfig, device="cuda", n_pages=None):
        self.cfg = cfg
        self.n_pages = n_pages
        c = cfg.c()
        if n_pages is None:
            total, self.offsets = cfg.layout()
        else:
            tot = ctypes.c_size_t()
            offs = (ctypes.c_size_t * 4)()
            _check(lib().kvq_paged_cache_layout(ctypes.byref(c), ctypes.byref(tot),
                                                ctypes.byref(offs)))
            total, self.offsets = tot.value, tuple(offs)
        self._raw = torch.empty(total + 256, dtype=torch.uint8, device=device)
        shift = (-self._raw.data_ptr()) % 256
        self.buffer = self._raw[shift:shift + total]
        self._c = _Cache()
        if n_pages is None:
            self.pool = None
            self.block_table = None
            _check(lib().kvq_cache_bind(ctypes.byref(c), ctypes.c_void_p(self.buffer.data_ptr()),
                                        ctypes.byref(self._c)))
        else:
            nbytes = lib().kvq_page_pool_bytes(ctypes.byref(c), int(n_pages))
            if nbytes == 0:
                raise KvqError(1, last_error())
            self.pool = torch.zeros(nbytes, dtype=torch.uint8, device=device)
            self.block_table = torch.full((cfg.batch, cfg.max_blocks), -1, dtype=torch.int32,
                                          device=device)
            _check(lib().kvq_paged_cache_bind(
                ctypes.byref(c), ctypes.c_void_p(self.buffer.data_ptr()),
                ctypes.c_void_p(self.pool.data_ptr()), int(n_pages),
                ctypes.c_void_p(self.block_table.data_ptr()), ctypes.byref(self._c)))
        self.reset()

    @property
    def paged(self):
        return self.n_pages is not None

    def map_blocks(self, b, blocks, page_sets):
        """Paged caches: block_table[b, blocks[i]] = page_sets[i] (a copy to
        the device on the current stream)."""
        if not self.paged:
            raise ValueError("map_blocks needs a paged cache")
        idx = torch.as_tensor(list(blocks), dtype=torch.long)
        val = torch.as_tensor(list(page_sets), dtype=torch.int32)
        self.block_table[b, idx.to(self.block_table.device)] = val.to(self.block_table.device)

    def reset(self, stream=None):
        c = self.cfg.c()
        _check(lib().kvq_cache_reset(ctypes.byref(c), ctypes.byref(self._c), _stream(stream)))

    # Views of the raw storage (layout of include/kvq.h).
    def pages(self):
        """Contiguous caches: the page array [batch, n_kv_heads, max_blocks,
        page_bytes]."""
        cfg = self.cfg
        if self.paged:
            raise ValueError("a paged cache has no page array: use head_pages")
        n = cfg.batch * cfg.n_kv_heads * cfg.max_blocks * cfg.page_bytes
        o = self.offsets[0]
        return self.buffer[o:o + n].view(cfg.batch, cfg.n_kv_heads, cfg.max_blocks,
                                         cfg.page_bytes)

    def pool_sets(self):
        """Paged caches: the pool as [n_pages, n_kv_heads, page_bytes]."""
        cfg = self.cfg
        return self.pool.view(self.n_pages, cfg.n_kv_heads, cfg.page_bytes)

    def head_pages(self, b, h, nb):
        """Blocks 0 .. nb - 1 of (sequence b, kv-head h) as [nb, page_bytes]
        (gathered through the block table for a paged cache)."""
        if not self.paged:
            return self.pages()[b, h, :nb]
        sets = self.block_table[b, :nb].long()
        return self.pool_sets()[sets, h]

    def resid(self):
        cfg = self.cfg
        n = cfg.batch * cfg.n_kv_heads * cfg.ring * cfg.head_dim * 2
        shape = (cfg.batch, cfg.n_kv_heads, cfg.ring, cfg.head_dim)
        k = self.buffer[self.offsets[1]:self.offsets[1] + n].view(torch.float16).view(shape)
        v = self.buffer[self.offsets[2]:self.offsets[2] + n].view(torch.float16).view(shape)
        return k, v

    def seq_region(self):
        o = self.offsets[3]
        return self.buffer[o:o + 4 * (2 * self.cfg.batch + 2)].view(torch.int32)

    def seq_lens(self):
        return self.seq_region()[:self.cfg.batch]

    def flags(self):
        return int(self.seq_region()[self.cfg.batch].item())


def blocks_written(L, n_new, residual=128, group=32):
    """Blocks a call that appends n_new tokens to a sequence of L tokens
    writes: [packed_len(L) / 32, packed_len(L + n_new) / 32)."""
    return range(packed_len(L, residual, group) // group,
                 packed_len(L + n_new, residual, group) // group)


def kvq_pack(cache: QuantKVCache, k_new, v_new, batch_begin=0, stream=None):
    """Append k_new/v_new fp16 [batch_count, n_kv_heads, n_new, 128] to
    sequences [batch_begin, batch_begin + batch_count)."""
    cfg = cache.cfg
    if k_new.dim() != 4 or k_new.shape != v_new.shape or k_new.shape[1] != cfg.n_kv_heads \
            or k_new.shape[3] != cfg.head_dim:
        raise ValueError("k_new/v_new must be [batch_count, n_kv_heads, n_new, 128]")
    c = cfg.c()
    _check(lib().kvq_pack(ctypes.byref(c), ctypes.byref(cache._c),
                          _dev(k_new, torch.float16, "k_new"), _dev(v_new, torch.float16, "v_new"),
                          k_new.shape[2], batch_begin, k_new.shape[0], _stream(stream)))


def attn_workspace(cfg: CacheConfig, n_splits=0, device="cuda"):
    c = cfg.c()
    n = lib().kvq_attn_workspace_bytes(ctypes.byref(c), n_splits)
    if n == 0:
        raise KvqError(1, last_error())
    return torch.zeros(n, dtype=torch.uint8, device=device)


def default_splits(cfg: CacheConfig):
    c = cfg.c()
    return lib().kvq_attn_default_splits(ctypes.byref(c))


def splits_for_lengths(cfg: CacheConfig, lengths):
    """kvq_attn_splits_for_lengths: the plan for host-known lengths, a split
    count (> 0, the split plan) or 0 (the flat plan)."""
    c = cfg.c()
    arr = (ctypes.c_int32 * cfg.batch)(*[int(x) for x in lengths])
    n = lib().kvq_attn_splits_for_lengths(ctypes.byref(c), arr)
    if n < 0:
        raise KvqError(1, last_error())
    return n


def _attn_out(q, out, out_dtype):
    """The output tensor and the entry-point suffix for its dtype."""
    if out is None:
        out = torch.empty(q.shape, dtype=out_dtype, device=q.device)
    if out.dtype == torch.float16:
        return out, ""
    if out.dtype == torch.float32:
        return out, "_f32"
    raise TypeError(f"out must be float16 or float32, got {out.dtype}")


def kvq_decode_attn(cache: QuantKVCache, q, out=None, softmax_scale=0.0, n_splits=0,
                    workspace=None, stream=None, out_dtype=torch.float16):
    """out = softmax(q K^T * scale) V over the cache; q fp16 [batch, n_q_heads, 128].

    out fp16 (the fp32 result rounded to nearest, kvq_decode_attn) or fp32
    (kvq_decode_attn_f32), picked by the dtype of ``out`` or ``out_dtype``."""
    cfg = cache.cfg
    if q.shape != (cfg.batch, cfg.n_q_heads, cfg.head_dim):
        raise ValueError(f"q must be [{cfg.batch}, {cfg.n_q_heads}, {cfg.head_dim}]")
    out, suffix = _attn_out(q, out, out_dtype)
    if out.shape != q.shape:
        raise ValueError("out must have the shape of q")
    if workspace is None:
        workspace = attn_workspace(cfg, n_splits, q.device)
    c = cfg.c()
    fn = getattr(lib(), "kvq_decode_attn" + suffix)
    _check(fn(ctypes.byref(c), ctypes.byref(cache._c), _dev(q, torch.float16, "q"),
              _dev(out, out.dtype, "out"), float(softmax_scale), n_splits,
              _dev(workspace, torch.uint8, "workspace"), workspace.numel(), _stream(stream)))
    return out


def kvq_decode_step(cache: QuantKVCache, k_new, v_new, q, out=None, softmax_scale=0.0,
                    n_splits=0, workspace=None, stream=None, out_dtype=torch.float16):
    """Append one token per sequence (k_new / v_new fp16 [batch, n_kv_heads, 128])
    and attend (q fp16 [batch, n_q_heads, 128] -> out fp16, or fp32 as in
    kvq_decode_attn) in one call: the same results as kvq_pack then
    kvq_decode_attn."""
    cfg = cache.cfg
    if q.shape != (cfg.batch, cfg.n_q_heads, cfg.head_dim):
        raise ValueError(f"q must be [{cfg.batch}, {cfg.n_q_heads}, {cfg.head_dim}]")
    for name, t in (("k_new", k_new), ("v_new", v_new)):
        if t.shape != (cfg.batch, cfg.n_kv_heads, cfg.head_dim):
            raise ValueError(f"{name} must be [{cfg.batch}, {cfg.n_kv_heads}, {cfg.head_dim}]")
    out, suffix = _attn_out(q, out, out_dtype)
    if out.shape != q.shape:
        raise ValueError("out must have the shape of q")
    if workspace is None:
        workspace = attn_workspace(cfg, n_splits, q.device)
    c = cfg.c()
    fn = getattr(lib(), "kvq_decode_step" + suffix)
    _check(fn(ctypes.byref(c), ctypes.byref(cache._c), _dev(k_new, torch.float16, "k_new"),
              _dev(v_new, torch.float16, "v_new"), _dev(q, torch.float16, "q"),
              _dev(out, out.dtype, "out"), float(softmax_scale), n_splits,
              _dev(workspace, torch.uint8, "workspace"), workspace.numel(), _stream(stream)))
    return out


def kvq_decode_attn_noalloc(cache: QuantKVCache, q, out, softmax_scale=0.0, n_splits=0,
                            stream=None):
    """kvq_decode_attn_f32 with the library's built-in scratch array instead of
    a workspace, for callers that cannot allocate device memory per step.
    ``out`` (fp32, the shape of q) is required: this wrapper allocates
    nothing either.  Calls share the array: do not let two of them overlap on
    the GPU."""
    cfg = cache.cfg
    if q.shape != (cfg.batch, cfg.n_q_heads, cfg.head_dim):
        raise ValueError(f"q must be [{cfg.batch}, {cfg.n_q_heads}, {cfg.head_dim}]")
    if out is None or out.shape != q.shape:
        raise ValueError("out must be a preallocated fp32 tensor of q's shape")
    c = cfg.c()
    _check(lib().kvq_decode_attn_noalloc(ctypes.byref(c), ctypes.byref(cache._c),
                                         _dev(q, torch.float16, "q"),
                                         _dev(out, torch.float32, "out"), float(softmax_scale),
                                         n_splits, _stream(stream)))
    return out


# ---------------------------------------------------------------------------
# DGAP epilogue
# ---------------------------------------------------------------------------


class DGAP:
    """Detector + corrector weights (device fp32) and the restore call."""

    def __init__(self, weights, K=32, tau=0.60, device="cuda"):
        self.K = int(K)
        self.tau = float(tau)
        self.w = {k: torch.as_tensor(v, dtype=torch.float32).to(device).contiguous()
                  for k, v in weights.items()}
        self.hidden = int(self.w["det_w1"].shape[0])
        nin = 5 * self.K + 8
        expect = {"det_w1": (self.hidden, 8), "det_b1": (self.hidden,),
                  "det_w2": (self.hidden,), "det_b2": (1,),
                  "cor_w1": (self.hidden, nin), "cor_b1": (self.hidden,),
                  "cor_w2": (self.K, self.hidden), "cor_b2": (self.K,)}
        for k, shp in expect.items():
            if tuple(self.w[k].shape) != shp:
                raise ValueError(f"{k} must have shape {shp}, got {tuple(self.w[k].shape)}")

    def params(self, tau=None):
        w = self.w
        return _DgapParams(self.K, self.hidden, float(self.tau if tau is None else tau),
                           *(ctypes.c_void_p(w[k].data_ptr()) for k in (
                               "det_w1", "det_b1", "det_w2", "det_b2",
                               "cor_w1", "cor_b1", "cor_w2", "cor_b2")))

    def workspace(self, batch, vocab, device="cuda"):
        p = self.params()
        n = lib().dgap_workspace_bytes(batch, vocab, ctypes.byref(p))
        if n == 0:
            raise KvqError(1, last_error())
        return torch.zeros(n, dtype=torch.uint8, device=device)

    def restore(self, logits, tau=None, outputs=None, workspace=None, features=True,
                next_token=True, stream=None):
        """Run dgap_restore on fp32 logits [batch, vocab] in place.

        Returns a dict of device tensors: topk_idx, topk_val, risk, gate,
        next_token, features (the last two may be None)."""
        if logits.dim() != 2:
            raise ValueError("logits must be [batch, vocab]")
        B, V = logits.shape
        dev = logits.device
        if outputs is None:
            outputs = dict(
                topk_idx=torch.empty(B, self.K, dtype=torch.int32, device=dev),
                topk_val=torch.empty(B, self.K, dtype=torch.float32, device=dev),
                risk=torch.empty(B, dtype=torch.float32, device=dev),
                gate=torch.empty(B, dtype=torch.uint8, device=dev),
                next_token=torch.empty(B, dtype=torch.int32, device=dev) if next_token else None,
                features=torch.empty(B, 8, dtype=torch.float32, device=dev) if features else None)
        if workspace is None:
            workspace = self.workspace(B, V, dev)
        p = self.params(tau)
        o = outputs

        def opt(t, dt, name):
            return ctypes.c_void_p(None) if t is None else _dev(t, dt, name)

        _check(lib().dgap_restore(
            ctypes.byref(p), _dev(logits, torch.float32, "logits"), B, V,
            _dev(o["topk_idx"], torch.int32, "topk_idx"),
            _dev(o["topk_val"], torch.float32, "topk_val"),
            _dev(o["risk"], torch.float32, "risk"), _dev(o["gate"], torch.uint8, "gate"),
            opt(o.get("next_token"), torch.int32, "next_token"),
            opt(o.get("features"), torch.float32, "features"),
            _dev(workspace, torch.uint8, "workspace"), workspace.numel(), _stream(stream)))
        return o


def logit(tau):
    """log(tau / (1 - tau)); the gate r > tau is f > logit(tau)."""
    if tau >= 1.0:
        return math.inf
    if tau <= 0.0:
        return -math.inf
    return math.log(tau / (1.0 - tau))


# ---------------------------------------------------------------------------
# Offline drift metrics (Sec. 4.1, Sec. 4.2)
# ---------------------------------------------------------------------------

def drift_metrics(z_fp, z_q, alpha, window, k_max, eps, rho_c, outputs=None, stream=None):
    """kvq_drift_metrics on paired fp32 logits [rows, vocab].

    Returns a dict of device tensors: m_t (int32), c_t, d_loc (fp32),
    y_t (uint8) per row and cov [rows, k_max] (fp32)."""
    if z_fp.dim() != 2 or z_fp.shape != z_q.shape:
        raise ValueError("z_fp and z_q must both be [rows, vocab]")
    R, V = z_fp.shape
    dev = z_fp.device
    if outputs is None:
        outputs = dict(m_t=torch.empty(R, dtype=torch.int32, device=dev),
                       c_t=torch.empty(R, dtype=torch.float32, device=dev),
                       d_loc=torch.empty(R, dtype=torch.float32, device=dev),
                       y_t=torch.empty(R, dtype=torch.uint8, device=dev),
                       cov=torch.empty(R, k_max, dtype=torch.float32, device=dev))
    o = outputs
    p = _DriftParams(float(alpha), int(window), int(k_max), float(eps), float(rho_c))
    _check(lib().kvq_drift_metrics(
        _dev(z_fp, torch.float32, "z_fp"), _dev(z_q, torch.float32, "z_q"), R, V, ctypes.byref(p),
        _dev(o["m_t"], torch.int32, "m_t"), _dev(o["c_t"], torch.float32, "c_t"),
        _dev(o["d_loc"], torch.float32, "d_loc"), _dev(o["y_t"], torch.uint8, "y_t"),
        _dev(o["cov"], torch.float32, "cov"), _stream(stream)))
    return o


def drift_window(cov, rho_k, stream=None):
    """kvq_drift_window: (K_b as a device int32 [1], mean coverage [k_max])."""
    if cov.dim() != 2:
        raise ValueError("cov must be [rows, k_max]")
    R, K = cov.shape
    mean = torch.empty(K, dtype=torch.float32, device=cov.device)
    kb = torch.empty(1, dtype=torch.int32, device=cov.device)
    _check(lib().kvq_drift_window(_dev(cov, torch.float32, "cov"), R, K, float(rho_k),
                                  _dev(mean, torch.float32, "mean_cov"),
                                  _dev(kb, torch.int32, "k_b"), _stream(stream)))
    return kb, mean


def selftest_wait_timeout(stream=None):
    """kvq_selftest_wait_timeout: the device flag word after a bounded wait on
    a copy that never arrives ran out (KVQ_FLAG_WAIT_TIMEOUT expected)."""
    flag = torch.zeros(1, dtype=torch.int32, device="cuda")
    _check(lib().kvq_selftest_wait_timeout(_dev(flag, torch.int32, "flag"), _stream(stream)))
    return flag
