"""ctypes binding of include/kvtier.h (argument marshalling only).

Every function here has the name of the C entry point it calls and passes
plain integers and device/host addresses through. All computation runs in
libkvtier.so's CUDA kernels; there is no fallback: importing this module
without the built library raises.

Device buffers may be given as torch tensors (their ``data_ptr()`` is passed)
or as integer addresses; streams as ``torch.cuda.Stream`` or raw handles.
"""
from __future__ import annotations

import ctypes as C
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libkvtier.so")

KV_OK = 0
KV_ERR_INVALID_ARG = -1
KV_ERR_BAD_STATE = -2
KV_ERR_NO_HOT_BLOCKS = -3
KV_ERR_NO_COLD_SPACE = -4
KV_ERR_CUDA = -5
KV_ERR_DEVICE_CHECK = -6
KV_SESSION_FREE, KV_SESSION_ACTIVE, KV_SESSION_PAUSED = 0, 1, 2
KV_POOL_HOST_LOGIC_ONLY = 1
KV_POOL_LRU_RESIDENCY = 2

_ERR_NAMES = {v: k for k, v in globals().items() if k.startswith("KV_ERR_")}

# Entry points declared in include/kvtier.h (checked by the export test).
EXPORTS = [
    "kv_pool_create", "kv_pool_destroy", "kv_block_bytes", "kv_token_bytes",
    "session_create", "session_create_paused", "session_destroy", "session_append",
    "decode_attention", "session_pause", "session_resume", "session_ready_event",
    "session_info", "session_block_table", "kv_pool_batch_tables", "kv_pool_shuffle_free",
    "kv_pool_free_list", "kv_pool_get_stats", "kv_pool_check_device",
    "kv_pool_inject_cuda_failure", "kv_last_error", "decode_attention_noalloc",
    "decode_attention_ex", "kv_pool_set_migration_limit", "kv_pool_batch_reserve",
    "decode_append_attention", "kv_pool_inject_decode_timeout", "kv_decode_splits",
    "session_block_table_device", "kv_pool_prefetch", "kv_pool_inject_stale_counter",
]

KV_DEVICE_BAD_BLOCK, KV_DEVICE_BAD_LENGTH, KV_DEVICE_TIMEOUT = 1, 2, 4
KV_DEVICE_STALE_COUNTERS = 8

KV_DECODE_OVERLAP_PREVIOUS = 1
KV_DECODE_OUT_BF16 = 2

KV_NOALLOC_SCRATCH_BYTES = 48 << 20


class kv_pool_config(C.Structure):
    _fields_ = [
        ("num_layers", C.c_int32), ("num_q_heads", C.c_int32), ("num_kv_heads", C.c_int32),
        ("head_dim", C.c_int32), ("block_tokens", C.c_int32), ("max_sessions", C.c_int32),
        ("max_batch", C.c_int32), ("device", C.c_int32), ("max_context", C.c_int64),
        ("num_hot_blocks", C.c_int64), ("hot_base", C.c_void_p), ("cold_bytes", C.c_int64),
        ("cold_base", C.c_void_p), ("alloc_seed", C.c_uint64), ("flags", C.c_uint32),
        ("reserved", C.c_uint32),
    ]


class kv_session_info(C.Structure):
    _fields_ = [
        ("state", C.c_int32), ("num_blocks", C.c_int32), ("tokens", C.c_int64),
        ("capacity", C.c_int64), ("cold_valid", C.c_int64), ("image", C.c_void_p),
    ]


class kv_pool_stats(C.Structure):
    _fields_ = [(n, C.c_int64) for n in (
        "free_blocks", "used_blocks", "cold_bytes_used", "bytes_unpacked", "bytes_packed",
        "bytes_appended", "resumes", "pauses", "appends", "decodes", "blocks_evicted",
        "resume_blocks_hit", "resume_blocks_missed", "batch_blocks_fetched",
        "blocks_prefetched", "prefetches")]


class KVError(RuntimeError):
    def __init__(self, code: int, where: str, msg: str):
        super().__init__(f"{where}: {_ERR_NAMES.get(code, code)}: {msg}")
        self.code = code


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is not built; run __graft_entry__.build() "
                          "(there is no CPU fallback for the CUDA path)")
    L = C.CDLL(LIB_PATH)
    p, i32, i64, u64 = C.c_void_p, C.c_int32, C.c_int64, C.c_uint64
    sig = {
        "kv_pool_create": [C.POINTER(kv_pool_config), C.POINTER(p)],
        "kv_pool_destroy": [p],
        "kv_block_bytes": [C.POINTER(kv_pool_config)],
        "kv_token_bytes": [C.POINTER(kv_pool_config)],
        "kv_decode_splits": [i64],
        "session_create": [p, i64, C.POINTER(i32)],
        "session_create_paused": [p, i64, i64, C.POINTER(i32)],
        "session_destroy": [p, i32],
        "session_append": [p, i32, p, p, i32, p],
        "kv_pool_batch_reserve": [p, p, i32, p, i32, p, p],
        "kv_pool_prefetch": [p, p, i32, p, i32, p],
        "decode_append_attention": [p, i32, p, p, p, p, p, i32, i32, C.c_float, p, C.c_uint32, p],
        "decode_attention": [p, i32, p, p, p, i32, i32, C.c_float, p, p],
        "decode_attention_ex": [p, i32, p, p, p, i32, i32, C.c_float, p, C.c_uint32, p],
        "session_pause": [p, i32, p],
        "session_resume": [p, i32, p],
        "session_ready_event": [p, i32, C.POINTER(p)],
        "session_info": [p, i32, C.POINTER(kv_session_info)],
        "session_block_table": [p, i32, p, i32, C.POINTER(i32)],
        "session_block_table_device": [p, i32, C.POINTER(p), C.POINTER(i32)],
        "kv_pool_batch_tables": [p, p, i32, p, i32, p, p],
        "kv_pool_shuffle_free": [p, u64],
        "kv_pool_free_list": [p, p, i64, C.POINTER(i64)],
        "kv_pool_get_stats": [p, C.POINTER(kv_pool_stats)],
        "kv_pool_check_device": [p, C.POINTER(i32)],
        "kv_pool_inject_cuda_failure": [p, i32],
        "kv_pool_inject_decode_timeout": [p, i32],
        "kv_pool_inject_stale_counter": [p],
        "kv_pool_set_migration_limit": [p, i32],
        "kv_last_error": [],
        "decode_attention_noalloc": [C.POINTER(kv_pool_config), i32, p, p, p, i32, i32,
                                     C.c_float, p, p],
    }
    for name, args in sig.items():
        f = getattr(L, name)
        f.argtypes = args
        f.restype = C.c_int
    L.kv_block_bytes.restype = i64
    L.kv_token_bytes.restype = i64
    L.kv_last_error.restype = C.c_char_p
    return L


lib = _load()


def _addr(x) -> int | None:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    if hasattr(x, "ctypes"):
        return x.ctypes.data
    raise TypeError(f"cannot take the address of {type(x)}")


def _stream(s) -> int | None:
    if s is None:
        return None
    if isinstance(s, int):
        return s
    return s.cuda_stream


def _check(rc: int, where: str) -> None:
    if rc != KV_OK:
        raise KVError(rc, where, kv_last_error())


def kv_last_error() -> str:
    return lib.kv_last_error().decode()


def kv_token_bytes(cfg: kv_pool_config) -> int:
    return int(lib.kv_token_bytes(C.byref(cfg)))


def kv_block_bytes(cfg: kv_pool_config) -> int:
    return int(lib.kv_block_bytes(C.byref(cfg)))


def kv_decode_splits(t: int) -> int:
    """Most KV splits a decode call makes per (session, head) for up to t tokens."""
    return int(lib.kv_decode_splits(t))


def kv_pool_create(cfg: kv_pool_config) -> int:
    out = C.c_void_p()
    _check(lib.kv_pool_create(C.byref(cfg), C.byref(out)), "kv_pool_create")
    return out.value


def kv_pool_destroy(pool: int) -> None:
    _check(lib.kv_pool_destroy(pool), "kv_pool_destroy")


def session_create(pool: int, max_tokens: int) -> int:
    sid = C.c_int32()
    _check(lib.session_create(pool, max_tokens, C.byref(sid)), "session_create")
    return sid.value


def session_create_paused(pool: int, max_tokens: int, tokens: int) -> int:
    sid = C.c_int32()
    _check(lib.session_create_paused(pool, max_tokens, tokens, C.byref(sid)),
           "session_create_paused")
    return sid.value


def session_destroy(pool: int, sid: int) -> None:
    _check(lib.session_destroy(pool, sid), "session_destroy")


def session_append(pool: int, sid: int, k, v, n: int, stream=None) -> None:
    _check(lib.session_append(pool, sid, _addr(k), _addr(v), n, _stream(stream)), "session_append")




def decode_append_attention(pool: int, layer: int, q, k_new, v_new, block_tables, seq_lens, B: int,
                            max_blocks: int, scale: float, out, flags: int = 0,
                            stream=None) -> None:
    _check(lib.decode_append_attention(pool, layer, _addr(q), _addr(k_new), _addr(v_new),
                                       _addr(block_tables), _addr(seq_lens), B, max_blocks, scale,
                                       _addr(out), flags, _stream(stream)),
           "decode_append_attention")


def decode_attention(pool: int, layer: int, q, block_tables, seq_lens, B: int, max_blocks: int,
                     scale: float, out, stream=None) -> None:
    _check(lib.decode_attention(pool, layer, _addr(q), _addr(block_tables), _addr(seq_lens), B,
                                max_blocks, scale, _addr(out), _stream(stream)),
           "decode_attention")


def decode_attention_ex(pool: int, layer: int, q, block_tables, seq_lens, B: int, max_blocks: int,
                        scale: float, out, flags: int, stream=None) -> None:
    _check(lib.decode_attention_ex(pool, layer, _addr(q), _addr(block_tables), _addr(seq_lens), B,
                                   max_blocks, scale, _addr(out), flags, _stream(stream)),
           "decode_attention_ex")


def session_pause(pool: int, sid: int, stream=None) -> None:
    _check(lib.session_pause(pool, sid, _stream(stream)), "session_pause")


def session_resume(pool: int, sid: int, stream=None) -> None:
    _check(lib.session_resume(pool, sid, _stream(stream)), "session_resume")


def session_ready_event(pool: int, sid: int) -> int | None:
    ev = C.c_void_p()
    _check(lib.session_ready_event(pool, sid, C.byref(ev)), "session_ready_event")
    return ev.value


def session_info(pool: int, sid: int) -> kv_session_info:
    info = kv_session_info()
    _check(lib.session_info(pool, sid, C.byref(info)), "session_info")
    return info


def session_block_table(pool: int, sid: int) -> list[int]:
    n = C.c_int32()
    _check(lib.session_block_table(pool, sid, None, 0, C.byref(n)), "session_block_table")
    buf = (C.c_int32 * max(1, n.value))()
    _check(lib.session_block_table(pool, sid, buf, n.value, C.byref(n)), "session_block_table")
    return list(buf[: n.value])


def session_block_table_device(pool: int, sid: int) -> tuple[int, int]:
    """(device address of the session's table row, number of logical blocks)."""
    row, n = C.c_void_p(), C.c_int32()
    _check(lib.session_block_table_device(pool, sid, C.byref(row), C.byref(n)),
           "session_block_table_device")
    return row.value, n.value


def kv_pool_batch_tables(pool: int, sids, block_tables, max_blocks: int, seq_lens,
                         stream=None) -> None:
    arr = (C.c_int32 * len(sids))(*sids)
    _check(lib.kv_pool_batch_tables(pool, arr, len(sids), _addr(block_tables), max_blocks,
                                    _addr(seq_lens), _stream(stream)), "kv_pool_batch_tables")


def kv_pool_batch_reserve(pool: int, sids, block_tables, max_blocks: int, seq_lens,
                          stream=None) -> None:
    arr = (C.c_int32 * len(sids))(*sids)
    _check(lib.kv_pool_batch_reserve(pool, arr, len(sids), _addr(block_tables), max_blocks,
                                     _addr(seq_lens), _stream(stream)), "kv_pool_batch_reserve")


def kv_pool_prefetch(pool: int, sids, busy=(), stream=None) -> None:
    arr = (C.c_int32 * len(sids))(*sids)
    barr = (C.c_int32 * len(busy))(*busy) if len(busy) else None
    _check(lib.kv_pool_prefetch(pool, arr, len(sids), barr, len(busy), _stream(stream)),
           "kv_pool_prefetch")


def kv_pool_shuffle_free(pool: int, seed: int) -> None:
    _check(lib.kv_pool_shuffle_free(pool, seed), "kv_pool_shuffle_free")


def kv_pool_free_list(pool: int) -> list[int]:
    n = C.c_int64()
    _check(lib.kv_pool_free_list(pool, None, 0, C.byref(n)), "kv_pool_free_list")
    buf = (C.c_int32 * max(1, n.value))()
    _check(lib.kv_pool_free_list(pool, buf, n.value, C.byref(n)), "kv_pool_free_list")
    return list(buf[: n.value])


def kv_pool_get_stats(pool: int) -> dict:
    st = kv_pool_stats()
    _check(lib.kv_pool_get_stats(pool, C.byref(st)), "kv_pool_get_stats")
    return {n: getattr(st, n) for n, _ in kv_pool_stats._fields_}


def kv_pool_check_device(pool: int) -> int:
    flags = C.c_int32()
    rc = lib.kv_pool_check_device(pool, C.byref(flags))
    if rc not in (KV_OK, KV_ERR_DEVICE_CHECK):
        _check(rc, "kv_pool_check_device")
    return flags.value


def kv_pool_inject_decode_timeout(pool: int, on: int = 1) -> None:
    _check(lib.kv_pool_inject_decode_timeout(pool, on), "kv_pool_inject_decode_timeout")


def kv_pool_inject_stale_counter(pool: int) -> None:
    _check(lib.kv_pool_inject_stale_counter(pool), "kv_pool_inject_stale_counter")


def kv_pool_set_migration_limit(pool: int, max_ctas: int) -> None:
    _check(lib.kv_pool_set_migration_limit(pool, max_ctas), "kv_pool_set_migration_limit")


def kv_pool_inject_cuda_failure(pool: int, n: int) -> None:
    _check(lib.kv_pool_inject_cuda_failure(pool, n), "kv_pool_inject_cuda_failure")


def decode_attention_noalloc(cfg: kv_pool_config, layer: int, q, block_tables, seq_lens, B: int,
                             max_blocks: int, scale: float, out, stream=None) -> None:
    """decode_attention for callers that cannot allocate: no pool, partials in
    the library's fixed device scratch (see include/kvtier.h)."""
    _check(lib.decode_attention_noalloc(C.byref(cfg), layer, _addr(q), _addr(block_tables),
                                        _addr(seq_lens), B, max_blocks, scale, _addr(out),
                                        _stream(stream)), "decode_attention_noalloc")


def make_config(*, num_layers: int, num_q_heads: int = 32, num_kv_heads: int = 4,
                head_dim: int = 128, block_tokens: int = 16, max_sessions: int = 64,
                max_batch: int = 64, device: int = 0, max_context: int = 32768,
                num_hot_blocks: int, hot_base=None, cold_bytes: int = 0, cold_base=None,
                alloc_seed: int = 0, flags: int = 0) -> kv_pool_config:
    c = kv_pool_config()
    c.num_layers, c.num_q_heads, c.num_kv_heads = num_layers, num_q_heads, num_kv_heads
    c.head_dim, c.block_tokens, c.max_sessions = head_dim, block_tokens, max_sessions
    c.max_batch, c.device, c.max_context = max_batch, device, max_context
    c.num_hot_blocks, c.hot_base = num_hot_blocks, _addr(hot_base)
    c.cold_bytes, c.cold_base = cold_bytes, _addr(cold_base)
    c.alloc_seed, c.flags = alloc_seed, flags
    return c
