"""CPU oracle for the hot/cold KV tiering hot path (test infrastructure).

Only the tests, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline
leg import this package; the CUDA library and its Python binding never do.
The arithmetic lives in ``oracle.c`` (plain C, double precision, OpenMP over
(layer, session, head)); this module compiles it with gcc and marshals numpy
arrays into it.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile liboracle.so with gcc (OpenMP when the compiler has it)."""
    if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC):
        return _LIB
    base = ["gcc", "-O2", "-std=c11", "-shared", "-fPIC", _SRC, "-o", _LIB + ".tmp", "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True, capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(_LIB + ".tmp", _LIB)
    return _LIB


def lib():
    global _lib
    if _lib is None:
        build()
        L = C.CDLL(_LIB)
        p = C.c_void_p
        i32, i64, u64 = C.c_int32, C.c_int64, C.c_uint64
        L.oracle_threads.restype = C.c_int
        L.oracle_kv_bytes_per_token.restype = i64
        L.oracle_kv_bytes_per_token.argtypes = [C.c_int, C.c_int, C.c_int]
        L.oracle_paged_decode.restype = C.c_int
        L.oracle_paged_decode.argtypes = [p, i64, C.c_int, C.c_int, C.c_int, C.c_int, C.c_int,
                                          C.c_int, C.c_int, p, p, C.c_int, p, C.c_int,
                                          C.c_double, p, C.c_int]
        L.oracle_unpack.restype = C.c_int
        L.oracle_unpack.argtypes = [p, i64, i64, p, p, i64, C.c_int, C.c_int, C.c_int, C.c_int]
        L.oracle_pack.restype = i64
        L.oracle_pack.argtypes = [p, i64, p, i64, i64, p, i64, C.c_int, C.c_int, C.c_int, C.c_int]
        L.oracle_append.restype = C.c_int
        L.oracle_append.argtypes = [p, i64, p, i64, C.c_int, p, p, C.c_int, C.c_int, C.c_int,
                                    C.c_int]
        L.oracle_splitmix64.restype = u64
        L.oracle_splitmix64.argtypes = [C.POINTER(u64)]
        L.oracle_shuffle.restype = None
        L.oracle_shuffle.argtypes = [p, i64, u64]
        L.oracle_free_list_init.restype = None
        L.oracle_free_list_init.argtypes = [p, i64, u64]
        L.oracle_free_list_pop.restype = i64
        L.oracle_free_list_pop.argtypes = [p, i64, i64, p]
        L.oracle_free_list_push.restype = i64
        L.oracle_free_list_push.argtypes = [p, i64, p, i64]
        del i32
        _lib = L
    return _lib


def _ptr(a: np.ndarray):
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(C.c_void_p)


def threads() -> int:
    return int(lib().oracle_threads())


def kv_bytes_per_token(L: int, Hkv: int, D: int) -> int:
    return int(lib().oracle_kv_bytes_per_token(L, Hkv, D))


def paged_decode(hot: np.ndarray, q: np.ndarray, tables: np.ndarray, seq_lens,
                 scale: float, num_q_heads: int, layer0: int = 0, nthreads: int = 0) -> np.ndarray:
    """hot [NB][L][2][Hkv][bt][D] uint16; q [nl][B][Hq][D] uint16 for layers
    layer0 .. layer0+nl-1; tables [B][max_blocks] int32. Returns float64
    out [nl][B][Hq][D]."""
    NB, L, two, Hkv, bt, D = hot.shape
    assert two == 2
    q = np.ascontiguousarray(q, dtype=np.uint16)
    nl, B, Hq, Dq = q.shape
    assert Hq == num_q_heads and Dq == D
    tables = np.ascontiguousarray(tables, dtype=np.int32)
    lens = np.ascontiguousarray(np.asarray(seq_lens, dtype=np.int32))
    out = np.zeros((nl, B, Hq, D), dtype=np.float64)
    hot = np.ascontiguousarray(hot, dtype=np.uint16)
    rc = lib().oracle_paged_decode(_ptr(hot), NB, L, Hq, Hkv, D, bt, layer0, nl, _ptr(q),
                                   _ptr(tables), tables.shape[1], _ptr(lens), B, float(scale),
                                   _ptr(out), int(nthreads))
    if rc != 0:
        raise ValueError("oracle_paged_decode rejected its arguments")
    return out


def unpack(img: np.ndarray, T: int, table_row, hot: np.ndarray) -> None:
    """In place: image tokens [0, T) into the blocks of table_row."""
    L, two, Hkv, T_cap, D = img.shape
    NB, L2, _, _, bt, _ = hot.shape
    row = np.ascontiguousarray(np.asarray(table_row, dtype=np.int32))
    rc = lib().oracle_unpack(_ptr(img), T_cap, T, _ptr(row), _ptr(hot), NB, L, Hkv, D, bt)
    if rc != 0:
        raise ValueError("oracle_unpack rejected its arguments")


def pack(hot: np.ndarray, table_row, t0: int, T: int, img: np.ndarray) -> int:
    """In place: hot tokens [t0, T) into the image; returns bytes written."""
    L, two, Hkv, T_cap, D = img.shape
    NB, _, _, _, bt, _ = hot.shape
    row = np.ascontiguousarray(np.asarray(table_row, dtype=np.int32))
    n = lib().oracle_pack(_ptr(hot), NB, _ptr(row), t0, T, _ptr(img), T_cap, L, Hkv, D, bt)
    if n < 0:
        raise ValueError("oracle_pack rejected its arguments")
    return int(n)


def append(hot: np.ndarray, table_row, pos0: int, k: np.ndarray, v: np.ndarray) -> None:
    """In place: k, v [L][n][Hkv][D] at logical positions pos0 .. pos0+n-1."""
    NB, L, _, Hkv, bt, D = hot.shape
    k = np.ascontiguousarray(k, dtype=np.uint16)
    v = np.ascontiguousarray(v, dtype=np.uint16)
    n = k.shape[1]
    row = np.ascontiguousarray(np.asarray(table_row, dtype=np.int32))
    rc = lib().oracle_append(_ptr(hot), NB, _ptr(row), pos0, n, _ptr(k), _ptr(v), L, Hkv, D, bt)
    if rc != 0:
        raise ValueError("oracle_append rejected its arguments")


def splitmix64_stream(seed: int, n: int) -> list[int]:
    st = C.c_uint64(seed)
    return [int(lib().oracle_splitmix64(C.byref(st))) for _ in range(n)]


def shuffle(lst: np.ndarray, seed: int) -> np.ndarray:
    a = np.ascontiguousarray(np.asarray(lst, dtype=np.int32)).copy()
    lib().oracle_shuffle(_ptr(a), len(a), seed)
    return a


class FreeList:
    """The placement contract: a list shuffled by seed, popped from the end."""

    def __init__(self, num_blocks: int, seed: int):
        self.buf = np.zeros(num_blocks, dtype=np.int32)
        lib().oracle_free_list_init(_ptr(self.buf), num_blocks, seed)
        self.n = num_blocks

    def pop(self, count: int) -> np.ndarray:
        out = np.zeros(count, dtype=np.int32)
        n = lib().oracle_free_list_pop(_ptr(self.buf), self.n, count, _ptr(out))
        if n < 0:
            raise MemoryError("free list exhausted")
        self.n = int(n)
        return out

    def push(self, blocks) -> None:
        b = np.ascontiguousarray(np.asarray(blocks, dtype=np.int32))
        self.n = int(lib().oracle_free_list_push(_ptr(self.buf), self.n, _ptr(b), len(b)))

    def shuffle(self, seed: int) -> None:
        lib().oracle_shuffle(_ptr(self.buf), self.n, seed)

    def contents(self) -> np.ndarray:
        return self.buf[: self.n].copy()
