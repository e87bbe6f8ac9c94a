"""Seeded synthetic decode workloads (inputs only; none of the method's arithmetic).

The generator recipe is documented in ``gen/ikvgen.h``.  Two compiled halves
draw identical numbers:

* ``libikvgen_host.so`` (gcc, OpenMP) -- used by the CPU oracle side;
* ``libikvgen_cuda.so`` (nvcc, sm_103a) -- fills multi-GB paged pools in HBM.

The five workload shapes follow the paper's two main backbones (Sec. 4.2:
Llama-3.1-8B with 8 KV heads / group 4, Qwen2.5-7B with 4 KV heads / group 7)
at 90% compression (10% budget, Sec. 4.3).  They stand in for the paper's
LongBench / RULER runs, whose datasets and model weights are not used here.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass, field, replace
from typing import List, Optional

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
HOST_LIB = os.path.join(HERE, "libikvgen_host.so")
CUDA_LIB = os.path.join(HERE, "libikvgen_cuda.so")

F32, BF16 = 0, 1


class Spec(ctypes.Structure):
    _fields_ = [
        ("seed", ctypes.c_uint64),
        ("batch", ctypes.c_int32),
        ("layers", ctypes.c_int32),
        ("kv_heads", ctypes.c_int32),
        ("head_dim", ctypes.c_int32),
        ("heavy_per_10000", ctypes.c_int32),
        ("n_sinks", ctypes.c_int32),
        ("sink_scale", ctypes.c_float),
        ("heavy_u_scale", ctypes.c_float),
        ("heavy_noise", ctypes.c_float),
    ]


def build(force: bool = False, cuda: bool = True, arch: str = "103a") -> None:
    """Compile the host and (optionally) device halves in place."""
    hdr = os.path.join(HERE, "ikvgen.h")
    jobs = []
    src = os.path.join(HERE, "ikvgen_host.c")
    if force or _stale(HOST_LIB, [src, hdr]):
        jobs.append(["gcc", "-O2", "-fPIC", "-shared", "-fopenmp", "-ffp-contract=off", "-std=c11",
                     "-o", HOST_LIB, src, "-lm"])
    csrc = os.path.join(HERE, "ikvgen_cuda.cu")
    if cuda and (force or _stale(CUDA_LIB, [csrc, hdr])):
        jobs.append(["nvcc", "-O3", "-shared", "-Xcompiler", "-fPIC", "-std=c++17",
                     f"-gencode=arch=compute_{arch},code=sm_{arch}", "-fmad=false",
                     "-o", CUDA_LIB, csrc])
    procs = [subprocess.Popen(j, stdout=subprocess.PIPE, stderr=subprocess.STDOUT) for j in jobs]
    for j, p in zip(jobs, procs):
        out, _ = p.communicate()
        if p.returncode != 0:
            raise RuntimeError("gen build failed: %s\n%s" % (" ".join(j), out.decode()))


def _stale(target: str, deps: List[str]) -> bool:
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(d) > t for d in deps)


_host = None
_cuda = None


def host_lib():
    global _host
    if _host is None:
        if not os.path.exists(HOST_LIB):
            build(cuda=False)
        lib = ctypes.CDLL(HOST_LIB)
        P, I32, I64, U64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint64
        lib.ikvgen_u_table.argtypes = [U64, I32, I32, I32, P]
        lib.ikvgen_kv_block.argtypes = [ctypes.POINTER(Spec), P, I32, I32, I64, I64, I32, P, P]
        lib.ikvgen_heavy_flags.argtypes = [ctypes.POINTER(Spec), I32, I64, I64, P]
        lib.ikvgen_kv_rows_at.argtypes = [ctypes.POINTER(Spec), P, I32, I32, P, I64, I32, P, P]
        lib.ikvgen_queries.argtypes = [U64, I32, I32, I32, I32, I32, P, I32, I32, I32, I32, P]
        lib.ikvgen_lengths.argtypes = [U64, I32, I32, I32, P]
        lib.ikvgen_normals.argtypes = [U64, U64, I64, P]
        lib.ikvgen_mix64_host.argtypes = [U64]
        lib.ikvgen_mix64_host.restype = U64
        _host = lib
    return _host


def cuda_lib():
    global _cuda
    if _cuda is None:
        if not os.path.exists(CUDA_LIB):
            raise RuntimeError("libikvgen_cuda.so missing: run __graft_entry__.build()")
        lib = ctypes.CDLL(CUDA_LIB)
        P, I32, I64, U64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint64
        lib.ikvgen_fill_paged_cuda.argtypes = [ctypes.POINTER(Spec), P, P, P, P, P, I32, I32, I32, I32, I32, P]
        lib.ikvgen_fill_tokens_cuda.argtypes = [ctypes.POINTER(Spec), P, P, I32, I32, I32, P, P, P]
        lib.ikvgen_normals_cuda.argtypes = [U64, U64, I64, P, P]
        for f in (lib.ikvgen_fill_paged_cuda, lib.ikvgen_fill_tokens_cuda, lib.ikvgen_normals_cuda):
            f.restype = ctypes.c_int
        _cuda = lib
    return _cuda


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data


@dataclass
class Workload:
    """One synthetic decode workload (shape, schedule and generator parameters)."""

    name: str
    batch: int
    layers: int
    q_heads: int
    kv_heads: int
    head_dim: int
    prefill: List[int]                 # L0 per sequence
    steps: int
    dtype: int = BF16
    alpha: float = 0.9
    budget_frac: float = 0.1
    refresh_period: int = 1
    score_free: bool = False
    seed: int = 0
    query_mode: int = 1                # 0: w_t = 0.5 eps_t (iid), 1: random walk, step noise 0.1
    n_sinks: int = 4
    sink_scale: float = 4.0
    heavy_per_10000: int = 100
    page_size: int = 64
    extra_cap: int = 0                 # spare slots per sequence beyond max(L0)+1

    @property
    def group(self) -> int:
        return self.q_heads // self.kv_heads

    def budgets(self) -> List[int]:
        """Decode budget per sequence: round-half-up of budget_frac * L0 (the paper's
        B = floor((1-rho) L0) differs by at most one; the library takes B explicitly)."""
        return [int(np.floor(self.budget_frac * L0 + 0.5)) for L0 in self.prefill]

    def budgets_floor(self) -> List[int]:
        return [int(np.floor(self.budget_frac * L0)) for L0 in self.prefill]

    def spec(self) -> Spec:
        return Spec(self.seed, self.batch, self.layers, self.kv_heads, self.head_dim, self.heavy_per_10000,
                    self.n_sinks, self.sink_scale, 3.0, 0.3)

    @property
    def cap(self) -> int:
        c = max(self.prefill) + 1 + self.extra_cap
        return (c + self.page_size - 1) // self.page_size * self.page_size

    @property
    def pages_per_seq(self) -> int:
        return self.cap // self.page_size

    # ---- host draws -------------------------------------------------------
    def u_table(self) -> np.ndarray:
        out = np.empty((self.layers, self.kv_heads, self.head_dim), np.float32)
        host_lib().ikvgen_u_table(self.seed, self.layers, self.kv_heads, self.head_dim, _ptr(out))
        return out

    def kv_block(self, b: int, layer: int, p0: int, count: int, u: Optional[np.ndarray] = None,
                 dtype: Optional[int] = None):
        """Keys and values [kv_heads][count][d] for positions [p0, p0+count): float32
        arrays holding exactly the values stored in the cache (bf16 values widened)."""
        u = self.u_table() if u is None else u
        dt = self.dtype if dtype is None else dtype
        sp = self.spec()
        shape = (self.kv_heads, count, self.head_dim)
        if dt == BF16:
            k = np.empty(shape, np.uint16)
            v = np.empty(shape, np.uint16)
        else:
            k = np.empty(shape, np.float32)
            v = np.empty(shape, np.float32)
        host_lib().ikvgen_kv_block(ctypes.byref(sp), _ptr(u), b, layer, p0, count, dt, _ptr(k), _ptr(v))
        if dt == BF16:
            return bf16_to_f32(k), bf16_to_f32(v)
        return k, v

    def kv_rows(self, b: int, layer: int, positions, u: Optional[np.ndarray] = None):
        """Keys and values [kv_heads][count][d] at arbitrary original positions (float32
        arrays holding exactly the stored values)."""
        u = self.u_table() if u is None else u
        pos = np.ascontiguousarray(np.asarray(positions, dtype=np.int64))
        n = pos.shape[0]
        shape = (self.kv_heads, n, self.head_dim)
        dt = np.uint16 if self.dtype == BF16 else np.float32
        k = np.empty(shape, dt)
        v = np.empty(shape, dt)
        sp = self.spec()
        host_lib().ikvgen_kv_rows_at(ctypes.byref(sp), _ptr(u), b, layer, _ptr(pos), n, self.dtype, _ptr(k), _ptr(v))
        if self.dtype == BF16:
            return bf16_to_f32(k), bf16_to_f32(v)
        return k, v

    def heavy_flags(self, b: int, p0: int, count: int) -> np.ndarray:
        out = np.empty(count, np.uint8)
        sp = self.spec()
        host_lib().ikvgen_heavy_flags(ctypes.byref(sp), b, p0, count, _ptr(out))
        return out

    def queries(self, t0: int, t1: int, u: Optional[np.ndarray] = None) -> np.ndarray:
        """Queries for decode steps [t0, t1): [t1-t0][layers][batch][q_heads][d] in the
        storage dtype (uint16 bf16 bits or float32)."""
        u = self.u_table() if u is None else u
        shape = (t1 - t0, self.layers, self.batch, self.q_heads, self.head_dim)
        out = np.empty(shape, np.uint16 if self.dtype == BF16 else np.float32)
        host_lib().ikvgen_queries(self.seed, self.batch, self.layers, self.q_heads, self.kv_heads, self.head_dim,
                                  _ptr(u), self.query_mode, t0, t1, self.dtype, _ptr(out))
        return out

    def new_tokens(self, t: int, u: Optional[np.ndarray] = None):
        """Appended K, V at decode step t: [layers][batch][kv_heads][d] float32 values."""
        u = self.u_table() if u is None else u
        K = np.empty((self.layers, self.batch, self.kv_heads, self.head_dim), np.float32)
        V = np.empty_like(K)
        for b in range(self.batch):
            for layer in range(self.layers):
                k, v = self.kv_block(b, layer, self.prefill[b] + t - 1, 1, u)
                K[layer, b] = k[:, 0]
                V[layer, b] = v[:, 0]
        return K, V

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    return (bits.astype(np.uint32) << 16).view(np.float32)


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round-to-nearest-even fp32 -> bf16 bits (finite inputs)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = u + 0x7FFF + ((u >> 16) & 1)
    return (u >> 16).astype(np.uint16)


def lengths(seed: int, batch: int, lo: int, hi: int) -> List[int]:
    out = np.empty(batch, np.int32)
    host_lib().ikvgen_lengths(seed, batch, lo, hi, _ptr(out))
    return [int(x) for x in out]


def config(i: int) -> Workload:
    """The five decode workloads (sizes of the paper's backbones; synthetic inputs)."""
    if i == 0:
        return Workload("tiny-fp32", 1, 2, 4, 2, 64, [512], 16, dtype=F32, alpha=0.9, seed=0, query_mode=0,
                        n_sinks=0, sink_scale=1.0)
    if i == 1:
        return Workload("llama8b-b1-32k", 1, 32, 32, 8, 128, [32768], 256, seed=1)
    if i == 2:
        return Workload("llama8b-b16-4k8k", 16, 32, 32, 8, 128, lengths(2, 16, 4096, 8192), 512, seed=2,
                        refresh_period=4)
    if i == 3:
        return Workload("llama8b-b8-64k", 8, 32, 32, 8, 128, [65536] * 8, 256, seed=3, score_free=True)
    if i == 4:
        return Workload("qwen7b-b32-16k", 32, 28, 28, 4, 128, [16384] * 32, 256, seed=4)
    raise ValueError(i)
