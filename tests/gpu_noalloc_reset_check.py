"""Child-process half of test_zz_no_alloc.py::test_permute_noalloc_after_device_reset.

moe_permute_noalloc keeps its scratch in an array compiled into the library, whose
device address belongs to the CUDA context that loaded the library's module. This
process calls it, resets the device (cudaDeviceReset ends this process's context;
the next runtime call creates a new one), and calls it again on buffers of the new
context: both times the results must equal the workspace-based moe_permute's. The
process uses the CUDA runtime directly (no torch), so nothing of its own outlives the
reset."""
import ctypes
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(HERE))

import numpy as np  # noqa: E402

from paper_2601_14327_gb300 import _lib as L  # noqa: E402


def cudart():
    """The CUDA runtime the library itself uses (found among the loaded libraries)."""
    L.load()
    with open("/proc/self/maps") as f:
        paths = sorted({ln.split()[-1] for ln in f if "libcudart.so" in ln})
    assert paths, "libcudart not loaded"
    rt = ctypes.CDLL(paths[0])
    rt.cudaMalloc.argtypes = [ctypes.POINTER(ctypes.c_void_p), ctypes.c_size_t]
    rt.cudaFree.argtypes = [ctypes.c_void_p]
    rt.cudaMemcpy.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int]
    return rt


def check(rt, ok, what):
    assert ok == 0, f"{what}: cuda error {ok}"


class Dev:
    def __init__(self, rt):
        self.rt, self.ptrs = rt, []

    def alloc(self, nbytes):
        p = ctypes.c_void_p()
        check(self.rt, self.rt.cudaMalloc(ctypes.byref(p), max(nbytes, 16)), "cudaMalloc")
        self.ptrs.append(p.value)
        return p.value

    def put(self, a):
        a = np.ascontiguousarray(a)
        p = self.alloc(a.nbytes)
        check(self.rt, self.rt.cudaMemcpy(p, a.ctypes.data, a.nbytes, 1), "H2D")
        return p

    def get(self, p, shape, dtype):
        out = np.empty(shape, dtype)
        check(self.rt, self.rt.cudaMemcpy(out.ctypes.data, p, out.nbytes, 2), "D2H")
        return out

    def free(self):
        for p in self.ptrs:
            self.rt.cudaFree(p)
        self.ptrs = []


def one_round(rt, T, d, E, k, seed):
    rng = np.random.default_rng(seed)
    x = rng.integers(0, 1 << 16, size=(T, d), dtype=np.uint16) & np.uint16(0xBFFF)  # finite bf16
    p = rng.dirichlet(np.full(E, 0.3))
    idx = np.stack([rng.choice(E, size=k, replace=False, p=p) for _ in range(T)]).astype(np.int32)
    R = L.moe_perm_rows_max(T, k, E)
    ws_bytes = L.moe_workspace_size(T, d, E, k, 128)
    dev = Dev(rt)
    xd, idd, ws = dev.put(x), dev.put(idx), dev.alloc(ws_bytes)
    outs = []
    for noalloc in (False, True):
        goff, gcnt = dev.alloc(4 * (E + 1)), dev.alloc(4 * E)
        row, xp = dev.alloc(4 * T * k), dev.alloc(2 * R * d)
        if noalloc:
            L.moe_permute_noalloc(xd, idd, None, T, d, E, k, R, goff, gcnt, row, xp, stream=0)
        else:
            L.moe_permute(xd, idd, None, T, d, E, k, R, goff, gcnt, row, xp, ws, ws_bytes,
                          stream=0)
        check(rt, rt.cudaDeviceSynchronize(), "synchronize")
        go = dev.get(goff, (E + 1,), np.int32)
        outs.append((go, dev.get(gcnt, (E,), np.int32), dev.get(row, (T, k), np.int32),
                     dev.get(xp, (R, d), np.uint16)[:go[-1]]))
    assert L.moe_device_error(clear=True) == 0
    for a, b in zip(*outs):
        assert np.array_equal(a, b)
    dev.free()


if __name__ == "__main__":
    rt = cudart()
    one_round(rt, 3000, 256, 64, 6, 21)
    check(rt, rt.cudaDeviceReset(), "cudaDeviceReset")  # this process's context ends
    one_round(rt, 4097, 128, 200, 8, 22)                 # buffers of the new context
    one_round(rt, 1000, 64, 16, 2, 23)
    print("noalloc across a device reset: ok")
