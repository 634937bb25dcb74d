"""moe_permute_noalloc: the permutation for callers that cannot allocate.

Some callers may not call cudaMalloc or pass a workspace (a plugin inside an
inference engine that planned and owns all device memory before running). For
them the library offers one entry point that keeps its scratch in a fixed
array compiled into the library. This test checks, through the C ABI, that
it returns exactly what the workspace-based moe_permute returns, on two
calls in a row (the second call reuses the array the first one left behind),
also after the process's CUDA context was replaced (the array's address belongs
to a context), and that a problem larger than the array is refused before any
launch.
"""
import os
import subprocess
import sys

import numpy as np
import pytest
import torch

from paper_2601_14327_gb300 import _lib as L
from paper_2601_14327_gb300 import synth

pytestmark = pytest.mark.gpu


def _buffers(T, d, E, k):
    R = L.moe_perm_rows_max(T, k, E)
    dev = "cuda"
    return {"goff": torch.empty(E + 1, dtype=torch.int32, device=dev),
            "gcnt": torch.empty(E, dtype=torch.int32, device=dev),
            "row": torch.empty(T, k, dtype=torch.int32, device=dev),
            "xp": torch.zeros(R, d, dtype=torch.bfloat16, device=dev), "R": R}


@pytest.mark.parametrize("calls", [[(3000, 256, 64, 6, 11), (4097, 128, 200, 8, 12)]])
def test_permute_noalloc_matches_workspace_permute_twice(calls):
    for T, d, E, k, seed in calls:
        x = synth.make_layer_inputs(T, d, E, k, 128, seed=seed, with_weights=False,
                                    backward=False)["x"].cuda()
        rng = np.random.default_rng(seed)
        p = rng.dirichlet(np.full(E, 0.3))
        idx = np.stack([rng.choice(E, size=k, replace=False, p=p) for _ in range(T)])
        ti = torch.from_numpy(idx.astype(np.int32)).cuda()
        ref, got = _buffers(T, d, E, k), _buffers(T, d, E, k)
        ws_bytes = L.moe_workspace_size(T, d, E, k, 128)
        ws = torch.empty(ws_bytes, dtype=torch.uint8, device="cuda")
        L.moe_permute(x, ti, None, T, d, E, k, ref["R"], ref["goff"], ref["gcnt"], ref["row"],
                      ref["xp"], ws, ws_bytes)
        L.moe_permute_noalloc(x, ti, None, T, d, E, k, got["R"], got["goff"], got["gcnt"],
                              got["row"], got["xp"])
        torch.cuda.synchronize()
        assert L.moe_device_error(clear=True) == 0
        for n in ("goff", "gcnt", "row"):
            assert torch.equal(ref[n], got[n]), n
        used = int(ref["goff"][-1])
        assert torch.equal(ref["xp"][:used], got["xp"][:used])


def test_permute_noalloc_refuses_problems_beyond_its_array():
    # 256 experts x ceil(131073*8/4096) = 257 blocks > 65536 entries: refused on the host
    with pytest.raises(L.MoEError) as e:
        L.moe_permute_noalloc(16, 16, None, 131073, 128, 256, 8, 131073 * 8 + 256 * 128,
                              16, 16, 16, 16)
    assert e.value.status == -2
    assert "scratch" in str(e.value)


def test_permute_noalloc_after_device_reset():
    """The array's device address is looked up per CUDA context: after cudaDeviceReset
    the new context gets its own lookup, and the results still equal moe_permute's. The
    reset would end this process's torch context, so it runs in a child process."""
    script = os.path.join(os.path.dirname(os.path.abspath(__file__)), "gpu_noalloc_reset_check.py")
    r = subprocess.run([sys.executable, script], capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-4000:]
