"""cure_tree_attn_noalloc against cure_tree_attn (GPU).

The no-allocation entry point serves callers that cannot allocate device
memory (for example a plugin whose host framework owns all of HBM and hands
it only its inputs and outputs): it keeps the split-KV workspace in a fixed
64 MiB static device array instead of a caller buffer.  It must give the
same attention output as the workspace-taking entry point, call after call,
even though every call reuses the array's previous contents.

This file is collected last so that a failure here stops a `-x` run only
after every other test has run.
"""
import ctypes as C
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2608_00531_gb300 import workload as W

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda:0")
TOL = 2e-2            # the absolute tolerance of the attention parity tests
SCRATCH = 64 * 1024 * 1024
CAPACITY = 2


@pytest.fixture(scope="module")
def env():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    from paper_2608_00531_gb300 import _lib, cure
    torch.cuda.set_device(DEV)
    lib = _lib.load()
    P, I32 = C.c_void_p, C.c_int32
    lib.cure_tree_attn_noalloc.argtypes = [P, P, P, P, P, C.POINTER(_lib.KVDesc), P, P, P, I32, I32, I32,
                                           C.c_float, P, P]
    lib.cure_tree_attn_noalloc.restype = C.c_int
    return lib, cure


def _inputs(seed, B=4, K=16, budget=16, Hq=28, Hkv=4, lens=(0, 37, 1500, 4000)):
    rng = np.random.default_rng(seed)
    margin = (rng.integers(0, 8, size=(B, K)) * 0.25).astype(np.float32)
    ids = rng.integers(0, 1000, size=(B, K, 3))
    L = np.asarray(lens, dtype=np.int32)
    t = oracle.build_tree(ids, margin, rng.integers(0, 1000, size=B), L, 1.0, budget, 3, 1)
    N = 1 + K + budget
    table, npages = W.block_table(L, K, seed)
    q = W.normal_bf16((B, N, Hq, 128), 1.0, rng).to(DEV)
    tk = W.normal_bf16((B, N, Hkv, 128), 1.0, rng).to(DEV)
    tv = W.normal_bf16((B, N, Hkv, 128), 1.0, rng).to(DEV)
    kc = W.normal_bf16((npages, 16, Hkv, 128), 1.0, rng).to(DEV)
    vc = W.normal_bf16((npages, 16, Hkv, 128), 1.0, rng).to(DEV)
    return dict(t=t, q=q, tk=tk, tv=tv, kc=kc, vc=vc, L=torch.from_numpy(L).to(DEV),
                table=torch.from_numpy(table).to(DEV), npages=npages, B=B, N=N, Hq=Hq, Hkv=Hkv,
                n=torch.from_numpy(t["n_nodes"].astype(np.int32)).to(DEV),
                anc=torch.from_numpy(t["anc"].view(np.int64)).to(DEV))


def _call_noalloc(lib, x, kv, out, in_place=False):
    s = C.c_void_p(torch.cuda.current_stream().cuda_stream)
    tk, tv = (None, None) if in_place else (x["tk"].data_ptr(), x["tv"].data_ptr())
    return lib.cure_tree_attn_noalloc(
        x["q"].data_ptr(), tk, tv, x["kc"].data_ptr(), x["vc"].data_ptr(),
        C.byref(kv), x["L"].data_ptr(), x["n"].data_ptr(), x["anc"].data_ptr(), x["B"], x["N"], x["Hq"],
        1.0 / math.sqrt(128), out.data_ptr(), s)


def test_noalloc_matches_workspace_entry_point_on_two_calls(env):
    lib, cure = env
    for call, seed in enumerate((1, 2)):     # two calls in a row, different inputs
        x = _inputs(seed)
        kv = cure.kv_desc(x["Hkv"], 128, x["table"].shape[1], x["table"], 16, x["npages"])
        assert cure.cure_tree_attn_workspace_size(x["B"], x["N"], x["Hq"], kv) <= SCRATCH
        ref = cure.cure_tree_attn(x["q"], x["tk"], x["tv"], x["kc"], x["vc"], kv, x["L"], x["n"], x["anc"],
                                  1.0 / math.sqrt(128))
        out = torch.full_like(ref, float("nan"))
        assert _call_noalloc(lib, x, kv, out) == 0
        torch.cuda.synchronize()
        assert cure.cure_device_error() == 0
        for b in range(x["B"]):
            nb = int(x["t"]["n_nodes"][b])
            got = out[b, :nb].float()
            want = ref[b, :nb].float()
            assert torch.isfinite(got).all(), (call, b)
            assert float((got - want).abs().max()) <= TOL, (call, b)


def test_noalloc_in_place_layout(env):
    """Both tree tensors NULL: the in-place layout (node j's rows at cache
    slot L + j), as in cure_tree_attn."""
    lib, cure = env
    x = _inputs(4)
    L = x["L"].cpu().numpy()
    table, npages = W.block_table(L, x["N"] - 1, 4)      # pages up to slot L + N - 1
    rng = np.random.default_rng(4)
    kc = W.normal_bf16((npages, 16, x["Hkv"], 128), 1.0, rng).to(DEV)
    vc = W.normal_bf16((npages, 16, x["Hkv"], 128), 1.0, rng).to(DEV)
    for b in range(x["B"]):
        for j in range(int(x["t"]["n_nodes"][b])):
            sl = int(L[b]) + j
            kc[int(table[b, sl // 16]), sl % 16] = x["tk"][b, j]
            vc[int(table[b, sl // 16]), sl % 16] = x["tv"][b, j]
    x = dict(x, kc=kc, vc=vc, table=torch.from_numpy(table).to(DEV), npages=npages)
    kv = cure.kv_desc(x["Hkv"], 128, table.shape[1], x["table"], 16, npages)
    ref = cure.cure_tree_attn(x["q"], None, None, kc, vc, kv, x["L"], x["n"], x["anc"], 1.0 / math.sqrt(128))
    sep = cure.cure_tree_attn(x["q"], x["tk"], x["tv"], kc, vc, kv, x["L"], x["n"], x["anc"],
                              1.0 / math.sqrt(128))
    out = torch.full_like(ref, float("nan"))
    assert _call_noalloc(lib, x, kv, out, in_place=True) == 0
    torch.cuda.synchronize()
    assert cure.cure_device_error() == 0
    for b in range(x["B"]):
        nb = int(x["t"]["n_nodes"][b])
        got = out[b, :nb].float()
        assert torch.isfinite(got).all(), b
        assert float((got - ref[b, :nb].float()).abs().max()) <= TOL, b
        assert float((got - sep[b, :nb].float()).abs().max()) <= TOL, b     # the same attention


def test_noalloc_rejects_shapes_beyond_its_scratch(env):
    lib, cure = env
    x = _inputs(3)
    # batch 200 with 28/4 heads needs more split-KV scratch than 64 MiB; the
    # buffers are too small for that batch, but nothing may be launched
    kv = cure.kv_desc(x["Hkv"], 128, x["table"].shape[1], x["table"], 16, x["npages"])
    assert cure.cure_tree_attn_workspace_size(200, x["N"], x["Hq"], kv) > SCRATCH
    out = torch.zeros_like(x["q"])
    big = dict(x, B=200)
    assert _call_noalloc(lib, big, kv, out) == CAPACITY
    torch.cuda.synchronize()
    assert int(out.abs().sum()) == 0      # nothing was launched
