"""The oracle's Philox4x32-10 against NVIDIA's implementation (cuRAND's
device function curand_Philox4x32_10, a library call): the raw four-word
outputs must be equal for every counter and key.  This pins the generator
both sides draw their random numbers from to an implementation written by
somebody else.  The test kernel is compiled here with nvcc; it is test
infrastructure and shares nothing with the library."""
import ctypes as C
import os
import shutil
import subprocess

import numpy as np
import pytest
import torch

import oracle as O

pytestmark = pytest.mark.gpu

SRC = r"""
#include <curand_kernel.h>
__global__ void philox_kernel(const uint4* c, const uint2* k, uint4* out, int n) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) out[i] = curand_Philox4x32_10(c[i], k[i]);
}
extern "C" int philox_launch(const void* c, const void* k, void* out, int n) {
  philox_kernel<<<(n + 127) / 128, 128>>>(static_cast<const uint4*>(c), static_cast<const uint2*>(k),
                                         static_cast<uint4*>(out), n);
  return (int)cudaGetLastError();
}
"""


def _build(tmp_path):
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    src = os.path.join(tmp_path, "philox_curand.cu")
    lib = os.path.join(tmp_path, "libphilox_curand.so")
    with open(src, "w") as f:
        f.write(SRC)
    subprocess.check_call([nvcc, "-shared", "-Xcompiler", "-fPIC", "-gencode", "arch=compute_103a,code=sm_103a",
                           "-o", lib, src])
    so = C.CDLL(lib)
    so.philox_launch.restype = C.c_int
    so.philox_launch.argtypes = [C.c_void_p, C.c_void_p, C.c_void_p, C.c_int]
    return so


def test_oracle_philox_matches_curand(tmp_path):
    so = _build(str(tmp_path))
    rng = np.random.default_rng(17)
    n = 4096
    ctr = rng.integers(0, 2**32, (n, 4), dtype=np.uint64).astype(np.uint32)
    key = rng.integers(0, 2**32, (n, 2), dtype=np.uint64).astype(np.uint32)
    # edge words: all-zero and all-one counters and keys, and the counters the
    # env draws use (env, step, iteration, purpose) with a 64-bit seed split
    ctr[0], key[0] = 0, 0
    ctr[1], key[1] = 0xFFFFFFFF, 0xFFFFFFFF
    ctr[2], key[2] = [12, 499, 3, 1], [0x9E3779B9, 0x7F4A7C15]
    c_d = torch.from_numpy(ctr.view(np.int32)).cuda()
    k_d = torch.from_numpy(key.view(np.int32)).cuda()
    out = torch.zeros((n, 4), dtype=torch.int32, device="cuda")
    assert so.philox_launch(c_d.data_ptr(), k_d.data_ptr(), out.data_ptr(), n) == 0
    torch.cuda.synchronize()
    got = out.cpu().numpy().view(np.uint32)
    for i in range(n):
        want = np.asarray(O.philox4x32_10([int(x) for x in ctr[i]], [int(x) for x in key[i]]), np.uint32)
        assert np.array_equal(got[i], want), (i, ctr[i], key[i], got[i], want)
