"""First calls of a process from two host threads at once.

The out-of-place gather and the tensor-core decode kernel need more than 48 KB
of dynamic shared memory, which a kernel attribute grants per device; the
library sets it once per device, recorded in an atomic per-device bit.  Here a
fresh child process makes its very first apack_compact call and its very first
apack_decode_attention call from two threads released together by a barrier
(ctypes drops the GIL during the calls), and checks both results: the gather
bit for bit against torch.index_select, the decode attention against the oracle.
"""

import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r"""
import sys, threading
import numpy as np, torch
sys.path.insert(0, sys.argv[1])
import __graft_entry__
__graft_entry__.build()
import paper_2608_08794_gb300 as ap
import oracle
from synth.gen import f32_to_bf16_bits

assert ap.apack_launch_count() == 0
dev = torch.device("cuda:0")
rng = np.random.default_rng(5)
# gather: 20000 rows of 1 KB, 3 planes, every third row kept
T, row = 20000, 1024
src = torch.randint(-30000, 30000, (3, T, row // 2), dtype=torch.int16, device=dev)
keep = torch.arange(0, T, 3, dtype=torch.int32, device=dev)
dst = torch.zeros((3, keep.numel(), row // 2), dtype=torch.int16, device=dev)
plane = ap.make_plane(src, dst, row, num_planes=3, src_plane_stride=T * row, dst_plane_stride=keep.numel() * row)
# decode attention: 28 query / 4 KV heads over 5000 cached tokens
cu = np.array([0, 5000], np.int32)
q = f32_to_bf16_bits(rng.standard_normal((1, 28, 128)).astype(np.float32))
k = f32_to_bf16_bits(rng.standard_normal((5000, 4, 128)).astype(np.float32))
v = f32_to_bf16_bits(rng.standard_normal((5000, 4, 128)).astype(np.float32))
qd = torch.from_numpy(q.view(np.int16)).to(dev)
kd = torch.from_numpy(k.reshape(5000, -1).view(np.int16)).to(dev)
vd = torch.from_numpy(v.reshape(5000, -1).view(np.int16)).to(dev)
out = torch.full((1, 28, 128), float("nan"), dtype=torch.float32, device=dev)
ws = torch.zeros(ap.apack_decode_workspace_size(cu, 28, 4), dtype=torch.uint8, device=dev)
torch.cuda.synchronize()

go = threading.Barrier(2)
errors = []

def gather():
    try:
        torch.cuda.set_device(dev)
        go.wait()
        ap.apack_compact(keep, keep.numel(), [plane])
    except Exception as e:
        errors.append(("compact", e))

def decode():
    try:
        torch.cuda.set_device(dev)
        go.wait()
        ap.apack_decode_attention(cu, qd, kd, vd, 4 * 256, 28, 4, out, ws)
    except Exception as e:
        errors.append(("decode", e))

ts = [threading.Thread(target=gather), threading.Thread(target=decode)]
for t in ts: t.start()
for t in ts: t.join()
torch.cuda.synchronize()
assert not errors, errors
assert torch.equal(dst, src.index_select(1, keep.long()))
assert ap.apack_device_error(ws) == ap.APACK_OK
np.testing.assert_allclose(out.cpu().numpy(), oracle.decode_attention(q, k, v, cu, 28, 4), atol=2e-4, rtol=2e-3)
print("first calls ok", ap.apack_launch_count())
"""


def test_first_compact_and_decode_calls_from_two_threads():
    r = subprocess.run([sys.executable, "-c", CHILD, ROOT], capture_output=True, text=True, cwd=ROOT, timeout=600)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-4000:]
    assert "first calls ok" in r.stdout
