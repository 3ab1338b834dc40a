"""In-tree build of the CUDA shared libraries with nvcc (sm_103a only).

``build_all()`` compiles every translation unit in parallel and links
``paper_2608_08794_gb300/_lib/libapack.so`` (the product) and
``synth/_lib/libsynth_fill.so`` (the device twin of the input generator).
Objects are rebuilt only when a source or header is newer.
"""

import os
import platform
import shutil
import subprocess
from concurrent.futures import ThreadPoolExecutor

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
INCLUDE = os.path.join(ROOT, "include")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC,-O2", "--expt-relaxed-constexpr"]


def _nvcc():
    exe = shutil.which("nvcc")
    if exe:
        return exe
    cand = "/usr/local/cuda/bin/nvcc"
    if os.path.exists(cand):
        return cand
    raise RuntimeError("nvcc not found")


def _newer(target, deps):
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(d) > t for d in deps)


def _compile(src, obj, deps, extra):
    if not _newer(obj, [src] + deps):
        return None
    cmd = [_nvcc()] + ARCH + NVCC_FLAGS + extra + ["-I", INCLUDE, "-c", src, "-o", obj]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
    return obj


def _link(objs, out):
    cmd = [_nvcc()] + ARCH + ["-shared", "-cudart", "shared", "-o", out] + objs
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed for {out}:\n{r.stdout}\n{r.stderr}")


def _build_lib(src_dir, names, headers, out_dir, lib_name, extra=()):
    build_dir = os.path.join(out_dir, "_obj_" + platform.machine())
    os.makedirs(build_dir, exist_ok=True)
    srcs = [os.path.join(src_dir, n) for n in names]
    objs = [os.path.join(build_dir, os.path.splitext(n)[0] + ".o") for n in names]
    with ThreadPoolExecutor(max_workers=len(srcs)) as ex:
        list(ex.map(lambda so: _compile(so[0], so[1], headers, list(extra)), zip(srcs, objs)))
    out = os.path.join(out_dir, lib_name)
    stamp = out + ".machine"          # the library in _lib was linked on this architecture
    if os.path.exists(out) and (not os.path.exists(stamp) or open(stamp).read() != platform.machine()):
        os.remove(out)
    if _newer(out, objs):
        _link(objs, out)
        with open(stamp, "w") as f:
            f.write(platform.machine())
    return out


def build_apack():
    csrc = os.path.join(HERE, "csrc")
    headers = [os.path.join(INCLUDE, "apack.h")] + [
        os.path.join(csrc, h) for h in os.listdir(csrc) if h.endswith((".cuh", ".h"))]
    return _build_lib(csrc, ["apack.cu", "score.cu", "score_narrow.cu", "score_narrow_tc.cu", "select.cu", "compact.cu", "compact_tma.cu", "compact_inplace.cu", "score_static.cu", "prellm.cu", "decode.cu", "decode_tc.cu", "schedule.cu"], headers,
                      os.path.join(HERE, "_lib"), "libapack.so")


def build_synth():
    sdir = os.path.join(ROOT, "synth")
    return _build_lib(sdir, ["fill.cu"], [], os.path.join(sdir, "_lib"), "libsynth_fill.so")


def build_all():
    with ThreadPoolExecutor(max_workers=2) as ex:
        a = ex.submit(build_apack)
        b = ex.submit(build_synth)
        return a.result(), b.result()


if __name__ == "__main__":
    print(build_all())
