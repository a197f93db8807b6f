"""Builds the CUDA libraries in-tree for sm_103a (GB300).

* ``libsplice.so``        -- the spliced decode-attention library (C ABI in
  ``include/splice.h``), from ``csrc/``.
* ``synth/libsplice_synth.so`` -- the device twin of the seeded input generator.

Each translation unit is compiled by its own ``nvcc`` process, in parallel,
then linked; a library is rebuilt only when a source or header is newer.
"""
from __future__ import annotations

import concurrent.futures as cf
import glob
import os
import shutil
import subprocess

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
CFLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-I", "/usr/local/cuda/include", "--expt-relaxed-constexpr",
          "-Xptxas", "-warn-spills"]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), "/usr/local/cuda/bin/nvcc", shutil.which("nvcc")):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA 13 toolkit is required to build the library")


def _stale(out: str, deps) -> bool:
    if not os.path.exists(out):
        return True
    t = os.path.getmtime(out)
    return any(os.path.getmtime(d) > t for d in deps)


def _run(cmd):
    r = subprocess.run(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)
    if r.returncode != 0:
        raise RuntimeError("build failed:\n" + " ".join(cmd) + "\n" + r.stdout)
    return r.stdout


def build_lib(name: str, sources, headers, out: str, force: bool = False, verbose: bool = False) -> str:
    if not force and not _stale(out, list(sources) + list(headers)):
        return out
    bdir = os.path.join(ROOT, "_build", name)
    os.makedirs(bdir, exist_ok=True)
    cc = nvcc()
    jobs = []
    for src in sources:
        obj = os.path.join(bdir, os.path.basename(src) + ".o")
        cmd = [cc, *ARCH, *CFLAGS, "-I", os.path.join(ROOT, "include"), "-c", src, "-o", obj]
        jobs.append((obj, cmd))
    with cf.ThreadPoolExecutor(max_workers=min(8, len(jobs))) as ex:
        logs = list(ex.map(lambda j: _run(j[1]), jobs))
    if verbose:
        for log in logs:
            if log.strip():
                print(log)
    tmp = out + ".tmp"
    _run([cc, *ARCH, "-shared", "-o", tmp, *[o for o, _ in jobs]])
    os.replace(tmp, out)
    return out


def splice_lib_path() -> str:
    return os.path.join(PKG, "libsplice.so")


def synth_lib_path() -> str:
    return os.path.join(PKG, "synth", "libsplice_synth.so")


def build(force: bool = False, verbose: bool = False) -> None:
    csrc = os.path.join(PKG, "csrc")
    sources = sorted(glob.glob(os.path.join(csrc, "*.cu")) + glob.glob(os.path.join(csrc, "*.cpp")))
    headers = sorted(glob.glob(os.path.join(csrc, "*.h")) + glob.glob(os.path.join(csrc, "*.cuh")) +
                     glob.glob(os.path.join(ROOT, "include", "*.h")))
    synth_src = [os.path.join(PKG, "synth", "synth.cu")]
    with cf.ThreadPoolExecutor(max_workers=2) as ex:
        a = ex.submit(build_lib, "splice", sources, headers, splice_lib_path(), force, verbose)
        b = ex.submit(build_lib, "synth", synth_src, [], synth_lib_path(), force, verbose)
        a.result()
        b.result()


if __name__ == "__main__":
    import sys
    build(force="--force" in sys.argv, verbose=True)
    print("built", splice_lib_path(), synth_lib_path())
