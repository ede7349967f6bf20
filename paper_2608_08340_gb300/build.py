"""Builds the CUDA library liboprag.so in-tree (paper_2608_08340_gb300/_build/).

Every translation unit is compiled by nvcc for sm_103a only, in parallel, and
linked against the shared CUDA runtime (so that the process shares one runtime
instance with PyTorch).  No cmake; the build reruns only when a source is newer
than the library.
"""
from __future__ import annotations

import concurrent.futures as cf
import glob
import os
import shutil
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(os.path.dirname(HERE), "include")
OUT_DIR = os.path.join(HERE, "_build")
LIB_PATH = os.path.join(OUT_DIR, "liboprag.so")
# The nvcc command lines of the last build, one per line (compiles, then the link).
COMMANDS_PATH = os.path.join(OUT_DIR, "nvcc_commands.txt")

ARCH = "-gencode=arch=compute_103a,code=sm_103a"


def _nvcc() -> str:
    cand = [os.environ.get("NVCC", ""), shutil.which("nvcc") or "", "/usr/local/cuda/bin/nvcc"]
    for c in cand:
        if c and os.path.exists(c):
            return c
    raise RuntimeError("nvcc not found")


def _cuda_lib_dir(nvcc: str) -> str:
    root = os.path.dirname(os.path.dirname(os.path.realpath(nvcc)))
    for sub in ("lib64", "lib", "targets/sbsa-linux/lib", "targets/x86_64-linux/lib"):
        p = os.path.join(root, sub)
        if os.path.exists(os.path.join(p, "libcudart.so")):
            return p
    return os.path.join(root, "lib64")


def sources() -> list[str]:
    return sorted(glob.glob(os.path.join(CSRC, "*.cu")))


def _stale() -> bool:
    if not os.path.exists(LIB_PATH):
        return True
    built = os.path.getmtime(LIB_PATH)
    deps = sources() + glob.glob(os.path.join(CSRC, "*.cuh")) + glob.glob(os.path.join(CSRC, "*.h"))
    deps += glob.glob(os.path.join(INCLUDE, "*.h"))
    return any(os.path.getmtime(p) > built for p in deps)


def build(force: bool = False, verbose: bool = False, extra_flags: list[str] | None = None,
          out_dir: str | None = None) -> str:
    """Compiles and links liboprag.so (into out_dir, default the in-tree
    _build/); returns its path."""
    if out_dir is not None and os.path.abspath(out_dir) != OUT_DIR:
        return _build_into(os.path.abspath(out_dir), verbose, extra_flags)
    if not force and not _stale():
        return LIB_PATH
    return _build_into(OUT_DIR, verbose, extra_flags)


def _build_into(out_dir: str, verbose: bool, extra_flags: list[str] | None) -> str:
    lib_path = os.path.join(out_dir, "liboprag.so")
    commands_path = os.path.join(out_dir, "nvcc_commands.txt")
    nvcc = _nvcc()
    os.makedirs(out_dir, exist_ok=True)
    flags = ["-O3", "-std=c++17", "-lineinfo", ARCH, "-Xcompiler", "-fPIC,-fvisibility=hidden",
             "-I", INCLUDE, "--expt-relaxed-constexpr"] + list(extra_flags or [])
    if verbose:
        flags += ["-Xptxas", "-v"]

    def compile_one(src: str) -> str:
        obj = os.path.join(out_dir, os.path.basename(src) + ".o")
        cmd = [nvcc, "-c", src, "-o", obj] + flags
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src}:\n{r.stderr}")
        if verbose and r.stderr:
            print(r.stderr)
        return obj

    commands = [[nvcc, "-c", src, "-o", os.path.join(out_dir, os.path.basename(src) + ".o")]
                + flags for src in sources()]
    with cf.ThreadPoolExecutor(max_workers=max(1, min(8, os.cpu_count() or 1))) as ex:
        objs = list(ex.map(compile_one, sources()))
    libdir = _cuda_lib_dir(nvcc)
    tmp = lib_path + f".tmp{os.getpid()}"
    cmd = [nvcc, "-shared", ARCH, "-o", tmp] + objs + [
        "-cudart", "shared", "-Xlinker", f"-rpath={libdir}"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stderr}")
    with open(commands_path, "w") as f:
        for c in commands + [cmd]:
            f.write(" ".join(c) + "\n")
    os.replace(tmp, lib_path)
    return lib_path


if __name__ == "__main__":
    import sys
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv))
