"""Build the C-ABI CUDA libraries for sm_103a, in-tree.

Each ``csrc/*.cu`` translation unit is compiled in parallel with
``nvcc -gencode arch=compute_103a,code=sm_103a``, then linked (static CUDA
runtime, no libcuda link: the driver's tensor-map encoders are fetched at run
time) into two libraries with the same entry points:
``paper_2509_26092_gb300/_build/libdbl.so`` stores activations, activation
gradients and weight copies as bfloat16, and ``_build/f16/libdbl_f16.so``
(compiled with DBL_ACT_F16) as IEEE binary16, for the fp16 mixed precision of
the paper's ImageNet runs.
"""
import concurrent.futures as cf
import glob
import hashlib
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
OUT_DIR = os.path.join(HERE, "_build")
LIB = os.path.join(OUT_DIR, "libdbl.so")
# storage format -> (extra nvcc flags, object directory, library)
VARIANTS = {"bf16": ([], OUT_DIR, LIB),
            "f16": (["-DDBL_ACT_F16"], os.path.join(OUT_DIR, "f16"), os.path.join(OUT_DIR, "f16", "libdbl_f16.so"))}
INCLUDE = os.path.join(os.path.dirname(HERE), "include")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-Xcompiler", "-fvisibility=hidden",
         "--expt-relaxed-constexpr", "-I", INCLUDE]


def _nvcc():
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libdbl.so")


def _sources():
    return sorted(glob.glob(os.path.join(CSRC, "*.cu")))


def _fingerprint(extra=()):
    h = hashlib.sha256()
    h.update(" ".join(extra).encode())
    for f in _sources() + sorted(glob.glob(os.path.join(CSRC, "*.cuh"))) + [os.path.join(INCLUDE, "dbl.h")]:
        with open(f, "rb") as fh:
            h.update(os.path.basename(f).encode())
            h.update(fh.read())
    h.update(" ".join(ARCH + FLAGS).encode())
    return h.hexdigest()


def build(force=False, verbose=False, jobs=None):
    """Compile and link both libraries if their sources changed; return the bf16 library's path."""
    todo = []
    for name, (extra, out_dir, lib) in VARIANTS.items():
        os.makedirs(out_dir, exist_ok=True)
        stamp = os.path.join(out_dir, os.path.basename(lib)[:-3] + ".stamp")
        fp = _fingerprint(extra)
        if force or not os.path.exists(lib) or not os.path.exists(stamp) or open(stamp).read() != fp:
            todo.append((extra, out_dir, lib, stamp, fp))
    if not todo:
        return LIB
    nvcc = _nvcc()

    def compile_one(job):
        extra, out_dir, src = job
        obj = os.path.join(out_dir, os.path.basename(src)[:-3] + ".o")
        cmd = [nvcc] + ARCH + FLAGS + list(extra) + ["-c", src, "-o", obj]
        if verbose:
            cmd.insert(1, "-Xptxas=-v")
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {os.path.basename(src)} {' '.join(extra)}:\n{r.stdout}\n{r.stderr}")
        return obj, r.stderr

    jobs_ = [(extra, out_dir, src) for extra, out_dir, _, _, _ in todo for src in _sources()]
    # the largest translation unit first, so that it is not the last to start
    jobs_.sort(key=lambda j: -os.path.getsize(j[2]))
    objs = {}
    with cf.ThreadPoolExecutor(max_workers=jobs or min(16, os.cpu_count() or 4)) as ex:
        for job, (obj, log) in zip(jobs_, ex.map(compile_one, jobs_)):
            objs.setdefault(job[1], []).append(obj)
            if verbose and log:
                print(log, file=sys.stderr)
    for extra, out_dir, lib, stamp, fp in todo:
        tmp = lib + f".tmp{os.getpid()}"
        r = subprocess.run([nvcc] + ARCH + ["-shared", "-o", tmp] + sorted(objs[out_dir]) + ["-lpthread"],
                           capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
        os.replace(tmp, lib)
        with open(stamp, "w") as f:
            f.write(fp)
    return LIB


def library_path(precision="bf16"):
    """Path of the library for a storage format ("bf16" or "f16")."""
    return VARIANTS[precision][2]


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv))
