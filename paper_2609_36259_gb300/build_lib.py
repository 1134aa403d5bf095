"""Build step of the CUDA library: compiles csrc/*.cu for sm_103a into libcyfa.so in-tree.

Each translation unit is compiled by its own nvcc process (in parallel) and the objects are
linked into one shared library with the C ABI of include/cyfa.h.  Runs on x86_64 (cross
build, no GPU needed) and on the aarch64 GPU hosts alike.
"""
import os
import shutil
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, 'csrc')
BUILD = os.path.join(HERE, '_build')
LIB = os.path.join(HERE, 'libcyfa.so')
ARCH = ['-gencode', 'arch=compute_103a,code=sm_103a']
FLAGS = ['-O3', '-lineinfo', '-std=c++17', '-Xcompiler', '-fPIC', '--expt-relaxed-constexpr',
         '-Xptxas', '-warn-spills']


def nvcc():
    exe = shutil.which('nvcc')
    if exe is None:
        cand = '/usr/local/cuda/bin/nvcc'
        if os.path.exists(cand):
            return cand
        raise RuntimeError('nvcc not found: the CUDA toolkit is required to build libcyfa.so')
    return exe


def sources():
    return sorted(os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith('.cu'))


def build(verbose=False, extra=()):
    os.makedirs(BUILD, exist_ok=True)
    cc = nvcc()
    srcs = sources()
    objs = [os.path.join(BUILD, os.path.basename(s)[:-3] + '.o') for s in srcs]

    def one(pair):
        src, obj = pair
        cmd = [cc, *ARCH, *FLAGS, *extra, '-c', src, '-o', obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        return src, r, cmd

    with ThreadPoolExecutor(max_workers=max(1, min(len(srcs), os.cpu_count() or 4))) as ex:
        results = list(ex.map(one, zip(srcs, objs)))
    failed = False
    for src, r, cmd in results:
        if verbose or r.returncode != 0:
            sys.stderr.write(' '.join(cmd) + '\n' + r.stdout + r.stderr)
        failed |= r.returncode != 0
    if failed:
        raise RuntimeError('nvcc failed to compile the CyFA kernels')
    tmp = LIB + '.tmp'
    cmd = [cc, *ARCH, '-shared', '-o', tmp, *objs]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        sys.stderr.write(' '.join(cmd) + '\n' + r.stdout + r.stderr)
        raise RuntimeError('linking libcyfa.so failed')
    os.replace(tmp, LIB)
    return LIB


if __name__ == '__main__':
    print(build(verbose='-v' in sys.argv))
