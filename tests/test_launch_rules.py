"""Static check of the dependent-launch rules in the CUDA sources (no GPU).

The kernels of a call after the table upload are launched with programmatic
stream serialisation (`launch_dep`, csrc/kernels.h), so a kernel may be
scheduled while the one before it drains.  The ordering that keeps this correct
rests on two rules stated in csrc/vc_common.cuh: a thread of every CTA returns
from dep_wait() before the CTA reads the previous kernel's output (or writes what
it reads or writes), and a CTA calls dep_launch() only after dep_wait().  This
test reads every kernel that a launch_dep call launches and checks that its body
calls dep_wait(), that no dep_launch() comes before the first dep_wait(), and
that no early `return` comes before the first dep_wait() (a CTA that exits
without waiting would let the kernel complete before its predecessor).
"""
import os
import re

CSRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "paper_2608_24063_gb300", "csrc")


def _sources():
    out = {}
    for f in sorted(os.listdir(CSRC)):
        if f.endswith((".cu", ".cuh", ".h", ".cpp")):
            with open(os.path.join(CSRC, f)) as fh:
                out[f] = fh.read()
    return out


def _strip_comments(s):
    s = re.sub(r"/\*.*?\*/", "", s, flags=re.S)
    return re.sub(r"//[^\n]*", "", s)


def _kernel_body(src, name):
    """Body of `__global__ ... name(...) { ... }` (braces matched), or None."""
    m = re.search(r"__global__[^;{]*?\b%s\s*\(" % re.escape(name), src)
    if not m:
        return None
    i = src.index("{", m.end())
    depth = 0
    for j in range(i, len(src)):
        if src[j] == "{":
            depth += 1
        elif src[j] == "}":
            depth -= 1
            if depth == 0:
                return src[i + 1:j]
    return None


def _launched_dependent(srcs):
    names = set()
    for f, s in srcs.items():
        if f == "kernels.h":
            continue
        for m in re.finditer(r"launch_dep\(\s*([A-Za-z_][\w:]*)", _strip_comments(s)):
            names.add(m.group(1).split("::")[-1])
    return names


def test_dependent_kernels_wait_before_they_launch_or_return():
    srcs = {f: _strip_comments(s) for f, s in _sources().items()}
    names = _launched_dependent(srcs)
    assert {"score_lse_tc_kernel", "score_colsum_tc_kernel", "chunk_sort_kernel", "chunk_rank_kernel",
            "gather_kv_kernel", "fuse_v_tcp_kernel"} <= names, names
    for name in sorted(names):
        bodies = [b for b in (_kernel_body(s, name) for s in srcs.values()) if b is not None]
        assert len(bodies) == 1, name
        body = bodies[0]
        w = body.find("dep_wait()")
        assert w >= 0, "%s never calls dep_wait()" % name
        launch = body.find("dep_launch()")
        assert launch < 0 or launch > w, "%s calls dep_launch() before dep_wait()" % name
        ret = re.search(r"\breturn\b", body[:w])
        assert ret is None, "%s may return before dep_wait()" % name


def test_the_first_kernel_of_a_call_is_an_ordinary_launch():
    srcs = {f: _strip_comments(s) for f, s in _sources().items()}
    assert "upload_kernel" not in _launched_dependent(srcs)
    assert re.search(r"upload_kernel<<<", srcs["upload.cu"])
