"""Source checks of the programmatic-dependent-launch discipline (no GPU needed).

A kernel launched with LUNA_LAUNCH_DEP may start while the previous kernel of
its stream is still running.  It is correct only if every block of it waits in
grid_dependency_sync() before it reads what an earlier kernel of the same call
writes and before its first global store, and if it never returns before that
wait (the wait of each kernel keeps the stream order transitive).  The only
data it may read earlier is the parameter table, so the launch is switched off
whenever the channel normalisation rewrites the table inside the call.  These
tests read the CUDA sources and check those rules for every such launch.
"""
import os
import re

import pytest

CSRC = os.path.join(os.path.dirname(__file__), "..", "paper_2512_08061_gb300", "csrc")

# AttnArgs fields a kernel may read before its dependency wait: the problem shape and the
# parameter table (written by luna_prepare before the call's first cudaMemsetAsync).
PRE_WAIT_FIELDS = {"lay", "table", "d", "dv", "n", "B", "H", "M", "L", "D"}


def _sources():
    out = {}
    for f in sorted(os.listdir(CSRC)):
        if f.endswith((".cu", ".cuh")):
            with open(os.path.join(CSRC, f)) as fh:
                out[f] = fh.read()
    return out


def _strip_comments(src: str) -> str:
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return re.sub(r"//[^\n]*", "", src)


def _dep_launches(srcs):
    """(file, tag, dep expression, kernel base name, enclosing source) of every LUNA_LAUNCH_DEP."""
    found = []
    for f, src in srcs.items():
        if not f.endswith(".cu"):
            continue
        code = _strip_comments(src)
        for m in re.finditer(r'LUNA_LAUNCH_DEP\(\s*"(\w+)"\s*,\s*([^,]+?)\s*,\s*\(?\s*(k_\w+)', code):
            found.append((f, m.group(1), m.group(2), m.group(3), code[: m.start()]))
    return found


def _kernel_body(srcs, name):
    for src in srcs.values():
        code = _strip_comments(src)
        m = re.search(r"__global__[^;{]*?\b" + name + r"\s*\(", code)
        if not m:
            continue
        i = code.index("{", m.end())
        depth, j = 0, i
        while True:
            if code[j] == "{":
                depth += 1
            elif code[j] == "}":
                depth -= 1
                if depth == 0:
                    return code[i + 1:j]
            j += 1
    raise AssertionError(f"no definition of kernel {name}")


SRCS = _sources()
LAUNCHES = _dep_launches(SRCS)


def test_dependent_launches_exist():
    kernels = {k for _, _, _, k, _ in LAUNCHES}
    assert {"k_tile_split", "k_tc_keys", "k_tc_query", "k_tc_causal", "k_seg_scan", "k_grad_sum",
            "k_mlp_grads"} <= kernels


@pytest.mark.parametrize("launch", LAUNCHES, ids=[f"{t}:{k}" for _, t, _, k, _ in LAUNCHES])
def test_dependent_launch_is_off_with_channel_normalisation(launch):
    f, tag, dep, kernel, before = launch
    if dep == "!a.ch_sigma":
        return
    assert dep == "dep", f"{tag}: dependency flag {dep!r}"
    func = before[before.rfind("\ncudaError_t "):]  # the enclosing host function
    assert re.search(r"\bdep\s*=\s*!a\.ch_sigma\s*;", func), f"{tag}: dep not derived from ch_sigma"


@pytest.mark.parametrize("kernel", sorted({k for _, _, _, k, _ in LAUNCHES}))
def test_kernel_waits_before_touching_dependent_memory(kernel):
    body = _kernel_body(SRCS, kernel)
    assert body.count("grid_dependency_sync()") == 1, f"{kernel}: exactly one dependency wait"
    pre = body[: body.index("grid_dependency_sync()")]
    assert not re.search(r"\breturn\b", pre), f"{kernel}: returns before its dependency wait"
    assert "Items it(" not in pre, f"{kernel}: reads the work split before its dependency wait"
    # a pointer field compared with nullptr reads the kernel parameter, not the memory behind it
    fields = set(re.findall(r"\ba\.(\w+)", re.sub(r"\ba\.\w+\s*[!=]=\s*nullptr", "", pre)))
    assert fields <= PRE_WAIT_FIELDS, f"{kernel}: reads {sorted(fields - PRE_WAIT_FIELDS)} before the wait"
    # no loop or branch may hide the wait: it sits at brace depth 0 of the kernel body
    assert pre.count("{") == pre.count("}"), f"{kernel}: dependency wait inside a block"
    # no global store before the wait: stores before it go to shared memory only
    for store in re.findall(r"(\w+)\s*\[[^\]]*\]\s*=(?!=)", pre):
        assert store in {"sk", "si", "w1t", "b1t", "w2t", "tyt", "rkt", "part", "bins", "sdW", "h"}, \
            f"{kernel}: store to {store} before the dependency wait"


def test_plain_launch_kernels_have_no_dangling_wait():
    """A kernel that calls grid_dependency_sync() is launched with LUNA_LAUNCH_DEP (else the wait is
    dead code that suggests an overlap that never happens)."""
    dep_kernels = {k for _, _, _, k, _ in LAUNCHES}
    for f, src in SRCS.items():
        code = _strip_comments(src)
        for m in re.finditer(r"__global__[^;{]*?\b(k_\w+)\s*\(", code):
            body = _kernel_body({f: src}, m.group(1))
            if "grid_dependency_sync()" in body:
                assert m.group(1) in dep_kernels, f"{m.group(1)} waits but is launched plainly"
