"""Every kernel launched as a programmatic dependent waits for the grid before it.

A kernel launched with launch_dependent may start while the previous kernel in its stream is
still running; it is correct only if it calls griddep_wait before it touches global memory. This
checks the sources: each kernel named in a launch_dependent call has griddep_wait in its body,
and no global load or store comes before it (the wait is the first statement that reads a kernel
argument or global memory).
"""
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2504_16795_gb300", "csrc")


def sources():
    for name in sorted(os.listdir(CSRC)):
        if name.endswith((".cu", ".cuh")):
            with open(os.path.join(CSRC, name)) as f:
                yield name, f.read()


def kernel_body(text, kernel):
    """The body of the __global__ function `kernel` (first definition), or None."""
    for m in re.finditer(r"__global__", text):
        head = text[m.start():]
        paren = head.find(kernel + "(")
        brace = head.find("{")
        if paren < 0 or brace < 0 or paren > brace:
            continue
        depth, i = 0, brace
        while True:
            if head[i] == "{":
                depth += 1
            elif head[i] == "}":
                depth -= 1
                if depth == 0:
                    return head[brace + 1:i]
            i += 1
    return None


def dependent_kernels():
    names = set()
    for name, text in sources():
        if not name.endswith(".cu"):
            continue  # the headers hold launch_dependent's own definition
        for m in re.finditer(r"launch_dependent\(\s*([A-Za-z_][A-Za-z_0-9]*)", text):
            names.add(m.group(1))
    return sorted(names)


def dereferences_an_argument(code):
    """True if `code` reads through a kernel argument: `*a.field` (not a product `x * a.field`),
    or `a.field[...]`."""
    if re.search(r"\ba\.[a-z_0-9]+\s*\[", code):
        return True
    for m in re.finditer(r"\*\s*a\.", code):
        prev = code[:m.start()].rstrip()[-1:]
        if not (prev.isalnum() or prev in ")]_"):
            return True
    return False


def test_some_kernels_are_launched_as_dependents():
    assert len(dependent_kernels()) >= 20


@pytest.mark.parametrize("kernel", dependent_kernels())
def test_dependent_kernel_waits_for_the_grid_before_it(kernel):
    bodies = [b for _, text in sources() for b in [kernel_body(text, kernel)] if b is not None]
    assert bodies, f"no definition of {kernel}"
    body = bodies[0]
    assert "griddep_wait()" in body, kernel
    before = body[:body.index("griddep_wait()")]
    # before the wait: declarations, shared-memory and tensor-memory setup only
    assert not dereferences_an_argument(before), kernel
    for pattern in (r"\bidx\s*\[", r"\boffsets\s*\[", r"\bentries\s*\[", r"\bq\s*\[", r"\bK\s*\[",
                    r"\bhist\s*\[", r"\bstart\s*\["):
        assert not re.search(pattern, before), (kernel, pattern)
