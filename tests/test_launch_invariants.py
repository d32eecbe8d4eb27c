"""Source-level invariant behind the library's stream order.

Kernels are launched with programmatic dependent launch (launch_pdl), which
lets a kernel's CTAs start before the previous kernel in the stream has
finished.  Stream order then holds only because every such kernel executes
griddep_wait() (griddepcontrol.wait) before it touches memory, and holds
transitively because its predecessor did the same.  This test reads the CUDA
sources and checks that every kernel passed to launch_pdl exists and that the
first statement of its body is griddep_wait(), and that no kernel triggers
its dependents early (griddepcontrol.launch_dependents).
"""
import pathlib
import re

CSRC = pathlib.Path(__file__).resolve().parents[1] / "paper_2509_26436_gb300" / "csrc"
SOURCES = sorted(CSRC.glob("*.cu"))


def _launched_kernels():
    names = set()
    for path in SOURCES:
        text = path.read_text()
        for m in re.finditer(r"launch_pdl\(\s*([A-Za-z_][A-Za-z_0-9]*)", text):
            names.add((path.name, m.group(1)))
    return names


def _kernel_body_start(text, name):
    """First statement of the body of __global__ kernel `name`, or None."""
    m = re.search(r"__global__[^;{]*?\b" + re.escape(name) + r"\s*\(", text, re.S)
    if not m:
        return None
    depth, i = 0, m.end() - 1
    while True:  # skip the parameter list
        if text[i] == "(":
            depth += 1
        elif text[i] == ")":
            depth -= 1
            if depth == 0:
                break
        i += 1
    brace = text.index("{", i)
    body = text[brace + 1:]
    stmt = body.lstrip().split(";", 1)[0]
    return stmt.strip()


def test_every_pdl_kernel_waits_first():
    launched = _launched_kernels()
    assert launched, "no launch_pdl call found"
    texts = {p.name: p.read_text() for p in SOURCES}
    for fname, name in sorted(launched):
        if name == "kern":  # the GEMM launch goes through a pointer to one of its instances
            name = "gemm_tcgen05_kernel"
        found = [f for f, t in texts.items() if _kernel_body_start(t, name) is not None]
        assert found, f"{fname}: launch_pdl of {name}, whose definition was not found"
        for f in found:
            first = _kernel_body_start(texts[f], name)
            assert first == "griddep_wait()", f"{f}: {name} starts with `{first}`, not griddep_wait()"


def test_no_early_dependent_trigger():
    for path in SOURCES:
        text = path.read_text()
        code = re.sub(r"//[^\n]*", "", text)
        assert "launch_dependents" not in code, f"{path.name} triggers dependents early"


def test_plain_launches_are_not_on_the_data_path():
    """Kernels still launched with <<< >>> are the measurement probes and the
    timeout self-test, which run alone and touch no tensor of the path."""
    allowed = {"probe_fp32_kernel", "probe_mma_f8_kernel", "selftest_timeout_kernel"}
    for path in SOURCES:
        for m in re.finditer(r"\b([A-Za-z_][A-Za-z_0-9]*)(?:<[^<>;]*>)?<<<", path.read_text()):
            assert m.group(1) in allowed, f"{path.name}: {m.group(1)} launched without launch_pdl"
