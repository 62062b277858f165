"""The usage example in the package docstring runs as written."""
import re

import pytest

import paper_2608_16336_gb300 as pkg

pytestmark = pytest.mark.gpu


def test_package_example_runs():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    doc = pkg.__doc__
    block = doc[doc.index("::\n") + 3:doc.index("Draining (Sec. 3.5)")]
    code = "\n".join(line[4:] if line.startswith("    ") else line for line in block.splitlines())
    assert "sim.run()" in code and re.search(r"latency_stats\(\)", code)
    exec(compile(code, "package-docstring-example", "exec"), {})
