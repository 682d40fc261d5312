"""The README's quick-start snippet runs as written (needs a GB300)."""
from __future__ import annotations

import os
import re

import pytest

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_readme_quick_start():
    from paper_2609_23314_gb300 import build
    build.build()
    with open(os.path.join(ROOT, "README.md")) as f:
        text = f.read()
    blocks = re.findall(r"```python\n(.*?)```", text, flags=re.S)
    assert blocks, "README has no python example"
    exec(compile(blocks[0], "README.md", "exec"), {})
