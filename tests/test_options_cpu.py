"""Every option name that prism_set_option accepts is documented in the
public header, and the header documents no option the library rejects."""
from __future__ import annotations

import os
import re

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _accepted():
    src = open(os.path.join(ROOT, "paper_2602_01762_gb300", "csrc", "prism_api.cu")).read()
    body = src[src.index("prism_status prism_set_option("):]
    body = body[:body.index("\n}\n")]
    return set(re.findall(r'strcmp\(name, "([a-z_0-9]+)"\)', body))


def _documented():
    hdr = open(os.path.join(ROOT, "include", "prism.h")).read()
    doc = hdr[:hdr.index("prism_status prism_set_option(")]
    doc = doc[doc.rindex("/*"):]
    return set(re.findall(r'"([a-z_0-9]+)"\s*(?:\*\s*)?\(', doc))


def test_every_accepted_option_is_documented():
    missing = _accepted() - _documented()
    assert not missing, sorted(missing)


def test_every_documented_option_is_accepted():
    extra = _documented() - _accepted()
    assert not extra, sorted(extra)
