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


def _code_defaults():
    """Initial values of the context's option fields named like their option."""
    src = open(os.path.join(ROOT, "paper_2602_01762_gb300", "csrc", "prism_api.cu")).read()
    block = src[src.index("    // execution\n"):src.index("    // tensor-core path")]
    out = {}
    for name in _accepted():
        m = re.search(r"\b%s\s*=\s*(true|false|-?\d+)" % re.escape(name), block)
        if m:
            v = m.group(1)
            out[name] = 1 if v == "true" else 0 if v == "false" else int(v)
    return out


def _documented_defaults():
    hdr = open(os.path.join(ROOT, "include", "prism.h")).read()
    doc = hdr[:hdr.index("prism_status prism_set_option(")]
    doc = re.sub(r"\s*\n\s*\*\s*", " ", doc[doc.rindex("/*"):])
    starts = [(m.start(), m.group(1)) for m in re.finditer(r'"([a-z_0-9]+)"\s*\(', doc)]
    out = {}
    for i, (pos, name) in enumerate(starts):
        text = doc[pos:starts[i + 1][0] if i + 1 < len(starts) else len(doc)]
        found = [(m.start(), int(m.group(1))) for m in re.finditer(r"(-?\d+), the default", text)]
        found += [(m.start(), int(m.group(1))) for m in re.finditer(r"default (-?\d+)", text)]
        if found:
            out[name] = min(found)[1]
    return out


def test_documented_defaults_match_the_code():
    code, doc = _code_defaults(), _documented_defaults()
    both = sorted(set(code) & set(doc))
    assert len(both) >= 15, both
    wrong = {n: (doc[n], code[n]) for n in both if doc[n] != code[n]}
    assert not wrong, wrong
