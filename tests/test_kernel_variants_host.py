"""The kernel-variant harness stays applicable: every variant's edits find
their anchors in the current sources (no GPU, nothing built)."""
import os

from tests import kernel_variants as K


def test_every_variant_anchor_is_in_the_sources():
    src = {f: open(os.path.join(K.CSRC, f)).read() for f in os.listdir(K.CSRC) if f.endswith((".cu", ".cuh"))}
    for fam, variants in K.VARIANTS.items():
        for name, spec in variants.items():
            edits, _flags = spec if isinstance(spec, tuple) else (spec, [])
            cur = dict(src)
            for e in edits:
                f, a, b = e if len(e) == 3 else ("hx_kernels.cu", *e)
                assert a in cur[f], f"{fam}/{name}: anchor not found in {f}: {a[:60]!r}"
                cur[f] = cur[f].replace(a, b)
