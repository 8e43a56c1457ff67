"""The per-role timeline utility still instruments the shipped kernel source (no GPU):
every probe anchor matches exactly once, so a kernel edit that breaks one fails here."""
import glob
import os
import shutil

from paper_2608_03893_gb300 import build as kbuild
from paper_2608_03893_gb300 import timeline


def test_every_probe_anchor_matches_the_kernel_source(tmp_path):
    for f in glob.glob(os.path.join(kbuild.CSRC, "*")):
        shutil.copy(f, tmp_path)
    events = timeline.instrument(str(tmp_path))
    assert sorted(events) == sorted(name for _, name, _ in timeline.PROBES)
    src = open(os.path.join(tmp_path, "kvx_tc.cu")).read()
    for name, ev in events.items():
        assert src.count("TR(%d);" % ev) == 1, name
    # every span's two events exist
    for a, b, _ in timeline.SPANS:
        assert a in events and b in events
