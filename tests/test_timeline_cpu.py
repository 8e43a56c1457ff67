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


def test_summary_of_a_fabricated_trace():
    """Stamps are (clock << 8) | event; a span (a, b) adds the time from the last a to each b."""
    import numpy as np
    ev = {name: i + 1 for i, (_, name, _) in enumerate(timeline.PROBES)}
    buf = np.zeros((timeline.N_CTAS, timeline.N_ROLES, 16), dtype=np.uint64)
    n = np.zeros((timeline.N_CTAS, timeline.N_ROLES), dtype=np.uint32)
    # issuer of the even layers, CTA 0: wait 100 cycles for a W stage, issue for 500, twice
    stamps = [(1000, "I_WFULL_W"), (1100, "I_WFULL_D"), (1600, "I_ISSUED"),
              (1700, "I_WFULL_W"), (1800, "I_WFULL_D"), (2300, "I_ISSUED")]
    for i, (t, e) in enumerate(stamps):
        buf[0, 0, i] = (t << 8) | ev[e]
    n[0, 0] = len(stamps)
    text = timeline.summarize(buf, n, ev, "fabricated", 1.0)
    span = 2300 - 1000
    assert "CTA 0, issuer, even layers (warp 1): %.2f M cycles" % (span / 1e6) in text
    assert "wait: W stage landed" in text and "%.1f %%  (2 intervals, mean 100 cycles)" % (100.0 * 200 / span) in text
    assert "%.1f %%  (2 intervals, mean 500 cycles)" % (100.0 * 1000 / span) in text
    assert "%.1f %%  (2 stages x 8 MMAs x 64 cycles)" % (100.0 * 2 * 512 / span) in text
