"""Host-side tools of bench.py that need no GPU."""
import os
import sys

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))


def test_trace_summary_on_synthetic_events(capsys):
    # bench.py --trace reduces clock stamps per (CTA, event, tile) to stage
    # medians; a synthetic timeline with fixed gaps must come back exactly.
    import numpy as np
    import bench

    ev = np.zeros((2, 128, 32), np.int64)
    for c in range(2):
        for it in range(6):
            t0 = 10_000 * it + 100 * c
            ev[c, 112:121, it] = t0 + np.arange(9) * 300   # QK chunks issued
            ev[c, 12, it] = t0 + 2_900                      # QK committed
            ev[c, 14, it] = t0 + 4_000                      # P seen
            ev[c, 15, it] = t0 + 5_600                      # PV issued
            ev[c, 24:28, it] = t0 + 5_500
            ev[c, 16, it] = t0 + 3_100
            ev[c, 19, it] = t0 + 3_900
            ev[c, 17, it] = t0 + 4_050
            ev[c, 18, it] = t0 + 4_100
            ev[c, 0, it] = t0 + 200
            ev[c, 105, it] = t0 + 500
            ev[c, 88:96, it] = t0 + 700
            ev[c, 32:40, it] = t0 + 2_500
            ev[c, 48:88, it] = t0 + 1_000
    bench.main_trace_summary(ev)
    out = capsys.readouterr().out
    assert "tile period (cycles, median over 6 tiles): 10000" in out
    assert "issuer 0: QK chunk 0 -> chunk 8 issued" in out and " 2400" in out
    assert "issuer 0: P seen -> PV issued" in out and " 1600" in out
