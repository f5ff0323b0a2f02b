"""Plain float64 CPU oracle for the sparse-prefill evidence probe.

TEST INFRASTRUCTURE ONLY. Nothing in the product path imports this package:
only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may call it. It shares no code with
the CUDA path; the only common module is the seeded input generator.

Every function here follows the paper's statement of the probe:
  * masked softmax attention restricted to retained blocks (Sec. 3.2,
    "Sparse Evidence Probing", Eq. 1 and the block-sparse attention it cites);
  * the frame-aligned block partition, text tokens partitioned independently
    (Appendix "Detailed Sparse Prefilling", the paragraph after Eq. 6);
  * logits q k^T / sqrt(d) (Eq. 8) and row-wise normalisation (Eq. 11);
  * head averaging, the query-frame cue A_qf, the intra-frame cue A_if and
    the cross-frame cue A_ff with its timestamp-aligned E_ff (Sec. 3.2,
    "Evidence Decomposition");
  * the top-p block retention of the sparse prefill (Appendix, Eq. 6-9),
    attention restricted to the retained blocks, and the coarse token-level
    map of Eq. 10-11 with its evidence (``topp``).
Parity pins for each function live in ``tests/test_oracle_pins.py``.
"""
from .attention import (  # noqa: F401
    token_layout, allowed_row, probe_rows, probe, text_probabilities, evidence, intra_frame, frame_mass_rows,
    cross_frame, e_ff,
)
from .topp import (  # noqa: F401
    block_layout, block_means, select_prefix, retained_blocks, attended_mask, probe_rows_topp, evidence_topp,
    coarse_evidence,
)
