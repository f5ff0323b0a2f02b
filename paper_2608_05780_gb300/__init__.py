"""GB300-native (sm_103a) sparse-prefill evidence probe.

The product is ``libevisel.so`` (C ABI in ``include/evisel.h``); this package
holds its sources (``csrc/``), the in-tree build and a thin ctypes binding with
the same entry-point names. ``workloads`` draws the seeded synthetic inputs.
"""
from ._binding import (  # noqa: F401
    EviselError, Workspace, evisel_evidence_reduce, evisel_free, evisel_probe_attention, evisel_probe_evidence_noalloc,
    evisel_intra_frame_evidence, evisel_cross_frame_evidence, evisel_topp_mask, tile_union_to_csr,
    evisel_coarse_evidence,
    evisel_selftest_wait, evisel_status, load,
)


def ensure_built(verbose: bool = True):
    """Builds the library if it does not hold the current tree's build id,
    loads it, and (``verbose``) reports the id of the binary that loaded."""
    import sys

    from .build import build
    path = build()
    lib = load()
    if verbose:
        sys.stderr.write(f"libevisel.so build {lib.evisel_build_id().decode()} ({path})\n")
    return lib
