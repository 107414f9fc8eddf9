"""Paged KV cache crop + suffix replay for one GB300 (sm_103a).

The hot path -- crop (restore of a metadata-only checkpoint), append of the
replayed suffix K/V and causal replay attention over the cropped cache -- is
the C-ABI library libpe.so (include/pe.h), built from the CUDA sources in
csrc/.  This package only binds it.
"""
from .binding import PagedKVCache, PEError, ProvenanceGraph, replay_schedule, version  # noqa: F401

__all__ = ["PagedKVCache", "PEError", "ProvenanceGraph", "replay_schedule", "version"]
