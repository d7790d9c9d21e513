"""Doubly pipelined, dual-root reduction-to-all on one GPU (Traff 2021,
arXiv 2109.12626): thin Python binding of the C ABI in ``include/dpdr.h``.

Argument marshalling only: every step of the reduction runs in the CUDA
kernels of ``libdpdr.so``.  Rank buffers are passed as torch tensors (or raw
device addresses); torch supplies device memory and streams.  If the
compiled library is missing the calls raise instead of falling back.
"""
from __future__ import annotations

from ._native import (DPDR_ERR_CUDA, DPDR_ERR_INVALID,  # noqa: F401
                      DPDR_ERR_NOT_COOPERATIVE, DPDR_ERR_OOM, DPDR_ERR_TIMEOUT,
                      DPDR_FLOAT32, DPDR_INT32, DPDR_MAT2X2_F32,
                      DPDR_MAT2X2_U32, DPDR_OK,
                      DPDR_OP_MATMUL, DPDR_OP_SUM, OPT_BLOCKS, OPT_FUSED_MODE,
                      OPT_HOST_CHUNK_BYTES, OPT_HOST_PATH,
                      OPT_SCHED_RANKS_PER_CTA, OPT_SCHED_SLICES,
                      OPT_SCHED_COPY, OPT_SCHED_LAYOUT, OPT_SCHED_THREADS, OPT_SCHED_TRANSPORT,
                      OPT_SKIP_RANK, OPT_SPLIT_DEPTH, OPT_WAIT_LIMIT_NS, DpdrError,
                      Plan,
                      block_count_rule, blocks, lib, tree)

__all__ = ["Plan", "DpdrError", "tree", "blocks", "block_count_rule", "lib"]
