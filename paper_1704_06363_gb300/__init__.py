"""GB300-native gater for hard mixtures of experts (arXiv 1704.06363, Section 2).

K-means (Lloyd) over feature vectors, the hard nearest-centre assignment of
Eq. 2, and the split of the data into per-expert shares, as hand-written
sm_103a CUDA kernels behind the C ABI in ``include/hme.h``.  ``hme`` is the thin
ctypes binding with the same entry-point names; PyTorch only provides device
memory and streams.
"""
from . import hme  # noqa: F401
from .hme import (HmeError, HME_F32, HME_BF16, hme_assign, hme_kmeans_init, hme_partition,  # noqa: F401
                  hme_prepare_features, hme_route, hme_sync_status, hme_update_centroids, hme_workspace_bytes,
                  hme_launch_count, hme_debug_bounded_wait, workspace)
