"""Worker functions for oracle runs in spawned processes.  This module imports
only numpy and the oracle (no torch, no GPU), so that a worker starts fast."""
import numpy as np

import oracle


def layer_stat(job):
    """The oracle's Eq. 5 statistic S_l of one layer."""
    q, k, modality, text_pos, w, scale, h_kv = job
    _, t = oracle.twr_scores_tvb_stat(oracle.widen_bf16(q[None]), oracle.widen_bf16(k[None]),
                                      modality, text_pos, w[None].astype(np.float64), scale, h_kv)
    return float(t[0])
