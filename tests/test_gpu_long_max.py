"""Max-sets of more than 32 members (max reductions over long dims) on the
GPU, against the oracle: cones, keys, verdicts, flags, export bytes and the
fp32 evaluation.  Keys of such max-sets come from the block-per-element
kernel (members loaded, sorted and deduplicated in shared memory).  Cases: a
max over all 128 output channels of a convolution (configuration 4's conv
and its candidate's weight-stride bug), a max over 1,024 row elements
against a max of the row's two parts (equal sets: discharged) and against
the row without its last element, a max over 33 members, and a max-shifted
softmax over 64 channels whose shift is broadcast back with explicit axes
(the rewrite to softmax does not apply, so the max stays).  One of the
channel cases reads its weights with a channel stride smaller than a
channel's weights, the overlapping strided reads the cone planner folds."""
import numpy as np
import pytest

from paper_2609_19611_gb300 import workloads as W

from .test_gpu_parity import Case, check_compare, check_cones, check_eval, check_keys

pytestmark = pytest.mark.gpu

CASES = {
    "channels128": lambda: W.channel_max(N=2, Ci=3, H=8, W=8, Co=128, bug_co=96),
    # the candidate's weight channel stride (Ci-1)*k*k = 18 is smaller than a
    # channel's 27 weights: at the padded borders its weight reads form
    # overlapping strided runs, which the cone planner folds into one lattice
    "channels128_overlapping_rows": lambda: W.channel_max(N=2, Ci=3, H=8, W=8, Co=128,
                                                           bug_co=96, bug_stride=18),
    "row1024_split": lambda: W.row_max(B=4, L=1024, split=333),
    "row1024_short": lambda: W.row_max(B=4, L=1024),
    "row33": lambda: W.row_max(B=5, L=33),
    "softmax64_broadcast_shift": lambda: W.softmax_shift_broadcast(N=3, C=64, L=5),
}


@pytest.mark.parametrize("name", list(CASES))
def test_long_max_sets(name):
    ref, cand = CASES[name]()
    case = Case(ref, cand, seed=17)
    locs = np.arange(case.R.out_numel, dtype=np.int64)
    check_cones(case, locs)
    kr, kc = check_keys(case, locs)
    v, f = check_compare(case, locs, budget=4)
    check_eval(case, locs)
    if name == "row1024_split":
        assert (v == 0).all()
    else:
        assert (v != 0).all()
