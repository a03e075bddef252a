import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")
    config.addinivalue_line("markers", "slow: long-running CPU test")


@pytest.fixture
def eogp_options():
    """Setter for the library's process-wide dispatch options
    (eogp_set_option); both are put back to their defaults afterwards."""
    from paper_2609_37842_gb300 import eogp as E

    def setter(score_operand=None, topk_path=None):
        if score_operand is not None:
            E.set_option(E.OPT_SCORE_OPERAND, score_operand)
        if topk_path is not None:
            E.set_option(E.OPT_TOPK_PATH, topk_path)

    yield setter
    E.set_option(E.OPT_SCORE_OPERAND, 0)
    E.set_option(E.OPT_TOPK_PATH, 0)
