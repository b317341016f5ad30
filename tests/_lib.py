"""Test helpers: build the library once and skip GPU tests without a GPU."""
import functools

import pytest
import torch


@functools.lru_cache(maxsize=1)
def built_lib():
    from paper_2605_11232_gb300 import build, pkv
    build.build()
    return pkv.load()


def need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    built_lib()
