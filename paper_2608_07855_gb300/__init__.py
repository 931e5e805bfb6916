"""CommitKV hot path on GB300 (sm_103a).

The CUDA library (csrc/, built in-tree into _build/libcommitkv.so) exposes
the C ABI of include/commitkv.h; ``commitkv`` is its Python binding and
``synth`` the seeded synthetic workload generator.
"""
from . import build  # noqa: F401
from .commitkv import (  # noqa: F401
    CommitKVError,
    Shape,
    Thresholds,
    Traj,
    TrajTensors,
    alloc_workspace,
    commitkv_classify,
    commitkv_compact,
    commitkv_joint_test,
    commitkv_page_effects,
    commitkv_workspace_init,
    commitkv_workspace_size,
    commitkv_workspace_status,
    load_library,
    make_shape,
    status_string,
)
