"""Ember optimizer step for V x D token tables on GB300 (sm_103a).

The computation lives in libember.so (CUDA, C ABI in include/ember.h); this
package is its ctypes binding, its build script and the seeded synthetic
input generators used by the tests and the benchmark.
"""
from .ember import (  # noqa: F401
    EMBER_BF16, EMBER_F32, EMBER_I32, EMBER_I64, EMBER_OK, Ember, EmberError,
    ember_abi_version, ember_bind_workspace, ember_create, ember_destroy,
    ember_get_device_status, ember_hparams, ember_hparams_default, ember_state_numel,
    ember_status_string, ember_step_dense, ember_step_sparse, ember_workspace_bytes,
)
