"""BeaconKV KV-cache compression step, GB300-native (sm_103a).

The work happens in libbkv.so (C ABI: include/bkv.h); ``bkv`` mirrors that
ABI in Python.  ``synth`` and ``workloads`` describe the synthetic workloads.
"""
from .workloads import WORKLOADS, Workload  # noqa: F401
