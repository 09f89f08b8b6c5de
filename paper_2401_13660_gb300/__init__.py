"""GB300-native selective-scan layer core of MambaByte (arXiv 2401.13660).

The compute path is libmbscan.so (hand-written sm_103a CUDA kernels behind a
C ABI, include/mbscan.h); `mbscan` is its Python binding. Names are imported
lazily so that `paper_2401_13660_gb300.inputs` can be used without loading the
library.
"""
_BINDING = ("mb_scan_prefill", "mb_scan_verify", "mb_rollback", "mb_step", "mb_step_resume", "mb_check",
            "mb_accept_topk", "mb_scan_prefill_ckpt", "mb_scan_backward", "mb_rmsnorm", "mb_conv1d_step",
            "mb_selftest_timeout", "mb_scan_verify_resume",
            "mb_workspace_size", "mb_status_string", "mb_version", "load_library", "MbError",
            "make_args", "new_workspace")

__all__ = list(_BINDING)


def __getattr__(name):
    if name in _BINDING:
        from . import mbscan
        return getattr(mbscan, name)
    raise AttributeError(name)
