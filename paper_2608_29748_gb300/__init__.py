"""GB300-native (sm_103a) per-round hot path of ReTrace.

``libretrace.so`` (built from ``csrc/``) exports the C ABI declared in
``include/retrace.h``; :mod:`paper_2608_29748_gb300.binding` is the thin
ctypes layer over it.  The binding is imported lazily so that the seeded
input generator (:mod:`paper_2608_29748_gb300.workloads`) works without a
built library.
"""

__version__ = "0.1.0"


def __getattr__(name):
    if name in ("retrace_verify", "retrace_align_refine", "retrace_gate_fuse", "retrace_round",
                "retrace_workspace_bytes", "retrace_workspace_init", "retrace_workspace_check",
                "Workspace", "lib", "RetraceError"):
        from . import binding

        return getattr(binding, name)
    raise AttributeError(name)
