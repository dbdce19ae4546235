"""libdlmrefine: one bidirectional refine step of speculative correction on GB300.

The compute lives in ``libdlmrefine.so`` (CUDA, sm_103a) behind a C ABI
(``include/dlmrefine.h``). This package is its thin Python binding
(``binding``), the seeded input generators (``synth`` and its device twin
``libdlmsynth.so``) and the workload recipes (``workloads``). Importing a
compute entry point loads the library and raises if it has not been built:
there is no fallback path.
"""
_BINDING_NAMES = {
    "dlm_bidir_attn", "dlm_vocab_confidence", "dlm_refine_update", "dlm_version",
    "dlm_status_string", "DlmError", "RefineParams", "library_path", "lib",
}


def __getattr__(name):
    if name in _BINDING_NAMES:
        from . import binding
        return getattr(binding, name)
    raise AttributeError(name)
