"""GB300-native draft-and-verify step of speculative sampling (sm_103a).

The two operations of the step live in the C-ABI library ``libcachespec.so``
built from ``csrc/``; ``binding`` exposes them to Python under the same
names (``cs_verify_attention``, ``cs_spec_accept``) and only marshals
arguments.  The library is loaded on first use: a missing or stale build is
an error, never a silent fallback.
"""

__all__ = ["binding", "workloads"]


def __getattr__(name):
    if name in ("cs_verify_attention", "cs_spec_accept", "cs_verify_attention_workspace_bytes",
                "cs_spec_accept_workspace_bytes", "load_library"):
        from . import binding
        return getattr(binding, name)
    raise AttributeError(name)
