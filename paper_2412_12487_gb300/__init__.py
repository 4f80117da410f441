"""GB300 (sm_103a) timeline composer for Echo-style training simulation (arXiv 2412.12487).

``Echo`` is the Python face of the C ABI in ``include/echo.h``; every step of the
hot path (CC estimation, composition, overlap adjustment) runs in ``libecho.so``.
``workloads`` builds seeded synthetic Megatron-shaped inputs.
"""
from .echo import Echo, EchoError, check_graph, load_library, library_path  # noqa: F401

__all__ = ["Echo", "EchoError", "check_graph", "load_library", "library_path"]
