"""GB300-native hot path of the latency-aware LLM query router.

The Serving Framework Simulation TTFT estimator (Sec. 4.1), the
accuracy-cost-latency objective (Sec. 3) and the per-query argmax, as CUDA
kernels for sm_103a behind a C ABI (``include/latency_router.h``).
``router`` is the thin Python binding; ``workloads`` draws seeded inputs.
"""
__all__ = ["router", "workloads"]
