"""FOCUS FP4 fake-quantizer for GB300 (sm_103a): Python binding of the C ABI.

The binding lives in `paper_2608_01847_gb300.focus` and is imported lazily so
that the synthetic-workload module can be used without a built library.
"""
