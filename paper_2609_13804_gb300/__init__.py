"""GB300-native StepPrune inference path: sequential visual-token selection,
compaction of the kept tokens and the language-model prefill over the packed
prefix, as hand-written sm_103a CUDA behind a C ABI (libstepprune.so).

Importing the package loads nothing; `binding` loads the library on first use
and raises if it has not been built.
"""
__all__ = ["binding", "synth"]
