"""GB300-native cached-search denoising step (arxiv 2607.23159).

The compute path is the C-ABI library built from ``csrc/`` (``libcachedsearch.so``);
``binding`` marshals arguments to it.  Importing the package loads nothing heavy.
"""
__all__ = ["synth", "binding"]
