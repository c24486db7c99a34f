"""GB300-native fork-tree decode attention for parallel reasoning branches.

Importing the package loads nothing native; the CUDA library is loaded on the
first call into ``paper_2608_24658_gb300.api`` and raises if it is missing.
"""
