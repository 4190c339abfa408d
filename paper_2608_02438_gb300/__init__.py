"""GB300-native implementation of the xPress refinement pass (arXiv 2608.02438)."""
