"""GB300-native (sm_103a) hot path of DART (arXiv 2608.02032)."""
