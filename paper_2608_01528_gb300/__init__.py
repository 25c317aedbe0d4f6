"""GB300-native (sm_103a) Gram-Space codebook path: C-ABI library + thin Python binding."""
