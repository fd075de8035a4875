"""GB300-native (sm_103a) Hydra-PPO experience-scoring library: Python binding."""
