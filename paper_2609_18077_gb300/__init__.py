"""GB300-native (sm_103a) softmax attention forward for video-DiT inference."""
