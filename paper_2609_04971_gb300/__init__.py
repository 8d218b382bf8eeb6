"""BeaconKV KV-cache compression step, GB300-native (sm_103a)."""
