"""GB300-native batched compliance checking for privacy intents (placement
selectors, flow-rule probe walks, jurisdiction-masked reachability)."""
