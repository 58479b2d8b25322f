"""GB300-native Elastic Shadow Pricing (ESP) solver: the tatonnement of Sec. 3.2 on one GPU."""
