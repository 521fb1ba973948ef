"""GB300-native SpeechKV decode hot path (speech-span KV pooling, text-token
append, split-K GQA decode attention) behind a C-ABI library."""
