// The fused preparation kernel built for DiT-MoE blocks (prep.cu with the
// block's work compiled in): u = x + a^{t0} while staging the token rows, the
// FFN-row map and the recomputing-token list in the compaction.
#define MOECA_PREP_ATTN 1
#include "prep.cu"
