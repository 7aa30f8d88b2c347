// The fused preparation kernel's two launches for token-sharded stacks
// (prep.cu, MODE 1 and MODE 2): routing and block partials before the
// all-gather of Eq. 11's sums, then decisions and compaction after it.
#define MOECA_PREP_SHARD 1
#include "prep.cu"
