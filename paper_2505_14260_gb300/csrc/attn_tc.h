// Tree-masked attention on the 5th-generation tensor cores (bf16 path): split
// bf16 operands (hi + lo planes, `lo` elements apart, a multiple of hd).
#pragma once

#include "kernels.h"

namespace msd {

struct AttnTcPlan;

// Per-context plan (tensor-map cache, SM count).
bool attn_tc_plan_create(AttnTcPlan **out);
void attn_tc_plan_destroy(AttnTcPlan *p);

// a.R rows grouped by request in blocks of rows_per_req; each row's visible
// prefix length comes from its row descriptor. B is the number of requests
// the cache buffers hold. order (nullable, a permutation of the a.R /
// rows_per_req blocks, used when there are at most 64): the blocks' launch
// order, longest first, so that the last wave holds the shortest CTAs (it
// changes no result). stamp (nullable): a profiling slot of three
// %globaltimer values (earliest entry, earliest return from the wait on the
// previous kernel, latest exit), min/min/max-updated by the CTAs. Returns false
// if the shape is not supported (the caller reports it).
bool launch_attention_tc(AttnTcPlan *p, const AttnArgs<bf16> &a, int B, int rows_per_req, const int *order,
                         int *status, cudaStream_t s, unsigned long long *stamp = nullptr);

}  // namespace msd
