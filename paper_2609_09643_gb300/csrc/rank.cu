// placeholder: the standalone ranking kernels are added next
#include "common.cuh"
extern "C" int unison_rank_batch(const unison_records *, const unison_rank_params *, const unison_rank_out *, int,
                                 void *) {
  return UNISON_ERR_ARG;
}
