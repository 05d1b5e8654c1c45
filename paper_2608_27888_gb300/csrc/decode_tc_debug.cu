// The debug instantiations of the tcgen05 gather-decode (decode_tc.cuh with
// DBG): the same kernels, launch configuration and bucketing, which also
// record every row their producers build (ntc_debug_decode_rows).
#include "decode_tc.cuh"

namespace ntc {

cudaError_t launch_decode_tc_debug(const Assets &A, const WeightImages &W, const Buckets &B, size_t n,
                                   void *out, unsigned long long *err, unsigned int *status, bool bf16,
                                   int num_sms, cudaStream_t st, int *launches, ntc_debug_row *rows) {
  *launches += 1;
  return dispatch_tm<true>(A, W, B, n, out, err, status, bf16, num_sms, st, rows);
}

}  // namespace ntc
