// Draft verification for reusing the lookahead prefix on a miss (section 3.3, "Speculative Decoding"): the number
// of leading draft tokens with P_f(t) >= P_g(t) for every query that is not served from the cache.
//
// One warp per query: each pass of 32 positions ballots the rejections (P_f < P_g); the first set bit, if any,
// ends the accepted prefix.
#include "internal.cuh"

namespace lc {

constexpr int kVerifyWarps = 8;

__global__ void __launch_bounds__(kVerifyWarps * 32)
    verify_draft_kernel(int B, int k, const float* __restrict__ pf, const float* __restrict__ pg,
                        const uint8_t* __restrict__ status, int32_t* __restrict__ accepted) {
  const int lane = threadIdx.x & 31;
  const int q = blockIdx.x * kVerifyWarps + (threadIdx.x >> 5);
  if (q >= B) return;
  if (status && status[q] == LACACHE_HIT) {
    if (lane == 0) accepted[q] = -1;
    return;
  }
  int n = k;
  for (int base = 0; base < k; base += 32) {
    const int i = base + lane;
    const bool reject = i < k && pf[(int64_t)q * k + i] < pg[(int64_t)q * k + i];
    const unsigned r = __ballot_sync(0xffffffffu, reject);
    if (r) {
      n = base + __ffs(r) - 1;
      break;
    }
  }
  if (lane == 0) accepted[q] = n;
}

}  // namespace lc

extern "C" lacache_status lacache_verify_draft(int32_t B, int32_t k, const float* p_target_dev,
                                               const float* p_draft_dev, const uint8_t* status_dev,
                                               int32_t* accepted_dev, void* cuda_stream) {
  lc::NvtxRange nvtx("lacache_verify_draft");
  if (B < 1 || k < 1 || k > lc::kMaxK || !p_target_dev || !p_draft_dev || !accepted_dev)
    return LACACHE_ERR_INVALID_ARG;
  const int blocks = (B + lc::kVerifyWarps - 1) / lc::kVerifyWarps;
  const cudaStream_t st = (cudaStream_t)cuda_stream;
  lc::verify_draft_kernel<<<blocks, lc::kVerifyWarps * 32, 0, st>>>(B, k, p_target_dev, p_draft_dev, status_dev,
                                                                   accepted_dev);
  return cudaGetLastError() == cudaSuccess ? LACACHE_OK : LACACHE_ERR_CUDA;
}
