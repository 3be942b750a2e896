// Threshold calibration (App. A.2, "Threshold Calibration"): the similarity of every benign pair, the nearest-rank
// percentile of those similarities, and the capped threshold min(cap, percentile).
//
//   pair_sim_kernel   one warp per pair: fp32 dot of two bf16 rows (16-byte loads, each lane's chunks in order,
//                     butterfly sum). HBM-bound: 4d bytes per pair.
//   select_*          the exact k-th smallest similarity by a three-pass radix select (11, 11, 10 bits) over the
//                     similarities mapped to order-preserving unsigned integers: per-pass counting over all CTAs
//                     (shared histograms, warp-aggregated adds) into a global histogram, then a one-CTA pick.
#include <math.h>

#include "internal.cuh"

namespace lc {
namespace {

constexpr int kPairWarps = 8;

__device__ __forceinline__ float dot8(const uint4& u, const uint4& v, float acc) {
  const __nv_bfloat162* a = reinterpret_cast<const __nv_bfloat162*>(&u);
  const __nv_bfloat162* b = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const float2 x = __bfloat1622float2(a[e]);
    const float2 y = __bfloat1622float2(b[e]);
    acc = fmaf(x.x, y.x, acc);
    acc = fmaf(x.y, y.y, acc);
  }
  return acc;
}

__global__ void __launch_bounds__(kPairWarps * 32)
    pair_sim_kernel(const uint4* __restrict__ x, const uint4* __restrict__ y, int64_t n, int d,
                    float* __restrict__ sims) {
  const int lane = threadIdx.x & 31;
  const int64_t i = (int64_t)blockIdx.x * kPairWarps + (threadIdx.x >> 5);
  if (i >= n) return;
  const int v = d / 8;
  float acc = 0.f;
  for (int c = lane; c < v; c += 32) acc = dot8(__ldg(x + i * v + c), __ldg(y + i * v + c), acc);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if (lane == 0) sims[i] = acc;
}

// Exact k-th smallest similarity: a radix select over the order-preserving integer image of the floats, 11, 11
// and 10 bits per pass. Each pass counts, over all CTAs, the elements whose higher bits equal the prefix chosen so
// far; a one-CTA kernel then picks the bin that holds the rank and narrows the prefix.
constexpr int kBins = 2048;
constexpr int kCountThreads = 1024;
constexpr int kPerThread = 8;

struct SelectState {
  uint32_t prefix;
  uint32_t mask;
  int64_t rank;   // rank still to find among the elements matching prefix under mask (0-based)
};

__device__ __forceinline__ unsigned int* ws_hist(void* ws) { return static_cast<unsigned int*>(ws); }
__device__ __forceinline__ SelectState* ws_state(void* ws) {
  return reinterpret_cast<SelectState*>(static_cast<unsigned char*>(ws) + kBins * 4);
}

__global__ void select_init(void* ws, int64_t rank) {
  for (int b = threadIdx.x; b < kBins; b += blockDim.x) ws_hist(ws)[b] = 0;
  if (threadIdx.x == 0) *ws_state(ws) = SelectState{0u, 0u, rank};
}

__global__ void __launch_bounds__(kCountThreads)
    select_count(const float* __restrict__ sims, int64_t n, void* ws, int shift, uint32_t bin_mask) {
  __shared__ unsigned int hist[kBins];
  const int lane = threadIdx.x & 31;
  for (int b = threadIdx.x; b < kBins; b += blockDim.x) hist[b] = 0;
  __syncthreads();
  const SelectState st = *ws_state(ws);
  const int64_t step = (int64_t)gridDim.x * blockDim.x * kPerThread;
  const int64_t n_round = (n + step - 1) / step * step;   // uniform trip count: every lane reaches __match_any_sync
  for (int64_t base = (int64_t)blockIdx.x * blockDim.x * kPerThread; base < n_round; base += step) {
    float v[kPerThread];
#pragma unroll
    for (int u = 0; u < kPerThread; ++u) {
      const int64_t i = base + (int64_t)u * blockDim.x + threadIdx.x;
      v[u] = i < n ? __ldg(sims + i) : 0.f;
    }
#pragma unroll
    for (int u = 0; u < kPerThread; ++u) {
      const int64_t i = base + (int64_t)u * blockDim.x + threadIdx.x;
      uint32_t bin = kBins;   // not counted
      if (i < n) {
        const uint32_t o = score_order(v[u]);
        if ((o & st.mask) == st.prefix) bin = (o >> shift) & bin_mask;
      }
      const unsigned peers = __match_any_sync(0xffffffffu, bin);
      if (bin < kBins && lane == __ffs(peers) - 1) atomicAdd(&hist[bin], __popc(peers));
    }
  }
  __syncthreads();
  for (int b = threadIdx.x; b < kBins; b += blockDim.x)
    if (hist[b]) atomicAdd(&ws_hist(ws)[b], hist[b]);
}

// One CTA of kBins / 2 threads: exclusive scan of the histogram, the bin holding the rank, the narrowed prefix;
// the histogram is cleared for the next pass. After the last pass the prefix is the value itself.
__global__ void __launch_bounds__(kBins / 2)
    select_pick(void* ws, int shift, uint32_t bin_mask, float cap, float* __restrict__ out, int last) {
  __shared__ unsigned long long part[kBins / 2];
  __shared__ int s_bin;
  __shared__ unsigned long long s_below;
  unsigned int* gh = ws_hist(ws);
  SelectState* st = ws_state(ws);
  const int t = threadIdx.x;
  const unsigned long long c0 = gh[2 * t], c1 = gh[2 * t + 1];
  part[t] = c0 + c1;
  __syncthreads();
  for (int off = 1; off < kBins / 2; off <<= 1) {   // inclusive scan (Hillis-Steele)
    const unsigned long long add = t >= off ? part[t - off] : 0;
    __syncthreads();
    part[t] += add;
    __syncthreads();
  }
  const unsigned long long before = t ? part[t - 1] : 0;
  const unsigned long long r = (unsigned long long)st->rank;
  if (r >= before && r < before + c0 + c1) {
    const bool first = r < before + c0;
    s_bin = 2 * t + (first ? 0 : 1);
    s_below = first ? before : before + c0;
  }
  __syncthreads();
  gh[2 * t] = 0;
  gh[2 * t + 1] = 0;
  if (t == 0) {
    SelectState nx = *st;
    nx.prefix |= (uint32_t)s_bin << shift;
    nx.mask |= bin_mask << shift;
    nx.rank = (int64_t)(r - s_below);
    *st = nx;
    if (last) {
      const float value = score_of_order(nx.prefix);
      out[0] = value;
      out[1] = fminf(cap, value);
    }
  }
}

}  // namespace

size_t calibrate_workspace_bytes() { return kBins * 4 + sizeof(SelectState); }

cudaError_t launch_calibrate(const void* x, const void* y, int64_t n, int d, int64_t rank, float cap, float* sims,
                             float* result, void* ws, int num_sms, cudaStream_t st) {
  const int64_t blocks = (n + kPairWarps - 1) / kPairWarps;
  pair_sim_kernel<<<(unsigned)blocks, kPairWarps * 32, 0, st>>>(static_cast<const uint4*>(x),
                                                                 static_cast<const uint4*>(y), n, d, sims);
  select_init<<<1, 1024, 0, st>>>(ws, rank);
  const int64_t want = (n + (int64_t)kCountThreads * kPerThread - 1) / ((int64_t)kCountThreads * kPerThread);
  const int grid = (int)(want < 2 * num_sms ? want : 2 * num_sms);
  const int shifts[3] = {21, 10, 0};
  const uint32_t masks[3] = {0x7FFu, 0x7FFu, 0x3FFu};
  for (int pass = 0; pass < 3; ++pass) {
    select_count<<<grid, kCountThreads, 0, st>>>(sims, n, ws, shifts[pass], masks[pass]);
    select_pick<<<1, kBins / 2, 0, st>>>(ws, shifts[pass], masks[pass], cap, result, pass == 2);
  }
  return cudaGetLastError();
}

}  // namespace lc

extern "C" size_t lacache_calibrate_workspace_bytes(void) { return lc::calibrate_workspace_bytes(); }

extern "C" lacache_status lacache_calibrate(int64_t n, int32_t d, const void* x_dev, const void* y_dev,
                                            double percentile, float cap, float* sims_dev, float* result_dev,
                                            void* workspace_dev, void* cuda_stream) {
  lc::NvtxRange nvtx("lacache_calibrate");
  if (n < 1 || n > (int64_t)INT32_MAX || d <= 0 || !x_dev || !y_dev || !sims_dev || !result_dev || !workspace_dev)
    return LACACHE_ERR_INVALID_ARG;
  if (!(percentile >= 0.0 && percentile <= 100.0) || isnan(cap)) return LACACHE_ERR_INVALID_ARG;
  if (d % 8 != 0 || d > lc::kMaxD) return LACACHE_ERR_UNSUPPORTED;
  if (((uintptr_t)x_dev & 15u) || ((uintptr_t)y_dev & 15u) || ((uintptr_t)workspace_dev & 15u))
    return LACACHE_ERR_INVALID_ARG;
  // nearest rank: ceil(percentile / 100 * n), at least 1 and at most n; the kernels take it 0-based
  int64_t rank = (int64_t)ceil(percentile / 100.0 * (double)n);
  if (rank < 1) rank = 1;
  if (rank > n) rank = n;
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return LACACHE_ERR_CUDA;
  return lc::launch_calibrate(x_dev, y_dev, n, d, rank - 1, cap, sims_dev, result_dev, workspace_dev, sms,
                              (cudaStream_t)cuda_stream) == cudaSuccess
             ? LACACHE_OK
             : LACACHE_ERR_CUDA;
}
