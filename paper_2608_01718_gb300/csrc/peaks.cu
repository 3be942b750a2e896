// Measurement kernels for the benchmark's roofline denominators; built into libpeaks.so, beside the lookup library
// and not part of it. Each launches asynchronously on the given stream; the caller times it with CUDA events.
//
//  lcpeaks_read: a read-only stream over a device buffer (128-bit ld.global.nc loads, four in flight per thread,
//    four 512-thread CTAs per SM), the rate at which this GPU's HBM delivers data to a kernel that only reads. The
//    copy figure of the peaks file moves the same bytes twice (read and write) and runs below it.
//  lcpeaks_popc: the SimHash scan's distance arithmetic with no memory traffic: every thread holds one entry's
//    signature words in registers and, per step, takes its Hamming distance to 32 query signatures read from shared
//    memory (XOR, three carry-save adders per 8 words, 5 population counts, compare with a radius), exactly as the
//    scan's inner loop does; the entry words change every step (one add per word) so nothing is loop-invariant.
//    The rate in signature words compared per second is the scan's integer-ALU ceiling.
#include <cuda_runtime.h>
#include <stdint.h>

namespace {

constexpr int kThreads = 512;

__global__ void __launch_bounds__(kThreads) read_stream_kernel(const uint4* __restrict__ buf, size_t n16,
                                                                unsigned* sink) {
  uint32_t acc = 0;
  const size_t stride = (size_t)gridDim.x * blockDim.x;
  size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x;
  for (; i + 3 * stride < n16; i += 4 * stride) {
    uint4 v[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) v[u] = __ldg(buf + i + u * stride);
#pragma unroll
    for (int u = 0; u < 4; ++u) acc ^= v[u].x ^ v[u].y ^ v[u].z ^ v[u].w;
  }
  for (; i < n16; i += stride) {
    const uint4 v = __ldg(buf + i);
    acc ^= v.x ^ v.y ^ v.z ^ v.w;
  }
  if (acc == 0x5EED5EEDu) *sink = acc;   // keeps the loads alive; the buffer never holds this pattern
}

__device__ __forceinline__ void csa(uint32_t& hi, uint32_t& lo, uint32_t a, uint32_t b, uint32_t c) {
  const uint32_t u = a ^ b;
  lo = u ^ c;
  hi = (a & b) | (u & c);
}

template <int W>
__device__ __forceinline__ int hamming(const uint32_t (&x)[W]) {
  int h = 0;
  if constexpr (W % 8 == 0) {
#pragma unroll
    for (int g = 0; g < W; g += 8) {
      uint32_t ca, sa, cb, sb, cc, sc;
      csa(ca, sa, x[g], x[g + 1], x[g + 2]);
      csa(cb, sb, x[g + 3], x[g + 4], x[g + 5]);
      csa(cc, sc, sa, sb, x[g + 6]);
      h += __popc(sc) + __popc(x[g + 7]) + 2 * (__popc(ca) + __popc(cb) + __popc(cc));
    }
  } else {
#pragma unroll
    for (int g = 0; g < W; g += 4) {
      uint32_t c, s;
      csa(c, s, x[g], x[g + 1], x[g + 2]);
      h += __popc(s) + __popc(x[g + 3]) + 2 * __popc(c);
    }
  }
  return h;
}

template <int W>
__global__ void __launch_bounds__(kThreads, 2) popc_mix_kernel(int steps, int radius, unsigned* sink) {
  __shared__ __align__(16) uint32_t qsig[32][W];
  for (int i = threadIdx.x; i < 32 * W; i += kThreads) qsig[i / W][i % W] = 0x9E3779B9u * (uint32_t)(i + 1);
  __syncthreads();
  uint32_t e[W];
#pragma unroll
  for (int w = 0; w < W; ++w) e[w] = 0x85EBCA6Bu * (uint32_t)(blockIdx.x * kThreads + threadIdx.x + w + 1);
  unsigned acc = 0;
  for (int s = 0; s < steps; ++s) {
    unsigned pend = 0;
#pragma unroll 1
    for (int g = 0; g < 32; g += 8) {
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int qq = g + u;
        const uint4* qs = reinterpret_cast<const uint4*>(qsig[qq]);
        uint32_t x[W];
#pragma unroll
        for (int w = 0; w < W / 4; ++w) {
          const uint4 v = qs[w];
          x[4 * w] = e[4 * w] ^ v.x;
          x[4 * w + 1] = e[4 * w + 1] ^ v.y;
          x[4 * w + 2] = e[4 * w + 2] ^ v.z;
          x[4 * w + 3] = e[4 * w + 3] ^ v.w;
        }
        pend |= (hamming<W>(x) <= radius ? 1u : 0u) << qq;
      }
    }
    acc += __popc(pend);
#pragma unroll
    for (int w = 0; w < W; ++w) e[w] += 0x27D4EB2Fu;   // the next entry
  }
  if (acc == 0xFFFFFFFFu) *sink = acc;
}

}  // namespace

extern "C" {

// Reads `bytes` (a multiple of 16) of the 16-byte aligned device buffer `buf` once. `sink` is a device word the
// kernel may write. Returns the cudaError_t of the launch.
int lcpeaks_read(const void* buf, size_t bytes, unsigned* sink, int num_sms, void* stream) {
  read_stream_kernel<<<4 * num_sms, kThreads, 0, (cudaStream_t)stream>>>(static_cast<const uint4*>(buf), bytes / 16,
                                                                        sink);
  return (int)cudaGetLastError();
}

// Two 512-thread CTAs per SM, each thread comparing `steps` entries of `words` signature words (4, 8 or 16) with 32
// queries: 2 * num_sms * 512 * steps * 32 * words signature words in all.
int lcpeaks_popc(int words, int steps, int radius, unsigned* sink, int num_sms, void* stream) {
  const dim3 grid(2 * num_sms);
  cudaStream_t st = (cudaStream_t)stream;
  switch (words) {
    case 4: popc_mix_kernel<4><<<grid, kThreads, 0, st>>>(steps, radius, sink); break;
    case 8: popc_mix_kernel<8><<<grid, kThreads, 0, st>>>(steps, radius, sink); break;
    case 16: popc_mix_kernel<16><<<grid, kThreads, 0, st>>>(steps, radius, sink); break;
    default: return (int)cudaErrorInvalidValue;
  }
  return (int)cudaGetLastError();
}

}  // extern "C"
