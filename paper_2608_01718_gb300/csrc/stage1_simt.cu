// Stage 1 on the CUDA cores: the key check sim(x, x') >= tau_c (Algorithm 1's cache search; section 4.1) as an
// FFMA scan, fused with the threshold and a per-query top_c, so no score matrix reaches memory.
//
// Grid: one CTA per split of the key range (contiguous rows). Block: 256 threads, one key per thread per tile.
// Queries are taken QC at a time and staged in shared memory as fp32. Each thread accumulates its key's QC
// scores in fp32, element 0..d-1 in order, so equal keys give bit-equal scores. Candidates that clear tau_c and
// beat the CTA's current c-th best go through a shared buffer. After every tile, one warp per query merges the
// buffer into the query's sorted list. Candidates are compared as packed (score, id) keys, so the lists do not
// depend on arrival order.
#include <string.h>

#include "internal.cuh"

namespace lc {
namespace {

constexpr int kThreads = 256;

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

template <int QC>
__global__ void __launch_bounds__(kThreads) stage1_simt_kernel(Stage1Args a, int splits) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int d = a.d;
  const int C = a.top_c;
  float* qs = reinterpret_cast<float*>(smem_raw);                       // [QC][d]
  uint64_t* list = reinterpret_cast<uint64_t*>(qs + QC * d);            // [QC][C]
  uint64_t* buf = list + QC * C;                                        // [QC][kThreads]
  int* cnt = reinterpret_cast<int*>(buf + QC * kThreads);               // [QC]
  unsigned int* best = reinterpret_cast<unsigned int*>(cnt + QC);       // [QC] score_order()

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int s = blockIdx.x;
  const int64_t j_begin = a.n * s / splits;
  const int64_t j_end = a.n * (s + 1) / splits;

  for (int q0 = 0; q0 < a.B; q0 += QC) {
    const int qn = min(QC, a.B - q0);
    for (int i = threadIdx.x; i < QC * d; i += kThreads) {
      const int qq = i / d;
      qs[i] = qq < qn ? __bfloat162float(a.q[(int64_t)(q0 + qq) * d + (i - qq * d)]) : 0.f;
    }
    for (int i = threadIdx.x; i < QC * C; i += kThreads) list[i] = 0;
    if (threadIdx.x < QC) {
      cnt[threadIdx.x] = 0;
      best[threadIdx.x] = score_order(-INFINITY);
    }
    __syncthreads();

    for (int64_t t0 = j_begin; t0 < j_end; t0 += kThreads) {
      const int64_t j = t0 + threadIdx.x;
      const bool valid = j < j_end;
      float acc[QC];
#pragma unroll
      for (int qq = 0; qq < QC; ++qq) acc[qq] = 0.f;
      if (valid) {
        const uint4* row = reinterpret_cast<const uint4*>(a.keys + j * d);
        for (int c8 = 0; c8 < d / 8; ++c8) {
          const uint4 v = __ldg(row + c8);
          const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&v);
          float kf[8];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float2 f = __bfloat1622float2(h2[e]);
            kf[2 * e] = f.x;
            kf[2 * e + 1] = f.y;
          }
#pragma unroll
          for (int qq = 0; qq < QC; ++qq) {
            const float4* qp = reinterpret_cast<const float4*>(qs + qq * d + c8 * 8);
            const float4 x0 = qp[0], x1 = qp[1];
            float t = acc[qq];
            t = fmaf(x0.x, kf[0], t);
            t = fmaf(x0.y, kf[1], t);
            t = fmaf(x0.z, kf[2], t);
            t = fmaf(x0.w, kf[3], t);
            t = fmaf(x1.x, kf[4], t);
            t = fmaf(x1.y, kf[5], t);
            t = fmaf(x1.z, kf[6], t);
            t = fmaf(x1.w, kf[7], t);
            acc[qq] = t;
          }
        }
      }
#pragma unroll
      for (int qq = 0; qq < QC; ++qq) {
        const float sc = valid ? acc[qq] : -INFINITY;
        const float wm = warp_max(sc);
        if (lane == 0 && qq < qn) atomicMax(&best[qq], score_order(wm));
        if (valid && qq < qn && sc >= a.tau_c) {
          const uint64_t key = pack_cand(sc, (uint32_t)j);
          if (key > list[qq * C + C - 1]) buf[qq * kThreads + atomicAdd(&cnt[qq], 1)] = key;
        }
      }
      __syncthreads();
      if (warp < QC && lane == 0) {
        uint64_t* L = list + warp * C;
        const int nb = cnt[warp];
        for (int i = 0; i < nb; ++i) {
          const uint64_t x = buf[warp * kThreads + i];
          if (x <= L[C - 1]) continue;
          int p = C - 1;
          while (p > 0 && L[p - 1] < x) {
            L[p] = L[p - 1];
            --p;
          }
          L[p] = x;
        }
        cnt[warp] = 0;
      }
      __syncthreads();
    }

    for (int i = threadIdx.x; i < qn * C; i += kThreads) {
      const int qq = i / C;
      a.part_cand[((int64_t)s * a.B + q0 + qq) * C + (i - qq * C)] = list[i];
    }
    if (threadIdx.x < qn) a.part_best[(int64_t)s * a.B + q0 + threadIdx.x] = score_of_order(best[threadIdx.x]);
    __syncthreads();
  }
}

template <int QC>
cudaError_t launch_qc(const Stage1Args& a, int splits, cudaStream_t st) {
  const size_t smem = (size_t)QC * a.d * 4 + (size_t)QC * a.top_c * 8 + (size_t)QC * kThreads * 8 + QC * 8;
  cudaError_t e = cudaFuncSetAttribute(stage1_simt_kernel<QC>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  stage1_simt_kernel<QC><<<splits, kThreads, smem, st>>>(a, splits);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_stage1_simt(const Stage1Args& a, int num_sms, int max_splits, cudaStream_t st, int* splits) {
  const int64_t tiles = (a.n + kThreads - 1) / kThreads;
  int s = (int)(tiles < (int64_t)num_sms ? tiles : (int64_t)num_sms);
  if (s > max_splits) s = max_splits;
  if (s < 1) s = 1;
  *splits = s;
  if (a.d <= 2048) return launch_qc<8>(a, s, st);
  if (a.d <= 4096) return launch_qc<4>(a, s, st);
  return launch_qc<2>(a, s, st);
}

}  // namespace lc
