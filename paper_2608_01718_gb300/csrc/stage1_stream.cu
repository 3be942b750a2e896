// Stage 1 on the CUDA cores, streaming: the key check sim(x, x') >= tau_c (Algorithm 1's cache search; section 4.1)
// for batches so small that reading the keys, not the arithmetic, bounds the scan. Threshold and per-query top_c are
// fused, so no score matrix reaches memory.
//
// Warp per key tile. A warp takes KT consecutive keys at a time. Each key row is cut into 16-byte chunks (8 bf16),
// and lane l owns chunks l, l + 32, l + 64, ...: for one key the 32 lanes read 512 contiguous bytes per 128-bit
// load (ld.global.nc.v4), so every load instruction of the warp is fully coalesced. The row goes in phases of PH
// chunks per lane, and all KT x PH loads of a phase are issued before any arithmetic. For one or two queries a phase
// is a whole row of up to 1024 elements (KT = 4 keys x PH = 4 chunks: 16 loads, 8 KB per warp in flight; KT = 8 for
// rows of at most 512 elements and one query); for 4 or 8 queries, 8 loads per phase, leaving registers for the sums.
//
// The queries of the launch sit in shared memory as fp32, split into the low and high halves of each chunk, so
// that lane l's reads of chunk l are contiguous across the warp (conflict-free 128-bit loads). They are taken QB
// at a time (a query group); each lane converts its key chunks to fp32 once per group and accumulates element
// pairs with packed fp32 FMAs (fma.rn.f32x2) into KT x QB partial sums.
//
// Reduction: one butterfly reduce-scatter over the warp turns the 32 lanes' V = KT x QB partials into full scores:
// lane l ends with value v = l / (32 / V), i.e. key v / QB of the tile and query v % QB of the group, after V - 1 +
// log2(32 / V) shuffles instead of 5 per score. Every score is summed in the same order (each lane's chunks in
// order, then the same butterfly tree), so equal keys give bit-equal scores.
//
// Threshold + top_c: every warp keeps, per query, a sorted list of packed (score, id) candidates in shared memory
// and a running threshold max(tau_c, c-th best). A lane whose score clears it inserts, one lane at a time
// (ballot order); the packed order makes the list independent of the order of arrival. At the end the CTA merges its
// warps' lists into the split's partial list (a record of its best score and candidate count, then the candidates).
// Grid: one CTA of 16 warps per SM, each CTA one contiguous split of the key range.
#include "internal.cuh"

namespace lc {
namespace {

constexpr int kWarps = 16;
constexpr int kThreads = kWarps * 32;
constexpr size_t kSmemBudget = 200 * 1024;   // queries + lists + thresholds, one CTA per SM

struct StreamParams {
  const __nv_bfloat16* keys;
  int64_t n;
  int d;
  int dc;             // 16-byte chunks per row, d / 8
  int nph;            // load phases per row: PH chunks per lane each
  const __nv_bfloat16* q;
  int B;              // row count of the partial lists
  int q0;             // first query of this launch
  int qn;             // queries of this launch
  int qpad;           // qn rounded up to the query group
  float tau_c;
  int top_c;
  int splits;
  uint64_t* part_cand;
  PartMeta* part_meta;
  int wait_first;     // the queries are written by the grid launched just before: wait before reading them
};

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

// d = a * b + c on both halves of a pair (one packed fp32 FMA)
__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) {
  float2 d;
  asm("{\n\t.reg .b64 ra, rb, rc, rd;\n\t"
      "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\tmov.b64 rc, {%6, %7};\n\t"
      "fma.rn.f32x2 rd, ra, rb, rc;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
  return d;
}

__device__ __forceinline__ uint4 load_chunk(const __nv_bfloat16* row, int c) {
  return __ldg(reinterpret_cast<const uint4*>(row) + c);
}

// Butterfly reduce-scatter of V = 2^m values per lane: afterwards each lane holds the warp-wide sum of value
// lane / (32 / V). Each step halves the vector (the lane keeps the half its lane bit selects and adds the partner's
// copy of it); once one value is left, the remaining steps add across the lanes that share it.
template <int V>
__device__ __forceinline__ float reduce_scatter(float (&x)[V], int lane) {
#pragma unroll
  for (int len = V, o = 16; len > 1; len >>= 1, o >>= 1) {
    const bool upper = (lane & o) != 0;
#pragma unroll
    for (int i = 0; i < len / 2; ++i) {
      const float keep = upper ? x[len / 2 + i] : x[i];
      const float send = upper ? x[i] : x[len / 2 + i];
      x[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
    }
  }
  float s = x[0];
#pragma unroll
  for (int o = 16 / V; o >= 1; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  return s;
}

// Insert packed candidate pk into the sorted (descending, 0-padded) list of C entries, and raise the threshold to
// the c-th best score once the list is full. Equal scores fall to the id order inside the packed key.
__device__ __forceinline__ void list_insert(uint64_t* lst, int C, uint64_t pk, float* thr, float tau_c) {
  if (pk <= lst[C - 1]) return;
  int i = C - 1;
  while (i > 0 && lst[i - 1] < pk) {
    lst[i] = lst[i - 1];
    --i;
  }
  lst[i] = pk;
  if (lst[C - 1] != 0) *thr = fmaxf(tau_c, cand_score(lst[C - 1]));
}

template <int QB, int KT, int PH>
__global__ void __launch_bounds__(kThreads, 1) stage1_stream_kernel(const StreamParams p) {
  extern __shared__ __align__(16) unsigned char smem[];
  const int dc = p.dc, qpad = p.qpad, C = p.top_c;
  float4* qlo = reinterpret_cast<float4*>(smem);                                 // [qpad][dc]
  float4* qhi = qlo + (size_t)qpad * dc;                                          // [qpad][dc]
  uint64_t* lists = reinterpret_cast<uint64_t*>(qhi + (size_t)qpad * dc);         // [kWarps][qpad][C]
  float* thr = reinterpret_cast<float*>(lists + (size_t)kWarps * qpad * C);       // [kWarps][qpad]
  float* best = thr + kWarps * qpad;                                              // [kWarps][qpad]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  // Launched as a programmatic dependent of the previous grid on the stream (the previous lookup's stage 2, which
  // reads the partial lists this grid writes and writes nothing it reads): the scan runs alongside it, and every
  // thread waits for it only before writing the partial lists. When the queries come from the grid just before
  // (the host-input gather), every thread waits here instead, before reading them.
  if (p.wait_first) asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  for (int i = threadIdx.x; i < qpad * dc; i += kThreads) {
    const int r = i / dc, c = i - r * dc;
    float4 lo = make_float4(0.f, 0.f, 0.f, 0.f), hi = lo;
    if (r < p.qn) {
      const uint4 v = load_chunk(p.q + (int64_t)(p.q0 + r) * p.d, c);
      lo = make_float4(bf_lo(v.x), bf_hi(v.x), bf_lo(v.y), bf_hi(v.y));
      hi = make_float4(bf_lo(v.z), bf_hi(v.z), bf_lo(v.w), bf_hi(v.w));
    }
    qlo[i] = lo;
    qhi[i] = hi;
  }
  for (int i = threadIdx.x; i < kWarps * qpad * C; i += kThreads) lists[i] = 0;
  for (int i = threadIdx.x; i < kWarps * qpad; i += kThreads) {
    thr[i] = p.tau_c;
    best[i] = -INFINITY;
  }
  __syncthreads();

  constexpr int V = KT * QB;           // scores per tile and query group
  constexpr int SPREAD = 32 / V;       // lanes that end the reduction with the same score
  constexpr int QS = QB < 4 ? QB : 4;  // queries whose chunk values sit in registers at once
  static_assert(V <= 32 && (V & (V - 1)) == 0, "KT * QB must be a power of two <= 32");
  const int my_v = lane / SPREAD;
  const int my_kt = my_v / QB, my_q = my_v % QB;
  const bool reporter = (lane % SPREAD) == 0;
  uint64_t* my_lists = lists + (size_t)warp * qpad * C;
  float* my_thr = thr + warp * qpad;
  float* my_best = best + warp * qpad;
  const int groups = qpad / QB;

  // one warp tile: keys [t0, t0 + KT), those at or past j_end absent
  auto tile = [&](int64_t t0, int64_t j_end) {
    for (int g = 0; g < groups; ++g) {
      float2 acc[KT][QB];
#pragma unroll
      for (int kt = 0; kt < KT; ++kt)
#pragma unroll
        for (int q = 0; q < QB; ++q) acc[kt][q] = make_float2(0.f, 0.f);
      for (int ph = 0; ph < p.nph; ++ph) {
        uint4 kv[KT][PH];
#pragma unroll
        for (int kt = 0; kt < KT; ++kt) {
          const int64_t j = t0 + kt;
          const __nv_bfloat16* row = p.keys + j * p.d;
#pragma unroll
          for (int i = 0; i < PH; ++i) {
            const int c = (ph * PH + i) * 32 + lane;
            kv[kt][i] = (j < j_end && c < dc) ? load_chunk(row, c) : make_uint4(0u, 0u, 0u, 0u);
          }
        }
#pragma unroll
        for (int i = 0; i < PH; ++i) {
          const int c = (ph * PH + i) * 32 + lane;
          if (c >= dc) continue;
#pragma unroll
          for (int qs = 0; qs < QB; qs += QS) {
            float2 qv[QS][4];
#pragma unroll
            for (int q = 0; q < QS; ++q) {
              const float4 a = qlo[(size_t)(g * QB + qs + q) * dc + c];
              const float4 b = qhi[(size_t)(g * QB + qs + q) * dc + c];
              qv[q][0] = make_float2(a.x, a.y);
              qv[q][1] = make_float2(a.z, a.w);
              qv[q][2] = make_float2(b.x, b.y);
              qv[q][3] = make_float2(b.z, b.w);
            }
#pragma unroll
            for (int kt = 0; kt < KT; ++kt) {
              const uint4 w = kv[kt][i];
              const float2 k0 = make_float2(bf_lo(w.x), bf_hi(w.x)), k1 = make_float2(bf_lo(w.y), bf_hi(w.y));
              const float2 k2 = make_float2(bf_lo(w.z), bf_hi(w.z)), k3 = make_float2(bf_lo(w.w), bf_hi(w.w));
#pragma unroll
              for (int q = 0; q < QS; ++q) {
                float2 t = acc[kt][qs + q];
                t = ffma2(k0, qv[q][0], t);
                t = ffma2(k1, qv[q][1], t);
                t = ffma2(k2, qv[q][2], t);
                t = ffma2(k3, qv[q][3], t);
                acc[kt][qs + q] = t;
              }
            }
          }
        }
      }
      // threshold, best score and top_c of the tile's scores for query group g
      float x[V];
#pragma unroll
      for (int kt = 0; kt < KT; ++kt)
#pragma unroll
        for (int q = 0; q < QB; ++q) x[kt * QB + q] = acc[kt][q].x + acc[kt][q].y;
      const float s = reduce_scatter<V>(x, lane);
      const int gq = g * QB + my_q;
      const int64_t j = t0 + my_kt;
      const bool valid = j < j_end && gq < p.qn;
      float m = valid ? s : -INFINITY;
#pragma unroll
      for (int o = SPREAD * QB; o < 32; o <<= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
      if (my_kt == 0 && reporter && gq < p.qn && m > my_best[gq]) my_best[gq] = m;
      const bool cand = valid && reporter && s >= my_thr[gq];
      unsigned mask = __ballot_sync(0xffffffffu, cand);
      while (mask) {
        const int src = __ffs(mask) - 1;
        mask &= mask - 1;
        if (lane == src)
          list_insert(my_lists + (size_t)gq * C, C, pack_cand(s, (uint32_t)j), my_thr + gq, p.tau_c);
        __syncwarp();
      }
    }
  };

  // the CTA's contiguous split of the keys, its warps interleaved over it
  const int64_t j_begin = p.n * blockIdx.x / p.splits, j_end = p.n * (blockIdx.x + 1) / p.splits;
  for (int64_t t0 = j_begin + (int64_t)warp * KT; t0 < j_end; t0 += (int64_t)kWarps * KT) tile(t0, j_end);

  __syncthreads();
  asm volatile("griddepcontrol.wait;" ::: "memory");
  // the split's partial list per query: merge of the warps' sorted lists
  for (int t = threadIdx.x; t < p.qn; t += kThreads) {
    int head[kWarps];
    float b = -INFINITY;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {
      head[w] = 0;
      b = fmaxf(b, best[w * qpad + t]);
    }
    uint64_t* dst = p.part_cand + ((int64_t)blockIdx.x * p.B + p.q0 + t) * C;
    int count = 0;
    for (; count < C; ++count) {
      uint64_t mx = 0;
      int mw = -1;
      for (int w = 0; w < kWarps; ++w) {
        const uint64_t x = head[w] < C ? lists[((size_t)w * qpad + t) * C + head[w]] : 0ull;
        if (x > mx) {
          mx = x;
          mw = w;
        }
      }
      if (mw < 0) break;   // every warp's list is exhausted
      dst[count] = mx;
      ++head[mw];
    }
    p.part_meta[(int64_t)blockIdx.x * p.B + p.q0 + t] = PartMeta{b, (uint32_t)count};
  }
}

size_t smem_bytes(int qpad, int d, int top_c) {
  return (size_t)qpad * d * 4 + (size_t)kWarps * qpad * ((size_t)8 * top_c + 8);
}

template <int QB, int KT, int PH>
cudaError_t launch_one(const StreamParams& p, cudaStream_t st) {
  const size_t smem = smem_bytes(p.qpad, p.d, p.top_c);
  cudaError_t e = cudaFuncSetAttribute(stage1_stream_kernel<QB, KT, PH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.splits);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, stage1_stream_kernel<QB, KT, PH>, p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

// Tile shape: KT keys per warp tile and PH chunks per lane per load phase, chosen so that the loads of a tile are
// in flight together (4-8 KB per warp) and the KT x QB packed partial sums fit beside them in 128 registers. Query
// groups of 1 or 2 load a whole row of up to 1024 elements in one phase (16 loads of 16 bytes per lane); rows of at
// most 512 elements take 8 keys per tile for one query (the partial sums of two queries would not fit beside them). Groups of 4 and 8 load 8 chunks per
// phase.
cudaError_t launch_shape(const StreamParams& p, int qb, cudaStream_t st) {
  const bool narrow = p.dc <= 64;
  switch (qb) {
    case 1: return narrow ? launch_one<1, 8, 2>(p, st) : launch_one<1, 4, 4>(p, st);
    case 2: return narrow ? launch_one<2, 4, 2>(p, st) : launch_one<2, 4, 4>(p, st);
    case 4: return launch_one<4, 4, 2>(p, st);
    default: return launch_one<8, 2, 4>(p, st);
  }
}
int shape_kt(int qb, int dc) { return qb == 1 ? (dc <= 64 ? 8 : 4) : qb <= 4 ? 4 : 2; }
int shape_ph(int qb, int dc) { return qb <= 2 ? (dc <= 64 ? 2 : 4) : qb == 4 ? 2 : 4; }

}  // namespace

cudaError_t launch_stage1_stream(const Stage1Args& a, int num_sms, int max_splits, cudaStream_t st, int* splits) {
  // query group: the batch rounded up to a power of two, at most 8; smaller if a group of fp32 query rows plus the
  // lists does not fit the shared-memory budget (d near its maximum)
  int qb = a.B <= 1 ? 1 : a.B <= 2 ? 2 : a.B <= 4 ? 4 : 8;
  while (qb > 1 && smem_bytes(qb, a.d, a.top_c) > kSmemBudget) qb >>= 1;
  if (smem_bytes(qb, a.d, a.top_c) > kSmemBudget) return cudaErrorInvalidValue;
  // queries per launch: as many whole groups as the budget holds; larger batches take several launches
  int qc = qb;
  while (qc < a.B && smem_bytes(qc + qb, a.d, a.top_c) <= kSmemBudget) qc += qb;
  StreamParams p{};
  p.keys = a.keys;
  p.n = a.n;
  p.d = a.d;
  p.dc = a.d / 8;
  const int kt = shape_kt(qb, p.dc), ph = shape_ph(qb, p.dc);
  p.nph = (p.dc + 32 * ph - 1) / (32 * ph);
  p.q = a.q;
  p.B = a.B;
  p.tau_c = a.tau_c;
  p.top_c = a.top_c;
  const int64_t tiles = (a.n + kt - 1) / kt;
  int64_t s = (tiles + kWarps - 1) / kWarps;
  if (s > num_sms) s = num_sms;
  if (s > max_splits) s = max_splits;
  if (s < 1) s = 1;
  p.splits = (int)s;
  p.part_cand = a.part_cand;
  p.part_meta = a.part_meta;
  *splits = p.splits;
  for (int q0 = 0; q0 < a.B; q0 += qc) {
    p.q0 = q0;
    p.qn = a.B - q0 < qc ? a.B - q0 : qc;
    p.qpad = (p.qn + qb - 1) / qb * qb;
    p.wait_first = q0 == 0 ? a.inputs_from_previous : 0;
    const cudaError_t e = launch_shape(p, qb, st);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace lc
