// Step A2 -- per-position reduction over the vocabulary logits.
//
// For each row x of V logits (the confidences that edits are thresholded on:
// Table 10's refine threshold, Appendix C.4's confident edits):
//   m = max x,  argmax = lowest index attaining m,
//   S = sum exp(x - m),  lse = m + ln S,  conf = 1 / S  (= exp(m - lse)).
//
// An HBM-bound stream: every logit is read exactly once, 16 bytes per load,
// coalesced across the block; with several waves of rows the loads go through
// a per-thread shared-memory staging ring (cp.async, eight vectors in flight
// per thread), otherwise straight into registers (four in flight). Each thread
// keeps an online (max, first index, scaled sum) triple; the sum is rescaled
// only when a 16-byte vector raises the running maximum, and the exponentials
// go two at a time through the packed fp32 FMA and add of the sm_100 family,
// so that the instruction stream stays below what HBM delivers per SM.
// Threads combine by warp shuffles, warps through shared memory, and -- with
// at most two rows per SM -- the CTAs of a thread-block cluster that split one
// row combine through distributed shared memory (no global scratch memory).
//
// The fused variant (vocab_step_kernel) also runs step A3: the CTA finishing a
// sequence's last row performs its update, counted with one int32 arrival
// counter per sequence in caller-provided scratch memory.
#include <cooperative_groups.h>

#include <cmath>
#include <cstdint>

#include "dlm_common.cuh"
#include "dlm_internal.h"
#include "update_impl.cuh"

namespace cg = cooperative_groups;

namespace dlm {
namespace {

constexpr int kThreads = 256;
constexpr int kUnroll = 4;
constexpr float kLog2e = 1.4426950408889634f;

struct Partial {
  float m;    // running maximum (exact logit value)
  int idx;    // lowest index attaining m
  float s;    // sum of exp(x - m)
};

// Combines two partials; the lower index wins ties of the maximum.
__device__ __forceinline__ Partial combine(Partial a, Partial b) {
  Partial r;
  r.m = fmaxf(a.m, b.m);
  if (a.m > b.m) r.idx = a.idx;
  else if (b.m > a.m) r.idx = b.idx;
  else r.idx = min(a.idx, b.idx);
  if (r.m == -INFINITY) {
    r.s = 0.f;
  } else {
    float sa = a.m == -INFINITY ? 0.f : a.s * ex2_approx((a.m - r.m) * kLog2e);
    float sb = b.m == -INFINITY ? 0.f : b.s * ex2_approx((b.m - r.m) * kLog2e);
    r.s = sa + sb;
  }
  return r;
}

__device__ __forceinline__ uint4 ld_stream16(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.L2::256B.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

// Elements of one 16-byte vector as fp32.
template <bool BF16>
struct Vec;

template <>
struct Vec<true> {
  static constexpr int kN = 8;
  __device__ __forceinline__ static void unpack(uint4 v, float (&x)[8]) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      x[2 * j] = __uint_as_float(w[j] << 16);
      x[2 * j + 1] = __uint_as_float(w[j] & 0xFFFF0000u);
    }
  }
  __device__ __forceinline__ static float load1(const void* base, int64_t i) {
    uint16_t h = static_cast<const uint16_t*>(base)[i];
    return __uint_as_float(static_cast<uint32_t>(h) << 16);
  }
};

template <>
struct Vec<false> {
  static constexpr int kN = 4;
  __device__ __forceinline__ static void unpack(uint4 v, float (&x)[4]) {
    x[0] = __uint_as_float(v.x);
    x[1] = __uint_as_float(v.y);
    x[2] = __uint_as_float(v.z);
    x[3] = __uint_as_float(v.w);
  }
  __device__ __forceinline__ static float load1(const void* base, int64_t i) {
    return static_cast<const float*>(base)[i];
  }
};

// Folds one value x at element index e into p (the scalar path: rows whose
// length or alignment rules out 16-byte vectors, and a row's ragged tail).
__device__ __forceinline__ void fold1(Partial& p, float& mL, float x, int e) {
  if (x > p.m) {
    p.s = (p.m == -INFINITY) ? 0.f : p.s * ex2_approx((p.m - x) * kLog2e);
    p.m = x;
    p.idx = e;
    mL = x * kLog2e;
  }
  if (p.m != -INFINITY) p.s += ex2_approx(fmaf(x, kLog2e, -mL));
}

// Folds one 16-byte vector of kN values starting at element index e0: the
// vector's maximum first (raising the running maximum rescales the sum, which
// is rare), then the kN exponentials in pairs with packed fp32 FMA and add
// into the two-lane running sum s2. mL is the running maximum times log2(e)
// and stays finite (0 until the first finite maximum): an entry of -inf then
// adds exp2(-inf) = 0 without a guard.
template <int kN>
__device__ __forceinline__ void fold_vec(Partial& p, float& mL, float2& s2, const float (&x)[kN], int e0) {
  float vm;
  if constexpr (kN == 8) vm = fmaxf(fmax3(fmax3(x[0], x[1], x[2]), fmax3(x[3], x[4], x[5]), x[6]), x[7]);
  else vm = fmaxf(fmax3(x[0], x[1], x[2]), x[3]);
  if (vm > p.m) {
    int first = kN - 1;
#pragma unroll
    for (int j = kN - 1; j >= 0; --j)
      if (x[j] == vm) first = j;
    const float f = (p.m == -INFINITY) ? 0.f : ex2_approx((p.m - vm) * kLog2e);
    s2 = make_float2(s2.x * f, s2.y * f);
    p.m = vm;
    p.idx = e0 + first;
    mL = vm * kLog2e;
  }
  const float2 k2 = make_float2(kLog2e, kLog2e), n2 = make_float2(-mL, -mL);
#pragma unroll
  for (int j = 0; j < kN; j += 2) {
    const float2 y = ffma2(make_float2(x[j], x[j + 1]), k2, n2);
    s2 = fadd2(s2, make_float2(ex2_approx(y.x), ex2_approx(y.y)));
  }
}

// Reduces the block's partials into thread 0's return value.
__device__ __forceinline__ Partial block_reduce(Partial p) {
  __shared__ Partial warp_part[kThreads / 32];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    Partial q;
    q.m = __shfl_xor_sync(0xffffffffu, p.m, o);
    q.idx = __shfl_xor_sync(0xffffffffu, p.idx, o);
    q.s = __shfl_xor_sync(0xffffffffu, p.s, o);
    p = combine(p, q);
  }
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (lane == 0) warp_part[warp] = p;
  __syncthreads();
  if (warp == 0) {
    p = lane < kThreads / 32 ? warp_part[lane] : Partial{-INFINITY, 0x7FFFFFFF, 0.f};
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      Partial q;
      q.m = __shfl_xor_sync(0xffffffffu, p.m, o);
      q.idx = __shfl_xor_sync(0xffffffffu, p.idx, o);
      q.s = __shfl_xor_sync(0xffffffffu, p.s, o);
      p = combine(p, q);
    }
  }
  return p;
}

// Scans elements [e_begin, e_end) of one row.
template <bool BF16, bool VEC>
__device__ __forceinline__ Partial scan_range(const char* row, int64_t e_begin, int64_t e_end) {
  using VT = Vec<BF16>;
  constexpr int kN = VT::kN;
  Partial p{-INFINITY, 0x7FFFFFFF, 0.f};
  float mL = 0.f;
  if constexpr (VEC) {
    // e_begin and e_end are multiples of kN except possibly the row's end.
    const int64_t v_begin = e_begin / kN;
    const int64_t v_end = e_end / kN;  // full vectors
    const uint4* vp = reinterpret_cast<const uint4*>(row);
    float2 s2 = make_float2(0.f, 0.f);
    int64_t vi = v_begin + threadIdx.x;
    for (; vi + (kUnroll - 1) * kThreads < v_end; vi += kUnroll * kThreads) {
      uint4 raw[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) raw[u] = ld_stream16(vp + vi + u * kThreads);
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        float x[kN];
        VT::unpack(raw[u], x);
        fold_vec<kN>(p, mL, s2, x, static_cast<int>((vi + u * kThreads) * kN));
      }
    }
    for (; vi < v_end; vi += kThreads) {
      float x[kN];
      VT::unpack(ld_stream16(vp + vi), x);
      fold_vec<kN>(p, mL, s2, x, static_cast<int>(vi * kN));
    }
    p.s = s2.x + s2.y;
    e_begin = v_end * kN;  // scalar tail (row length not a multiple of kN)
  }
  for (int64_t e = e_begin + threadIdx.x; e < e_end; e += kThreads)
    fold1(p, mL, VT::load1(row, e), static_cast<int>(e));
  return p;
}

// 16-byte asynchronous copy global -> shared (bypassing L1), and its groups.
__device__ __forceinline__ void cp_async16(void* smem_dst, const void* gsrc) {
  asm volatile("cp.async.cg.shared.global.L2::256B [%0], [%1], 16;" ::"r"(smem_u32(smem_dst)), "l"(gsrc) : "memory");
}
// The same copy, issued only once `after` holds its value: passing a register
// loaded from the destination slot orders the slot's read before its refill.
__device__ __forceinline__ void cp_async16_after(void* smem_dst, const void* gsrc, uint32_t after) {
  asm volatile("cp.async.cg.shared.global.L2::256B [%0], [%1], 16;" ::"r"(smem_u32(smem_dst)), "l"(gsrc), "r"(after)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// scan_range for 16-byte aligned rows with the loads staged through shared
// memory: each thread keeps kStages of its vectors in flight in its own slots
// of `ring` ([kStages][kThreads]), reads back only what it copied itself (so
// no block barrier), and refills a slot as soon as its value is in registers:
// twice the bytes in flight of the register-loaded scan, with no registers
// held for them.
template <bool BF16, int kStages>
__device__ __forceinline__ Partial scan_range_staged(const char* row, int64_t e_begin, int64_t e_end, uint4* ring) {
  using VT = Vec<BF16>;
  constexpr int kN = VT::kN;
  Partial p{-INFINITY, 0x7FFFFFFF, 0.f};
  float mL = 0.f;
  float2 s2 = make_float2(0.f, 0.f);
  const uint4* vp = reinterpret_cast<const uint4*>(row);
  const int64_t v_end = e_end / kN;
  const int64_t first = e_begin / kN + threadIdx.x;
  const int nk = first < v_end ? static_cast<int>((v_end - first + kThreads - 1) / kThreads) : 0;
  uint4* mine = ring + threadIdx.x;
#pragma unroll
  for (int k = 0; k < kStages; ++k) {
    if (k < nk) cp_async16(mine + k * kThreads, vp + first + static_cast<int64_t>(k) * kThreads);
    cp_async_commit();
  }
  for (int k = 0; k < nk; ++k) {
    cp_async_wait<kStages - 1>();  // the group of vector k has landed
    uint4* slot = mine + (k % kStages) * kThreads;
    const uint4 v = *slot;
    if (k + kStages < nk) cp_async16_after(slot, vp + first + static_cast<int64_t>(k + kStages) * kThreads, v.w);
    cp_async_commit();
    float x[kN];
    VT::unpack(v, x);
    fold_vec<kN>(p, mL, s2, x, static_cast<int>((first + static_cast<int64_t>(k) * kThreads) * kN));
  }
  cp_async_wait<0>();
  p.s = s2.x + s2.y;
  for (int64_t e = v_end * kN + threadIdx.x; e < e_end; e += kThreads)  // ragged tail
    fold1(p, mL, VT::load1(row, e), static_cast<int>(e));
  return p;
}

__device__ __forceinline__ void write_out(const VocabArgs& a, int64_t rowi, Partial p) {
  // A NaN entry makes the sum NaN; a row of only -inf leaves the maximum -inf.
  if (kCheckBounds && (isnan(p.s) || p.m == -INFINITY)) set_device_error(a.err, DLM_DEVERR_INPUT);
  a.argmax[rowi] = p.idx;
  a.conf[rowi] = 1.0f / p.s;
  a.lse[rowi] = p.m + logf(p.s);
}

// One CTA per row (grid-stride over rows). kStaged: the loads go through the
// shared-memory staging ring of scan_range_staged (16-byte aligned rows only).
constexpr int kStages = 8;
template <bool BF16, bool VEC, bool kStaged>
__global__ void __launch_bounds__(kThreads, 4) vocab_rows_kernel(VocabArgs a) {
  __shared__ uint4 ring[kStaged ? kStages * kThreads : 1];
  const int esz = BF16 ? 2 : 4;
  for (int64_t rowi = blockIdx.x; rowi < a.N; rowi += gridDim.x) {
    const char* row = static_cast<const char*>(a.logits) + rowi * a.row_stride * esz;
    Partial p = kStaged ? scan_range_staged<BF16, kStages>(row, 0, a.V, ring) : scan_range<BF16, VEC>(row, 0, a.V);
    p = block_reduce(p);
    if (threadIdx.x == 0) write_out(a, rowi, p);
    __syncthreads();
  }
}

// Fused A2 + A3: one CTA per row as above; the CTA that completes the last
// row of a sequence (an arrival counter per sequence in `counters`) then runs
// that sequence's refine update, reading the predictions the other CTAs wrote
// around L1. The counter of a sequence is returned to zero by its last CTA,
// so `counters` must be zero before the first launch and is zero after each
// complete launch.
template <bool BF16, bool VEC>
__global__ void __launch_bounds__(kThreads, 4) vocab_step_kernel(VocabArgs a, UpdateArgs u, int* counters, int* err) {
  __shared__ UpdateShared<kThreads> ush;
  __shared__ int last;
  __shared__ uint4 ring[VEC ? kStages * kThreads : 1];
  const int esz = BF16 ? 2 : 4;
  for (int64_t rowi = blockIdx.x; rowi < a.N; rowi += gridDim.x) {
    const char* row = static_cast<const char*>(a.logits) + rowi * a.row_stride * esz;
    Partial p = VEC ? scan_range_staged<BF16, kStages>(row, 0, a.V, ring) : scan_range<BF16, VEC>(row, 0, a.V);
    p = block_reduce(p);
    const int b = static_cast<int>(rowi / u.L);
    if (threadIdx.x == 0) {
      write_out(a, rowi, p);
      __threadfence();  // the predictions are visible before the arrival is
      last = atomicAdd(&counters[b], 1) == u.L - 1;
    }
    __syncthreads();
    if (last) {
      if (threadIdx.x == 0) counters[b] = 0;
      __threadfence();
      refine_sequence<kThreads, true>(u, b, err, ush);
    }
    __syncthreads();
  }
}

// Rows split over a cluster of `csize` CTAs: CTA c of a cluster scans chunk c
// of the row, rank 0 combines the chunk partials through distributed shared
// memory. Persistent: cluster k takes rows k, k + clusters, ..., so a launch is
// one wave of resident CTAs, with no per-row launch and ramp-up; the partial
// slots alternate between rows, so one cluster barrier per row suffices (rank
// 0 reads row i's partials before it scans row i + 1, whose barrier the other
// CTAs must pass before they overwrite that slot with row i + 2's).
template <bool BF16, bool VEC>
__global__ void __launch_bounds__(kThreads, 4) vocab_cluster_kernel(VocabArgs a) {
  __shared__ Partial cta_part[2];
  cg::cluster_group cluster = cg::this_cluster();
  const int csize = static_cast<int>(cluster.num_blocks());
  const int crank = static_cast<int>(cluster.block_rank());
  const int64_t nclusters = gridDim.x / csize;
  const int esz = BF16 ? 2 : 4;
  const int kN = BF16 ? 8 : 4;
  // Chunk boundaries on whole vectors.
  const int64_t nvec = (a.V + kN - 1) / kN;
  const int64_t per = (nvec + csize - 1) / csize;
  int64_t e0 = crank * per * kN;
  int64_t e1 = (crank + 1) * per * kN;
  if (e0 > a.V) e0 = a.V;
  if (e1 > a.V) e1 = a.V;
  int it = 0;
  for (int64_t rowi = blockIdx.x / csize; rowi < a.N; rowi += nclusters, ++it) {
    const char* row = static_cast<const char*>(a.logits) + rowi * a.row_stride * esz;
    Partial p = scan_range<BF16, VEC>(row, e0, e1);
    p = block_reduce(p);
    if (threadIdx.x == 0) cta_part[it & 1] = p;
    cluster.sync();
    if (crank == 0 && threadIdx.x < 32) {
      Partial q{-INFINITY, 0x7FFFFFFF, 0.f};
      if (static_cast<int>(threadIdx.x) < csize) q = *cluster.map_shared_rank(&cta_part[it & 1], threadIdx.x);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        Partial t;
        t.m = __shfl_xor_sync(0xffffffffu, q.m, o);
        t.idx = __shfl_xor_sync(0xffffffffu, q.idx, o);
        t.s = __shfl_xor_sync(0xffffffffu, q.s, o);
        q = combine(q, t);
      }
      if (threadIdx.x == 0) write_out(a, rowi, q);
    }
  }
  cluster.sync();  // keep every CTA's shared memory alive until rank 0 has read it
}

// Probability of a given token of each row: one gathered logit per row.
template <bool BF16>
__global__ void __launch_bounds__(256) token_prob_kernel(VocabArgs a, const int32_t* tokens, const float* lse,
                                                         float* prob) {
  const int64_t r = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (r >= a.N) return;
  const int32_t t = tokens[r];
  float p = 0.f;
  if (kCheckBounds && (t < 0 || t >= a.V)) set_device_error(a.err, DLM_DEVERR_INPUT);
  if (t >= 0 && t < a.V) {
    const int64_t off = r * a.row_stride + t;
    const float x = BF16 ? __bfloat162float(static_cast<const __nv_bfloat16*>(a.logits)[off])
                         : static_cast<const float*>(a.logits)[off];
    p = expf(x - lse[r]);
  }
  prob[r] = p;
}

template <bool BF16, bool VEC>
int launch_typed(const VocabArgs& a, cudaStream_t stream) {
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int esz = BF16 ? 2 : 4;
  const int64_t row_bytes = a.V * esz;
  const int64_t want_ctas = 4LL * sms;  // resident CTAs at 4 per SM
  // One CTA per row wherever there are rows enough to keep more than two CTAs
  // per SM streaming: measured on this GPU (V = 151552, bf16), splitting rows
  // over clusters wins only up to about 2 rows per SM (64 rows: 16 us against
  // 21; 304: 22.6 against 24.9), and loses beyond (512 rows: 49.6 against 31.3,
  // as each CTA's short chunks pay the memory latency once per row).
  if (row_bytes < 65536 || a.N > 2LL * sms) {
    const int64_t grid = a.N < 64LL * want_ctas ? a.N : 64LL * want_ctas;
    if (VEC && a.N > want_ctas) {
      // Several waves of rows: stage the loads through shared memory
      // (measured at 32 x 512 x 151552: 0.692 ms against 0.722-0.733 for the
      // register-loaded scan; with a single wave of rows the latter is as fast).
      vocab_rows_kernel<BF16, VEC, true><<<static_cast<unsigned>(grid), kThreads, 0, stream>>>(a);
    } else {
      vocab_rows_kernel<BF16, VEC, false><<<static_cast<unsigned>(grid), kThreads, 0, stream>>>(a);
    }
  } else {
    // Few long rows: split each over a cluster. Choose the cluster size that
    // minimises the rows' share per CTA, ceil(N / clusters) / csize, with
    // clusters = resident CTAs / csize (never more clusters than rows).
    int csize = 2;
    int64_t nclusters = 1;
    double best = 1e30;
    for (int c = 2; c <= 8; c *= 2) {
      int64_t nc = want_ctas / c;
      if (nc > a.N) nc = a.N;
      const double cost = static_cast<double>((a.N + nc - 1) / nc) / c;
      if (cost < best - 1e-9) {
        best = cost;
        csize = c;
        nclusters = nc;
      }
    }
    cudaLaunchConfig_t cfg = {};
    cfg.blockDim = dim3(kThreads);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = csize;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    // No more clusters than can be resident at once (one wave).
    cfg.gridDim = dim3(static_cast<unsigned>(nclusters * csize));
    int active = 0;
    if (cudaOccupancyMaxActiveClusters(&active, vocab_cluster_kernel<BF16, VEC>, &cfg) == cudaSuccess && active > 0 &&
        nclusters > active) {
      nclusters = active;
      cfg.gridDim = dim3(static_cast<unsigned>(nclusters * csize));
    }
    cudaGetLastError();  // an occupancy query that failed leaves the grid as computed
    cudaError_t e = cudaLaunchKernelEx(&cfg, vocab_cluster_kernel<BF16, VEC>, a);
    if (e != cudaSuccess)
      return fail(DLM_ERR_CUDA, "vocab_confidence cluster launch: %s", cudaGetErrorString(e));
  }
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return fail(DLM_ERR_CUDA, "vocab_confidence launch: %s", cudaGetErrorString(e));
  return DLM_OK;
}

}  // namespace

int launch_vocab_confidence(const VocabArgs& a, cudaStream_t stream) {
  if (a.N == 0) return DLM_OK;
  const int esz = a.is_bf16 ? 2 : 4;
  const bool vec = (reinterpret_cast<uintptr_t>(a.logits) % 16 == 0) && ((a.row_stride * esz) % 16 == 0);
  if (a.is_bf16) return vec ? launch_typed<true, true>(a, stream) : launch_typed<true, false>(a, stream);
  return vec ? launch_typed<false, true>(a, stream) : launch_typed<false, false>(a, stream);
}

int launch_token_prob(const VocabArgs& a, const int32_t* tokens, const float* lse, float* prob,
                      cudaStream_t stream) {
  if (a.N == 0) return DLM_OK;
  const unsigned grid = static_cast<unsigned>((a.N + 255) / 256);
  if (a.is_bf16) token_prob_kernel<true><<<grid, 256, 0, stream>>>(a, tokens, lse, prob);
  else token_prob_kernel<false><<<grid, 256, 0, stream>>>(a, tokens, lse, prob);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return fail(DLM_ERR_CUDA, "token_prob launch: %s", cudaGetErrorString(e));
  return DLM_OK;
}

int launch_vocab_step(const VocabArgs& a, const UpdateArgs& u, int* counters, cudaStream_t stream) {
  if (a.N == 0) return DLM_OK;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t cap = 2LL * 64 * sms;
  const unsigned grid = static_cast<unsigned>(a.N < cap ? a.N : cap);
  const int esz = a.is_bf16 ? 2 : 4;
  const bool vec = (reinterpret_cast<uintptr_t>(a.logits) % 16 == 0) && ((a.row_stride * esz) % 16 == 0);
  int* err = device_error_word();
  if (a.is_bf16) {
    if (vec) vocab_step_kernel<true, true><<<grid, kThreads, 0, stream>>>(a, u, counters, err);
    else vocab_step_kernel<true, false><<<grid, kThreads, 0, stream>>>(a, u, counters, err);
  } else {
    if (vec) vocab_step_kernel<false, true><<<grid, kThreads, 0, stream>>>(a, u, counters, err);
    else vocab_step_kernel<false, false><<<grid, kThreads, 0, stream>>>(a, u, counters, err);
  }
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return fail(DLM_ERR_CUDA, "refine_step launch: %s", cudaGetErrorString(e));
  return DLM_OK;
}

}  // namespace dlm
