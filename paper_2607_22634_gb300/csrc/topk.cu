// presto_topk: single-pass streaming log-softmax + top-k over the drafter's
// per-position logits (§2.3 marginals q_d, §4.3 top-k candidate extraction).
//
// Design (HBM-bound; roofline = B*L*V*elem bytes read once):
//   * Each row is split into `parts` contiguous spans so that the grid holds about
//     three CTAs per SM.  A CTA stages its span through shared memory with
//     cp.async.bulk copies (TMA, 16 KB stages, 4 in flight) tracked by mbarriers.
//   * Every lane keeps an online (max, sum-exp) pair; every warp keeps a sorted
//     top-k list spread over lanes 0..k-1 and a shared threshold, so only the
//     rare elements that beat the threshold cost an insertion (ballot + shuffle).
//   * Warp lists and (max, sum) pairs merge in shared memory; spans of one row
//     merge in the CTA that finishes last (atomic ticket), which writes the row.
#include <cuda_bf16.h>

#include <mutex>

#include "common.cuh"

namespace presto {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kStageBytes = 16384;
constexpr int kStages = 4;
constexpr int kSweepBytes = kThreads * 16;
constexpr int kCtasPerSm = 3;
constexpr float kLog2e = 1.4426950408889634f;
constexpr unsigned kFull = 0xffffffffu;

template <typename T>
struct Elem;
template <>
struct Elem<float> {
  static constexpr int kPerVec = 4;
  static constexpr int kBytes = 4;
  __device__ static float load(const float* p) { return *p; }
  __device__ static void unpack(const uint4& u, float (&v)[4]) {
    v[0] = __uint_as_float(u.x);
    v[1] = __uint_as_float(u.y);
    v[2] = __uint_as_float(u.z);
    v[3] = __uint_as_float(u.w);
  }
};
template <>
struct Elem<__nv_bfloat16> {
  static constexpr int kPerVec = 8;
  static constexpr int kBytes = 2;
  __device__ static float load(const __nv_bfloat16* p) { return __bfloat162float(*p); }
  __device__ static void unpack(const uint4& u, float (&v)[8]) {
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      v[2 * i] = __uint_as_float(w[i] << 16);
      v[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
    }
  }
};

struct Plan {
  int rows, parts, stages_per_row, stages_per_part;
  long long row_bytes, aligned_bytes;
};

Plan make_plan(int B, int L, int V, int elem_bytes) {
  Plan p;
  p.rows = B * L;
  p.row_bytes = static_cast<long long>(V) * elem_bytes;
  p.aligned_bytes = p.row_bytes / 16 * 16;
  p.stages_per_row = static_cast<int>((p.aligned_bytes + kStageBytes - 1) / kStageBytes);
  if (p.stages_per_row < 1) p.stages_per_row = 1;
  const int target = sm_count() * kCtasPerSm;
  int parts = (target + p.rows - 1) / p.rows;
  if (parts < 1) parts = 1;
  if (parts > p.stages_per_row) parts = p.stages_per_row;
  p.stages_per_part = (p.stages_per_row + parts - 1) / parts;
  p.parts = (p.stages_per_row + p.stages_per_part - 1) / p.stages_per_part;
  return p;
}

struct Workspace {
  float* val;       // [rows][parts][k]
  int* id;          // [rows][parts][k]
  float2* ms;       // [rows][parts] (max, sum-exp relative to max)
  unsigned* ticket; // [rows]
};

size_t workspace_layout(const Plan& p, int k, char* base, Workspace* w) {
  size_t off = 0;
  const size_t n = static_cast<size_t>(p.rows) * p.parts;
  auto take = [&](size_t bytes) {
    char* ptr = base ? base + off : nullptr;
    off = align_up(off + bytes, 256);
    return ptr;
  };
  char* val = take(n * k * sizeof(float));
  char* id = take(n * k * sizeof(int));
  char* ms = take(n * sizeof(float2));
  char* ticket = take(static_cast<size_t>(p.rows) * sizeof(unsigned));
  if (w) {
    w->val = reinterpret_cast<float*>(val);
    w->id = reinterpret_cast<int*>(id);
    w->ms = reinterpret_cast<float2*>(ms);
    w->ticket = reinterpret_cast<unsigned*>(ticket);
  }
  return off;
}

struct Args {
  const void* logits;
  long long row_stride;  // elements
  int V, k, parts, stages_per_part;
  long long aligned_bytes;
  int use_bulk;
  int32_t* topk_ids;
  float* topk_logq;
  float* lse;
  Workspace ws;
  int32_t* dev_status;
};

__device__ __forceinline__ long long llmin(long long a, long long b) { return a < b ? a : b; }

// (v1, id1) ranks before (v2, id2): larger value, then lower id.
__device__ __forceinline__ bool beats(float v1, int id1, float v2, int id2) {
  return v1 > v2 || (v1 == v2 && id1 < id2);
}

// Per-warp sorted top-k list: lane j < k holds the j-th entry; (tv, tid) is entry k-1.
struct WarpTopk {
  float lv;
  int lid;
  float tv;
  int tid;
  int k, lane;

  __device__ void init(int k_, int lane_) {
    k = k_;
    lane = lane_;
    lv = -INFINITY;
    lid = 0x7fffffff;
    tv = -INFINITY;
    tid = 0x7fffffff;
  }
  __device__ __forceinline__ void insert(float cv, int cid) {
    const unsigned better = __ballot_sync(kFull, lane < k && beats(lv, lid, cv, cid));
    const int pos = __popc(better);
    if (pos < k) {
      const float uv = __shfl_up_sync(kFull, lv, 1);
      const int uid = __shfl_up_sync(kFull, lid, 1);
      if (lane > pos) {
        lv = uv;
        lid = uid;
      }
      if (lane == pos) {
        lv = cv;
        lid = cid;
      }
      tv = __shfl_sync(kFull, lv, k - 1);
      tid = __shfl_sync(kFull, lid, k - 1);
    }
  }
  // Offer one element per lane (valid lanes only); filter against the threshold.
  __device__ __forceinline__ void offer(float v, int id, bool valid, float floor_v) {
    unsigned lanes = __ballot_sync(kFull, valid && v >= fmaxf(tv, floor_v) && beats(v, id, tv, tid));
    while (lanes) {
      const int src = __ffs(lanes) - 1;
      lanes &= lanes - 1;
      const float cv = __shfl_sync(kFull, v, src);
      const int cid = __shfl_sync(kFull, id, src);
      insert(cv, cid);
      lanes &= __ballot_sync(kFull, valid && beats(v, id, tv, tid));
    }
  }
};

struct LaneSum {
  float m = -INFINITY;
  float s = 0.f;
  template <int n>
  __device__ __forceinline__ void add(const float (&v)[n]) {
    float bm = v[0];
#pragma unroll
    for (int e = 1; e < n; ++e) bm = fmaxf(bm, v[e]);
    if (bm > m) {
      s *= ex2((m - bm) * kLog2e);
      m = bm;
    }
    if (m != -INFINITY) {
#pragma unroll
      for (int e = 0; e < n; ++e) s += ex2((v[e] - m) * kLog2e);
    }
  }
};

__device__ __forceinline__ void merge_ms(float& m, float& s, float m2, float s2) {
  const float M = fmaxf(m, m2);
  if (M == -INFINITY) return;
  s = s * ex2((m - M) * kLog2e) + s2 * ex2((m2 - M) * kLog2e);
  m = M;
}

__device__ __forceinline__ void warp_merge_ms(float& m, float& s) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const float m2 = __shfl_xor_sync(kFull, m, off);
    const float s2 = __shfl_xor_sync(kFull, s, off);
    merge_ms(m, s, m2, s2);
  }
}

// k-th largest per-lane maximum: no element below it can be in this warp's top-k,
// since at least k lane maxima (distinct elements) are >= it.
__device__ __forceinline__ float seed_floor(float lane_max, int k, int lane) {
  int rank = 0;
#pragma unroll 8
  for (int l = 0; l < 32; ++l) {
    const float o = __shfl_sync(kFull, lane_max, l);
    rank += (o > lane_max) || (o == lane_max && l < lane);
  }
  const unsigned at = __ballot_sync(kFull, rank == k - 1);
  return __shfl_sync(kFull, lane_max, __ffs(at) - 1);
}

template <typename T>
__device__ __forceinline__ void process_vec(const float (&v)[Elem<T>::kPerVec], int id0,
                                            int nvalid, WarpTopk& wt, LaneSum& ls,
                                            bool& seeded) {
  constexpr int n = Elem<T>::kPerVec;
  float x[n];
#pragma unroll
  for (int e = 0; e < n; ++e) x[e] = e < nvalid ? v[e] : -INFINITY;
  ls.add(x);
  float floor_v = -INFINITY;
  if (!seeded) {
    float lm = x[0];
#pragma unroll
    for (int e = 1; e < n; ++e) lm = fmaxf(lm, x[e]);
    floor_v = seed_floor(lm, wt.k, wt.lane);
    seeded = true;
  }
  float lm = x[0];
#pragma unroll
  for (int e = 1; e < n; ++e) lm = fmaxf(lm, x[e]);
  // Common case: no lane holds anything that can enter the list.
  if (!__any_sync(kFull, nvalid > 0 && lm >= fmaxf(wt.tv, floor_v))) return;
#pragma unroll
  for (int e = 0; e < n; ++e) wt.offer(x[e], id0 + e, e < nvalid, floor_v);
}

template <typename T>
__global__ void __launch_bounds__(kThreads) topk_kernel(const Args a) {
  constexpr int n = Elem<T>::kPerVec;
  constexpr int eb = Elem<T>::kBytes;
  extern __shared__ __align__(1024) uint8_t stage_mem[];
  __shared__ uint64_t full[kStages];
  __shared__ float s_val[kWarps][kMaxK];
  __shared__ int s_id[kWarps][kMaxK];
  __shared__ float2 s_ms[kWarps];
  __shared__ int s_last;

  const int row = blockIdx.x / a.parts;
  const int part = blockIdx.x % a.parts;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const T* rowp = static_cast<const T*>(a.logits) + static_cast<long long>(row) * a.row_stride;

  WarpTopk wt;
  wt.init(a.k, lane);
  LaneSum ls;
  bool seeded = false;

  const long long b0 = static_cast<long long>(part) * a.stages_per_part * kStageBytes;
  long long b1 = b0 + static_cast<long long>(a.stages_per_part) * kStageBytes;
  if (b1 > a.aligned_bytes) b1 = a.aligned_bytes;
  const int nst = b1 > b0 ? static_cast<int>((b1 - b0 + kStageBytes - 1) / kStageBytes) : 0;

  bool timed_out = false;
  if (a.use_bulk) {
    if (tid == 0) {
      for (int s = 0; s < kStages; ++s) mbar_init(&full[s], 1);
      fence_barrier_init();
    }
    __syncthreads();
    auto issue = [&](int st) {
      const long long off = b0 + static_cast<long long>(st) * kStageBytes;
      const uint32_t bytes = static_cast<uint32_t>(llmin(kStageBytes, b1 - off));
      uint8_t* dst = stage_mem + (st % kStages) * kStageBytes;
      mbar_arrive_expect_tx(&full[st % kStages], bytes);
      bulk_g2s(dst, reinterpret_cast<const uint8_t*>(rowp) + off, bytes, &full[st % kStages]);
    };
    if (tid == 0)
      for (int st = 0; st < nst && st < kStages; ++st) issue(st);
    for (int st = 0; st < nst; ++st) {
      const int slot = st % kStages;
      const bool ok = mbar_wait(&full[slot], (st / kStages) & 1);
      if (__syncthreads_or(!ok)) {  // CTA-uniform decision
        timed_out = true;
        if (tid == 0)  // drain the copies still in flight, again bounded
          for (int s2 = st + 1; s2 < nst && s2 < st + kStages; ++s2)
            mbar_wait(&full[s2 % kStages], (s2 / kStages) & 1);
        break;
      }
      const long long off = b0 + static_cast<long long>(st) * kStageBytes;
      const int valid_bytes = static_cast<int>(llmin(kStageBytes, b1 - off));
      const uint8_t* sp = stage_mem + slot * kStageBytes;
      for (int sw = 0; sw < kStageBytes; sw += kSweepBytes) {
        const int boff = sw + tid * 16;
        float v[n];
        int nvalid = 0;
        if (boff < valid_bytes) {
          Elem<T>::unpack(*reinterpret_cast<const uint4*>(sp + boff), v);
          nvalid = n;
        } else {
#pragma unroll
          for (int e = 0; e < n; ++e) v[e] = -INFINITY;
        }
        process_vec<T>(v, static_cast<int>((off + boff) / eb), nvalid, wt, ls, seeded);
      }
      __syncthreads();  // every thread is done with this slot before it is refilled
      if (tid == 0 && st + kStages < nst) issue(st + kStages);
    }
  } else {
    // Unaligned rows: plain loads over the same element range.
    const long long e0 = b0 / eb, e1 = b1 / eb;
    for (long long sb = e0; sb < e1; sb += static_cast<long long>(kThreads) * n) {
      const long long id0 = sb + static_cast<long long>(tid) * n;
      float v[n];
      int nvalid = 0;
#pragma unroll
      for (int e = 0; e < n; ++e) {
        const bool ok = id0 + e < e1;
        v[e] = ok ? Elem<T>::load(rowp + id0 + e) : -INFINITY;
        nvalid += ok;
      }
      process_vec<T>(v, static_cast<int>(id0), nvalid, wt, ls, seeded);
    }
  }
  // Row tail not covered by 16-byte units: the last part reads it directly.
  if (part == a.parts - 1) {
    const long long t0 = a.aligned_bytes / eb;
    if (t0 < a.V) {
      const long long id0 = t0 + static_cast<long long>(tid) * n;
      float v[n];
      int nvalid = 0;
#pragma unroll
      for (int e = 0; e < n; ++e) {
        const bool ok = id0 + e < a.V;
        v[e] = ok ? Elem<T>::load(rowp + id0 + e) : -INFINITY;
        nvalid += ok;
      }
      process_vec<T>(v, static_cast<int>(id0), nvalid, wt, ls, seeded);
    }
  }
  if (timed_out) report(a.dev_status, PRESTO_DEV_TIMEOUT);

  // ---- CTA merge: warp lists and (max, sum) pairs -> warp 0.
  float m = ls.m, s = ls.s;
  warp_merge_ms(m, s);
  if (lane < a.k) {
    s_val[warp][lane] = wt.lv;
    s_id[warp][lane] = wt.lid;
  }
  if (lane == 0) s_ms[warp] = make_float2(m, s);
  __syncthreads();
  if (warp != 0) return;
  for (int w = 1; w < kWarps; ++w) {
    const bool ok = lane < a.k;
    wt.offer(ok ? s_val[w][lane] : -INFINITY, ok ? s_id[w][lane] : 0x7fffffff, ok, -INFINITY);
  }
  m = lane < kWarps ? s_ms[lane].x : -INFINITY;
  s = lane < kWarps ? s_ms[lane].y : 0.f;
  warp_merge_ms(m, s);

  if (a.parts > 1) {
    const size_t slot = static_cast<size_t>(row) * a.parts + part;
    if (lane < a.k) {
      a.ws.val[slot * a.k + lane] = wt.lv;
      a.ws.id[slot * a.k + lane] = wt.lid;
    }
    if (lane == 0) a.ws.ms[slot] = make_float2(m, s);
    __threadfence();
    __syncwarp();
    if (lane == 0) s_last = atomicAdd(&a.ws.ticket[row], 1u) == static_cast<unsigned>(a.parts - 1);
    __syncwarp();
    if (!s_last) return;
    __threadfence();
    // Last CTA of the row: merge every span's list and (max, sum).
    wt.init(a.k, lane);
    const int total = a.parts * a.k;
    const size_t base = static_cast<size_t>(row) * a.parts * a.k;
    for (int i0 = 0; i0 < total; i0 += 32) {
      const int i = i0 + lane;
      const bool ok = i < total;
      const float v = ok ? __ldcg(a.ws.val + base + i) : -INFINITY;
      const int id = ok ? __ldcg(a.ws.id + base + i) : 0x7fffffff;
      wt.offer(v, id, ok, -INFINITY);
    }
    m = -INFINITY;
    s = 0.f;
    for (int p = lane; p < a.parts; p += 32) {
      const float2 ms = __ldcg(a.ws.ms + static_cast<size_t>(row) * a.parts + p);
      merge_ms(m, s, ms.x, ms.y);
    }
    warp_merge_ms(m, s);
  }
  // ---- write the row
  const float logs = logf(s);
  if (!(m > -INFINITY && m < INFINITY)) {
    if (lane == 0) report(a.dev_status, PRESTO_DEV_NONFINITE);
  }
  if (lane < a.k) {
    a.topk_ids[static_cast<size_t>(row) * a.k + lane] = wt.lid;
    a.topk_logq[static_cast<size_t>(row) * a.k + lane] = (wt.lv - m) - logs;
  }
  if (lane == 0 && a.lse) a.lse[row] = m + logs;
}

}  // namespace
}  // namespace presto

using namespace presto;

extern "C" size_t presto_topk_workspace(int B, int L, int V, int k) {
  if (B < 1 || L < 1 || V < 1 || k < 1 || k > kMaxK) return 0;
  // Sized for the larger element type (float32 rows give the most spans).
  const Plan p = make_plan(B, L, V, 4);
  return workspace_layout(p, k, nullptr, nullptr);
}

extern "C" int presto_topk(const void* logits, int dtype, int B, int L, int V,
                           long long row_stride, int k, int32_t* topk_ids, float* topk_logq,
                           float* lse, void* ws, size_t ws_bytes, int32_t* dev_status,
                           presto_stream_t stream) {
  PRESTO_CHECK_ARG(logits && topk_ids && topk_logq);
  PRESTO_CHECK_ARG(dtype == PRESTO_F32 || dtype == PRESTO_BF16);
  PRESTO_CHECK_ARG(B >= 1 && L >= 1 && V >= 1 && k >= 1 && row_stride >= V);
  PRESTO_CHECK_ARG(k <= V);
  PRESTO_CHECK_LIMIT(k <= kMaxK && V < kMaxV && L <= kMaxL);
  const int eb = dtype == PRESTO_F32 ? 4 : 2;
  const Plan p = make_plan(B, L, V, eb);
  Workspace w{};
  if (p.parts > 1) {
    if (!ws || ws_bytes < workspace_layout(p, k, nullptr, nullptr)) return PRESTO_ERR_WORKSPACE;
    if (reinterpret_cast<uintptr_t>(ws) % 256) return PRESTO_ERR_WORKSPACE;
    workspace_layout(p, k, static_cast<char*>(ws), &w);
    if (cudaMemsetAsync(w.ticket, 0, sizeof(unsigned) * p.rows, stream) != cudaSuccess)
      return PRESTO_ERR_CUDA;
  }
  Args a;
  a.logits = logits;
  a.row_stride = row_stride;
  a.V = V;
  a.k = k;
  a.parts = p.parts;
  a.stages_per_part = p.stages_per_part;
  a.aligned_bytes = p.aligned_bytes;
  a.use_bulk = (reinterpret_cast<uintptr_t>(logits) % 16 == 0) && ((row_stride * eb) % 16 == 0);
  a.topk_ids = topk_ids;
  a.topk_logq = topk_logq;
  a.lse = lse;
  a.ws = w;
  a.dev_status = dev_status;
  const dim3 grid(static_cast<unsigned>(p.rows) * p.parts);
  const size_t smem = a.use_bulk ? static_cast<size_t>(kStages) * kStageBytes : 0;
  static bool attr_set = [] {
    cudaFuncSetAttribute(topk_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         kStages * kStageBytes);
    cudaFuncSetAttribute(topk_kernel<__nv_bfloat16>,
                         cudaFuncAttributeMaxDynamicSharedMemorySize, kStages * kStageBytes);
    return true;
  }();
  (void)attr_set;
  if (dtype == PRESTO_F32)
    topk_kernel<float><<<grid, kThreads, smem, stream>>>(a);
  else
    topk_kernel<__nv_bfloat16><<<grid, kThreads, smem, stream>>>(a);
  return launch_status();
}

// ---------------------------------------------------------------------------
// Allocation-free top-k.
//
// Some callers cannot hand this library a workspace: a plugin running inside an
// inference server whose device memory all belongs to the host framework's
// allocator, a C caller with no allocator handle at all, or a latency-critical
// loop that must not call cudaMalloc (which can block on device-wide
// synchronisation and fail under fragmentation).  For them this entry point
// keeps the span partials of presto_topk in a fixed file-scope device array
// instead of a caller workspace, and otherwise runs the same code.
//
// The array costs kStaticScratchBytes on every GPU that loads this library, for
// the life of the process.  All calls on one device share it: two calls whose
// kernels overlap on the GPU (different streams, no ordering between them) race
// on it.  Its contents persist between calls; the per-row tickets that must
// start at zero are cleared by an async memset on the caller's stream at every
// call, and everything else is written before it is read.
// ---------------------------------------------------------------------------
namespace presto {
namespace {

constexpr size_t kStaticScratchBytes = PRESTO_TOPK_STATIC_SCRATCH_BYTES;
__device__ __align__(256) unsigned char g_topk_scratch[kStaticScratchBytes];

std::mutex g_scratch_mutex;
void* g_scratch_addr[64] = {};

// Device address of g_topk_scratch for the current device.  Host code cannot use
// the symbol itself (its host-side name is only a stand-in), so the address is
// looked up once per device, with that device current, and cached.
void* static_scratch() {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  std::lock_guard<std::mutex> lock(g_scratch_mutex);
  if (!g_scratch_addr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_topk_scratch) != cudaSuccess || !p) return nullptr;
    g_scratch_addr[dev] = p;
  }
  return g_scratch_addr[dev];
}

}  // namespace
}  // namespace presto

extern "C" int presto_topk_noalloc(const void* logits, int dtype, int B, int L, int V,
                                   long long row_stride, int k, int32_t* topk_ids,
                                   float* topk_logq, float* lse, int32_t* dev_status,
                                   presto_stream_t stream) {
  PRESTO_CHECK_ARG(logits && topk_ids && topk_logq);
  PRESTO_CHECK_ARG(dtype == PRESTO_F32 || dtype == PRESTO_BF16);
  PRESTO_CHECK_ARG(B >= 1 && L >= 1 && V >= 1 && k >= 1 && k <= V && row_stride >= V);
  PRESTO_CHECK_LIMIT(k <= kMaxK && V < kMaxV && L <= kMaxL);
  const size_t need = presto_topk_workspace(B, L, V, k);
  if (need > kStaticScratchBytes) return PRESTO_ERR_UNSUPPORTED;
  void* ws = static_scratch();
  if (!ws) return PRESTO_ERR_CUDA;
  return presto_topk(logits, dtype, B, L, V, row_stride, k, topk_ids, topk_logq, lse, ws,
                     kStaticScratchBytes, dev_status, stream);
}
