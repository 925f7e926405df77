// presto_topk: single-pass streaming log-softmax + top-k over the drafter's
// per-position logits (§2.3 marginals q_d, §4.3 top-k candidate extraction).
//
// Design (HBM-bound; roofline = B*L*V*elem bytes read once):
//   * A row is split into `parts` contiguous spans.  Spans of one row form a
//     thread-block cluster (<= 8 CTAs) and merge through distributed shared memory;
//     only when very few rows would leave the GPU idle does a row take more spans,
//     which then merge through a workspace in the CTA that finishes last.
//   * Each warp of a CTA streams its own 2 KB chunks of the span through shared
//     memory (cp.async.bulk = TMA, 4 chunks in flight per warp, one mbarrier per
//     slot), so the stream needs no CTA-wide barrier.
//   * Elements are ordered by a 64-bit key (value bits mapped to an ordered integer,
//     then the complement of the token id), so "larger value, then lower id" is
//     plain integer order and every key is unique.
//   * Per chunk, pass A accumulates each lane's online (max, sum exp) and its
//     largest key; the chunk's candidates are the keys above the warp's current
//     k-th best, raised when needed to the k-th largest lane maximum (no element
//     below that can be among the chunk's k best, and at most k lanes x 32 elements
//     can reach it).  Pass B re-reads the chunk from shared memory and collects the
//     candidates; a rank count merges them with the warp's list.  The CTA merges
//     its warps' lists once at the end.
#include <cuda_bf16.h>

#include <cooperative_groups.h>

#include <mutex>

#include "common.cuh"

namespace presto {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kStageBytes = 16384;                  // planning unit: bytes per CTA stage
constexpr int kChunkBytes = 2048;                   // one warp's bulk copy
constexpr int kWarpSlots = 4;                       // chunks in flight per warp
constexpr int kVecs = kChunkBytes / (32 * 16);      // 16-byte vectors per lane per chunk
constexpr int kWarpRoom = 512;                      // candidate keys per warp and chunk
constexpr int kMaxCluster = 8;
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

enum Mode { kDirect = 0, kCluster = 1, kGlobal = 2 };

struct Plan {
  int rows, parts, stages_per_row, stages_per_part, mode;
  long long row_bytes, aligned_bytes;
};

Plan make_plan(int B, int L, int V, int elem_bytes) {
  Plan p;
  p.rows = B * L;
  p.row_bytes = static_cast<long long>(V) * elem_bytes;
  p.aligned_bytes = p.row_bytes / 16 * 16;
  p.stages_per_row = static_cast<int>((p.aligned_bytes + kStageBytes - 1) / kStageBytes);
  if (p.stages_per_row < 1) p.stages_per_row = 1;
  const int sms = sm_count();
  int parts = (3 * sms / 2 + p.rows - 1) / p.rows;  // about 1.5 CTAs per SM
  if (parts < 1) parts = 1;
  if (parts > p.stages_per_row) parts = p.stages_per_row;
  // clusters of up to 8 CTAs while that still gives half the SMs a CTA; only a
  // handful of rows spreads wider, merging through the workspace
  if (parts > kMaxCluster && 2 * p.rows * kMaxCluster >= sms) parts = kMaxCluster;
  p.stages_per_part = (p.stages_per_row + parts - 1) / parts;
  p.parts = (p.stages_per_row + p.stages_per_part - 1) / p.stages_per_part;
  p.mode = p.parts == 1 ? kDirect : (p.parts <= kMaxCluster ? kCluster : kGlobal);
  return p;
}

struct Workspace {
  unsigned long long* keys;  // [rows][parts][k]
  float2* ms;                // [rows][parts] (max, sum exp relative to max)
  unsigned* ticket;          // [rows]
};

size_t workspace_layout(const Plan& p, int k, char* base, Workspace* w) {
  if (p.mode != kGlobal) return 256;
  size_t off = 0;
  const size_t n = static_cast<size_t>(p.rows) * p.parts;
  auto take = [&](size_t bytes) {
    char* ptr = base ? base + off : nullptr;
    off = align_up(off + bytes, 256);
    return ptr;
  };
  char* keys = take(n * k * sizeof(unsigned long long));
  char* ms = take(n * sizeof(float2));
  char* ticket = take(static_cast<size_t>(p.rows) * sizeof(unsigned));
  if (w) {
    w->keys = reinterpret_cast<unsigned long long*>(keys);
    w->ms = reinterpret_cast<float2*>(ms);
    w->ticket = reinterpret_cast<unsigned*>(ticket);
  }
  return off;
}

struct Args {
  const void* logits;
  long long row_stride;  // elements
  int V, k, parts, stages_per_part, mode;
  long long aligned_bytes;
  int use_bulk;
  int32_t* topk_ids;
  float* topk_logq;
  float* lse;
  Workspace ws;
  int32_t* dev_status;
};

__device__ __forceinline__ uint32_t ordered(float f) {
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float unordered(uint32_t o) {
  return __uint_as_float((o & 0x80000000u) ? (o & 0x7fffffffu) : ~o);
}
// Larger key = earlier in (value desc, id asc).  0 marks "no element".
__device__ __forceinline__ unsigned long long elem_key(float v, int id) {
  return (static_cast<unsigned long long>(ordered(v)) << 32) |
         static_cast<uint32_t>(0xFFFFFFFFu - static_cast<uint32_t>(id));
}
__device__ __forceinline__ float key_value(unsigned long long key) {
  return unordered(static_cast<uint32_t>(key >> 32));
}
__device__ __forceinline__ int key_id(unsigned long long key) {
  return static_cast<int>(0xFFFFFFFFu - static_cast<uint32_t>(key));
}
__device__ __forceinline__ long long llmin(long long a, long long b) { return a < b ? a : b; }

// Online (max, sum exp) of one thread, kept in the log2 domain: m2 = max * log2(e),
// s = sum 2^(x*log2(e) - m2).
struct LaneSum {
  float m2 = -INFINITY;
  float s = 0.f;
  template <int n>
  __device__ __forceinline__ void add(const float (&v)[n], float bm) {
    const float bm2 = bm * kLog2e;
    if (bm2 > m2) {
      s *= ex2(m2 - bm2);
      m2 = bm2;
    }
    if (m2 != -INFINITY) {
#pragma unroll
      for (int e = 0; e < n; ++e) s += ex2(fmaf(v[e], kLog2e, -m2));
    }
  }
  __device__ __forceinline__ float max_value() const { return m2 * (1.f / kLog2e); }
};

// Merge two (max, sum) pairs of the log2 domain.
__device__ __forceinline__ void merge_ms(float& m2, float& s, float n2, float t) {
  const float M = fmaxf(m2, n2);
  if (M == -INFINITY) return;
  s = s * ex2(m2 - M) + t * ex2(n2 - M);
  m2 = M;
}

__device__ __forceinline__ void warp_merge_ms(float& m, float& s) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const float m2 = __shfl_xor_sync(kFull, m, off);
    const float s2 = __shfl_xor_sync(kFull, s, off);
    merge_ms(m, s, m2, s2);
  }
}

struct WarpTopk {
  unsigned long long cand[kWarpRoom + kMaxK];  // chunk candidates, then the list
  unsigned long long list[kMaxK];              // running top-k of the warp, descending
  int n_cand;
  int n_list;
};

struct TopkSmem {
  WarpTopk w[kWarps];
  unsigned long long cand[kWarps * kMaxK + kMaxCluster * kMaxK];
  unsigned long long list[kMaxK];      // top-k of the CTA (then of the row), descending
  unsigned long long part[kMaxCluster][kMaxK];  // leader: lists of the cluster's CTAs
  float2 part_ms[kMaxCluster];
  float2 warp_ms[kWarps];
  int last;
  int count;
};

// Keys e[0..M) (unique apart from zeros, 0 = none) -> their descending top-k in
// out[0..k) by rank counting; returns how many were written (all threads).
// Block-wide; ends with a barrier.
__device__ int rank_select(const unsigned long long* e, int M, int k, unsigned long long* out,
                           int* counter, int tid) {
  if (tid == 0) *counter = 0;
  __syncthreads();
  int nz = 0;
  for (int i = tid; i < M; i += kThreads) {
    const unsigned long long ki = e[i];
    if (ki == 0ull) continue;
    ++nz;
    int r = 0;
    for (int j = 0; j < M; ++j) r += e[j] > ki;
    if (r < k) out[r] = ki;
  }
  if (nz) atomicAdd(counter, nz);
  __syncthreads();
  const int valid = *counter;
  __syncthreads();
  return valid < k ? valid : k;
}

// One chunk of elements [elem0, elem0 + count), processed by one warp: lane owns
// vectors (i * 32 + lane) for i < kVecs.  `ld(v, off, n)` loads n elements at
// element offset `off` of the chunk into v (missing elements as -inf).
template <typename T, typename Load>
__device__ __forceinline__ void warp_chunk(WarpTopk& wt, long long elem0, int count, int k,
                                          int lane, LaneSum& ls, Load ld) {
  constexpr int n = Elem<T>::kPerVec;
  // pass A: sum of exponentials, and the lane's largest element (lowest index on ties)
  float tmax = -INFINITY;
  int targ = -1;
#pragma unroll
  for (int i = 0; i < kVecs; ++i) {
    const int off = (i * 32 + lane) * n;
    if (off < count) {
      float v[n];
      const int nv = min(n, count - off);
      ld(v, off, nv);
      float bm = v[0];
#pragma unroll
      for (int e = 1; e < n; ++e) bm = fmaxf(bm, v[e]);
      ls.add(v, bm);
      if (bm > tmax || targ < 0) {
#pragma unroll
        for (int e = n - 1; e >= 0; --e)
          if (e < nv && v[e] == bm) targ = off + e;
        tmax = bm;
      }
    }
  }
  const unsigned long long tkey =
      targ < 0 ? 0ull : elem_key(tmax, static_cast<int>(elem0 + targ));
  const int nl = wt.n_list;
  const unsigned long long list_thr = nl >= k ? wt.list[k - 1] + 1ull : 1ull;
  const unsigned busy = __ballot_sync(kFull, tkey >= list_thr);
  if (busy == 0u) return;  // common case once the list has settled
  unsigned long long thr = list_thr;
  if (__popc(busy) * kVecs * n > kWarpRoom) {
    // raise the threshold to the k-th largest lane key of the chunk
    int r = 0;
#pragma unroll 8
    for (int l = 0; l < 32; ++l) {
      const unsigned long long o = __shfl_sync(kFull, tkey, l);
      r += o > tkey || (o == tkey && l < lane);
    }
    const int src = __ffs(__ballot_sync(kFull, r == k - 1)) - 1;
    const unsigned long long thr0 = __shfl_sync(kFull, tkey, src);
    thr = thr0 > thr ? thr0 : thr;
  }
  // pass B: collect the chunk's keys at or above the threshold (<= kWarpRoom)
  if (lane == 0) wt.n_cand = 0;
  __syncwarp();
  if (tkey >= thr) {
#pragma unroll
    for (int i = 0; i < kVecs; ++i) {
      const int off = (i * 32 + lane) * n;
      if (off < count) {
        float v[n];
        const int nv = min(n, count - off);
        ld(v, off, nv);
#pragma unroll
        for (int e = 0; e < n; ++e)
          if (e < nv) {
            const unsigned long long key = elem_key(v[e], static_cast<int>(elem0 + off + e));
            if (key >= thr) {
              const int slot = atomicAdd(&wt.n_cand, 1);
              if (slot < kWarpRoom) wt.cand[slot] = key;
            }
          }
      }
    }
  }
  __syncwarp();
  // merge: candidates + the current list, ranked by counting
  const int nc = min(wt.n_cand, kWarpRoom);
  if (lane < nl) wt.cand[nc + lane] = wt.list[lane];
  __syncwarp();
  const int M = nc + nl;
  for (int i = lane; i < M; i += 32) {
    const unsigned long long ki = wt.cand[i];
    int r = 0;
    for (int j = 0; j < M; ++j) r += wt.cand[j] > ki;
    if (r < k) wt.list[r] = ki;
  }
  __syncwarp();
  if (lane == 0) wt.n_list = M < k ? M : k;
  __syncwarp();
}

template <typename T>
__global__ void __launch_bounds__(kThreads, 2) topk_kernel(const Args a) {
  namespace cg = cooperative_groups;
  constexpr int n = Elem<T>::kPerVec;
  constexpr int eb = Elem<T>::kBytes;
  constexpr int kRoom = static_cast<int>(sizeof(TopkSmem::cand) / 8) - kMaxK;
  extern __shared__ __align__(1024) uint8_t stage_mem[];  // [warp][slot][kChunkBytes]
  __shared__ uint64_t full[kWarps][kWarpSlots];
  __shared__ TopkSmem sh;

  const int row = blockIdx.x / a.parts;
  const int part = blockIdx.x % a.parts;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int k = a.k;
  const T* rowp = static_cast<const T*>(a.logits) + static_cast<long long>(row) * a.row_stride;
  WarpTopk& wt = sh.w[warp];
  if (lane == 0) {
    wt.n_list = 0;
    wt.n_cand = 0;
  }
  __syncwarp();
  LaneSum ls;

  const long long b0 = static_cast<long long>(part) * a.stages_per_part * kStageBytes;
  long long b1 = b0 + static_cast<long long>(a.stages_per_part) * kStageBytes;
  if (b1 > a.aligned_bytes) b1 = a.aligned_bytes;
  const int nchunks = b1 > b0 ? static_cast<int>((b1 - b0 + kChunkBytes - 1) / kChunkBytes) : 0;
  const int my_n = nchunks > warp ? (nchunks - warp + kWarps - 1) / kWarps : 0;  // chunks warp + 8i

  auto generic = [&](long long e0, int count) {  // plain loads from global memory
    warp_chunk<T>(wt, e0, count, k, lane, ls, [&](float (&v)[n], int off, int nv) {
#pragma unroll
      for (int e = 0; e < n; ++e) v[e] = e < nv ? Elem<T>::load(rowp + e0 + off + e) : -INFINITY;
    });
  };
  bool timed_out = false;
  if (a.use_bulk) {
    if (tid == 0) {
      for (int w = 0; w < kWarps; ++w)
        for (int sl = 0; sl < kWarpSlots; ++sl) mbar_init(&full[w][sl], 1);
      fence_barrier_init();
    }
    __syncthreads();
    uint8_t* wbuf = stage_mem + warp * kWarpSlots * kChunkBytes;
    auto issue = [&](int i) {  // lane 0: chunk i of this warp into slot i % kWarpSlots
      const long long off = b0 + static_cast<long long>(warp + kWarps * i) * kChunkBytes;
      const uint32_t bytes = static_cast<uint32_t>(llmin(kChunkBytes, b1 - off));
      const int slot = i % kWarpSlots;
      mbar_arrive_expect_tx(&full[warp][slot], bytes);
      bulk_g2s(wbuf + slot * kChunkBytes, reinterpret_cast<const uint8_t*>(rowp) + off, bytes,
               &full[warp][slot]);
    };
    if (lane == 0)
      for (int i = 0; i < my_n && i < kWarpSlots; ++i) issue(i);
    for (int i = 0; i < my_n; ++i) {
      const int slot = i % kWarpSlots;
      const bool ok = mbar_wait(&full[warp][slot], (i / kWarpSlots) & 1);
      if (__any_sync(kFull, !ok)) {  // warp-uniform decision
        timed_out = true;
        if (lane == 0)  // drain the copies still in flight, again bounded
          for (int i2 = i + 1; i2 < my_n && i2 < i + kWarpSlots; ++i2)
            mbar_wait(&full[warp][i2 % kWarpSlots], (i2 / kWarpSlots) & 1);
        break;
      }
      const long long off = b0 + static_cast<long long>(warp + kWarps * i) * kChunkBytes;
      const int count = static_cast<int>(llmin(kChunkBytes, b1 - off)) / eb;
      const uint8_t* sp = wbuf + slot * kChunkBytes;
      warp_chunk<T>(wt, off / eb, count, k, lane, ls, [&](float (&v)[n], int eoff, int nv) {
        (void)nv;  // bulk chunks hold whole 16-byte vectors
        Elem<T>::unpack(*reinterpret_cast<const uint4*>(sp + static_cast<size_t>(eoff) * eb), v);
      });
      __syncwarp();  // every lane is done with this slot before it is refilled
      if (lane == 0 && i + kWarpSlots < my_n) issue(i + kWarpSlots);
    }
  } else {
    for (int i = 0; i < my_n; ++i) {
      const long long off = b0 + static_cast<long long>(warp + kWarps * i) * kChunkBytes;
      generic(off / eb, static_cast<int>(llmin(kChunkBytes, b1 - off) / eb));
    }
  }
  // row tail not covered by 16-byte units: warp 0 of the last part reads it directly
  if (part == a.parts - 1 && warp == 0) {
    const long long t0 = a.aligned_bytes / eb;
    if (t0 < a.V) generic(t0, static_cast<int>(a.V - t0));
  }
  if (timed_out && lane == 0) report(a.dev_status, PRESTO_DEV_TIMEOUT);

  // ---- the CTA: (max, sum exp) in the log2 domain, and the top-k of its warps
  float m = ls.m2, s = ls.s;
  warp_merge_ms(m, s);
  if (lane == 0) sh.warp_ms[warp] = make_float2(m, s);
  if (lane < k) sh.cand[warp * k + lane] = lane < wt.n_list ? wt.list[lane] : 0ull;
  __syncthreads();
  if (warp == 0) {
    m = lane < kWarps ? sh.warp_ms[lane].x : -INFINITY;
    s = lane < kWarps ? sh.warp_ms[lane].y : 0.f;
    warp_merge_ms(m, s);
  }
  const int got = rank_select(sh.cand, kWarps * k, k, sh.list, &sh.count, tid);

  // ---- combine the spans of the row
  if (a.mode == kCluster) {
    cg::cluster_group cluster = cg::this_cluster();
    TopkSmem* leader = cluster.map_shared_rank(&sh, 0);
    if (tid < k) leader->part[part][tid] = tid < got ? sh.list[tid] : 0ull;
    if (tid == 0) leader->part_ms[part] = make_float2(m, s);
    cluster.sync();
    if (part != 0) return;
    m = -INFINITY;
    s = 0.f;
    if (warp == 0) {
      if (lane < a.parts) {
        m = sh.part_ms[lane].x;
        s = sh.part_ms[lane].y;
      }
      warp_merge_ms(m, s);
    }
    for (int i = tid; i < a.parts * k; i += kThreads) sh.cand[i] = sh.part[i / k][i % k];
    __syncthreads();
    rank_select(sh.cand, a.parts * k, k, sh.list, &sh.count, tid);
  } else if (a.mode == kGlobal) {
    const size_t slot = static_cast<size_t>(row) * a.parts + part;
    if (tid < k) a.ws.keys[slot * k + tid] = tid < got ? sh.list[tid] : 0ull;
    if (tid == 0) a.ws.ms[slot] = make_float2(m, s);
    __threadfence();
    __syncthreads();
    if (tid == 0) sh.last = atomicAdd(&a.ws.ticket[row], 1u) == static_cast<unsigned>(a.parts - 1);
    __syncthreads();
    if (!sh.last) return;
    __threadfence();
    const size_t base = static_cast<size_t>(row) * a.parts * k;
    const int M = a.parts * k;
    m = -INFINITY;
    s = 0.f;
    if (warp == 0) {
      for (int p2 = lane; p2 < a.parts; p2 += 32) {
        const float2 ms = __ldcg(a.ws.ms + static_cast<size_t>(row) * a.parts + p2);
        merge_ms(m, s, ms.x, ms.y);
      }
      warp_merge_ms(m, s);
    }
    int nl = 0;  // merge the spans' lists in groups that fit the buffer
    for (int g = 0; g < M; g += kRoom) {
      const int cnt = min(kRoom, M - g);
      for (int i = tid; i < cnt; i += kThreads) sh.cand[i] = __ldcg(a.ws.keys + base + g + i);
      if (tid < nl) sh.cand[cnt + tid] = sh.list[tid];
      __syncthreads();
      nl = rank_select(sh.cand, cnt + nl, k, sh.list, &sh.count, tid);
    }
  }
  // ---- write the row (warp 0 holds the row's (max, sum exp))
  if (warp == 0) {
    // natural-log normaliser: lse = (m2 + log2 s) * ln 2; log q = (x - max) - ln s
    const float mx = m * (1.f / kLog2e);
    const float logs = logf(s);
    if (lane == 0 && !(mx > -INFINITY && mx < INFINITY)) report(a.dev_status, PRESTO_DEV_NONFINITE);
    if (lane < k) {
      const unsigned long long key = sh.list[lane];
      a.topk_ids[static_cast<size_t>(row) * k + lane] = key_id(key);
      a.topk_logq[static_cast<size_t>(row) * k + lane] = (key_value(key) - mx) - logs;
    }
    if (lane == 0 && a.lse) a.lse[row] = mx + logs;
  }
}

}  // namespace
}  // namespace presto

using namespace presto;

extern "C" size_t presto_topk_workspace(int B, int L, int V, int k) {
  if (B < 1 || L < 1 || V < 1 || k < 1 || k > kMaxK) return 0;
  size_t w = 0;
  for (int eb : {2, 4}) {  // the larger of the two element types' needs
    const size_t x = workspace_layout(make_plan(B, L, V, eb), k, nullptr, nullptr);
    w = x > w ? x : w;
  }
  return w;
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
  if (p.mode == kGlobal) {
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
  a.mode = p.mode;
  a.aligned_bytes = p.aligned_bytes;
  a.use_bulk = (reinterpret_cast<uintptr_t>(logits) % 16 == 0) && ((row_stride * eb) % 16 == 0);
  a.topk_ids = topk_ids;
  a.topk_logq = topk_logq;
  a.lse = lse;
  a.ws = w;
  a.dev_status = dev_status;
  static bool attr_set = [] {
    cudaFuncSetAttribute(topk_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         kWarps * kWarpSlots * kChunkBytes);
    cudaFuncSetAttribute(topk_kernel<__nv_bfloat16>,
                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                         kWarps * kWarpSlots * kChunkBytes);
    return true;
  }();
  (void)attr_set;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(static_cast<unsigned>(p.rows) * p.parts);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = a.use_bulk ? static_cast<size_t>(kWarps) * kWarpSlots * kChunkBytes : 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = p.mode == kCluster ? p.parts : 1;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e = dtype == PRESTO_F32 ? cudaLaunchKernelEx(&cfg, topk_kernel<float>, a)
                                      : cudaLaunchKernelEx(&cfg, topk_kernel<__nv_bfloat16>, a);
  if (e != cudaSuccess) return PRESTO_ERR_CUDA;
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
