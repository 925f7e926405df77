// presto_topk: single-pass log-softmax + top-k over the drafter's per-position
// logits (§2.3 marginals q_d, §4.3 top-k candidate extraction).
//
// Design (HBM-bound; roofline = B*L*V*elem bytes read once):
//   * A row is split into `parts` spans (<= 8), one CTA of 512 threads each; the
//     spans of a row form a thread-block cluster and merge through distributed
//     shared memory, so no workspace is needed.
//   * Every thread loads its whole share of the span (up to kMaxVpt 16-byte vectors)
//     into registers with one burst of non-caching vector loads, then:
//       - its maximum (packed bf16x2 max for bf16) and Σ exp(x - max) (one exp2 per
//         element, four independent accumulators fed by packed float32x2 FMA/add);
//       - the CTA's threshold tau = the k-th largest of the 16 warp maxima: at least
//         k elements of the span are >= tau, so the span's top-k are among them;
//       - the elements >= tau (vectors whose maximum is below tau are skipped) become
//         64-bit keys (value as an ordered integer, then the complement of the id,
//         so "larger value, then lower id" is integer order) in a candidate buffer,
//         ranked by counting.  A span has few of them, so only the threads holding
//         one work: one shared atomic each reserves their slots.  If the buffer
//         overflows (massive ties), an exact fallback raises a key threshold over
//         the register-resident data until the survivors fit.
//   * The leader CTA of the cluster merges the spans' (max, Σexp) pairs (warp 0) and
//     ranks their top-k lists (the other warps, at the same time), and writes the row.
//   * With ENT the same pass also yields the row's entropy (App. F): next to
//     s = Σ 2^u, u = x log2e - max2, each thread sums t = Σ 2^u u, and the merges
//     carry t along (when the reference maximum drops by δ, t -> 2^δ (t + δ s)).
//     Then H = ln s - ln2 t / s, and lambda_d = beta H / (H + C).
//   * Problems of more rows than one wave of this kernel holds go to the streaming
//     kernel further down (per-warp bulk-copy rings over longer spans).
//   * With slot rows (self-speculative rounds, App. C (II)) row j of sequence b is
//     read in place from slot slot_off + j of the deepest accepted node a*_b =
//     accept_path[b][accept_len[b]], looked up on the device after the accept
//     kernel that precedes it on the stream: no gather copy, no host round trip.
#include <cuda_bf16.h>

#include <cooperative_groups.h>

#include <algorithm>
#include <cmath>
#include <mutex>

#include "common.cuh"

namespace presto {
namespace {

constexpr int kThreads = 512;
constexpr int kWarps = kThreads / 32;
constexpr int kMaxParts = 8;     // spans of a row = CTAs of its (portable) cluster
constexpr int kCandCap = 1024;   // candidate keys per CTA and round
constexpr size_t kPrefetchCap = 48ull << 20;  // bytes a streaming launch asks L2 to prefetch
constexpr float kLog2e = 1.4426950408889634f;
constexpr unsigned kFull = 0xffffffffu;
static_assert(kWarps >= kMaxK, "tau needs at least k warp maxima");
static_assert(kWarps <= 32 && (kWarps & (kWarps - 1)) == 0, "the warp merge is a butterfly over kWarps lanes");
static_assert(kMaxParts <= 32 && (kMaxParts & (kMaxParts - 1)) == 0, "the span merge is a butterfly over kMaxParts lanes");

template <typename T>
struct Elem;
template <>
struct Elem<float> {
  static constexpr int kPerVec = 4;
  static constexpr int kBytes = 4;
  static constexpr int kPairs = 2;
  static constexpr uint32_t kNegInfWord = 0xff800000u;
  __device__ static float load(const float* p) { return *p; }
  // elements 2q and 2q + 1 of a vector
  __device__ static float2 pair(const uint4& u, int q) {
    return q == 0 ? make_float2(__uint_as_float(u.x), __uint_as_float(u.y))
                  : make_float2(__uint_as_float(u.z), __uint_as_float(u.w));
  }
  __device__ static float value(const uint4& u, int e) {
    return __uint_as_float(e == 0 ? u.x : e == 1 ? u.y : e == 2 ? u.z : u.w);
  }
  __device__ static float vmax(const uint4& u) {
    float m;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(m) : "f"(__uint_as_float(u.x)), "f"(__uint_as_float(u.y)),
        "f"(__uint_as_float(u.z)));
    return fmaxf(m, __uint_as_float(u.w));
  }
  // maximum of N vectors (two independent three-input chains)
  template <int N>
  __device__ static float max_of(const uint4 (&d)[N]) {
    float a = fmaxf(__uint_as_float(d[0].x), __uint_as_float(d[0].y));
    float b = fmaxf(__uint_as_float(d[0].z), __uint_as_float(d[0].w));
#pragma unroll
    for (int i = 1; i < N; ++i) {
      asm("max.f32 %0, %0, %1, %2;" : "+f"(a) : "f"(__uint_as_float(d[i].x)), "f"(__uint_as_float(d[i].y)));
      asm("max.f32 %0, %0, %1, %2;" : "+f"(b) : "f"(__uint_as_float(d[i].z)), "f"(__uint_as_float(d[i].w)));
    }
    return fmaxf(a, b);
  }
};
template <>
struct Elem<__nv_bfloat16> {
  static constexpr int kPerVec = 8;
  static constexpr int kBytes = 2;
  static constexpr int kPairs = 4;
  static constexpr uint32_t kNegInfWord = 0xff80ff80u;
  __device__ static float load(const __nv_bfloat16* p) { return __bfloat162float(*p); }
  // elements 2q and 2q + 1 of a vector (the two halves of word q)
  __device__ static float2 pair(const uint4& u, int q) {
    const uint32_t w = q == 0 ? u.x : q == 1 ? u.y : q == 2 ? u.z : u.w;
    return make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xffff0000u));
  }
  __device__ static float value(const uint4& u, int e) {
    const uint32_t w = (e >> 1) == 0 ? u.x : (e >> 1) == 1 ? u.y : (e >> 1) == 2 ? u.z : u.w;
    return __uint_as_float((e & 1) ? (w & 0xffff0000u) : (w << 16));
  }
  __device__ static float vmax(const uint4& u) {
    uint32_t a, b;
    asm("max.bf16x2 %0, %1, %2;" : "=r"(a) : "r"(u.x), "r"(u.y));
    asm("max.bf16x2 %0, %1, %2;" : "=r"(b) : "r"(u.z), "r"(u.w));
    asm("max.bf16x2 %0, %0, %1;" : "+r"(a) : "r"(b));
    return fmaxf(__uint_as_float(a << 16), __uint_as_float(a & 0xffff0000u));
  }
  // maximum of N vectors: packed maxima along four independent word chains
  template <int N>
  __device__ static float max_of(const uint4 (&d)[N]) {
    uint32_t m0 = d[0].x, m1 = d[0].y, m2 = d[0].z, m3 = d[0].w;
#pragma unroll
    for (int i = 1; i < N; ++i) {
      asm("max.bf16x2 %0, %0, %1;" : "+r"(m0) : "r"(d[i].x));
      asm("max.bf16x2 %0, %0, %1;" : "+r"(m1) : "r"(d[i].y));
      asm("max.bf16x2 %0, %0, %1;" : "+r"(m2) : "r"(d[i].z));
      asm("max.bf16x2 %0, %0, %1;" : "+r"(m3) : "r"(d[i].w));
    }
    asm("max.bf16x2 %0, %0, %1;" : "+r"(m0) : "r"(m1));
    asm("max.bf16x2 %0, %0, %1;" : "+r"(m2) : "r"(m3));
    asm("max.bf16x2 %0, %0, %1;" : "+r"(m0) : "r"(m2));
    return fmaxf(__uint_as_float(m0 << 16), __uint_as_float(m0 & 0xffff0000u));
  }
};

// 16 bytes at a shared-memory address (an explicit shared load: a pointer computed
// through integer arithmetic would otherwise be read with a generic one).
__device__ __forceinline__ uint4 lds128(uint32_t saddr) {
  uint4 r;
  asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "r"(saddr)
               : "memory");
  return r;
}

__device__ __forceinline__ uint4 ldg_stream(const uint4* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

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

// Merge two (max, sum) pairs of the log2 domain: sum = Σ 2^(x log2e - max).
__device__ __forceinline__ void merge_ms(float& m2, float& s, float n2, float t) {
  const float M = fmaxf(m2, n2);
  if (M == -INFINITY) return;
  s = s * ex2(m2 - M) + t * ex2(n2 - M);
  m2 = M;
}
// The same with the entropy sums t = Σ 2^u u, u = x log2e - max: moving a pair's
// reference maximum from m to M scales s by 2^(m-M) and t to 2^(m-M) (t + (m-M) s).
// A pair with maximum -inf holds nothing (s = t = 0) and is skipped.
__device__ __forceinline__ void merge_mst(float& m2, float& s, float& t, float n2, float s2,
                                          float t2) {
  const float M = fmaxf(m2, n2);
  if (M == -INFINITY) return;
  float so = 0.f, to = 0.f;
  if (m2 != -INFINITY) {
    const float f = ex2(m2 - M);
    so = s * f;
    to = f * fmaf(m2 - M, s, t);
  }
  if (n2 != -INFINITY) {
    const float f = ex2(n2 - M);
    so = fmaf(s2, f, so);
    to = fmaf(f, fmaf(n2 - M, s2, t2), to);
  }
  s = so;
  t = to;
  m2 = M;
}

struct Plan {
  int rows, parts, vpt, vmax;  // vpt: vectors per thread; vmax: the kernel's register bound
  int epv;                     // elements per 16-byte vector
  bool stream;                 // streaming kernel (then vpt = vectors per span)
};

struct Args {
  const void* logits;
  long long row_stride;  // elements
  int V, k, parts, vpt;
  uint32_t pf_bytes;  // streaming kernel: L2 prefetch budget of each warp (bytes)
  int32_t* topk_ids;
  float* topk_logq;
  float* lse;
  float* entropy;   // ENT: [rows] H in nats, nullable
  float* lambda_d;  // ENT: [rows] beta H / (H + C), nullable
  float beta, C;
  // slot rows (acc_len non-null): logits = [B][n_prev][n_slots][row_stride]
  const int32_t* acc_len;    // [B]
  const int32_t* acc_path;   // [B][path_len]
  int path_len, n_prev, n_slots, slot_off, Lrows;
  const int32_t* node_token;  // [B][n_prev], nullable (with bonus, ctx2_next)
  const int32_t* bonus;       // [B]
  int32_t* ctx2_next;         // [B][2]
  int32_t* dev_status;
};

// Row `row` of the launch: a plain row of the logits, or (slot rows) slot
// slot_off + j of the accepted node of sequence b, row = b * Lrows + j.  Slot rows
// read the accept results, so the caller has passed the grid dependency wait.  A
// path entry out of range is reported and reads the root's slots instead.
template <typename T>
__device__ __forceinline__ const T* row_base(const Args& a, int row, bool first) {
  const T* base = static_cast<const T*>(a.logits);
  if (!a.acc_len) return base + static_cast<long long>(row) * a.row_stride;
  const int b = row / a.Lrows, j = row - b * a.Lrows;
  const int len = ld_chain(a.acc_len + b);
  int node = -1;
  if (len >= 0 && len < a.path_len) node = ld_chain(a.acc_path + static_cast<long long>(b) * a.path_len + len);
  if (node < 0 || node >= a.n_prev) {
    if (first) report(a.dev_status, PRESTO_DEV_BAD_PATH);
    node = 0;
  }
  if (first && j == 0 && a.ctx2_next) {
    a.ctx2_next[2 * b] = a.node_token[static_cast<long long>(b) * a.n_prev + node];
    a.ctx2_next[2 * b + 1] = a.bonus[b];
  }
  const long long slot = (static_cast<long long>(b) * a.n_prev + node) * a.n_slots + a.slot_off + j;
  return base + slot * a.row_stride;
}

struct Smem {
  unsigned long long cand[kCandCap];
  unsigned long long list[kMaxK];               // the CTA's top-k, descending
  unsigned long long part[kMaxParts * kMaxK];   // leader: the cluster's lists, span p at p * k
  float2 part_ms[kMaxParts];                    // leader: the cluster's (max, sum)
  float2 warp_ms[kWarps];                       // (max log2, sum) per warp
  float warp_t[kWarps];                         // ENT: entropy sum per warp
  float part_t[kMaxParts];                      // ENT leader: the cluster's entropy sums
  float warp_max[kWarps];                       // plain maxima, for tau
  unsigned long long thr;                       // key threshold of the current round
  int count;
  float tau;
};

// Keys e[0..M) (unique, nonzero) -> their descending top-k in out[0..min(M, k)).
// NT threads: every thread takes keys tid, tid + NT, ...; no barrier inside.
template <int NT = kThreads>
__device__ __forceinline__ void rank_keys(const unsigned long long* e, int M, int k,
                                          unsigned long long* out, int tid) {
  for (int i = tid; i < M; i += NT) {
    const unsigned long long ki = e[i];
    int r = 0;
    int j = 0;
    for (; j + 8 <= M; j += 8) {
#pragma unroll
      for (int u = 0; u < 8; ++u) r += e[j + u] > ki;
    }
    for (; j < M; ++j) r += e[j] > ki;
    if (r < k) out[r] = ki;
  }
}

// Warp 0 writes a row: its top-k ids and log q from the k keys in `list`, lse and
// (ENT) the entropy and lambda_d, from the row's (max log2, Σ 2^u[, Σ 2^u u]).
template <bool ENT>
__device__ __forceinline__ void write_row(const Args& a, const unsigned long long* list, int row,
                                          float m_row, float s_row, float t_row) {
  const int lane = threadIdx.x & 31;
  const int k = a.k;
  // natural-log normaliser: lse = (m2 + log2 s) ln 2 = max + ln s; log q = (x - max) - ln s
  const float mx = m_row * (1.f / kLog2e);
  const float logs = logf(s_row);
  if (lane == 0 && !(mx > -INFINITY && mx < INFINITY)) report(a.dev_status, PRESTO_DEV_NONFINITE);
  if (lane < k) {
    const unsigned long long key = list[lane];
    a.topk_ids[static_cast<size_t>(row) * k + lane] = key_id(key);
    a.topk_logq[static_cast<size_t>(row) * k + lane] = (key_value(key) - mx) - logs;
  }
  if (lane == 0 && a.lse) a.lse[row] = mx + logs;
  if constexpr (ENT) {
    if (lane == 0) {
      // H = -Σ q ln q = ln s - ln2 (t / s); q ln q -> 0 where q underflows.  H >= 0
      // exactly; rounding can take a near-one-hot row a hair below, so clamp (this
      // also keeps lambda_d >= 0, as the tree build requires)
      const float H = fmaxf(logs - 0.6931471805599453f * __fdiv_rn(t_row, s_row), 0.f);
      if (a.entropy) a.entropy[row] = H;
      if (a.lambda_d) a.lambda_d[row] = __fdiv_rn(__fmul_rn(a.beta, H), __fadd_rn(H, a.C));
    }
  }
}

// Combine the spans of a row in the leader CTA of its cluster (keys, (max, sum) and
// the entropy sums), then write the row.  Every thread of the CTA calls this; the
// first NT take part in ranking; warp 0 holds the CTA's (m, s, t) on entry.
template <bool ENT, int NT, typename SM>
__device__ __forceinline__ void finish_row(const Args& a, SM& sh, int row, int part, float m_cta,
                                           float s_cta, float t_cta, int got) {
  namespace cg = cooperative_groups;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int k = a.k;
  // ---- combine the spans of the row in the leader CTA
  float m_row = m_cta, s_row = s_cta, t_row = t_cta;
  if (a.parts > 1) {
    cg::cluster_group cluster = cg::this_cluster();
    SM* leader = cluster.map_shared_rank(&sh, 0);
    if (tid < k) leader->part[part * k + tid] = tid < got ? sh.list[tid] : 0ull;
    if (tid == 0) {
      leader->part_ms[part] = make_float2(m_cta, s_cta);
      if constexpr (ENT) leader->part_t[part] = t_cta;
    }
    cluster.sync();
    if (part != 0) return;
    // the leader: warps 1.. rank the spans' keys (zeros pad a span with fewer than k
    // and rank below every real key), beside warp 0's merge of the spans' (max, sum)
    const int P = a.parts * k;
    if (warp != 0) {
      rank_keys<NT - 32>(sh.part, P, k, sh.list, tid - 32);
    } else {
      // lanes >= parts hold nothing: the butterfly stays within kMaxParts lanes
      float mw = lane < a.parts ? sh.part_ms[lane].x : -INFINITY;
      float sw = lane < a.parts ? sh.part_ms[lane].y : 0.f;
      float tw = 0.f;
      if constexpr (ENT) tw = lane < a.parts ? sh.part_t[lane] : 0.f;
#pragma unroll
      for (int off = kMaxParts / 2; off > 0; off >>= 1) {
        const float m_o = __shfl_xor_sync(kFull, mw, off);
        const float s_o = __shfl_xor_sync(kFull, sw, off);
        if constexpr (ENT) {
          const float t_o = __shfl_xor_sync(kFull, tw, off);
          merge_mst(mw, sw, tw, m_o, s_o, t_o);
        } else {
          merge_ms(mw, sw, m_o, s_o);
        }
      }
      // write_row reads the pair in lanes 0..k-1
      m_row = __shfl_sync(kFull, mw, 0);
      s_row = __shfl_sync(kFull, sw, 0);
      if constexpr (ENT) t_row = __shfl_sync(kFull, tw, 0);
    }
    __syncthreads();
  }
  // ---- write the row (warp 0 holds the row's (max, sum))
  if (warp == 0) write_row<ENT>(a, sh.list, row, m_row, s_row, t_row);
}

template <typename T, int VMAX, bool ENT>
__global__ void __launch_bounds__(kThreads, VMAX <= 4 ? 2 : 1) topk_kernel(const Args a) {
  namespace cg = cooperative_groups;
  using E = Elem<T>;
  static_assert(VMAX <= 31, "vector hit bits and the scalar hit bit share one word");
  constexpr int n = E::kPerVec;
  constexpr int eb = E::kBytes;
  __shared__ Smem sh;
  pdl_launch_dependents();
  const int row = blockIdx.x / a.parts;
  const int part = blockIdx.x % a.parts;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int k = a.k, V = a.V;
  if (a.acc_len) pdl_wait();  // slot rows: the accept results come from the previous kernel
  const T* rowp = row_base<T>(a, row, part == 0 && tid == 0);
  // the row's 16-byte-aligned vectors [head, head + nvec * n); the few elements
  // before and after are read one by one
  const int mis = static_cast<int>(reinterpret_cast<uintptr_t>(rowp) & 15);
  const int head = min(V, mis == 0 ? 0 : (16 - mis) / eb);
  const int nvec = (V - head) / n;
  const int tail0 = head + nvec * n;
  const uint4* vecp = reinterpret_cast<const uint4*>(rowp + head);
  const int per_part = a.vpt * kThreads;
  const int v0 = part * per_part;
  const int v1 = min(nvec, v0 + per_part);
  // extra scalar element of this thread: threads 0-6 of part 0 take the head (< 8
  // elements), threads 8-14 of the last part the tail (< 8 elements)
  int xid = -1;
  if (part == 0 && tid < head) xid = tid;
  if (part == a.parts - 1 && tid >= 8 && tid - 8 < V - tail0) xid = tail0 + (tid - 8);
  // before the dependency wait, ask L2 for the span (slot rows are only known after
  // it): a hint that reads nothing into the SM, so it cannot return data older than
  // the loads below, and its DRAM latency overlaps the previous kernel
  if (!a.acc_len && tid < kWarps && v1 > v0) {
    const int per = (v1 - v0 + kWarps - 1) / kWarps;
    const int b = v0 + tid * per, e = min(v1, b + per);
    if (e > b) prefetch_l2_bulk(vecp + b, static_cast<uint32_t>(e - b) * 16u);
  }

  pdl_wait();  // the logits may come from the previous kernel on the stream
  uint4 d[VMAX];
#pragma unroll
  for (int i = 0; i < VMAX; ++i) {
    const int vi = v0 + i * kThreads + tid;
    const uint32_t ni = E::kNegInfWord;
    d[i] = (i < a.vpt && vi < v1) ? ldg_stream(vecp + vi) : make_uint4(ni, ni, ni, ni);
  }
  const float xval = xid >= 0 ? E::load(rowp + xid) : -INFINITY;

  // ---- the thread's maximum and Σ 2^(x log2e - m2)
  float mt = xval;
#pragma unroll
  for (int i = 0; i < VMAX; ++i) mt = fmaxf(mt, E::vmax(d[i]));
  const float m2 = mt * kLog2e;
  float st = 0.f, tt = 0.f;  // tt (ENT): Σ 2^u u
  if (mt != -INFINITY) {
    // element e of a vector goes to accumulator e & 3, as pairs: packed float32x2
    // FMA and add (each half rounds exactly as the scalar instruction)
    const float2 l2 = make_float2(kLog2e, kLog2e), nm = make_float2(-m2, -m2);
    float2 acc[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
    if constexpr (!ENT) {
#pragma unroll
      for (int i = 0; i < VMAX; ++i) {
#pragma unroll
        for (int q = 0; q < E::kPairs; ++q) {
          const float2 u = __ffma2_rn(E::pair(d[i], q), l2, nm);
          acc[q & 1] = __fadd2_rn(acc[q & 1], make_float2(ex2(u.x), ex2(u.y)));
        }
      }
      st = (acc[0].x + acc[0].y) + (acc[1].x + acc[1].y);
      if (xid >= 0) st += ex2(fmaf(xval, kLog2e, -m2));
    } else {
      // u is clamped at -256: 2^u flushes to 0 there, so -inf entries add 0 to both
      float2 tac[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
      for (int i = 0; i < VMAX; ++i) {
#pragma unroll
        for (int q = 0; q < E::kPairs; ++q) {
          float2 u = __ffma2_rn(E::pair(d[i], q), l2, nm);
          u.x = fmaxf(u.x, -256.f);
          u.y = fmaxf(u.y, -256.f);
          const float2 p = make_float2(ex2(u.x), ex2(u.y));
          acc[q & 1] = __fadd2_rn(acc[q & 1], p);
          tac[q & 1] = __ffma2_rn(p, u, tac[q & 1]);
        }
      }
      st = (acc[0].x + acc[0].y) + (acc[1].x + acc[1].y);
      tt = (tac[0].x + tac[0].y) + (tac[1].x + tac[1].y);
      if (xid >= 0) {
        const float u = fmaxf(fmaf(xval, kLog2e, -m2), -256.f);
        const float p = ex2(u);
        st += p;
        tt = fmaf(p, u, tt);
      }
    }
  }
  // ---- warp: (max, sum) and the plain maximum
  const uint32_t wm_o = __reduce_max_sync(kFull, ordered(mt));
  const float wm = unordered(wm_o);
  const float wm2 = wm * kLog2e;
  const float fw = (mt == -INFINITY) ? 0.f : ex2(m2 - wm2);
  float ws = st * fw;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) ws += __shfl_xor_sync(kFull, ws, off);
  float wt = 0.f;
  if constexpr (ENT) {
    wt = (mt == -INFINITY) ? 0.f : fw * fmaf(m2 - wm2, st, tt);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) wt += __shfl_xor_sync(kFull, wt, off);
  }
  if (lane == 0) {
    sh.warp_ms[warp] = make_float2(wm == -INFINITY ? -INFINITY : wm2, ws);
    sh.warp_max[warp] = wm;
    if constexpr (ENT) sh.warp_t[warp] = wt;
  }
  if (tid == 0) sh.count = 0;
  __syncthreads();
  // ---- tau: the k-th largest warp maximum (ties by warp index)
  if (tid < kWarps) {
    const float x = sh.warp_max[tid];
    int r = 0;
#pragma unroll
    for (int u = 0; u < kWarps; ++u) {
      const float y = sh.warp_max[u];
      r += y > x || (y == x && u < tid);
    }
    if (r == k - 1) sh.tau = x;
  }
  __syncthreads();
  const float tau = sh.tau;
  // ---- candidates: the elements >= tau (then, on overflow, keys >= thr)
  // vectors holding a value >= tau, as a bit mask (no branches); most warps have none
  uint32_t hits = 0u;
#pragma unroll
  for (int i = 0; i < VMAX; ++i) {
    const int vi = v0 + i * kThreads + tid;  // the -inf padding of absent vectors is skipped
    hits |= (i < a.vpt && vi < v1 && E::vmax(d[i]) >= tau) ? (1u << i) : 0u;
  }
  const bool xhit = xid >= 0 && xval >= tau;
  // the elements of vector i that are >= tau, as a bit mask from independent compares
  auto ge_tau = [&](int i) {
    uint32_t em = 0u;
#pragma unroll
    for (int e = 0; e < n; ++e) em |= (E::value(d[i], e) >= tau) ? (1u << e) : 0u;
    return em;
  };
  // every element >= tau becomes a candidate key.  Only the threads holding one (a
  // few per span) do any work: each counts its elements, reserves their slots with
  // one shared atomic and writes their keys
  if (hits | static_cast<uint32_t>(xhit)) {
    int mine = xhit ? 1 : 0;
#pragma unroll
    for (int i = 0; i < VMAX; ++i)
      if ((hits >> i) & 1u) mine += __popc(ge_tau(i));
    int slot = atomicAdd(&sh.count, mine);
#pragma unroll
    for (int i = 0; i < VMAX; ++i) {
      if ((hits >> i) & 1u) {
        uint32_t em = ge_tau(i);
        const int id0 = head + (v0 + i * kThreads + tid) * n;
        while (em) {
          const int e = __ffs(em) - 1;
          em &= em - 1u;
          if (slot < kCandCap) sh.cand[slot] = elem_key(E::value(d[i], e), id0 + e);
          ++slot;
        }
      }
    }
    if (xhit && slot < kCandCap) sh.cand[slot] = elem_key(xval, xid);
  }
  __syncthreads();
  int M = sh.count;
  if (M > kCandCap) {
    // overflow (massive ties; uniform across the CTA): the k-th largest of the keys
    // collected is <= the span's k-th largest key, so the keys below it can go.  The
    // rounds below collect the keys >= a threshold thr and raise it the same way
    // until they fit; keys are unique, so it rises strictly and the rounds end
    const uint32_t warp_hits = __reduce_or_sync(kFull, hits | (xhit ? 0x80000000u : 0u));
    unsigned long long thr = 0ull;
    for (;;) {
      rank_keys(sh.cand, kCandCap, k, sh.list, tid);
      __syncthreads();
      if (tid == 0) {
        sh.thr = sh.list[k - 1];
        sh.count = 0;
      }
      __syncthreads();
      thr = sh.thr;
      // count this thread's keys >= thr, reserve their slots with one atomic per
      // warp, then write them; vectors are visited under warp-uniform votes
      auto visit = [&](auto&& emit) {
#pragma unroll
        for (int i = 0; i < VMAX; ++i) {
          if ((warp_hits >> i) & 1u) {  // warp-uniform
            uint32_t em = ((hits >> i) & 1u) ? ge_tau(i) : 0u;
            const int id0 = head + (v0 + i * kThreads + tid) * n;
            while (em) {
              const int e = __ffs(em) - 1;
              em &= em - 1u;
              const unsigned long long key = elem_key(E::value(d[i], e), id0 + e);
              emit(key >= thr, key);
            }
          }
        }
        if (warp_hits >> 31) {
          const unsigned long long key = elem_key(xval, xid);
          emit(xhit && key >= thr, key);
        }
      };
      int mine = 0;
      if (warp_hits) visit([&](bool take, unsigned long long) { mine += take; });
      int incl = mine;  // inclusive prefix over the warp
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const int y = __shfl_up_sync(kFull, incl, off);
        if (lane >= off) incl += y;
      }
      int base = 0;
      if (lane == 31 && incl > 0) base = atomicAdd(&sh.count, incl);
      base = __shfl_sync(kFull, base, 31) + incl - mine;
      if (warp_hits)
        visit([&](bool take, unsigned long long key) {
          if (take && base < kCandCap) sh.cand[base] = key;
          base += take;
        });
      __syncthreads();
      M = sh.count;
      if (M <= kCandCap) break;
    }
  }
  // ---- the span's top-k (warps 1..), beside warp 0's merge of the warps' (max, sum)
  if (warp != 0) rank_keys<kThreads - 32>(sh.cand, M, k, sh.list, tid - 32);
  float m_cta = -INFINITY, s_cta = 0.f, t_cta = 0.f;
  if (warp == 0) {
    float mw = lane < kWarps ? sh.warp_ms[lane].x : -INFINITY;
    float sw = lane < kWarps ? sh.warp_ms[lane].y : 0.f;
    float tw = 0.f;
    if constexpr (ENT) tw = lane < kWarps ? sh.warp_t[lane] : 0.f;
    // lanes >= kWarps hold nothing: merging them changes no bit, so the butterfly
    // stays within the first kWarps lanes
#pragma unroll
    for (int off = kWarps / 2; off > 0; off >>= 1) {
      const float m_o = __shfl_xor_sync(kFull, mw, off);
      const float s_o = __shfl_xor_sync(kFull, sw, off);
      if constexpr (ENT) {
        const float t_o = __shfl_xor_sync(kFull, tw, off);
        merge_mst(mw, sw, tw, m_o, s_o, t_o);
      } else {
        merge_ms(mw, sw, m_o, s_o);
      }
    }
    // lanes 0..kWarps-1 hold the span's pair (write_row reads it in lanes 0..k-1)
    m_cta = mw;
    s_cta = sw;
    t_cta = tw;
  }
  __syncthreads();
  const int got = M < k ? M : k;

  finish_row<ENT, kThreads>(a, sh, row, part, m_cta, s_cta, t_cta, got);
}

// ---------------------------------------------------------------------------
// Streaming variant, for problems of more than one wave of the kernel above (many
// rows).  The CTA's span is cut into one contiguous piece per warp, and each warp
// streams its piece in 4 KB chunks: its lane 0 keeps kWStages bulk copies in flight
// in a ring of the warp's own.  Every lane keeps an online (max, Σ 2^u) pair and
// every warp its own top-k, sorted across lanes 0..k-1.  A candidate must reach
// theta: first the k-th largest of all lanes' first-chunk maxima in the CTA (each a
// real element), then the largest k-th value any warp of the CTA has published (a
// warp's list holds k elements at or above its k-th value); nothing below theta is
// in the row's top-k.  A lane whose chunk maximum is below theta costs one compare;
// a candidate enters the warp's list by a warp-wide sorted insertion.  When its
// piece is done, every warp sends its (max, sum) pair and the keys of its list at or
// above theta straight to the leader CTA of the row's cluster, which merges them,
// in warp order, after one cluster barrier.
// ---------------------------------------------------------------------------
constexpr int kWThreads = 256;
constexpr int kWWarps = kWThreads / 32;
constexpr int kWVec = 8;                    // 16-byte vectors per lane and chunk
constexpr int kWChunkVec = 32 * kWVec;      // 256 vectors
constexpr int kWChunkBytes = kWChunkVec * 16;
constexpr int kWStages = 3;
constexpr size_t kWDynBytes = static_cast<size_t>(kWWarps) * kWStages * kWChunkBytes + 128;
constexpr int kWCtasPerSm = 2;  // ~106 KB of shared memory and <= 128 registers a thread
constexpr int kWSlots = kMaxParts * kWWarps;  // (part, warp) results gathered in the leader

struct WSmem {
  uint64_t full[kWWarps][kWStages];
  unsigned long long keys[kWSlots * kMaxK];  // leader: every warp's kept keys (0 = none)
  unsigned long long list[kMaxK];            // leader: the row's top-k, descending
  float2 ms[kWSlots];                        // leader: every warp's (max log2, Σ 2^u)
  float ts[kWSlots];                         // leader, ENT: every warp's Σ 2^u u
  uint32_t first[kWWarps * kMaxK];           // every warp's k largest first-chunk lane maxima
  float theta[kWWarps];                      // every warp's published k-th value
  float theta0;                              // the CTA's first threshold
  int abort;                                 // set by any warp whose bounded wait ran out
};

// Insert `key` (uniform across the warp, larger than the k-th key) into the warp's
// descending list lst (lane j < k holds the j-th key, 0 = none); returns the new
// k-th key.
__device__ __forceinline__ unsigned long long warp_insert(unsigned long long& lst,
                                                          unsigned long long key, int k,
                                                          int lane) {
  const int pos = __popc(__ballot_sync(kFull, lane < k && lst > key));
  const unsigned long long up = __shfl_up_sync(kFull, lst, 1);
  if (lane < k) lst = lane == pos ? key : (lane > pos ? up : lst);
  return __shfl_sync(kFull, lst, k - 1);
}

// A warp's top-k state: lane j < k holds the j-th key in lst (0 = none), thr is the
// k-th key (0 until k are held), theta the candidate threshold.
struct WarpTop {
  unsigned long long lst, thr;
  float theta;
};

// The candidates of one vector (bit e of m: element e reaches theta, id0 + e its id),
// one at a time through the warp's list; a raised theta is published to *pub_slot.
// Out of line: the chunk loop's rare path, kept out of its instruction stream.  All
// lanes of the warp call it.
template <typename E>
__device__ __noinline__ WarpTop drain_vector(WarpTop t, uint4 di, unsigned m, int id0, int k,
                                             volatile float* pub_slot) {
  const int lane = threadIdx.x & 31;
  for (unsigned w = __ballot_sync(kFull, m != 0u); w; w = __ballot_sync(kFull, m != 0u)) {
    const int src = __ffs(w) - 1;
    const int e = __ffs(m) - 1;
    const unsigned long long mine = m ? elem_key(E::value(di, e), id0 + e) : 0ull;
    const unsigned long long key = __shfl_sync(kFull, mine, src);
    if (lane == src) m &= m - 1u;
    if (key > t.thr) {
      t.thr = warp_insert(t.lst, key, k, lane);
      if (t.thr) {
        const float tv = key_value(t.thr);
        if (tv > t.theta) {
          t.theta = tv;
          if (lane == 0) *pub_slot = tv;
        }
      }
    }
  }
  return t;
}

// Move a lane's online (max, Σ 2^u[, Σ 2^u u]) pair to the maximum cm of new elements
// when that is larger (u = x log2e - max2).
template <bool ENT>
__device__ __forceinline__ void rescale_to(float& mt, float& st, float& tt, float cm) {
  if (cm > mt) {
    if (mt != -INFINITY) {
      const float dl = mt * kLog2e - cm * kLog2e;  // the old reference minus the new
      const float f = ex2(dl);
      if constexpr (ENT) tt = f * fmaf(dl, st, tt);
      st *= f;
    }
    mt = cm;
  }
}

// Merge pairs (m2_j, s_j[, t_j]) (log2-domain maxima, Σ 2^u, Σ 2^u u) held by the
// lanes of a warp into one, the same in every lane: the maximum by a reduction, then
// each pair moved to it and summed.  Pairs with m2 = -inf hold nothing.
template <bool ENT>
__device__ __forceinline__ void warp_merge_pairs(float& m2, float& s, float& t) {
  const float M = unordered(__reduce_max_sync(kFull, ordered(m2)));
  float so = 0.f, to = 0.f;
  if (m2 != -INFINITY) {
    const float f = ex2(m2 - M);
    so = s * f;
    if constexpr (ENT) to = f * fmaf(m2 - M, s, t);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    so += __shfl_xor_sync(kFull, so, off);
    if constexpr (ENT) to += __shfl_xor_sync(kFull, to, off);
  }
  m2 = M;
  s = so;
  t = to;
}

template <typename T, bool ENT>
__global__ void __launch_bounds__(kWThreads, 2) topk_stream_kernel(const Args a) {
  namespace cg = cooperative_groups;
  using E = Elem<T>;
  constexpr int n = E::kPerVec;
  constexpr int eb = E::kBytes;
  __shared__ WSmem sh;
  extern __shared__ unsigned char dyn_raw[];
  pdl_launch_dependents();
  const int row = blockIdx.x / a.parts;
  const int part = blockIdx.x % a.parts;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int k = a.k, V = a.V;
  unsigned char* const ring =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(dyn_raw) + 127) &
                                       ~static_cast<uintptr_t>(127)) +
      warp * kWStages * kWChunkBytes;
  const uint32_t ring_s = smem_u32(ring);  // read with shared-memory loads, not generic ones
  if (lane == 0) {
    for (int s = 0; s < kWStages; ++s) mbar_init(&sh.full[warp][s], 1);
    sh.theta[warp] = -INFINITY;
    fence_barrier_init();
  }
  if (tid == 0) sh.abort = 0;
  __syncthreads();
  // the warp's piece [wb, we) of the row's aligned vectors
  auto geometry = [&](const T* rp, int& head, int& tail0, const uint4*& vecp, int& wb, int& we) {
    const int mis = static_cast<int>(reinterpret_cast<uintptr_t>(rp) & 15);
    head = min(V, mis == 0 ? 0 : (16 - mis) / eb);
    const int nvec = (V - head) / n;
    tail0 = head + nvec * n;
    vecp = reinterpret_cast<const uint4*>(rp + head);
    const int v0 = min(nvec, part * a.vpt);  // vpt: vectors per span here
    const int v1 = min(nvec, v0 + a.vpt);
    const int per = (v1 - v0 + kWWarps - 1) / kWWarps;
    wb = min(v1, v0 + warp * per);
    we = min(v1, wb + per);
  };
  // before the dependency wait (plain rows only; slot rows are known after it), ask
  // L2 for the head of the warp's piece: a hint that reads nothing into the SM, so
  // it cannot return data older than the copies below
  if (!a.acc_len && lane == 0 && a.pf_bytes > 0) {
    int h0, t0, b0, e0;
    const uint4* vp;
    geometry(row_base<T>(a, row, false), h0, t0, vp, b0, e0);
    const uint32_t bytes = min(a.pf_bytes, static_cast<uint32_t>(max(0, e0 - b0)) * 16u);
    for (uint32_t o = 0; o < bytes; o += 65536u)
      prefetch_l2_bulk(reinterpret_cast<const char*>(vp + b0) + o, min(65536u, bytes - o));
  }
  pdl_wait();  // the logits (and slot rows' accept results) come from earlier kernels
  const T* rowp = row_base<T>(a, row, part == 0 && tid == 0);
  int head, tail0, wb, we;
  const uint4* vecp;
  geometry(rowp, head, tail0, vecp, wb, we);
  const int nch = (we - wb + kWChunkVec - 1) / kWChunkVec;  // chunks of the piece
  volatile int* abort = &sh.abort;
  volatile float* pub = sh.theta;

  auto issue = [&](int c) {  // lane 0: chunk c of the piece into ring slot c % kWStages
    const int st2 = c % kWStages;
    const int vb = wb + c * kWChunkVec;
    const uint32_t bytes = static_cast<uint32_t>(min(kWChunkVec, we - vb)) * 16u;
    mbar_arrive_expect_tx(&sh.full[warp][st2], bytes);
    bulk_g2s(ring + st2 * kWChunkBytes, vecp + vb, bytes, &sh.full[warp][st2]);
  };
  if (lane == 0)
    for (int c = 0; c < nch && c < kWStages; ++c) issue(c);

  float mt = -INFINITY, st = 0.f, tt = 0.f;  // the lane's running max (plain), Σ 2^u, Σ 2^u u
  float theta = -INFINITY;                   // candidates: value >= theta ...
  unsigned long long thr = 0ull;             // ... and key > thr, the warp's k-th key
  unsigned long long lst = 0ull;             // lane j < k: the warp's j-th key

  // one candidate of each lane (key 0: none) at a time through the warp's list
  auto drain = [&](unsigned& m, auto key_of) {
    for (unsigned w = __ballot_sync(kFull, m != 0u); w; w = __ballot_sync(kFull, m != 0u)) {
      const int src = __ffs(w) - 1;
      const unsigned long long mine = m ? key_of(__ffs(m) - 1) : 0ull;
      const unsigned long long key = __shfl_sync(kFull, mine, src);
      if (lane == src) m &= m - 1u;
      if (key > thr) {
        thr = warp_insert(lst, key, k, lane);
        if (thr) {
          const float tv = key_value(thr);
          if (tv > theta) {
            theta = tv;
            if (lane == 0) pub[warp] = tv;
          }
        }
      }
    }
  };
  // chunk c: wait for its copy, take it into registers and refill its slot with
  // chunk c + kWStages; false (for the whole warp) when the wait gave up
  auto take = [&](uint4 (&d)[kWVec], int c) -> bool {
    const int sg = c % kWStages;
    const bool ok = mbar_wait(&sh.full[warp][sg], (c / kWStages) & 1, abort);
    if (!__all_sync(kFull, ok)) {
      if (lane == 0) {
        *abort = 1;
        report(a.dev_status, PRESTO_DEV_TIMEOUT);
      }
      return false;
    }
    const int nv = min(kWChunkVec, we - (wb + c * kWChunkVec));
    const uint32_t ni = E::kNegInfWord;
#pragma unroll
    for (int i = 0; i < kWVec; ++i) {
      const int vi = i * 32 + lane;
      d[i] = vi < nv ? lds128(ring_s + sg * kWChunkBytes + vi * 16) : make_uint4(ni, ni, ni, ni);
    }
    __syncwarp();
    if (lane == 0 && c + kWStages < nch) {  // the slot is free again: refill it
      fence_proxy_async();
      issue(c + kWStages);
    }
    return true;
  };
  // the chunk's lane maximum (returned) and the lane's online (max, Σ 2^u) pair, log2
  // domain; eight independent accumulators
  auto reduce = [&](const uint4 (&d)[kWVec]) -> float {
    const float cm = E::template max_of<kWVec>(d);
    rescale_to<ENT>(mt, st, tt, cm);
    if (mt != -INFINITY) {
      const float m2 = mt * kLog2e;
      // element e of vector i goes to accumulator (i n + e) & 7, as pairs: packed
      // float32x2 FMA and add (each half rounds exactly as the scalar instruction)
      const float2 l2 = make_float2(kLog2e, kLog2e), nm = make_float2(-m2, -m2);
      float2 acc[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) acc[j] = make_float2(0.f, 0.f);
      if constexpr (!ENT) {
#pragma unroll
        for (int i = 0; i < kWVec; ++i)
#pragma unroll
          for (int q = 0; q < E::kPairs; ++q) {
            const int j = (i * n / 2 + q) & 3;
            const float2 u = __ffma2_rn(E::pair(d[i], q), l2, nm);
            acc[j] = __fadd2_rn(acc[j], make_float2(ex2(u.x), ex2(u.y)));
          }
      } else {
        // u clamped at -256: 2^u flushes to 0 there, so -inf adds 0 to both sums
        float2 tac[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) tac[j] = make_float2(0.f, 0.f);
#pragma unroll
        for (int i = 0; i < kWVec; ++i)
#pragma unroll
          for (int q = 0; q < E::kPairs; ++q) {
            const int j = (i * n / 2 + q) & 3;
            float2 u = __ffma2_rn(E::pair(d[i], q), l2, nm);
            u.x = fmaxf(u.x, -256.f);
            u.y = fmaxf(u.y, -256.f);
            const float2 p = make_float2(ex2(u.x), ex2(u.y));
            acc[j] = __fadd2_rn(acc[j], p);
            tac[j] = __ffma2_rn(p, u, tac[j]);
          }
        tt += ((tac[0].x + tac[0].y) + (tac[1].x + tac[1].y)) +
              ((tac[2].x + tac[2].y) + (tac[3].x + tac[3].y));
      }
      st += ((acc[0].x + acc[0].y) + (acc[1].x + acc[1].y)) +
            ((acc[2].x + acc[2].y) + (acc[3].x + acc[3].y));
    }
    return cm;
  };
  // theta = the best k-th value any warp of the CTA has published so far
  auto refresh = [&]() {
    float tp = lane < kWWarps ? pub[lane] : -INFINITY;
#pragma unroll
    for (int off = 4; off > 0; off >>= 1) tp = fmaxf(tp, __shfl_xor_sync(kFull, tp, off));
    theta = fmaxf(theta, __shfl_sync(kFull, tp, 0));
  };
  // candidates of chunk c (cm: the lane's chunk maximum; padding vectors hold -inf
  // and are never taken)
  auto collect = [&](const uint4 (&d)[kWVec], float cm, int c) {
    const bool lane_hit = cm >= theta;
    if (!__any_sync(kFull, lane_hit)) return;
    const int vb = wb + c * kWChunkVec;
    const int nv = min(kWChunkVec, we - vb);
    unsigned hits = 0u;
    if (lane_hit) {
#pragma unroll
      for (int i = 0; i < kWVec; ++i)
        if (i * 32 + lane < nv && E::vmax(d[i]) >= theta) hits |= 1u << i;
    }
    if (!__any_sync(kFull, hits != 0u)) return;
#pragma unroll
    for (int i = 0; i < kWVec; ++i) {
      if (!__any_sync(kFull, (hits >> i) & 1u)) continue;
      unsigned m = 0u;
      if ((hits >> i) & 1u) {
#pragma unroll
        for (int e = 0; e < n; ++e)
          if (E::value(d[i], e) >= theta) m |= 1u << e;
      }
      const WarpTop t = drain_vector<E>(WarpTop{lst, thr, theta}, d[i], m,
                                        head + (vb + i * 32 + lane) * n, k, &pub[warp]);
      lst = t.lst;
      thr = t.thr;
      theta = t.theta;
    }
  };

  // ---- every warp's first chunk, then the CTA's first threshold: the k-th largest
  // of all lanes' first-chunk maxima (as ordered integers; -inf where a lane had no
  // data).  Each warp's k largest come from k warp-wide maximum reductions; then a
  // thread per value counts the larger ones.
  uint4 d[kWVec];
  bool alive = true;
  float cm0 = -INFINITY;
  int failed = -1;  // the chunk whose wait gave up
  if (nch > 0) {
    alive = take(d, 0);
    if (alive) cm0 = reduce(d);
    else failed = 0;
  }
  {
    uint32_t o = ordered(cm0);  // >= ordered(-inf) > 0: a taken lane's 0 never wins
    for (int s2 = 0; s2 < k; ++s2) {
      const uint32_t mx = __reduce_max_sync(kFull, o);
      if (lane == 0) sh.first[warp * k + s2] = mx;
      const unsigned win = __ballot_sync(kFull, o == mx);
      if (lane == __ffs(win) - 1) o = 0u;
    }
  }
  __syncthreads();
  if (tid < kWWarps * k) {
    const uint32_t v = sh.first[tid];
    const int nf = kWWarps * k;
    int r = 0;
    int u = 0;
    for (; u + 8 <= nf; u += 8) {
#pragma unroll
      for (int z = 0; z < 8; ++z) {
        const uint32_t y = sh.first[u + z];
        r += y > v || (y == v && u + z < tid);
      }
    }
    for (; u < nf; ++u) {
      const uint32_t y = sh.first[u];
      r += y > v || (y == v && u < tid);
    }
    if (r == k - 1) sh.theta0 = unordered(v);
  }
  __syncthreads();
  theta = sh.theta0;
  if (lane == 0 && theta > pub[warp]) pub[warp] = theta;

  // ---- scalar elements (warp 0): the head of part 0 (lanes 0-6) and the tail of
  // the last part (lanes 8-14), each < 8 elements, join the lanes' online pairs
  if (warp == 0) {
    int xid = -1;
    if (part == 0 && lane < head) xid = lane;
    if (part == a.parts - 1 && lane >= 8 && lane - 8 < V - tail0) xid = tail0 + (lane - 8);
    const float x = xid >= 0 ? E::load(rowp + xid) : -INFINITY;
    rescale_to<ENT>(mt, st, tt, x);
    if (xid >= 0 && mt != -INFINITY) {
      const float u = fmaxf(fmaf(x, kLog2e, -mt * kLog2e), -256.f);
      const float p = ex2(u);
      st += p;
      if constexpr (ENT) tt = fmaf(p, u, tt);
    }
    unsigned m = (xid >= 0 && x >= theta) ? 1u : 0u;
    drain(m, [&](int) { return elem_key(x, xid); });
  }

  // ---- the chunks
  if (alive && nch > 0) collect(d, cm0, 0);
  for (int c = 1; alive && c < nch; ++c) {
    if (!take(d, c)) {
      alive = false;
      failed = c;
      break;
    }
    const float cm = reduce(d);
    refresh();
    collect(d, cm, c);
  }
  if (failed >= 0 && lane == 0) {
    // gave up: no copy of this warp may still be landing when the CTA exits (chunks
    // failed .. failed + kWStages - 1 were issued and not taken)
    for (int c2 = failed; c2 < nch && c2 < failed + kWStages; ++c2)
      mbar_wait(&sh.full[warp][c2 % kWStages], (c2 / kWStages) & 1, nullptr);
  }

  // ---- the warp's (max, Σ) pair and its keys at or above theta, into the leader
  refresh();
  {
    float m2 = mt == -INFINITY ? -INFINITY : mt * kLog2e;
    float sw = st, tw = tt;
    warp_merge_pairs<ENT>(m2, sw, tw);
    WSmem* ld = &sh;
    if (a.parts > 1) ld = cg::this_cluster().map_shared_rank(&sh, 0);
    const int slot = part * kWWarps + warp;
    if (lane < k) ld->keys[slot * k + lane] = (lst != 0ull && key_value(lst) >= theta) ? lst : 0ull;
    if (lane == 0) {
      ld->ms[slot] = make_float2(m2, sw);
      if constexpr (ENT) ld->ts[slot] = tw;
    }
  }
  if (a.parts > 1)
    cg::this_cluster().sync();
  else
    __syncthreads();
  if (part != 0) return;

  // ---- leader: the row's top-k among the kept keys (every one of the row's top-k is
  // kept, so at least k are real), and its (max, Σ) from the warps' pairs
  const int M = a.parts * kWWarps * k;
  for (int i = tid; i < M; i += kWThreads) {
    const unsigned long long ki = sh.keys[i];
    if (ki == 0ull) continue;
    int r = 0;
    int u = 0;
    for (; u + 8 <= M; u += 8) {
#pragma unroll
      for (int z = 0; z < 8; ++z) r += sh.keys[u + z] > ki;
    }
    for (; u < M; ++u) r += sh.keys[u] > ki;
    if (r < k) sh.list[r] = ki;
  }
  float m_row = -INFINITY, s_row = 0.f, t_row = 0.f;
  if (warp == 0) {
    // lane l folds slots l and l + 32 (<= 64 slots), then the warp merges the lanes
    const int P = a.parts * kWWarps;
    float ma = lane < P ? sh.ms[lane].x : -INFINITY;
    float sa = lane < P ? sh.ms[lane].y : 0.f;
    float ta = 0.f;
    if constexpr (ENT) ta = lane < P ? sh.ts[lane] : 0.f;
    const float mb = lane + 32 < P ? sh.ms[lane + 32].x : -INFINITY;
    const float sb = lane + 32 < P ? sh.ms[lane + 32].y : 0.f;
    if constexpr (ENT) {
      const float tb = lane + 32 < P ? sh.ts[lane + 32] : 0.f;
      merge_mst(ma, sa, ta, mb, sb, tb);
    } else {
      merge_ms(ma, sa, mb, sb);
    }
    warp_merge_pairs<ENT>(ma, sa, ta);
    m_row = ma;
    s_row = sa;
    t_row = ta;
  }
  __syncthreads();  // the row's list is complete
  if (warp == 0) write_row<ENT>(a, sh.list, row, m_row, s_row, t_row);
}

template <typename T, int VMAX, bool ENT>
int max_active_clusters(int parts) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(static_cast<unsigned>(parts));
  cfg.blockDim = dim3(kThreads);
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = parts;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, topk_kernel<T, VMAX, ENT>, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

template <bool ENT>
int max_active_clusters_of(int eb, int vmax, int parts) {
  if (eb == 4)
    return vmax == 4 ? max_active_clusters<float, 4, ENT>(parts)
           : vmax == 8 ? max_active_clusters<float, 8, ENT>(parts)
                       : max_active_clusters<float, 16, ENT>(parts);
  return vmax == 4 ? max_active_clusters<__nv_bfloat16, 4, ENT>(parts)
         : vmax == 8 ? max_active_clusters<__nv_bfloat16, 8, ENT>(parts)
                     : max_active_clusters<__nv_bfloat16, 16, ENT>(parts);
}

// Resident clusters of `parts` CTAs for the kernel of element size eb, register
// bound vmax and entropy flag ent, queried once per device.
int active_clusters(int eb, int vmax, int parts, bool ent) {
  static std::mutex mu;
  static int cache[64][2][3][2][kMaxParts + 1];
  static bool done[64][2][3][2][kMaxParts + 1];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) dev = 0;
  const int ti = eb == 4 ? 0 : 1, vi = vmax == 4 ? 0 : (vmax == 8 ? 1 : 2), ei = ent ? 1 : 0;
  std::lock_guard<std::mutex> lock(mu);
  if (!done[dev][ti][vi][ei][parts]) {
    cache[dev][ti][vi][ei][parts] = ent ? max_active_clusters_of<true>(eb, vmax, parts)
                                        : max_active_clusters_of<false>(eb, vmax, parts);
    done[dev][ti][vi][ei][parts] = true;
  }
  return cache[dev][ti][vi][ei][parts];
}

// Spans per row (= cluster size) and vectors per thread: the estimated time is
// waves of resident clusters x (fixed cost + cost per vector per thread).
Plan make_plan(int B, int L, int V, int elem_bytes, bool ent) {
  Plan p;
  p.rows = B * L;
  p.epv = 16 / elem_bytes;
  const int nvec = V / p.epv + 1;  // upper bound on a row's aligned vectors
  double best = 1e30;
  p.parts = 1;
  p.vpt = 1;
  for (int parts = 1; parts <= kMaxParts; ++parts) {
    const int vpt = (nvec + parts * kThreads - 1) / (parts * kThreads);
    if (vpt > 16) continue;
    if (parts > 1 && (nvec + vpt * kThreads - 1) / (vpt * kThreads) < parts) continue;  // empty span
    const int vmax = vpt <= 4 ? 4 : (vpt <= 8 ? 8 : 16);
    int act = active_clusters(elem_bytes, vmax, parts, ent);
    if (act < 1) act = parts == 1 ? sm_count() : 0;
    if (act < 1) continue;
    const double waves = std::ceil(static_cast<double>(p.rows) / act);
    const double cost = waves * (4.0 + 0.3 * vpt);
    if (cost < best - 1e-9) {
      best = cost;
      p.parts = parts;
      p.vpt = vpt;
    }
  }
  p.vmax = p.vpt <= 4 ? 4 : (p.vpt <= 8 ? 8 : 16);
  p.stream = false;
  // More than one wave of the register kernel: stream instead, with about one CTA
  // per SM or more (a row's spans still form one cluster of <= 8 CTAs)
  const int act = active_clusters(elem_bytes, p.vmax, p.parts, ent);
  if (act >= 1 && p.rows > act) {
    const int slots = kWCtasPerSm * sm_count();  // resident CTAs of the streaming kernel
    int parts = slots / p.rows;
    parts = parts < 1 ? 1 : (parts > kMaxParts ? kMaxParts : parts);
    const int nv = V / p.epv;  // a row's aligned vectors, up to one
    while (parts > 1 && (nv + parts - 1) / parts < kWWarps * kWChunkVec / 2) --parts;  // no tiny spans
    p.stream = true;
    p.parts = parts;
    p.vpt = (nv + 1 + parts - 1) / parts;
  }
  return p;
}

template <typename T, int VMAX, bool ENT>
cudaError_t launch(const Plan& p, const Args& a, cudaStream_t stream) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(static_cast<unsigned>(p.rows) * p.parts);
  cfg.blockDim = dim3(kThreads);
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = p.parts;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1] = pdl_attribute();
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, topk_kernel<T, VMAX, ENT>, a);
}

template <typename T, bool ENT>
cudaError_t launch_stream(const Plan& p, const Args& a, cudaStream_t stream) {
  static PerDeviceOnce attr;
  const cudaError_t ae = attr.run([] {
    return cudaFuncSetAttribute(topk_stream_kernel<T, ENT>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize,
                                static_cast<int>(kWDynBytes));
  });
  if (ae != cudaSuccess) return ae;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(static_cast<unsigned>(p.rows) * p.parts);
  cfg.blockDim = dim3(kWThreads);
  cfg.dynamicSmemBytes = kWDynBytes;
  cfg.stream = stream;
  cudaLaunchAttribute at[2];
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = p.parts;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  at[1] = pdl_attribute();
  cfg.attrs = at;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, topk_stream_kernel<T, ENT>, a);
}

template <bool ENT>
cudaError_t dispatch(int dtype, const Plan& p, const Args& a, cudaStream_t stream) {
  if (p.stream)
    return dtype == PRESTO_F32 ? launch_stream<float, ENT>(p, a, stream)
                               : launch_stream<__nv_bfloat16, ENT>(p, a, stream);
  if (dtype == PRESTO_F32)
    return p.vmax == 4 ? launch<float, 4, ENT>(p, a, stream)
           : p.vmax == 8 ? launch<float, 8, ENT>(p, a, stream)
                         : launch<float, 16, ENT>(p, a, stream);
  return p.vmax == 4 ? launch<__nv_bfloat16, 4, ENT>(p, a, stream)
         : p.vmax == 8 ? launch<__nv_bfloat16, 8, ENT>(p, a, stream)
                       : launch<__nv_bfloat16, 16, ENT>(p, a, stream);
}

// Slot-row source of presto_topk_slots (see Args).
struct SlotRows {
  const int32_t* acc_len;
  const int32_t* acc_path;
  int path_len, n_prev, n_slots, slot_off;
  const int32_t* node_token;
  const int32_t* bonus;
  int32_t* ctx2_next;
};

// Checks and launch shared by presto_topk, presto_topk_entropy and presto_topk_slots
// (B x L output rows; `slots` null: row r of the logits is output row r).
int topk_common(const void* logits, int dtype, int B, int L, int V, long long row_stride, int k,
                int32_t* topk_ids, float* topk_logq, float* lse, float* entropy, float* lambda_d,
                float beta, float C, const SlotRows* slots, int32_t* dev_status,
                cudaStream_t stream) {
  PRESTO_CHECK_ARG(logits && topk_ids && topk_logq);
  PRESTO_CHECK_ARG(dtype == PRESTO_F32 || dtype == PRESTO_BF16);
  PRESTO_CHECK_ARG(B >= 1 && L >= 1 && V >= 1 && k >= 1 && row_stride >= V);
  PRESTO_CHECK_ARG(k <= V);
  PRESTO_CHECK_LIMIT(k <= kMaxK && V < kMaxV && L <= kMaxL);
  const int eb = dtype == PRESTO_F32 ? 4 : 2;
  PRESTO_CHECK_ARG(reinterpret_cast<uintptr_t>(logits) % eb == 0);
  const bool ent = entropy || lambda_d;
  const Plan p = make_plan(B, L, V, eb, ent);
  Args a{};
  a.logits = logits;
  a.row_stride = row_stride;
  a.V = V;
  a.k = k;
  a.parts = p.parts;
  a.vpt = p.vpt;
  if (p.stream && !slots) {
    // the whole problem up to kPrefetchCap bytes, the head of every warp's piece beyond
    const size_t total = static_cast<size_t>(B) * L * V * eb;
    const size_t warps = static_cast<size_t>(p.rows) * p.parts * kWWarps;
    const size_t per = total <= kPrefetchCap ? total : kPrefetchCap / warps;
    a.pf_bytes = static_cast<uint32_t>(std::min<size_t>(per, 0x7fffffffu) / 16 * 16);
  }
  a.topk_ids = topk_ids;
  a.topk_logq = topk_logq;
  a.lse = lse;
  a.entropy = entropy;
  a.lambda_d = lambda_d;
  a.beta = beta;
  a.C = C;
  if (slots) {
    a.acc_len = slots->acc_len;
    a.acc_path = slots->acc_path;
    a.path_len = slots->path_len;
    a.n_prev = slots->n_prev;
    a.n_slots = slots->n_slots;
    a.slot_off = slots->slot_off;
    a.Lrows = L;
    a.node_token = slots->node_token;
    a.bonus = slots->bonus;
    a.ctx2_next = slots->ctx2_next;
  }
  a.dev_status = dev_status;
  const cudaError_t e = ent ? dispatch<true>(dtype, p, a, stream) : dispatch<false>(dtype, p, a, stream);
  if (e != cudaSuccess) return PRESTO_ERR_CUDA;
  return launch_status();
}

}  // namespace
}  // namespace presto

using namespace presto;

extern "C" size_t presto_topk_workspace(int B, int L, int V, int k) {
  if (B < 1 || L < 1 || V < 1 || k < 1 || k > kMaxK) return 0;
  // spans merge inside thread-block clusters: no device workspace is needed
  return 256;
}

extern "C" int presto_topk(const void* logits, int dtype, int B, int L, int V,
                           long long row_stride, int k, int32_t* topk_ids, float* topk_logq,
                           float* lse, void* ws, size_t ws_bytes, int32_t* dev_status,
                           presto_stream_t stream) {
  (void)ws;
  (void)ws_bytes;
  return topk_common(logits, dtype, B, L, V, row_stride, k, topk_ids, topk_logq, lse, nullptr,
                     nullptr, 0.f, 0.f, nullptr, dev_status, stream);
}

extern "C" int presto_topk_entropy(const void* logits, int dtype, int B, int L, int V,
                                   long long row_stride, int k, float beta, float C,
                                   int32_t* topk_ids, float* topk_logq, float* lse,
                                   float* entropy, float* lambda_d, void* ws, size_t ws_bytes,
                                   int32_t* dev_status, presto_stream_t stream) {
  (void)ws;
  (void)ws_bytes;
  PRESTO_CHECK_ARG(entropy || lambda_d);
  if (lambda_d) PRESTO_CHECK_ARG(beta > 0.f && beta < INFINITY && C > 0.f && C < INFINITY);
  return topk_common(logits, dtype, B, L, V, row_stride, k, topk_ids, topk_logq, lse, entropy,
                     lambda_d, beta, C, nullptr, dev_status, stream);
}

extern "C" int presto_topk_slots(const void* slot_logits, int dtype, int B, int n_prev,
                                 int n_slots, int V, long long row_stride,
                                 const int32_t* accept_len, const int32_t* accept_path,
                                 int path_len, int slot_offset, int L, int k,
                                 const int32_t* node_token, const int32_t* bonus,
                                 int32_t* ctx2_next, int32_t* topk_ids, float* topk_logq,
                                 float* lse, void* ws, size_t ws_bytes, int32_t* dev_status,
                                 presto_stream_t stream) {
  (void)ws;
  (void)ws_bytes;
  PRESTO_CHECK_ARG(accept_len && accept_path);
  PRESTO_CHECK_ARG(B >= 1 && n_prev >= 1 && n_slots >= 1 && path_len >= 1 && L >= 1);
  PRESTO_CHECK_ARG(slot_offset >= 0 && slot_offset <= n_slots - L);
  PRESTO_CHECK_ARG((node_token && bonus && ctx2_next) || (!node_token && !bonus && !ctx2_next));
  PRESTO_CHECK_LIMIT(static_cast<long long>(B) * n_prev * n_slots < (1ll << 31));
  const SlotRows sr{accept_len, accept_path, path_len, n_prev, n_slots, slot_offset,
                    node_token, bonus, ctx2_next};
  return topk_common(slot_logits, dtype, B, L, V, row_stride, k, topk_ids, topk_logq, lse,
                     nullptr, nullptr, 0.f, 0.f, &sr, dev_status, stream);
}
