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
//         element, four independent accumulators);
//       - the CTA's threshold tau = the k-th largest of the 16 warp maxima: at least
//         k elements of the span are >= tau, so the span's top-k are among them;
//       - the elements >= tau (vectors whose maximum is below tau are skipped) become
//         64-bit keys (value as an ordered integer, then the complement of the id,
//         so "larger value, then lower id" is integer order) in a candidate buffer,
//         ranked by counting.  If the buffer overflows (massive ties), an exact
//         fallback raises a key threshold over the register-resident data until the
//         survivors fit.
//   * The leader CTA of the cluster merges the spans' (max, Σexp) pairs and top-k
//     lists and writes the row.
//   * With ENT the same pass also yields the row's entropy (App. F): next to
//     s = Σ 2^u, u = x log2e - max2, each thread sums t = Σ 2^u u, and the merges
//     carry t along (when the reference maximum drops by δ, t -> 2^δ (t + δ s)).
//     Then H = ln s - ln2 t / s, and lambda_d = beta H / (H + C).
//   * With slot rows (self-speculative rounds, App. C (II)) row j of sequence b is
//     read in place from slot slot_off + j of the deepest accepted node a*_b =
//     accept_path[b][accept_len[b]], looked up on the device after the accept
//     kernel that precedes it on the stream: no gather copy, no host round trip.
#include <cuda_bf16.h>

#include <cooperative_groups.h>

#include <cmath>
#include <mutex>

#include "common.cuh"

namespace presto {
namespace {

constexpr int kThreads = 512;
constexpr int kWarps = kThreads / 32;
constexpr int kMaxParts = 8;     // spans of a row = CTAs of its (portable) cluster
constexpr int kCandCap = 1024;   // candidate keys per CTA and round
constexpr float kLog2e = 1.4426950408889634f;
constexpr unsigned kFull = 0xffffffffu;
static_assert(kWarps >= kMaxK, "tau needs at least k warp maxima");

template <typename T>
struct Elem;
template <>
struct Elem<float> {
  static constexpr int kPerVec = 4;
  static constexpr int kBytes = 4;
  static constexpr uint32_t kNegInfWord = 0xff800000u;
  __device__ static float load(const float* p) { return *p; }
  __device__ static float value(const uint4& u, int e) {
    return __uint_as_float(e == 0 ? u.x : e == 1 ? u.y : e == 2 ? u.z : u.w);
  }
  __device__ static float vmax(const uint4& u) {
    float m;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(m) : "f"(__uint_as_float(u.x)), "f"(__uint_as_float(u.y)),
        "f"(__uint_as_float(u.z)));
    return fmaxf(m, __uint_as_float(u.w));
  }
};
template <>
struct Elem<__nv_bfloat16> {
  static constexpr int kPerVec = 8;
  static constexpr int kBytes = 2;
  static constexpr uint32_t kNegInfWord = 0xff80ff80u;
  __device__ static float load(const __nv_bfloat16* p) { return __bfloat162float(*p); }
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
};

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
  const int len = a.acc_len[b];
  int node = -1;
  if (len >= 0 && len < a.path_len) node = a.acc_path[static_cast<long long>(b) * a.path_len + len];
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
  unsigned long long part[kMaxParts][kMaxK];    // leader: the cluster's lists
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
    for (int j = 0; j < M; ++j) r += e[j] > ki;
    if (r < k) out[r] = ki;
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
    if (tid < k) leader->part[part][tid] = tid < got ? sh.list[tid] : 0ull;
    if (tid == 0) {
      leader->part_ms[part] = make_float2(m_cta, s_cta);
      if constexpr (ENT) leader->part_t[part] = t_cta;
    }
    cluster.sync();
    if (part != 0) return;
    // the parts' keys: zeros (fewer than k in a span) rank below every real key and
    // are dropped below
    const int P = a.parts * k;
    for (int i = tid; i < P; i += NT) sh.cand[i] = sh.part[i / k][i % k];
    if (warp == 0) {
      float mw = lane < a.parts ? sh.part_ms[lane].x : -INFINITY;
      float sw = lane < a.parts ? sh.part_ms[lane].y : 0.f;
      float tw = 0.f;
      if constexpr (ENT) tw = lane < a.parts ? sh.part_t[lane] : 0.f;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        const float m_o = __shfl_xor_sync(kFull, mw, off);
        const float s_o = __shfl_xor_sync(kFull, sw, off);
        if constexpr (ENT) {
          const float t_o = __shfl_xor_sync(kFull, tw, off);
          merge_mst(mw, sw, tw, m_o, s_o, t_o);
        } else {
          merge_ms(mw, sw, m_o, s_o);
        }
      }
      m_row = mw;
      s_row = sw;
      t_row = tw;
    }
    __syncthreads();
    rank_keys<NT>(sh.cand, P, k, sh.list, tid);
    __syncthreads();
  }
  // ---- write the row (warp 0 holds the row's (max, sum))
  if (warp == 0) {
    // natural-log normaliser: lse = (m2 + log2 s) ln 2 = max + ln s; log q = (x - max) - ln s
    const float mx = m_row * (1.f / kLog2e);
    const float logs = logf(s_row);
    if (lane == 0 && !(mx > -INFINITY && mx < INFINITY)) report(a.dev_status, PRESTO_DEV_NONFINITE);
    if (lane < k) {
      const unsigned long long key = sh.list[lane];
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
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    if constexpr (!ENT) {
#pragma unroll
      for (int i = 0; i < VMAX; ++i) {
#pragma unroll
        for (int e = 0; e < n; ++e) acc[e & 3] += ex2(fmaf(E::value(d[i], e), kLog2e, -m2));
      }
      st = (acc[0] + acc[1]) + (acc[2] + acc[3]);
      if (xid >= 0) st += ex2(fmaf(xval, kLog2e, -m2));
    } else {
      // u is clamped at -256: 2^u flushes to 0 there, so -inf entries add 0 to both
      float tac[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int i = 0; i < VMAX; ++i) {
#pragma unroll
        for (int e = 0; e < n; ++e) {
          const float u = fmaxf(fmaf(E::value(d[i], e), kLog2e, -m2), -256.f);
          const float p = ex2(u);
          acc[e & 3] += p;
          tac[e & 3] = fmaf(p, u, tac[e & 3]);
        }
      }
      st = (acc[0] + acc[1]) + (acc[2] + acc[3]);
      tt = (tac[0] + tac[1]) + (tac[2] + tac[3]);
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
  const uint32_t warp_hits = __reduce_or_sync(kFull, hits | (xhit ? 0x80000000u : 0u));
  unsigned long long thr = 1ull;  // every real key is >= 1
  int M;
  for (;;) {
    // count this thread's candidates, reserve their slots with one atomic per warp,
    // then write them.  Vectors are visited under warp-uniform votes; a visited
    // vector's elements >= tau form a bit mask from independent compares, and only
    // those elements become keys
    auto elem_mask = [&](int i) {
      uint32_t em = 0u;
#pragma unroll
      for (int e = 0; e < n; ++e) em |= (E::value(d[i], e) >= tau) ? (1u << e) : 0u;
      return ((hits >> i) & 1u) ? em : 0u;
    };
    auto visit = [&](auto&& emit) {
#pragma unroll
      for (int i = 0; i < VMAX; ++i) {
        if ((warp_hits >> i) & 1u) {  // warp-uniform
          uint32_t em = elem_mask(i);
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
    if (warp_hits && thr == 1ull) {  // every key passes: count the mask bits
#pragma unroll
      for (int i = 0; i < VMAX; ++i)
        if ((warp_hits >> i) & 1u) mine += __popc(elem_mask(i));
      mine += xhit;
    } else if (warp_hits) {
      visit([&](bool take, unsigned long long) { mine += take; });
    }
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
    // overflow: the k-th largest of the collected keys is <= the span's k-th largest
    // key, so raising the threshold to it keeps the span's top-k; keys are unique, so
    // it rises strictly and the rounds end
    rank_keys(sh.cand, kCandCap, k, sh.list, tid);
    __syncthreads();
    if (tid == 0) {
      sh.thr = sh.list[k - 1];
      sh.count = 0;
    }
    __syncthreads();
    thr = sh.thr;
  }
  // ---- the span's top-k
  rank_keys(sh.cand, M, k, sh.list, tid);
  // the span's (max, sum) from the warps'
  float m_cta = -INFINITY, s_cta = 0.f, t_cta = 0.f;
  if (warp == 0) {
    float mw = lane < kWarps ? sh.warp_ms[lane].x : -INFINITY;
    float sw = lane < kWarps ? sh.warp_ms[lane].y : 0.f;
    float tw = 0.f;
    if constexpr (ENT) tw = lane < kWarps ? sh.warp_t[lane] : 0.f;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const float m_o = __shfl_xor_sync(kFull, mw, off);
      const float s_o = __shfl_xor_sync(kFull, sw, off);
      if constexpr (ENT) {
        const float t_o = __shfl_xor_sync(kFull, tw, off);
        merge_mst(mw, sw, tw, m_o, s_o, t_o);
      } else {
        merge_ms(mw, sw, m_o, s_o);
      }
    }
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
// rows): one producer thread keeps a ring of kSStages bulk copies (32 KB each) of
// the CTA's span in flight while eight consumer warps work on the chunk before, so
// HBM stays busy for the whole life of the CTA.  A consumer thread takes 8 vectors
// of each chunk into registers and updates its online (max, Σexp) pair; the
// candidates are the elements at or above a threshold taken from the first chunk
// (the k-th largest of its 16 half-warp maxima: at least k elements of the span
// reach it), kept in a shared buffer that is cut back to the running top-k (and
// the threshold raised to its k-th key) whenever it passes half full.  A chunk whose
// candidates overflow the buffer is re-scanned from registers with a raised key
// threshold, as in the kernel above.
// ---------------------------------------------------------------------------
constexpr int kSCons = 256;                 // consumer threads (8 warps)
constexpr int kSWarps = kSCons / 32;
constexpr int kSThreads = kSCons + 32;      // + the producer warp
constexpr int kSVec = 8;                    // 16-byte vectors per consumer thread and chunk
constexpr int kSChunkVec = kSCons * kSVec;  // 2048 vectors
constexpr int kSChunkBytes = kSChunkVec * 16;
constexpr int kSStages = 3;

constexpr size_t kSDynBytes = static_cast<size_t>(kSStages) * kSChunkBytes + 128;
static_assert(2 * kSWarps >= kMaxK, "theta needs at least k half-warp maxima");
constexpr int kSCap = 1024;                 // candidate buffer
constexpr int kSCompact = kSCap / 2;        // cut back above this many
static_assert(kSCompact % kSCons == 0, "old candidates are re-read in whole rounds");

struct SSmem {
  uint64_t full[kSStages], empty[kSStages];
  unsigned long long cand[kSWarps * kMaxK];  // the warps' top-k; the parts' in the leader
  unsigned long long list[kMaxK];
  unsigned long long part[kMaxParts][kMaxK];
  float2 part_ms[kMaxParts];
  float part_t[kMaxParts];
  float2 warp_ms[kSWarps];
  float warp_t[kSWarps];
  unsigned long long cand2[kSCap];  // the span's candidates
  float gmax[2 * kSWarps];  // half-warp maxima of the first chunk
  float theta;              // the first chunk's threshold, for every consumer
  int cnt[3];               // candidates appended by chunk c, at cnt[c % 3]
  int fcnt;                 // the same on the overflow path
  int abort;                // set by any thread whose bounded wait ran out
  int stop[2];              // the consumers' common copy of abort at chunk c's end
};

__device__ __forceinline__ void consumers_sync() {
  asm volatile("bar.sync 1, %0;" ::"n"(kSCons) : "memory");
}

template <typename T, bool ENT>
__global__ void __launch_bounds__(kSThreads, 2) topk_stream_kernel(const Args a) {
  using E = Elem<T>;
  constexpr int n = E::kPerVec;
  constexpr int eb = E::kBytes;
  __shared__ SSmem sh;
  extern __shared__ unsigned char dyn_raw[];
  unsigned char* const ring = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(dyn_raw) + 127) & ~static_cast<uintptr_t>(127));
  pdl_launch_dependents();
  const int row = blockIdx.x / a.parts;
  const int part = blockIdx.x % a.parts;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int k = a.k, V = a.V;
  if (tid == 0) {
    for (int st = 0; st < kSStages; ++st) {
      mbar_init(&sh.full[st], 1);
      mbar_init(&sh.empty[st], kSWarps);
    }
    for (int i = 0; i < 3; ++i) sh.cnt[i] = 0;
    sh.abort = 0;
    sh.theta = -INFINITY;
    fence_barrier_init();
  }
  __syncthreads();
  pdl_wait();  // the logits (and slot rows' accept results) come from earlier kernels
  const T* rowp = row_base<T>(a, row, part == 0 && tid == 0);
  const int mis = static_cast<int>(reinterpret_cast<uintptr_t>(rowp) & 15);
  const int head = min(V, mis == 0 ? 0 : (16 - mis) / eb);
  const int nvec = (V - head) / n;
  const int tail0 = head + nvec * n;
  const uint4* vecp = reinterpret_cast<const uint4*>(rowp + head);
  const int v0 = min(nvec, part * a.vpt);  // vpt: vectors per span here
  const int v1 = min(nvec, v0 + a.vpt);
  const int nch = (v1 - v0 + kSChunkVec - 1) / kSChunkVec;
  volatile int* abort = &sh.abort;

  float m_cta = -INFINITY, s_cta = 0.f, t_cta = 0.f;
  int got = 0;
  if (warp == kSWarps) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      int c = 0;
      for (; c < nch; ++c) {
        const int st = c % kSStages;
        if (c >= kSStages && !mbar_wait(&sh.empty[st], (c / kSStages - 1) & 1, abort)) {
          *abort = 1;
          report(a.dev_status, PRESTO_DEV_TIMEOUT);
          break;
        }
        const int vb = v0 + c * kSChunkVec;
        const int nv = min(kSChunkVec, v1 - vb);
        mbar_arrive_expect_tx(&sh.full[st], static_cast<uint32_t>(nv) * 16u);
        bulk_g2s(ring + st * kSChunkBytes, vecp + vb, static_cast<uint32_t>(nv) * 16u,
                 &sh.full[st]);
      }
      // no copy may still be landing when the CTA exits (the consumers have waited
      // for every one already unless they gave up)
      for (int c2 = c > kSStages ? c - kSStages : 0; c2 < c; ++c2)
        mbar_wait(&sh.full[c2 % kSStages], (c2 / kSStages) & 1, nullptr);
    }
  } else {
    // ------------------------------------------------------------ consumers
    // extra scalar element: threads 0-6 of part 0 take the head, 8-14 of the last
    // part the tail (each < 8 elements), with the first chunk
    int xid = -1;
    if (part == 0 && tid < head) xid = tid;
    if (part == a.parts - 1 && tid >= 8 && tid - 8 < V - tail0) xid = tail0 + (tid - 8);
    const float xval0 = xid >= 0 ? E::load(rowp + xid) : -INFINITY;
    float mt = -INFINITY, st = 0.f, tt = 0.f;  // running max (plain), Σ 2^u, Σ 2^u u
    float theta = -INFINITY;                   // candidates: value >= theta ...
    unsigned long long thr = 1ull;             // ... and key >= thr (every real key is >= 1)
    int base = 0;                              // candidates kept from earlier chunks
    const int nloop = nch > 0 ? nch : 1;       // one round for the scalars alone
    for (int c = 0; c < nloop; ++c) {
      const int sg = c % kSStages;
      const int vb = v0 + c * kSChunkVec;
      const int nv = c < nch ? min(kSChunkVec, v1 - vb) : 0;
      bool ok = true;
      if (c < nch && !mbar_wait(&sh.full[sg], (c / kSStages) & 1, abort)) {
        ok = false;
        *abort = 1;
        report(a.dev_status, PRESTO_DEV_TIMEOUT);
      }
      uint4 d[kSVec];
      const uint32_t ni = E::kNegInfWord;
      auto load_chunk = [&]() {
#pragma unroll
        for (int i = 0; i < kSVec; ++i) {
          const int vi = i * kSCons + tid;
          d[i] = (ok && vi < nv)
                     ? *reinterpret_cast<const uint4*>(ring + sg * kSChunkBytes + vi * 16)
                     : make_uint4(ni, ni, ni, ni);
        }
      };
      load_chunk();  // the slot is released once the chunk's candidates are taken
      const float xval = c == 0 ? xval0 : -INFINITY;
      const bool xin = c == 0 && xid >= 0;

      // ---- the chunk's maximum and the online (max, Σ 2^u) pair, log2 domain
      float cm = xval;
#pragma unroll
      for (int i = 0; i < kSVec; ++i) cm = fmaxf(cm, E::vmax(d[i]));
      if (cm > mt) {
        if (mt != -INFINITY) {
          const float dl = mt * kLog2e - cm * kLog2e;  // the old reference minus the new
          const float f = ex2(dl);
          if constexpr (ENT) tt = f * fmaf(dl, st, tt);
          st *= f;
        }
        mt = cm;
      }
      if (mt != -INFINITY) {
        const float m2 = mt * kLog2e;
        float acc[4] = {0.f, 0.f, 0.f, 0.f};
        if constexpr (!ENT) {
#pragma unroll
          for (int i = 0; i < kSVec; ++i)
#pragma unroll
            for (int e = 0; e < n; ++e) acc[e & 3] += ex2(fmaf(E::value(d[i], e), kLog2e, -m2));
          if (xin) acc[0] += ex2(fmaf(xval, kLog2e, -m2));
        } else {
          // u clamped at -256: 2^u flushes to 0 there, so -inf adds 0 to both sums
          float tac[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
          for (int i = 0; i < kSVec; ++i)
#pragma unroll
            for (int e = 0; e < n; ++e) {
              const float u = fmaxf(fmaf(E::value(d[i], e), kLog2e, -m2), -256.f);
              const float p = ex2(u);
              acc[e & 3] += p;
              tac[e & 3] = fmaf(p, u, tac[e & 3]);
            }
          if (xin) {
            const float u = fmaxf(fmaf(xval, kLog2e, -m2), -256.f);
            const float p = ex2(u);
            acc[0] += p;
            tac[0] = fmaf(p, u, tac[0]);
          }
          tt += (tac[0] + tac[1]) + (tac[2] + tac[3]);
        }
        st += (acc[0] + acc[1]) + (acc[2] + acc[3]);
      }

      // ---- first chunk: theta = the k-th largest half-warp maximum (CTA-wide, once)
      if (c == 0) {
        float hm = cm;
#pragma unroll
        for (int off = 8; off > 0; off >>= 1) hm = fmaxf(hm, __shfl_xor_sync(kFull, hm, off));
        if ((lane & 15) == 0) sh.gmax[warp * 2 + (lane >> 4)] = hm;
        consumers_sync();
        if (warp == 0 && lane < 2 * kSWarps) {
          const float x = sh.gmax[lane];
          int r = 0;
#pragma unroll
          for (int u = 0; u < 2 * kSWarps; ++u) {
            const float y = sh.gmax[u];
            r += y > x || (y == x && u < lane);
          }
          if (r == k - 1) sh.theta = x;
        }
        consumers_sync();
        theta = sh.theta;
      } else {
        // later chunks: every warp publishes its half-warps' running maxima (real
        // elements, so the k-th largest of the 16 published values still has k
        // elements at or above it) and raises its own threshold to that k-th largest,
        // with no barrier: a value another warp has not yet raised is only a looser
        // bound
        volatile float* gm = sh.gmax;
        float hm = mt;
#pragma unroll
        for (int off = 8; off > 0; off >>= 1) hm = fmaxf(hm, __shfl_xor_sync(kFull, hm, off));
        if ((lane & 15) == 0) gm[warp * 2 + (lane >> 4)] = hm;
        __syncwarp();
        const float x = lane < 2 * kSWarps ? gm[lane] : -INFINITY;
        int r = 0;
#pragma unroll
        for (int u = 0; u < 2 * kSWarps; ++u) {
          const float y = __shfl_sync(kFull, x, u);
          r += y > x || (y == x && u < lane);
        }
        const unsigned who = __ballot_sync(kFull, lane < 2 * kSWarps && r == k - 1);
        theta = fmaxf(theta, __shfl_sync(kFull, x, __ffs(who) - 1));
      }

      // ---- candidates of the chunk (value >= theta, key >= thr), appended one by one
      // (they are rare) at base + a per-chunk counter.  The counter of chunk c + 2
      // is cleared right after chunk c's barrier: every thread read it (as chunk
      // c - 1's) before that barrier, and appends to it only after the next one.
      auto emit_chunk = [&](unsigned long long thr_k, int* ctr, int at) {
#pragma unroll
        for (int i = 0; i < kSVec; ++i) {
          const int vi = i * kSCons + tid;
          if (vi < nv && E::vmax(d[i]) >= theta) {
            const int id0 = head + (vb + vi) * n;
#pragma unroll
            for (int e = 0; e < n; ++e) {
              const float x = E::value(d[i], e);
              const unsigned long long key = elem_key(x, id0 + e);
              if (x >= theta && key >= thr_k) {
                const int j = at + atomicAdd(ctr, 1);
                if (j < kSCap) sh.cand2[j] = key;
              }
            }
          }
        }
        if (xin && xval >= theta) {
          const unsigned long long key = elem_key(xval, xid);
          if (key >= thr_k) {
            const int j = at + atomicAdd(ctr, 1);
            if (j < kSCap) sh.cand2[j] = key;
          }
        }
      };
      const int cs = c % 3;
      emit_chunk(thr, &sh.cnt[cs], base);
      if (tid == 0) sh.stop[c & 1] = *abort;  // one reading for all consumers
      consumers_sync();
      int M = base + sh.cnt[cs];
      const int stop = sh.stop[c & 1];
      if (tid == 0) sh.cnt[(c + 2) % 3] = 0;
      while (M > kSCap) {
        // overflow: the k-th largest of the buffer's keys bounds the span's top-k
        // from below; keep the earlier chunks' keys above it and re-scan this one
        rank_keys<kSCons>(sh.cand2, kSCap, k, sh.list, tid);
        consumers_sync();
        thr = sh.list[k - 1];
        unsigned long long keep[kSCompact / kSCons];
#pragma unroll
        for (int j = 0; j < kSCompact / kSCons; ++j) {
          const int e = j * kSCons + tid;
          keep[j] = (e < base && sh.cand2[e] >= thr) ? sh.cand2[e] : 0ull;
        }
        if (tid == 0) sh.fcnt = 0;
        consumers_sync();
#pragma unroll
        for (int j = 0; j < kSCompact / kSCons; ++j)
          if (keep[j]) sh.cand2[atomicAdd(&sh.fcnt, 1)] = keep[j];
        consumers_sync();
        base = sh.fcnt;
        consumers_sync();
        if (tid == 0) sh.fcnt = 0;
        consumers_sync();
        load_chunk();  // the chunk again, from its ring slot
        emit_chunk(thr, &sh.fcnt, base);
        consumers_sync();
        M = base + sh.fcnt;
        consumers_sync();  // every thread has read the counter
      }
      __syncwarp();
      if (c < nch && lane == 0) mbar_arrive(&sh.empty[sg]);  // the slot may be refilled
      if (M > kSCompact) {
        // cut back to the running top-k and raise the thresholds to its k-th key
        rank_keys<kSCons>(sh.cand2, M, k, sh.list, tid);
        consumers_sync();
        thr = sh.list[k - 1];
        if (tid < k) sh.cand2[tid] = sh.list[tid];
        M = k;
        consumers_sync();
      }
      if (thr > 1ull) theta = fmaxf(theta, key_value(thr));
      base = M;
      if (stop) break;
    }
    // ---- the span's top-k and its (max, sum) pair
    rank_keys<kSCons>(sh.cand2, base, k, sh.list, tid);
    got = base < k ? base : k;
    const uint32_t wm_o = __reduce_max_sync(kFull, ordered(mt));
    const float wm = unordered(wm_o);
    const float wm2 = wm * kLog2e;
    const float m2 = mt * kLog2e;
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
      if constexpr (ENT) sh.warp_t[warp] = wt;
    }
    consumers_sync();
    if (warp == 0) {
      float mw = lane < kSWarps ? sh.warp_ms[lane].x : -INFINITY;
      float sw = lane < kSWarps ? sh.warp_ms[lane].y : 0.f;
      float tw = 0.f;
      if constexpr (ENT) tw = lane < kSWarps ? sh.warp_t[lane] : 0.f;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        const float m_o = __shfl_xor_sync(kFull, mw, off);
        const float s_o = __shfl_xor_sync(kFull, sw, off);
        if constexpr (ENT) {
          const float t_o = __shfl_xor_sync(kFull, tw, off);
          merge_mst(mw, sw, tw, m_o, s_o, t_o);
        } else {
          merge_ms(mw, sw, m_o, s_o);
        }
      }
      m_cta = mw;
      s_cta = sw;
      t_cta = tw;
    }
  }
  __syncthreads();  // producer and consumers
  finish_row<ENT, kSCons>(a, sh, row, part, m_cta, s_cta, t_cta, got);
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
    const int sms = sm_count();
    int parts = (sms + p.rows - 1) / p.rows;
    parts = parts < 1 ? 1 : (parts > kMaxParts ? kMaxParts : parts);
    const int nv = V / p.epv;  // a row's aligned vectors, up to one
    while (parts > 1 && (nv + parts - 1) / parts < kSChunkVec / 2) --parts;  // no tiny spans
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
  static const cudaError_t attr = cudaFuncSetAttribute(
      topk_stream_kernel<T, ENT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
      static_cast<int>(kSDynBytes));
  if (attr != cudaSuccess) return attr;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(static_cast<unsigned>(p.rows) * p.parts);
  cfg.blockDim = dim3(kSThreads);
  cfg.dynamicSmemBytes = kSDynBytes;
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

// ---------------------------------------------------------------------------
// Allocation-free top-k.
//
// Some callers cannot hand this library a workspace: a plugin running inside an
// inference server whose device memory all belongs to the host framework's
// allocator, a C caller with no allocator handle at all, or a latency-critical
// loop that must not call cudaMalloc (which can block on device-wide
// synchronisation and fail under fragmentation).  For them this entry point
// hands presto_topk a fixed file-scope device array as its workspace, and
// otherwise runs the same code.  (The current plan merges a row's spans inside a
// thread-block cluster and uses no workspace, so the array is reserved rather
// than used.)
//
// The array costs kStaticScratchBytes on every GPU that loads this library, for
// the life of the process.  All calls on one device share it: should a plan use
// it, two calls whose kernels overlap on the GPU (different streams, no ordering
// between them) would race on it.
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
