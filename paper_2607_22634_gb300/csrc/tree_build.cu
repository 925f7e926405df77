// presto_score_build_tree: prefix-aligned token scores (§4.1, Eq. path-score)
// and best-first tree construction (§4.2, Alg. 2; a node is committed when it is
// popped), plus the device-side trigram table (presto_ngram3_*).
//
// One thread-block cluster of 8 CTAs per sequence:
//   phase 1 (all CTAs): each CTA takes a share of the context pairs reachable in
//     the candidate tree and computes, for every candidate j of depth d+1 under
//     that context, s = log q + lambda log rho (hash-table probes, batched so their
//     loads overlap), keeps the top-b by (s desc, token asc) as 8-byte records that
//     already hold the child's key bits, and notes whether fp32 rounding can reorder
//     two kept siblings; it writes them into the leader CTA's shared memory
//     (distributed shared memory), then the cluster synchronises once.
//   phase 2 (leader, warp 0): the pop loop.  A frontier entry carries a 64-bit key packing
//     the total order (S desc, depth asc, token asc, parent index asc), so two
//     warp-wide max reductions find the next node.  Each committed node owns one
//     entry (its next child not yet taken), held in a fixed register slot of a fixed
//     lane: popping a child advances its parent's entry to the next sibling and
//     gives the new node an entry for its first child (lazy sibling enumeration).
#include <cooperative_groups.h>

#include <initializer_list>

#include "common.cuh"

namespace presto {
namespace {

constexpr int kThreads = 512;
constexpr unsigned kFull = 0xffffffffu;

__host__ __device__ inline uint64_t fmix64(uint64_t k) {
  // MurmurHash3 64-bit finaliser (Appleby, public domain).
  k ^= k >> 33;
  k *= 0xff51afd7ed558ccdull;
  k ^= k >> 33;
  k *= 0xc4ceb9fe1a85ec53ull;
  k ^= k >> 33;
  return k;
}

// Linear probe for `key` starting at slot h.
__device__ __noinline__ float probe_from(const uint64_t* keys, const float* logrho,
                                         uint32_t mask, float miss, uint64_t key, uint32_t h) {
  for (uint32_t it = 0; it <= mask; ++it) {
    const uint64_t kk = __ldg(keys + h);
    if (kk == key) return __ldg(logrho + h);
    if (kk == PRESTO_NGRAM3_EMPTY) return miss;
    h = (h + 1) & mask;
  }
  return miss;
}

__global__ void ngram_insert_kernel(uint64_t* keys, float* logrho, uint32_t mask,
                                    const uint64_t* in_keys, const float* in_val, int n,
                                    int32_t* dev_status) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const uint64_t key = in_keys[i];
  if (key == PRESTO_NGRAM3_EMPTY) return;
  uint32_t h = static_cast<uint32_t>(fmix64(key)) & mask;
  for (uint32_t it = 0; it <= mask; ++it) {
    const unsigned long long prev = atomicCAS(reinterpret_cast<unsigned long long*>(keys + h),
                                              PRESTO_NGRAM3_EMPTY, key);
    if (prev == PRESTO_NGRAM3_EMPTY || prev == key) {
      logrho[h] = in_val[i];
      return;
    }
    h = (h + 1) & mask;
  }
  report(dev_status, PRESTO_DEV_TABLE_FULL);
}

struct Args {
  const int32_t* ids;
  const float* logq;
  const int32_t* ctx2;
  const uint64_t* keys;
  const float* logrho;
  uint32_t cap_mask;
  float miss;
  float lambda;
  int use_table;
  int L, k, bf, N;
  int nctx_all;      // contexts of one sequence over all depths
  int per_cta;       // contexts each CTA of the cluster scores
  int tables_in_smem;
  unsigned char* g_tables;  // [B][tables_bytes] when the tables do not fit in smem
  int32_t* node_token;
  int32_t* node_parent;
  int32_t* node_depth;
  float* node_score;
  int32_t* n_nodes;
  int32_t* dev_status;
};

// Order-preserving map float -> uint32 (larger float -> larger integer) and back.
__device__ __forceinline__ uint32_t ordered(float f) {
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float unordered(uint32_t o) {
  return __uint_as_float((o & 0x80000000u) ? (o & 0x7fffffffu) : ~o);
}
// Frontier key: larger key = earlier in the total order (S desc, depth asc, token
// asc, parent index asc).  Zero never occurs for a real node (ordered(-inf) > 0).
__device__ __forceinline__ uint64_t make_key(float S, int depth, int token, int parent) {
  return (static_cast<uint64_t>(ordered(S)) << 32) |
         (static_cast<uint64_t>(63 - depth) << 26) |
         (static_cast<uint64_t>(0x3FFFF - token) << 8) | static_cast<uint64_t>(255 - parent);
}

struct Smem {
  int tok[kMaxN];
  int par[kMaxN];
  int dep[kMaxN];
  float S[kMaxN];
  int cid[kMaxL][kMaxK];          // candidate tokens of every depth
  float clq[kMaxL][kMaxK];        // their log q
  int ctx0, ctx1;
};

// Tables of one sequence, indexed by context c = d * ctx_stride + ci (d = depth of
// the children - 1, ci = context pair index):
//   kid  uint2[c][b]  the top-b candidates of the context in (s desc, token asc)
//                     order: x = bits of s, y = the key bits of (depth d+1, token)
//                     with the candidate index in the low byte (the parent field
//                     of the key, filled in when the child is generated)
//   info float2[c]    (smallest gap between s-adjacent kept candidates whose tokens
//                     are in descending order, largest |s| among them)
// With a prefix signal ctx_stride = k*k (contexts (t_{d-1}, t_d) as index pairs);
// marginal-only scoring has one context per depth.
struct TableLayout {
  int cs, nctx;
  size_t info_off, bytes;
  __host__ __device__ TableLayout(int L, int k, int bf, int use_table) {
    cs = use_table ? k * k : 1;
    nctx = L * cs;
    info_off = static_cast<size_t>(nctx) * bf * 8;
    bytes = align_up(info_off + static_cast<size_t>(nctx) * 8, 16);
  }
};
__host__ __device__ inline size_t child_bytes(int N, int bf) {
  return align_up(static_cast<size_t>(N) * bf * 9, 16);  // uint64 keys + payload bytes
}
// Flat context id g (over live contexts only) -> (d, ci).
__device__ __forceinline__ void decode_ctx(int g, int k, int use_table, int& d, int& ci) {
  if (!use_table) {
    d = g;
    ci = 0;
  } else if (g == 0) {
    d = 0;
    ci = 0;
  } else if (g <= k) {
    d = 1;
    ci = g - 1;
  } else {
    const int r = g - 1 - k;
    d = 2 + r / (k * k);
    ci = r - (d - 2) * k * k;
  }
}
constexpr size_t kDynSmemBudget = 200 * 1024;
constexpr int kCluster = 8;
constexpr float kTieMargin = 4.8e-7f;  // 2^-21: fp32 sums closer than this may round equal

// Best-first pop loop of the leader CTA's warp 0 (see file header).
// SLOTS = frontier register slots per lane (ceil(N / 32), a power of two).
template <int SLOTS>
__device__ __forceinline__ int pop_loop(const Args& a, Smem& sm, const uint2* kids,
                                        const float2* info, uint64_t* chkey,
                                        unsigned char* chpay, int lane) {
  const int L = a.L, k = a.k, N = a.N, nb = a.bf;
  const int cs = a.use_table ? k * k : 1;
  uint64_t fk[SLOTS];
  uint32_t fp[SLOTS];
#pragma unroll
  for (int r = 0; r < SLOTS; ++r) {
    fk[r] = 0ull;
    fp[r] = 0u;
  }
  uint64_t best = 0ull;
  uint32_t best_pay = 0u;
  int best_slot = 0;
  // lane-local maximum over the slots, as a tree of independent comparisons
  auto rescan = [&]() {
    uint64_t kb[SLOTS];
    uint32_t pb[SLOTS];
    int sb[SLOTS];
#pragma unroll
    for (int r = 0; r < SLOTS; ++r) {
      kb[r] = fk[r];
      pb[r] = fp[r];
      sb[r] = r;
    }
#pragma unroll
    for (int w = 1; w < SLOTS; w *= 2)
#pragma unroll
      for (int r = 0; r + w < SLOTS; r += 2 * w)
        if (kb[r + w] > kb[r]) {
          kb[r] = kb[r + w];
          pb[r] = pb[r + w];
          sb[r] = sb[r + w];
        }
    best = kb[0];
    best_pay = pb[0];
    best_slot = sb[0];
  };
  auto set_slot = [&](int slot, uint64_t key, uint32_t pay) {
#pragma unroll
    for (int r = 0; r < SLOTS; ++r)
      if (r == slot) {
        fk[r] = key;
        fp[r] = pay;
      }
  };
  // Children of committed node n (depth d, score Sn, context ci of its children,
  // own candidate index jn): the kept candidates of depth d+1 in s order, stored by
  // key order (S desc, token asc) as n's child list.  Every lane gets the first
  // child's key and payload (child order | candidate index << 8 | jn << 16).
  auto expand = [&](int n, int d, float Sn, int ci, int jn, uint64_t& key0, uint32_t& pay0) {
    key0 = 0ull;
    pay0 = 0u;
    if (d >= L) return;
    const int c = d * cs + ci;
    const bool on = lane < nb;
    const uint2 kd = on ? kids[c * nb + lane] : make_uint2(0u, 0u);
    const float2 inf = info[c];
    const int j = static_cast<int>(kd.y & 0xFFu);
    const uint64_t key = on ? (static_cast<uint64_t>(ordered(__fadd_rn(Sn, __uint_as_float(kd.x))))
                               << 32) | (kd.y & ~0xFFu) | static_cast<uint32_t>(255 - n)
                            : 0ull;
    // In s order the fp32 path scores are non-increasing; siblings can leave key
    // order only if two of them round to the same S.  `safe` rules that out.
    const bool safe = inf.x > kTieMargin * (fabsf(Sn) + inf.y);
    int pos = lane, src = 0;
    if (!safe) {  // rank by key; equal keys (duplicate tokens) by lane
      pos = 0;
      for (int i = 0; i < nb; ++i) {
        const uint64_t ki = __shfl_sync(kFull, key, i);
        pos += ki > key || (ki == key && i < lane);
      }
      src = __ffs(__ballot_sync(kFull, on && pos == 0)) - 1;
    }
    if (on) {
      chkey[n * nb + pos] = key;
      chpay[n * nb + pos] = static_cast<unsigned char>(j);
    }
    key0 = __shfl_sync(kFull, key, src);
    pay0 = (static_cast<uint32_t>(__shfl_sync(kFull, j, src)) << 8) |
           (static_cast<uint32_t>(jn) << 16);
  };

  if (lane == 0) {
    sm.tok[0] = sm.ctx1;
    sm.par[0] = -1;
    sm.dep[0] = 0;
    sm.S[0] = 0.f;
  }
  {
    uint64_t k0;
    uint32_t p0;
    expand(0, 0, 0.f, 0, 0, k0, p0);
    if (lane == 0) {
      set_slot(0, k0, p0);
      rescan();
    }
  }
  __syncwarp();
  int n = 1;
  while (n < N) {
    const unsigned hi = static_cast<unsigned>(best >> 32), lo = static_cast<unsigned>(best);
    const unsigned mh = __reduce_max_sync(kFull, hi);
    if (mh == 0u) break;  // frontier empty
    const unsigned cand = __ballot_sync(kFull, hi == mh);
    int win;
    unsigned ml;
    if ((cand & (cand - 1u)) == 0u) {  // one lane holds the largest S (common case)
      win = __ffs(cand) - 1;
      ml = __shfl_sync(kFull, lo, win);
    } else {
      ml = __reduce_max_sync(kFull, hi == mh ? lo : 0u);
      win = __ffs(__ballot_sync(kFull, hi == mh && lo == ml)) - 1;
    }
    const uint32_t pay = __shfl_sync(kFull, best_pay, win);
    const float S = unordered(mh);
    const int d = 63 - static_cast<int>((ml >> 26) & 63u);
    const int t = 0x3FFFF - static_cast<int>((ml >> 8) & 0x3FFFFu);
    const int p = 255 - static_cast<int>(ml & 255u);
    const int c = static_cast<int>(pay & 0xFFu);
    const int j = static_cast<int>((pay >> 8) & 0xFFu);
    const int jp = static_cast<int>((pay >> 16) & 0xFFu);
    if (p >= n || d < 1 || d > L || j >= k || c >= nb) {  // cannot happen on valid input
      if (lane == 0) report(a.dev_status, PRESTO_DEV_BAD_PARENT);
      break;
    }
    // p's next child (every parent of a frontier entry has b children; the loads
    // are issued now and used after the expansion below)
    const int c2 = c + 1;
    const bool more = c2 < nb;
    const uint64_t nk = more ? chkey[p * nb + c2] : 0ull;
    const uint32_t np = more ? static_cast<uint32_t>(c2) |
                                   (static_cast<uint32_t>(chpay[p * nb + c2]) << 8) |
                                   (static_cast<uint32_t>(jp) << 16)
                             : 0u;
    if (lane == 0) {
      sm.tok[n] = t;
      sm.par[n] = p;
      sm.dep[n] = d;
      sm.S[n] = S;
    }
    // children of n see the context (t_{d-1}, t_d)
    const int ci = !a.use_table ? 0 : (d == 1 ? j : jp * k + j);
    uint64_t k0;
    uint32_t p0;
    expand(n, d, S, ci, j, k0, p0);
    // frontier update: p's entry moves on to its next child (lane win), n gets an
    // entry for its first child (lane n % 32)
    const bool upd_win = lane == win, upd_own = lane == (n & 31) && k0 != 0ull;
    if (upd_win || upd_own) {
      if (upd_win) set_slot(best_slot, nk, np);
      if (upd_own) set_slot(n >> 5, k0, p0);
      rescan();
    }
    ++n;
    __syncwarp();  // node arrays and child lists written above are read later
  }
  return n;
}

template <int SLOTS>
__global__ void __launch_bounds__(kThreads, 1) build_kernel(const Args a) {
  namespace cg = cooperative_groups;
  extern __shared__ __align__(16) unsigned char dyn[];
  __shared__ Smem sm;
  cg::cluster_group cluster = cg::this_cluster();
  const int rank = static_cast<int>(cluster.block_rank());
  const int b = blockIdx.x / kCluster;
  const int tid = threadIdx.x, lane = tid & 31;
  const int L = a.L, k = a.k, N = a.N, nb = a.bf, use_table = a.use_table;
  const TableLayout tl(L, k, nb, use_table);
  // leader's tables: in its shared memory (seen through DSMEM) or in the workspace
  const size_t cb = child_bytes(N, nb);
  unsigned char* tables;
  if (a.tables_in_smem)
    tables = static_cast<unsigned char*>(cluster.map_shared_rank(static_cast<void*>(dyn + cb), 0));
  else
    tables = a.g_tables + static_cast<size_t>(b) * tl.bytes;
  uint2* kids = reinterpret_cast<uint2*>(tables);
  float2* info = reinterpret_cast<float2*>(tables + tl.info_off);
  // this CTA's staging area: scores and order of its share of the contexts
  const size_t stage_off = cb + (a.tables_in_smem ? tl.bytes : 0);
  float* st_s = reinterpret_cast<float*>(dyn + stage_off);
  unsigned char* st_o = dyn + stage_off + static_cast<size_t>(a.per_cta) * k * 4;

  // ---- candidates and context
  for (int i = tid; i < L * k; i += kThreads) {
    const int d = i / k, j = i - d * k;
    int t = a.ids[(static_cast<size_t>(b) * L + d) * k + j];
    if (t < 0 || t >= kMaxV) {
      if (rank == 0) report(a.dev_status, PRESTO_DEV_BAD_TOKEN);
      t = 0;
    }
    sm.cid[d][j] = t;
    sm.clq[d][j] = a.logq[(static_cast<size_t>(b) * L + d) * k + j];
  }
  if (tid == 0) {
    sm.ctx0 = a.ctx2[2 * b];
    sm.ctx1 = a.ctx2[2 * b + 1];
    if (rank == 0 && (sm.ctx0 < 0 || sm.ctx0 >= kMaxV || sm.ctx1 < 0 || sm.ctx1 >= kMaxV))
      report(a.dev_status, PRESTO_DEV_BAD_TOKEN);
  }
  __syncthreads();
  if (rank == 0)
    for (int i = tid; i < L * k * k; i += kThreads) {  // sibling tokens must be distinct
      const int d = i / (k * k), r = i - d * k * k, j1 = r / k, j2 = r - j1 * k;
      if (j1 < j2 && sm.cid[d][j1] == sm.cid[d][j2]) report(a.dev_status, PRESTO_DEV_DUP_SIBLING);
    }

  // ---- phase 1: this CTA scores contexts [g0, g1) of the sequence
  const int g0 = rank * a.per_cta;
  const int g1 = min(a.nctx_all, g0 + a.per_cta);
  const int my = g1 > g0 ? (g1 - g0) * k : 0;
  constexpr int kBatch = 4;
  for (int f0 = tid; f0 < my; f0 += kThreads * kBatch) {
    uint64_t key[kBatch];
    uint32_t h[kBatch];
    float lq[kBatch];
#pragma unroll
    for (int q = 0; q < kBatch; ++q) {
      const int f = f0 + q * kThreads;
      key[q] = PRESTO_NGRAM3_EMPTY;
      h[q] = 0;
      lq[q] = 0.f;
      if (f >= my) continue;
      const int gl = f / k, j = f - gl * k;
      int d, ci;
      decode_ctx(g0 + gl, k, use_table, d, ci);
      lq[q] = sm.clq[d][j];
      if (!use_table) continue;
      int ta, tb;
      if (d == 0) {
        ta = sm.ctx0;
        tb = sm.ctx1;
      } else if (d == 1) {
        ta = sm.ctx1;
        tb = sm.cid[0][ci];
      } else {
        ta = sm.cid[d - 2][ci / k];
        tb = sm.cid[d - 1][ci % k];
      }
      key[q] = (static_cast<uint64_t>(ta & 0x3FFFF) << 36) |
               (static_cast<uint64_t>(tb & 0x3FFFF) << 18) |
               static_cast<uint64_t>(sm.cid[d][j] & 0x3FFFF);
      h[q] = static_cast<uint32_t>(fmix64(key[q])) & a.cap_mask;
    }
    uint64_t kv[kBatch];
    float vv[kBatch];
#pragma unroll
    for (int q = 0; q < kBatch; ++q) {
      const bool live = key[q] != PRESTO_NGRAM3_EMPTY;
      kv[q] = live ? __ldg(a.keys + h[q]) : PRESTO_NGRAM3_EMPTY;
      vv[q] = live ? __ldg(a.logrho + h[q]) : 0.f;
    }
#pragma unroll
    for (int q = 0; q < kBatch; ++q) {
      const int f = f0 + q * kThreads;
      if (f >= my) continue;
      float sc = lq[q];  // marginal-only: s = log q
      if (key[q] != PRESTO_NGRAM3_EMPTY) {
        float lr;
        if (kv[q] == key[q])
          lr = vv[q];
        else if (kv[q] == PRESTO_NGRAM3_EMPTY)
          lr = a.miss;
        else  // collision: continue the linear probe from the next slot
          lr = probe_from(a.keys, a.logrho, a.cap_mask, a.miss, key[q], (h[q] + 1) & a.cap_mask);
        sc = __fadd_rn(__fmul_rn(a.lambda, lr), lq[q]);
      }
      if (sc > 0.f) report(a.dev_status, PRESTO_DEV_POSITIVE_SCORE);
      st_s[f] = sc;
    }
  }
  __syncthreads();
  // rank of each candidate within its context, strict total order (float bits as
  // integers, then token, then index) so ranks form a permutation even for
  // duplicate tokens or NaN
  for (int f = tid; f < my; f += kThreads) {
    const int gl = f / k, j = f - gl * k;
    int d, ci;
    decode_ctx(g0 + gl, k, use_table, d, ci);
    const float* row = st_s + gl * k;
    const uint32_t sj = ordered(row[j]);
    const int tj = sm.cid[d][j];
    int rk = 0;
    for (int i = 0; i < k; ++i) {
      const uint32_t si = ordered(row[i]);
      const int ti = sm.cid[d][i];
      rk += (si > sj) || (si == sj && (ti < tj || (ti == tj && i < j)));
    }
    st_o[gl * k + rk] = static_cast<unsigned char>(j);
  }
  __syncthreads();
  // kept children of every context, in s order, into the leader's tables
  for (int f = tid; f < (g1 - g0) * nb; f += kThreads) {
    const int gl = f / nb, r = f - gl * nb;
    int d, ci;
    decode_ctx(g0 + gl, k, use_table, d, ci);
    const int j = st_o[gl * k + r];
    const uint32_t lowbits = (static_cast<uint32_t>(63 - (d + 1)) << 26) |
                             (static_cast<uint32_t>(0x3FFFF - sm.cid[d][j]) << 8) |
                             static_cast<uint32_t>(j);
    kids[(d * tl.cs + ci) * nb + r] = make_uint2(__float_as_uint(st_s[gl * k + j]), lowbits);
  }
  // per context: can fp32 rounding reorder two kept siblings?
  for (int gl = tid; gl < g1 - g0; gl += kThreads) {
    int d, ci;
    decode_ctx(g0 + gl, k, use_table, d, ci);
    float gap = INFINITY, mag = 0.f;
    for (int r = 0; r < nb; ++r) {
      const int jr = st_o[gl * k + r];
      const float sr = st_s[gl * k + jr];
      mag = fmaxf(mag, fabsf(sr));
      if (r + 1 < nb) {
        const int jn = st_o[gl * k + r + 1];
        if (sm.cid[d][jr] > sm.cid[d][jn]) gap = fminf(gap, sr - st_s[gl * k + jn]);
      }
    }
    if (!(mag < INFINITY)) gap = 0.f;  // non-finite scores: always rank by key
    info[d * tl.cs + ci] = make_float2(gap, mag);
  }
  if (!a.tables_in_smem) __threadfence();
  cluster.sync();  // the leader's tables are complete
  if (rank != 0 || tid >= 32) return;

  // ---- phase 2: best-first pop loop (leader, warp 0)
  uint64_t* chkey = reinterpret_cast<uint64_t*>(dyn);
  unsigned char* chpay = dyn + static_cast<size_t>(N) * nb * 8;
  int n;
  if (a.tables_in_smem)  // separate instance so the table loads are shared-memory loads
    n = pop_loop<SLOTS>(a, sm, reinterpret_cast<const uint2*>(dyn + cb),
                        reinterpret_cast<const float2*>(dyn + cb + tl.info_off), chkey, chpay,
                        lane);
  else
    n = pop_loop<SLOTS>(a, sm, kids, info, chkey, chpay, lane);
  // ---- write the tree
  for (int i = lane; i < N; i += 32) {
    const size_t o = static_cast<size_t>(b) * N + i;
    const bool used = i < n;
    a.node_token[o] = used ? sm.tok[i] : -1;
    a.node_parent[o] = used ? sm.par[i] : -1;
    a.node_depth[o] = used ? sm.dep[i] : -1;
    a.node_score[o] = used ? sm.S[i] : -INFINITY;
  }
  if (lane == 0) a.n_nodes[b] = n;
}

}  // namespace
}  // namespace presto

using namespace presto;

extern "C" int presto_ngram3_clear(const presto_ngram3* t, presto_stream_t stream) {
  PRESTO_CHECK_ARG(t && t->keys && t->logrho);
  PRESTO_CHECK_ARG(t->log2_cap >= 4 && t->log2_cap <= 30);
  const size_t cap = size_t{1} << t->log2_cap;
  if (cudaMemsetAsync(t->keys, 0xFF, cap * sizeof(uint64_t), stream) != cudaSuccess)
    return PRESTO_ERR_CUDA;
  return PRESTO_OK;
}

extern "C" int presto_ngram3_insert(const presto_ngram3* t, const uint64_t* keys,
                                    const float* logrho, int n, int32_t* dev_status,
                                    presto_stream_t stream) {
  PRESTO_CHECK_ARG(t && t->keys && t->logrho);
  PRESTO_CHECK_ARG(t->log2_cap >= 4 && t->log2_cap <= 30);
  PRESTO_CHECK_ARG(n >= 0);
  if (n == 0) return PRESTO_OK;
  PRESTO_CHECK_ARG(keys && logrho);
  const uint32_t mask = (1u << t->log2_cap) - 1u;
  ngram_insert_kernel<<<(n + 255) / 256, 256, 0, stream>>>(t->keys, t->logrho, mask, keys,
                                                            logrho, n, dev_status);
  return launch_status();
}

namespace {
size_t stage_bytes(int per_cta, int k) { return align_up(static_cast<size_t>(per_cta) * k * 5, 16); }
int contexts_all(int L, int k, int use_table) {
  if (!use_table) return L;
  return 1 + (L > 1 ? k : 0) + (L > 2 ? (L - 2) * k * k : 0);
}
}  // namespace

extern "C" size_t presto_build_workspace(int B, int L, int k, int N) {
  if (B < 1 || L < 1 || k < 1 || N < 1) return 0;
  // The leader CTA keeps the tables in shared memory when they fit; otherwise they
  // live here (sized for the prefix-signal case, the larger one).
  const TableLayout tl(L, k, k, 1);
  const int per = (contexts_all(L, k, 1) + kCluster - 1) / kCluster;
  const size_t smem = child_bytes(N, k) + tl.bytes + stage_bytes(per, k);
  return smem <= kDynSmemBudget ? 256 : align_up(B * tl.bytes, 256);
}

extern "C" int presto_score_build_tree(const int32_t* topk_ids, const float* topk_logq, int B,
                                       int L, int k, int b, const int32_t* ctx2,
                                       const presto_ngram3* ngram, float lambda, int N,
                                       int32_t* node_token, int32_t* node_parent,
                                       int32_t* node_depth, float* node_score,
                                       int32_t* n_nodes, void* ws, size_t ws_bytes,
                                       int32_t* dev_status, presto_stream_t stream) {
  PRESTO_CHECK_ARG(topk_ids && topk_logq && ctx2 && node_token && node_parent && node_depth &&
                   node_score && n_nodes);
  PRESTO_CHECK_ARG(B >= 1 && L >= 1 && k >= 1 && b >= 1 && N >= 1 && b <= k);
  PRESTO_CHECK_ARG(lambda >= 0.f && lambda == lambda);
  PRESTO_CHECK_LIMIT(L <= kMaxL && k <= kMaxK && N <= kMaxN);
  if (ngram) {
    PRESTO_CHECK_ARG(ngram->keys && ngram->logrho);
    PRESTO_CHECK_ARG(ngram->log2_cap >= 4 && ngram->log2_cap <= 30);
    PRESTO_CHECK_ARG(ngram->miss_logrho <= 0.f);
  }
  Args a{};
  a.ids = topk_ids;
  a.logq = topk_logq;
  a.ctx2 = ctx2;
  a.use_table = ngram != nullptr;
  if (ngram) {
    a.keys = ngram->keys;
    a.logrho = ngram->logrho;
    a.cap_mask = (1u << ngram->log2_cap) - 1u;
    a.miss = ngram->miss_logrho;
  }
  a.lambda = lambda;
  a.L = L;
  a.k = k;
  a.bf = b;
  a.N = N;
  a.nctx_all = contexts_all(L, k, a.use_table);
  a.per_cta = (a.nctx_all + kCluster - 1) / kCluster;
  const TableLayout tl(L, k, b, a.use_table);
  const size_t cb = child_bytes(N, b), sb = stage_bytes(a.per_cta, k);
  a.tables_in_smem = cb + tl.bytes + sb <= kDynSmemBudget;
  if (!a.tables_in_smem) {
    if (!ws || reinterpret_cast<uintptr_t>(ws) % 16 || ws_bytes < static_cast<size_t>(B) * tl.bytes)
      return PRESTO_ERR_WORKSPACE;
    a.g_tables = static_cast<unsigned char*>(ws);
  }
  a.node_token = node_token;
  a.node_parent = node_parent;
  a.node_depth = node_depth;
  a.node_score = node_score;
  a.n_nodes = n_nodes;
  a.dev_status = dev_status;
  const size_t smem = cb + (a.tables_in_smem ? tl.bytes : 0) + sb;
  if (smem > kDynSmemBudget) return PRESTO_ERR_UNSUPPORTED;
  void (*kernel)(Args);
  const int slots = (N + 31) / 32;
  kernel = slots <= 1 ? build_kernel<1> : slots <= 2 ? build_kernel<2>
         : slots <= 4 ? build_kernel<4> : build_kernel<8>;
  static bool attr_set = [] {
    for (auto fn : {build_kernel<1>, build_kernel<2>, build_kernel<4>, build_kernel<8>})
      cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(kDynSmemBudget));
    return true;
  }();
  (void)attr_set;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(static_cast<unsigned>(B) * kCluster);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = kCluster;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (cudaLaunchKernelEx(&cfg, kernel, a) != cudaSuccess) return PRESTO_ERR_CUDA;
  return launch_status();
}
