// presto_score_build_tree: prefix-aligned token scores (§4.1, Eq. path-score)
// and best-first tree construction (§4.2, Alg. 2; a node is committed when it is
// popped), plus the device-side trigram table (presto_ngram3_*).
//
// One CTA per sequence:
//   phase 1 (all 256 threads): the score table s[d][ctx][j] for every context pair
//     reachable in the candidate tree, d = 1..L, j over the k candidates of depth d
//     (hash-table probes, fully parallel), into shared memory.
//   phase 2 (warp 0): the pop loop.  Every frontier entry carries a 64-bit key that
//     packs the total order (S desc, depth asc, token asc, parent index asc), so
//     one warp-wide max reduction finds the next node.  A committed node pushes only
//     its best child, and a popped child pushes its next sibling, so the frontier
//     holds at most one entry per committed node (lazy sibling enumeration).
#include "common.cuh"

namespace presto {
namespace {

constexpr int kThreads = 512;
constexpr unsigned kFull = 0xffffffffu;
constexpr int kSlotsPerLane = 12;       // frontier capacity 384 >= N + 1 (see push)
constexpr size_t kMaxTableSmem = 160 * 1024;

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
  int table_in_smem;
  float* g_table;  // [B][L*k^3] when the table does not fit in shared memory
  int32_t* node_token;
  int32_t* node_parent;
  int32_t* node_depth;
  float* node_score;
  int32_t* n_nodes;
  int32_t* dev_status;
};

// Order-preserving map float -> uint32 (larger float -> larger integer).
__device__ __forceinline__ uint32_t ordered(float f) {
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ uint64_t make_key(float S, int depth, int token, int parent) {
  return (static_cast<uint64_t>(ordered(S)) << 32) |
         (static_cast<uint64_t>(63 - depth) << 26) |
         (static_cast<uint64_t>(0x3FFFF - token) << 8) | static_cast<uint64_t>(255 - parent);
}

struct Smem {
  // node arrays
  int tok[kMaxN];
  int par[kMaxN];
  int dep[kMaxN];
  int rank[kMaxN];      // candidate index j of the node within its depth's top-k
  int cix[kMaxN];       // context index of the node's children
  float S[kMaxN];
  unsigned char nch[kMaxN];
  unsigned char chj[kMaxN][kMaxK];   // children in key order (candidate indices)
  // frontier: slot-major so lane l owns fkey[*][l]
  unsigned long long fkey[kSlotsPerLane][32];
  unsigned fpay[kSlotsPerLane][32];
  // candidates of every depth
  int cid[kMaxL][kMaxK];
  float clq[kMaxL][kMaxK];
  int ctx0, ctx1;
  int n_committed;
};

// s for candidate j of depth d (1-based) under context index ci.
__device__ __forceinline__ float score_at(const Args& a, const Smem& sm, const float* table,
                                          int d, int ci, int j) {
  if (!a.use_table) return sm.clq[d - 1][j];
  const int k = a.k;
  return table[((static_cast<size_t>(d - 1) * k * k) + ci) * k + j];
}

__global__ void __launch_bounds__(kThreads) build_kernel(const Args a) {
  extern __shared__ __align__(16) unsigned char dyn[];
  __shared__ Smem sm;
  const int b = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31;
  const int L = a.L, k = a.k, N = a.N;
  const size_t tsize = static_cast<size_t>(L) * k * k * k;
  float* table = a.table_in_smem ? reinterpret_cast<float*>(dyn) : a.g_table + b * tsize;

  // ---- load candidates and context
  for (int i = tid; i < L * k; i += kThreads) {
    const int d = i / k, j = i % k;
    int t = a.ids[(static_cast<size_t>(b) * L + d) * k + j];
    if (t < 0 || t >= kMaxV) {
      report(a.dev_status, PRESTO_DEV_BAD_TOKEN);
      t = 0;
    }
    sm.cid[d][j] = t;
    sm.clq[d][j] = a.logq[(static_cast<size_t>(b) * L + d) * k + j];
  }
  if (tid == 0) {
    sm.ctx0 = a.ctx2[2 * b];
    sm.ctx1 = a.ctx2[2 * b + 1];
    if (sm.ctx0 < 0 || sm.ctx0 >= kMaxV || sm.ctx1 < 0 || sm.ctx1 >= kMaxV)
      report(a.dev_status, PRESTO_DEV_BAD_TOKEN);
  }
  __syncthreads();
  // duplicate tokens among one depth's candidates break sibling uniqueness
  for (int i = tid; i < L * k * k; i += kThreads) {
    const int d = i / (k * k), j1 = (i / k) % k, j2 = i % k;
    if (j1 < j2 && sm.cid[d][j1] == sm.cid[d][j2]) report(a.dev_status, PRESTO_DEV_DUP_SIBLING);
  }

  // ---- phase 1: score table s = fl(fl(lambda * log rho) + log q).
  // Each thread resolves kBatch probes at once so their first loads overlap.
  if (a.use_table) {
    constexpr int kBatch = 8;
    for (size_t e0 = tid; e0 < tsize; e0 += static_cast<size_t>(kThreads) * kBatch) {
      uint64_t key[kBatch];
      uint32_t h[kBatch];
      bool live[kBatch];
#pragma unroll
      for (int q = 0; q < kBatch; ++q) {
        const size_t e = e0 + static_cast<size_t>(q) * kThreads;
        live[q] = false;
        key[q] = 0;
        h[q] = 0;
        if (e >= tsize) continue;
        const int j = static_cast<int>(e % k);
        const int ci = static_cast<int>((e / k) % (k * k));
        const int d = static_cast<int>(e / (static_cast<size_t>(k) * k * k)) + 1;
        const int nctx = d == 1 ? 1 : (d == 2 ? k : k * k);
        if (ci >= nctx) continue;
        int ta, tb;
        if (d == 1) {
          ta = sm.ctx0;
          tb = sm.ctx1;
        } else if (d == 2) {
          ta = sm.ctx1;
          tb = sm.cid[0][ci];
        } else {
          ta = sm.cid[d - 3][ci / k];
          tb = sm.cid[d - 2][ci % k];
        }
        const int t = sm.cid[d - 1][j];
        key[q] = (static_cast<uint64_t>(ta & 0x3FFFF) << 36) |
                 (static_cast<uint64_t>(tb & 0x3FFFF) << 18) | static_cast<uint64_t>(t & 0x3FFFF);
        h[q] = static_cast<uint32_t>(fmix64(key[q])) & a.cap_mask;
        live[q] = true;
      }
      uint64_t kk[kBatch];
      float vv[kBatch];
#pragma unroll
      for (int q = 0; q < kBatch; ++q) {
        kk[q] = live[q] ? __ldg(a.keys + h[q]) : PRESTO_NGRAM3_EMPTY;
        vv[q] = live[q] ? __ldg(a.logrho + h[q]) : 0.f;
      }
#pragma unroll
      for (int q = 0; q < kBatch; ++q) {
        if (!live[q]) continue;
        float lr;
        if (kk[q] == key[q])
          lr = vv[q];
        else if (kk[q] == PRESTO_NGRAM3_EMPTY)
          lr = a.miss;
        else  // collision: continue the linear probe from the next slot
          lr = probe_from(a.keys, a.logrho, a.cap_mask, a.miss, key[q], (h[q] + 1) & a.cap_mask);
        const size_t e = e0 + static_cast<size_t>(q) * kThreads;
        const int j = static_cast<int>(e % k);
        const int d = static_cast<int>(e / (static_cast<size_t>(k) * k * k)) + 1;
        const float sc = __fadd_rn(__fmul_rn(a.lambda, lr), sm.clq[d - 1][j]);
        if (sc > 0.f) report(a.dev_status, PRESTO_DEV_POSITIVE_SCORE);
        table[e] = sc;
      }
    }
  } else {
    for (int i = tid; i < L * k; i += kThreads)
      if (sm.clq[i / k][i % k] > 0.f) report(a.dev_status, PRESTO_DEV_POSITIVE_SCORE);
  }
  if (!a.table_in_smem) __threadfence_block();
  __syncthreads();
  if (tid >= 32) return;

  // ---- phase 2: best-first pop loop (warp 0)
  // Per-lane frontier state: number of entries, best key and its slot.
  int cnt = 0;
  unsigned long long best = 0ull;
  int best_slot = -1;

  auto rescan = [&]() {
    best = 0ull;
    best_slot = -1;
    for (int s2 = 0; s2 < cnt; ++s2) {
      const unsigned long long kk = sm.fkey[s2][lane];
      if (kk > best) {
        best = kk;
        best_slot = s2;
      }
    }
  };
  // Push (key, payload) to the lane holding the fewest entries (warp-uniform call).
  auto push = [&](unsigned long long key, unsigned pay) {
    const unsigned sel = __reduce_min_sync(kFull, (static_cast<unsigned>(cnt) << 5) | lane);
    if (lane == static_cast<int>(sel & 31)) {
      if (cnt < kSlotsPerLane) {
        sm.fkey[cnt][lane] = key;
        sm.fpay[cnt][lane] = pay;
        if (key > best) {
          best = key;
          best_slot = cnt;
        }
        ++cnt;
      }
    }
  };
  // Children of committed node n (depth d < L): top-b of the k candidates of depth
  // d+1 by (s desc, token asc), stored in key order (S desc, token asc).
  auto expand = [&](int n) {
    const int d = sm.dep[n];
    if (d >= L) {
      if (lane == 0) sm.nch[n] = 0;
      __syncwarp();
      return;
    }
    const int ci = sm.cix[n];
    const bool on = lane < k;
    const float s = on ? score_at(a, sm, table, d + 1, ci, lane) : -INFINITY;
    const int t = on ? sm.cid[d][lane] : 0x7fffffff;
    const float Sc = __fadd_rn(sm.S[n], s);
    unsigned selmask = __ballot_sync(kFull, on);
    if (a.bf < k) {  // keep the top-b by (s desc, token asc)
      int rs = 0;
      for (int i = 0; i < k; ++i) {
        const float si = __shfl_sync(kFull, s, i);
        const int ti = __shfl_sync(kFull, t, i);
        rs += (si > s) || (si == s && ti < t);
      }
      selmask = __ballot_sync(kFull, on && rs < a.bf);
    }
    // order of the kept children by key: S desc, then token asc
    int rk = 0;
    for (int i = 0; i < k; ++i) {
      const float Si = __shfl_sync(kFull, Sc, i);
      const int ti = __shfl_sync(kFull, t, i);
      rk += ((selmask >> i) & 1u) && ((Si > Sc) || (Si == Sc && ti < t));
    }
    if ((selmask >> lane) & 1u) sm.chj[n][rk] = static_cast<unsigned char>(lane);
    const int nsel = __popc(selmask);
    if (lane == 0) sm.nch[n] = static_cast<unsigned char>(nsel);
    __syncwarp();
    if (nsel > 0) {
      const int j0 = sm.chj[n][0];
      const float S0 = __fadd_rn(sm.S[n], score_at(a, sm, table, d + 1, ci, j0));
      push(make_key(S0, d + 1, sm.cid[d][j0], n), static_cast<unsigned>(n) << 8);
    }
  };

  if (lane == 0) {
    sm.tok[0] = sm.ctx1;
    sm.par[0] = -1;
    sm.dep[0] = 0;
    sm.rank[0] = -1;
    sm.cix[0] = 0;
    sm.S[0] = 0.f;
  }
  __syncwarp();
  expand(0);
  int n = 1;
  while (n < N) {
    const unsigned hi = static_cast<unsigned>(best >> 32), lo = static_cast<unsigned>(best);
    const unsigned mh = __reduce_max_sync(kFull, hi);
    const unsigned ml = __reduce_max_sync(kFull, hi == mh ? lo : 0u);
    if (mh == 0u) break;  // frontier empty (real keys have hi >= 0x007fffff)
    const int win = __ffs(__ballot_sync(kFull, hi == mh && lo == ml)) - 1;
    const unsigned pay = __shfl_sync(kFull, best_slot >= 0 ? sm.fpay[best_slot][lane] : 0u, win);
    if (lane == win) {  // remove the entry: move the lane's last entry into its slot
      --cnt;
      if (best_slot != cnt) {
        sm.fkey[best_slot][lane] = sm.fkey[cnt][lane];
        sm.fpay[best_slot][lane] = sm.fpay[cnt][lane];
      }
      rescan();
    }
    const int p = static_cast<int>(pay >> 8), c = static_cast<int>(pay & 0xFF);
    const int d = sm.dep[p] + 1;
    const int j = sm.chj[p][c];
    const int pci = sm.cix[p];
    const float s = score_at(a, sm, table, d, pci, j);
    const float Sn = __fadd_rn(sm.S[p], s);
    if (lane == 0) {
      sm.tok[n] = sm.cid[d - 1][j];
      sm.par[n] = p;
      sm.dep[n] = d;
      sm.rank[n] = j;
      sm.S[n] = Sn;
      // children of n (depth d+1) see context (t_{d-1}, t_d)
      sm.cix[n] = d == 1 ? j : sm.rank[p] * k + j;
    }
    __syncwarp();
    // next sibling of n under p
    if (c + 1 < sm.nch[p]) {
      const int j2 = sm.chj[p][c + 1];
      const float S2 = __fadd_rn(sm.S[p], score_at(a, sm, table, d, pci, j2));
      push(make_key(S2, d, sm.cid[d - 1][j2], p), (static_cast<unsigned>(p) << 8) | (c + 1));
    }
    expand(n);
    ++n;
  }
  __syncwarp();
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
size_t table_bytes(int L, int k) { return static_cast<size_t>(L) * k * k * k * sizeof(float); }
}  // namespace

extern "C" size_t presto_build_workspace(int B, int L, int k, int N) {
  (void)N;
  if (B < 1 || L < 1 || k < 1) return 0;
  // The score table lives in shared memory when it fits; otherwise here.
  return table_bytes(L, k) <= kMaxTableSmem ? 256 : align_up(B * table_bytes(L, k), 256);
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
  const size_t tb = table_bytes(L, k);
  a.table_in_smem = !a.use_table || tb <= kMaxTableSmem;
  if (a.use_table && !a.table_in_smem) {
    if (!ws || ws_bytes < static_cast<size_t>(B) * tb) return PRESTO_ERR_WORKSPACE;
    a.g_table = static_cast<float*>(ws);
  }
  a.node_token = node_token;
  a.node_parent = node_parent;
  a.node_depth = node_depth;
  a.node_score = node_score;
  a.n_nodes = n_nodes;
  a.dev_status = dev_status;
  const size_t smem = (a.use_table && a.table_in_smem) ? tb : 0;
  static bool attr_set = [] {
    cudaFuncSetAttribute(build_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         static_cast<int>(kMaxTableSmem));
    return true;
  }();
  (void)attr_set;
  build_kernel<<<B, kThreads, smem, stream>>>(a);
  return launch_status();
}
