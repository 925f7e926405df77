// presto_score_build_tree: prefix-aligned token scores (§4.1, Eq. path-score)
// and best-first tree construction (§4.2, Alg. 2; a node is committed when it is
// popped), plus the device-side trigram table (presto_ngram3_*).
//
// One thread-block cluster per sequence: 16 CTAs when every cluster of the launch fits
// on the device at once, else 8 (the trigram probes of phase 1 are bound by the
// issue of their scattered loads, one L1 wavefront per lane, so they spread over as
// many SMs as the launch can hold):
//   phase 1 (all CTAs): each CTA takes a share of the context pairs reachable in
//     the candidate tree and computes, for every candidate j of depth d+1 under
//     that context, s = log q + lambda log rho (hash-table probes, batched so their
//     loads overlap), keeps the top-b by (s desc, token asc) as 8-byte records that
//     already hold the child's key bits, and writes them into the leader CTA's
//     shared memory (distributed shared memory); the cluster then synchronises once.
//   phase 2 (leader CTA): the nodes the best-first loop commits are the N - 1
//     largest keys of the candidate tree (key = S desc, depth asc, token asc, parent
//     index asc, packed into 64 bits), because a child's key is always below its
//     parent's.  They are found level by level with the whole CTA: the N - 1
//     largest keys among nodes of depth <= d are kept sorted; the children of the
//     newest level that beat the smallest kept key are ranked against them.  L
//     block-wide steps replace N - 1 dependent pops, with the same nodes in the
//     same order.
#include <cooperative_groups.h>

#include <initializer_list>
#include <mutex>

#include "common.cuh"

namespace presto {
namespace {

constexpr int kThreads = 512;

__host__ __device__ inline uint64_t fmix64(uint64_t k) {
  // MurmurHash3 64-bit finaliser (Appleby, public domain).
  k ^= k >> 33;
  k *= 0xff51afd7ed558ccdull;
  k ^= k >> 33;
  k *= 0xc4ceb9fe1a85ec53ull;
  k ^= k >> 33;
  return k;
}

// Loads of the trigram table with an L2 evict-last policy: the table is model state that
// every round probes, while the round's logits and KV cache stream through L2 once, so
// its recently probed slots should outlive them there.  A cache policy is a hint.
__device__ __forceinline__ uint64_t l2_keep_policy() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_last.L2::evict_unchanged.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}
__device__ __forceinline__ uint64_t ld_table(const uint64_t* p, uint64_t pol) {
  uint64_t v;
  asm volatile("ld.global.nc.L2::cache_hint.u64 %0, [%1], %2;" : "=l"(v) : "l"(p), "l"(pol));
  return v;
}
__device__ __forceinline__ float ld_table(const float* p, uint64_t pol) {
  float v;
  asm volatile("ld.global.nc.L2::cache_hint.f32 %0, [%1], %2;" : "=f"(v) : "l"(p), "l"(pol));
  return v;
}

// Linear probe for `key` starting at slot h.
__device__ __noinline__ float probe_from(const uint64_t* keys, const float* logrho,
                                         uint32_t mask, float miss, uint64_t key, uint32_t h) {
  const uint64_t pol = l2_keep_policy();
  for (uint32_t it = 0; it <= mask; ++it) {
    const uint64_t kk = ld_table(keys + h, pol);
    if (kk == key) return ld_table(logrho + h, pol);
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
  const float* lambda_d;  // [B, L] per-row lambda, or null (use `lambda`)
  int policy, W;          // PRESTO_SEARCH_*, beam width
  int use_table;
  int L, k, bf, N;
  int nctx_all;      // contexts of one sequence over all depths
  int csize;         // CTAs of a sequence's cluster
  int per_cta;       // contexts each CTA of the cluster scores
  int tables_in_smem;
  unsigned char* g_tables;  // [B][tables_bytes] when the tables do not fit in smem
  int p2_in_smem;
  unsigned char* g_p2;      // [B][p2_stride] when the selection scratch does not
  size_t tables_stride, p2_stride;  // workspace bytes per sequence
  int32_t* node_token;
  int32_t* node_parent;
  int32_t* node_depth;
  float* node_score;
  int32_t* n_nodes;
  const int32_t* kv_len;  // fused mask (nullable together with mask, pos_ids)
  uint32_t* mask;         // [B][N][ceil(N / 32)]
  int32_t* pos_ids;       // [B][N]
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

struct Smem {
  int cid[kMaxL][kMaxK];          // candidate tokens of every depth
  int trk[kMaxL][kMaxK];          // their ranks by token id within the depth
  int rtok[kMaxL][kMaxK];         // the token of each rank
  float clq[kMaxL][kMaxK];        // their log q
  int ctx0, ctx1;
  float lam[kMaxL];               // lambda of every drafter row
  int nc[2];                      // candidates of a level (phase 2, double-buffered)
  unsigned long long tau;         // the smallest key of a full A (phase 2)
  int16_t par[kMaxN];             // the output tree's parents (for the fused mask)
};

// Tables of one sequence, indexed by context c = d * ctx_stride + ci (d = depth of
// the children - 1, ci = context pair index):
//   kid  uint2[c][b]  the top-b candidates of the context by (s desc, token asc),
//                     in no particular order: x = bits of s, y = the key bits of
//                     (depth d+1, token) with the candidate index in the low byte
//                     (the parent field of the key, filled in when the child is
//                     generated)
// With a prefix signal ctx_stride = k*k (contexts (t_{d-1}, t_d) as index pairs);
// marginal-only scoring has one context per depth.
struct TableLayout {
  int cs, nctx;
  size_t bytes;
  __host__ __device__ TableLayout(int L, int k, int bf, int use_table) {
    cs = use_table ? k * k : 1;
    nctx = L * cs;
    bytes = align_up(static_cast<size_t>(nctx) * bf * 8, 16);
  }
};
// Low word of a node key: 63 - depth (6 bits), 15 - the token's rank among its
// depth's k candidates by token id (4 bits: all nodes of one depth draw their tokens
// from the same k candidates, so for equal S and depth this orders by token id), then
// kPMask - the parent field (22 bits).  In a child record the low field holds the
// candidate index j instead.
constexpr uint32_t kPMask = 0x3FFFFFu;
constexpr int kTRankShift = 22;
// Child record of candidate j (token rank tr) of depth d+1 under some context, score s.
__device__ __forceinline__ uint2 kid_record(float s, int d, int tr, int j) {
  return make_uint2(__float_as_uint(s), (static_cast<uint32_t>(63 - (d + 1)) << 26) |
                                            (static_cast<uint32_t>(15 - tr) << kTRankShift) |
                                            static_cast<uint32_t>(j));
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
constexpr int kCluster = 8;       // CTAs of a sequence's cluster (portable size) ...
constexpr int kClusterWide = 16;  // ... or, when every cluster of a launch fits at once, this

// Phase-2 scratch of the leader CTA (aliases the phase-1 staging area).  The kept
// set A (non-root nodes, sorted by key, so A[r] is node r + 1) and the candidate
// set C of a level are double-buffered.  Per entry: key, the index of its own children's
// context (kNoCtx at depth L), its candidate index j, and its parent's node index.
struct P2Layout {
  size_t akey, axc, apid, aj, ckey, cxc, cpid, cj, rk, rkc, skey, sidx, bytes;
  int nc;  // capacity of one candidate buffer: every child of max(N, W) parents
  int np;  // the sort buffer: the power of two >= nc
  __host__ __device__ P2Layout(int N, int bf, int W) {
    const size_t na = N;
    nc = (N > W ? N : W) * bf;
    np = 1;
    while (np < nc) np <<= 1;
    size_t o = 0;
    akey = o;  o += 2 * na * 8;
    ckey = o;  o += 2 * static_cast<size_t>(nc) * 8;
    axc = o;   o += 2 * na * 4;
    cxc = o;   o += 2 * static_cast<size_t>(nc) * 4;
    apid = o;  o += align_up(2 * na * 2, 4);
    cpid = o;  o += align_up(2 * static_cast<size_t>(nc) * 2, 4);
    rk = o;    o += align_up((na + nc) * 2, 4);
    rkc = o;   o += align_up(static_cast<size_t>(nc) * 2, 4);
    aj = o;    o += align_up(2 * na, 4);
    cj = o;    o += align_up(2 * static_cast<size_t>(nc), 8);
    skey = o;  o += static_cast<size_t>(np) * 8;
    sidx = o;  o += static_cast<size_t>(np) * 2;
    bytes = align_up(o, 16);
  }
};
constexpr uint32_t kNoCtx = 0xFFFFFFFFu;
constexpr int kSortMin = 256;  // candidates of a level above which they are sorted first
static_assert(kSortMin < (1 << 16) && kMaxN < (1 << 15), "two counts share one int in the ranking");

// Top-N selection of the candidate tree, level by level (leader CTA, all threads).
//
// Best-first expansion with lazy commits pops nodes in decreasing key order (a
// child's key is below its parent's: S does not grow along a path and ties go to
// the shallower node), so its N - 1 committed nodes are the N - 1 largest keys of
// the whole tree.  After step d, A holds the N - 1 largest keys among nodes of
// depth <= d.  Step d + 1 only needs the children of A's depth-d nodes: any node
// of depth d + 1 among the N - 1 largest of depth <= d + 1 has its parent among the
// N - 1 largest of depth <= d, and its key exceeds tau, the smallest key of a full
// A.  The candidates that pass are ranked against A and the N - 1 largest kept.
// A node's final index is its rank, so the parent index in the key (the last tie
// break) is the parent's rank in A, consistent across steps.
// Returns the node count (root included).
__device__ __forceinline__ int select_levels(const Args& a, Smem& sm, const uint2* kids,
                                             unsigned char* p2,
                             int tid) {
  const int L = a.L, k = a.k, N = a.N, nb = a.bf, W = a.W;
  const bool beam = a.policy == PRESTO_SEARCH_BEAM;
  const int cs = a.use_table ? k * k : 1;
  const int cap = N - 1;  // non-root nodes
  const int lane = tid & 31;
  const P2Layout ly(N, nb, W);
  const int NC = ly.nc;
  // buffer u of each A field starts at u * N, of each C field at u * NC
  uint64_t* const akey = reinterpret_cast<uint64_t*>(p2 + ly.akey);
  uint32_t* const axc = reinterpret_cast<uint32_t*>(p2 + ly.axc);
  int16_t* const apid = reinterpret_cast<int16_t*>(p2 + ly.apid);
  uint8_t* const aj = p2 + ly.aj;
  uint64_t* const ckey = reinterpret_cast<uint64_t*>(p2 + ly.ckey);
  uint32_t* const cxc = reinterpret_cast<uint32_t*>(p2 + ly.cxc);
  int16_t* const cpid = reinterpret_cast<int16_t*>(p2 + ly.cpid);
  uint8_t* const cj = p2 + ly.cj;
  int16_t* const rk = reinterpret_cast<int16_t*>(p2 + ly.rk);
  int16_t* const rkc = reinterpret_cast<int16_t*>(p2 + ly.rkc);
  uint64_t* const skey = reinterpret_cast<uint64_t*>(p2 + ly.skey);
  int16_t* const sidx = reinterpret_cast<int16_t*>(p2 + ly.sidx);

  // Child c of a node with score Sp, children context x and candidate index pj, at
  // depth dc; `pfield` fills the key's last field (kPMask - the parent's position among
  // the parents of its level).  Returns the key, context and candidate index.
  const int nkid = L * cs * nb;  // child records in the tables
  auto child = [&](uint32_t x, float Sp, int pj, int pfield, int dc, int c, uint64_t& key,
                   uint32_t& xc, int& jc) {
    const int ik = static_cast<int>(x) * nb + c;
    const uint2 kd = PRESTO_IN_BOUNDS(ik, nkid, a.dev_status) ? kids[ik] : make_uint2(0u, 0u);
    key = (static_cast<uint64_t>(ordered(__fadd_rn(Sp, __uint_as_float(kd.x)))) << 32) |
          (kd.y & ~kPMask) | (kPMask - static_cast<uint32_t>(pfield));
    jc = static_cast<int>(kd.y & kPMask);
    xc = dc >= L ? kNoCtx
                 : static_cast<uint32_t>(dc * cs + (!a.use_table ? 0 : (dc == 1 ? jc : pj * k + jc)));
  };
  // Reserve `keep`-many candidate slots of buffer u, one atomic per warp (all lanes).
  auto reserve = [&](bool keep, int u) {
    const unsigned bal = __ballot_sync(0xffffffffu, keep);
    int base = 0;
    if (lane == 0 && bal) base = atomicAdd(&sm.nc[u], __popc(bal));
    return __shfl_sync(0xffffffffu, base, 0) + __popc(bal & ((1u << lane) - 1u));
  };

  // level 1: the root's children (A is empty, so every one is a candidate)
  if (cap > 0 && tid < nb) {
    uint64_t key;
    uint32_t xc;
    int jc;
    child(0u, 0.f, 0, 0, 1, tid, key, xc, jc);
    ckey[tid] = key;
    cxc[tid] = xc;
    cpid[tid] = 0;
    cj[tid] = static_cast<uint8_t>(jc);
  }
  if (tid == 0) sm.nc[1] = 0;
  __syncthreads();
  int na = 0, m = cap > 0 ? nb : 0, cur = 0, cc = 0;
  int tsize = 1 + m;    // |T|, root included (beam search stops once it reaches N)
  uint64_t tau = 0ull;  // the smallest key of A once A is full (0: not yet full)
  for (int step = 0; m > 0; ++step) {
    // ---- ranks in A u C by (key desc, position asc); A is sorted.  rkc: the rank of
    // a candidate among the candidates alone (beam search keeps the W best)
    const uint64_t* C = ckey + cc * NC;
    const int ne = na + m;
    if (m > kSortMin) {
      // many candidates: sort them once (bitonic, descending; keys are unique and
      // nonzero, zeros pad to a power of two) and take every rank by binary search
      int P = 1;
      while (P < m) P <<= 1;
      for (int i = tid; i < P; i += kThreads) {
        skey[i] = i < m ? C[i] : 0ull;
        sidx[i] = static_cast<int16_t>(i);
      }
      __syncthreads();
      for (int size = 2; size <= P; size <<= 1) {
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
          for (int t = tid; t < P / 2; t += kThreads) {
            const int i = 2 * t - (t & (stride - 1)), l = i + stride;
            const uint64_t ki = skey[i], kl = skey[l];
            const bool desc = (i & size) == 0;  // this block's direction
            if (desc ? ki < kl : ki > kl) {
              skey[i] = kl;
              skey[l] = ki;
              const int16_t x = sidx[i];
              sidx[i] = sidx[l];
              sidx[l] = x;
            }
          }
          __syncthreads();
        }
      }
      for (int q = tid; q < m; q += kThreads) rkc[sidx[q]] = static_cast<int16_t>(q);
      __syncthreads();
      for (int e = tid; e < ne; e += kThreads) {
        int r;
        if (e < na) {
          const uint64_t ke = akey[cur * N + e];
          int lo = 0, hi = m;  // sorted candidates with key > ke
          while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (skey[mid] > ke) lo = mid + 1;
            else hi = mid;
          }
          r = e + lo;
        } else {
          const int ci = e - na;
          const uint64_t ke = C[ci];
          int lo = 0, hi = na;  // A entries with key >= ke
          while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (akey[cur * N + mid] >= ke) lo = mid + 1;
            else hi = mid;
          }
          r = lo + rkc[ci];
        }
        rk[e] = static_cast<int16_t>(r < cap ? r : cap);
        if (r == cap - 1) sm.tau = e < na ? akey[cur * N + e] : C[e - na];  // the new A's last key
      }
    } else {
      // each entry's count of candidates above it is split over a group of G lanes
      // (candidates g, g + G, ...; G a power of two, as many as the block holds) and
      // summed across the group, so no thread runs a chain of m compares
      int G = 1;
      while (G < 32 && ne * (2 * G) <= kThreads) G *= 2;
      const int total = ne * G;
      for (int base = tid & ~31; base < total; base += kThreads) {  // warp-uniform
        const int idx = base + lane;
        const bool act = idx < total;
        const int e = idx / G, g = idx & (G - 1);
        uint64_t ke = 0ull;
        int ci = -1;  // a candidate's own index (ties to the lower index); -1 for A entries
        if (act) {
          if (e < na) {
            ke = akey[cur * N + e];
          } else {
            ci = e - na;
            ke = C[ci];
          }
        }
        // low half: candidates above the entry; high half (candidates only): entries of
        // A with key >= ke, i.e. the candidate's position in the sorted A
        int cnt = 0;
        if (act) {
          for (int i = g; i < m; i += G) {
            const uint64_t ki = C[i];
            cnt += ki > ke || (ki == ke && i < ci);
          }
          if (ci >= 0)
            for (int i = g; i < na; i += G) cnt += (akey[cur * N + i] >= ke) << 16;
        }
        for (int off = G >> 1; off > 0; off >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, off);
        if (act && g == 0) {
          int r;
          const int rc = cnt & 0xFFFF;
          if (e < na) {
            r = e + rc;
          } else {
            rkc[ci] = static_cast<int16_t>(rc);
            r = (cnt >> 16) + rc;
          }
          rk[e] = static_cast<int16_t>(r < cap ? r : cap);
          if (r == cap - 1) sm.tau = ke;  // the new A's last key
        }
      }
    }
    if (tid == 0) sm.nc[cc ^ 1] = 0;  // the next level's counter (last read a level ago)
    __syncthreads();
    if (ne >= cap) tau = sm.tau;  // the new A is full: its smallest key
    // ---- the cap largest become the new A (parent indices follow their ranks), and
    // the next level's candidates are generated:
    //   best-first: children of the new nodes that entered A, with key > tau;
    //   beam: children of the W best candidates (the beam), all of them, while |T| < N
    const int nxt = cur ^ 1, cn = cc ^ 1;
    for (int e = tid; e < ne; e += kThreads) {
      const int r = rk[e];
      if (r >= cap) continue;
      int pid;
      if (e < na) {
        akey[nxt * N + r] = akey[cur * N + e];
        axc[nxt * N + r] = axc[cur * N + e];
        aj[nxt * N + r] = aj[cur * N + e];
        pid = apid[cur * N + e];
      } else {
        akey[nxt * N + r] = C[e - na];
        axc[nxt * N + r] = cxc[cc * NC + e - na];
        aj[nxt * N + r] = cj[cc * NC + e - na];
        pid = cpid[cc * NC + e - na];
      }
      if (pid > 0) {
        const int pr = rk[pid - 1];
        if (pr >= cap || pr >= r) report(a.dev_status, PRESTO_DEV_BAD_PARENT);  // s > 0 input
        pid = pr < cap ? pr + 1 : 0;
      } else if (pid < 0) {  // a parent outside A: cannot happen when every s <= 0
        report(a.dev_status, PRESTO_DEV_BAD_PARENT);
        pid = 0;
      }
      apid[nxt * N + r] = static_cast<int16_t>(pid);
    }
    const bool grow = !beam || tsize < N;  // warp-uniform
    const int pairs = grow ? m * nb : 0;
    const int iters = (pairs + kThreads - 1) / kThreads;  // uniform, for the warp scans
    for (int it = 0; it < iters; ++it) {
      const int q = it * kThreads + tid;
      const int ci = q / nb, c = q - ci * nb;
      const int r = q < pairs ? rk[na + ci] : cap;
      const int rc = q < pairs ? rkc[ci] : W;
      const bool parent = beam ? rc < W : r < cap;
      const uint32_t xe = parent ? cxc[cc * NC + ci] : kNoCtx;
      uint64_t key = 0ull;
      uint32_t xc = kNoCtx;
      int jc = 0;
      if (xe != kNoCtx) {  // a parent below depth L
        const uint64_t ke = C[ci];
        const int dc = 64 - static_cast<int>((ke >> 26) & 63u);  // the children's depth
        child(xe, unordered(static_cast<uint32_t>(ke >> 32)), cj[cc * NC + ci],
              beam ? rc : r + 1, dc, c, key, xc, jc);
      }
      const bool keep = key != 0ull && (beam || key > tau);
      const int slot = reserve(keep, cn);
      if (keep && PRESTO_IN_BOUNDS(slot, NC, a.dev_status)) {
        ckey[cn * NC + slot] = key;
        cxc[cn * NC + slot] = xc;
        cpid[cn * NC + slot] = static_cast<int16_t>(r < cap ? r + 1 : -1);
        cj[cn * NC + slot] = static_cast<uint8_t>(jc);
      }
    }
    na = ne < cap ? ne : cap;
    cur = nxt;
    cc = cn;
    __syncthreads();
    m = sm.nc[cc];
    tsize += m;
  }

  // ---- Alg. 2 as printed: the nodes are expanded in the lazy order above (node 0
  // the root, node r + 1 = A[r]) until |T| = 1 + (their children) reaches N; the
  // output is those X nodes, then the best of their children not expanded
  int head = na + 1, ntail = 0;  // rows from A (root included), rows from the tail
  if (a.policy == PRESTO_SEARCH_EAGER) {
    __syncthreads();  // every thread has read the loop's last counter
    if (tid == 0) {
      int cnt = 1, x = 0;
      while (cnt < N && x <= na) {
        const int d = x == 0 ? 0 : 63 - static_cast<int>((akey[cur * N + x - 1] >> 26) & 63u);
        cnt += d < L ? nb : 0;
        ++x;
      }
      sm.nc[0] = x;
      sm.nc[1] = 0;
    }
    __syncthreads();
    const int X = sm.nc[0];
    // X = 0 (N = 1): nothing expanded, the root alone; X > na: the whole tree
    if (X >= 1 && X <= na) {
      head = X;
      // the children of nodes 0 .. X-1 that are not among nodes 1 .. X-1
      const int pairs = X * nb;
      const int iters = (pairs + kThreads - 1) / kThreads;
      uint64_t* const F = ckey + cc * NC;  // the last level's buffer is free now
      for (int it = 0; it < iters; ++it) {
        const int q = it * kThreads + tid;
        const int i = q / nb, c = q - i * nb;
        uint64_t key = 0ull;
        uint32_t xc = kNoCtx;
        int jc = 0;
        if (q < pairs) {
          uint64_t ke = 0ull;
          uint32_t x = 0u;
          int pj = 0, d = 0;
          if (i > 0) {
            ke = akey[cur * N + i - 1];
            x = axc[cur * N + i - 1];
            pj = aj[cur * N + i - 1];
            d = 63 - static_cast<int>((ke >> 26) & 63u);
          }
          if (d < L) {
            child(x, i == 0 ? 0.f : unordered(static_cast<uint32_t>(ke >> 32)), pj, i, d + 1, c,
                  key, xc, jc);
            // expanded already: one of A[0 .. X-2], the same (S, depth, token) under the
            // same parent (A's last key field dates from its own level, so compare
            // the node's parent instead)
            int lo = 0, hi = X - 1;
            while (lo < hi) {
              const int mid = (lo + hi) >> 1;
              if ((akey[cur * N + mid] >> kTRankShift) > (key >> kTRankShift)) lo = mid + 1;
              else hi = mid;
            }
            for (; lo < X - 1 && (akey[cur * N + lo] >> kTRankShift) == (key >> kTRankShift); ++lo)
              if (apid[cur * N + lo] == i) key = 0ull;
          }
        }
        const bool keep = key != 0ull;
        const int slot = reserve(keep, 1);
        if (keep && PRESTO_IN_BOUNDS(slot, NC, a.dev_status)) {
          F[slot] = key;
          cpid[cc * NC + slot] = static_cast<int16_t>(i);
        }
      }
      __syncthreads();
      const int nf = sm.nc[1];
      ntail = nf < N - X ? nf : N - X;
      for (int e = tid; e < nf; e += kThreads) {
        const uint64_t ke = F[e];
        int r = 0;
        for (int i2 = 0; i2 < nf; ++i2) r += F[i2] > ke || (F[i2] == ke && i2 < e);
        rk[e] = static_cast<int16_t>(r);
      }
      __syncthreads();
      // the tail rows, in rank order, into A's buffer beyond the head
      for (int e = tid; e < nf; e += kThreads) {
        const int r = rk[e];
        if (r >= ntail) continue;
        akey[(cur ^ 1) * N + r] = F[e];
        apid[(cur ^ 1) * N + r] = cpid[cc * NC + e];
      }
      __syncthreads();
    }
  }

  // ---- write the tree: node 0 is the root, node r + 1 is A[r] for r + 1 < head, then
  // the tail rows
  for (int i = tid; i < N; i += kThreads) {
    const size_t o = static_cast<size_t>(blockIdx.x / a.csize) * N + i;
    uint64_t ke = 0ull;
    int pid = -1;
    if (i > 0 && i < head) {
      ke = akey[cur * N + i - 1];
      pid = apid[cur * N + i - 1];
    } else if (i >= head && i < head + ntail) {
      ke = akey[(cur ^ 1) * N + i - head];
      pid = apid[(cur ^ 1) * N + i - head];
    }
    sm.par[i] = static_cast<int16_t>(i == 0 || ke == 0ull ? -1 : pid);
    if (i == 0) {
      a.node_token[o] = sm.ctx1;
      a.node_parent[o] = -1;
      a.node_depth[o] = 0;
      a.node_score[o] = 0.f;
    } else if (ke != 0ull) {
      const uint32_t lo = static_cast<uint32_t>(ke);
      const int dd = 63 - static_cast<int>((lo >> 26) & 63u);
      const int tr = 15 - static_cast<int>((lo >> kTRankShift) & 15u);
      a.node_token[o] = PRESTO_IN_BOUNDS(dd - 1, L, a.dev_status) && PRESTO_IN_BOUNDS(tr, k, a.dev_status)
                            ? sm.rtok[dd - 1][tr]
                            : -1;
      a.node_depth[o] = dd;
      a.node_parent[o] = pid;
      a.node_score[o] = unordered(static_cast<uint32_t>(ke >> 32));
    } else {
      a.node_token[o] = -1;
      a.node_parent[o] = -1;
      a.node_depth[o] = -1;
      a.node_score[o] = -INFINITY;
    }
  }
  return head + ntail;
}

__global__ void __launch_bounds__(kThreads, 1) build_kernel(const Args a) {
  namespace cg = cooperative_groups;
  pdl_launch_dependents();
  extern __shared__ __align__(16) unsigned char dyn[];
  __shared__ Smem sm;
  cg::cluster_group cluster = cg::this_cluster();
  const int rank = static_cast<int>(cluster.block_rank());
  const int b = blockIdx.x / a.csize;
  const int tid = threadIdx.x;
  const int L = a.L, k = a.k, nb = a.bf, use_table = a.use_table;
  const TableLayout tl(L, k, nb, use_table);
  // leader's tables: in its shared memory (seen through DSMEM) or in the workspace
  unsigned char* tables;
  if (a.tables_in_smem)
    tables = static_cast<unsigned char*>(cluster.map_shared_rank(static_cast<void*>(dyn), 0));
  else
    tables = a.g_tables + static_cast<size_t>(b) * a.tables_stride;
  uint2* kids = reinterpret_cast<uint2*>(tables);
  // this CTA's staging area: scores and order of its share of the contexts
  const size_t stage_off = a.tables_in_smem ? tl.bytes : 0;
  float* st_s = reinterpret_cast<float*>(dyn + stage_off);

  // ---- candidates and context (produced by the previous kernel on the stream)
  pdl_wait();
  // every load first (one round trip: L * k <= 2 kThreads, L <= kThreads), then the
  // checks, so that no status report sits between two loads
  static_assert(kMaxL * kMaxK <= 2 * kThreads && kMaxL <= kThreads, "one pass of loads");
  int t_in[2] = {0, 0};
  float lq_in[2] = {0.f, 0.f};
#pragma unroll
  for (int u = 0; u < 2; ++u) {
    const int i = tid + u * kThreads;
    if (i < L * k) {
      t_in[u] = ld_chain(a.ids + static_cast<size_t>(b) * L * k + i);
      lq_in[u] = ld_chain(a.logq + static_cast<size_t>(b) * L * k + i);
    }
  }
  float lam = a.lambda;
  if (tid < L && a.lambda_d) lam = ld_chain(a.lambda_d + static_cast<size_t>(b) * L + tid);
  int c0 = 0, c1 = 0;
  if (tid == 0) {
    c0 = ld_chain(a.ctx2 + 2 * b);
    c1 = ld_chain(a.ctx2 + 2 * b + 1);
  }
#pragma unroll
  for (int u = 0; u < 2; ++u) {
    const int i = tid + u * kThreads;
    if (i < L * k) {
      const int d = i / k, j = i - d * k;
      int t = t_in[u];
      if (t < 0 || t >= kMaxV) {
        if (rank == 0) report(a.dev_status, PRESTO_DEV_BAD_TOKEN);
        t = 0;
      }
      sm.cid[d][j] = t;
      sm.clq[d][j] = lq_in[u];
    }
  }
  if (tid < L) {
    if (!(lam >= 0.f)) {  // negative or NaN: scores could turn positive
      if (rank == 0) report(a.dev_status, PRESTO_DEV_POSITIVE_SCORE);
      lam = 0.f;
    }
    sm.lam[tid] = lam;
  }
  if (tid == 0) {
    sm.ctx0 = c0;
    sm.ctx1 = c1;
    if (rank == 0 && (c0 < 0 || c0 >= kMaxV || c1 < 0 || c1 >= kMaxV))
      report(a.dev_status, PRESTO_DEV_BAD_TOKEN);
  }
  __syncthreads();
  if (rank == 0)
    for (int i = tid; i < L * k * k; i += kThreads) {  // sibling tokens must be distinct
      const int d = i / (k * k), r = i - d * k * k, j1 = r / k, j2 = r - j1 * k;
      if (j1 < j2 && sm.cid[d][j1] == sm.cid[d][j2]) report(a.dev_status, PRESTO_DEV_DUP_SIBLING);
    }
  // every candidate's rank by (token, index) within its depth (a permutation even
  // with duplicate tokens), and the inverse map
  for (int i = tid; i < L * k; i += kThreads) {
    const int d = i / k, j = i - d * k;
    const int t = sm.cid[d][j];
    int r = 0;
    for (int u = 0; u < k; ++u) {
      const int tu = sm.cid[d][u];
      r += tu < t || (tu == t && u < j);
    }
    sm.trk[d][j] = r;
    sm.rtok[d][r] = t;
  }
  __syncthreads();

  // ---- phase 1: this CTA scores contexts [g0, g1) of the sequence
  const int g0 = rank * a.per_cta;
  const int g1 = min(a.nctx_all, g0 + a.per_cta);
  const int my = g1 > g0 ? (g1 - g0) * k : 0;
  // each probe first reads its home slot (key and value); the probes that meet
  // another key (about a quarter at the tables' load factor) then read the next kWin
  // slots in one round; only a longer chain continues slot by slot
  constexpr int kBatch = 2;
  constexpr int kWin = 4;
  const uint64_t pol = l2_keep_policy();
  for (int f0 = tid; f0 < my; f0 += kThreads * kBatch) {
    uint64_t key[kBatch];
    uint32_t h[kBatch];
    float lq[kBatch], lam[kBatch];
#pragma unroll
    for (int q = 0; q < kBatch; ++q) {
      const int f = f0 + q * kThreads;
      key[q] = PRESTO_NGRAM3_EMPTY;
      h[q] = 0;
      lq[q] = 0.f;
      lam[q] = 0.f;
      if (f >= my) continue;
      const int gl = f / k, j = f - gl * k;
      int d, ci;
      decode_ctx(g0 + gl, k, use_table, d, ci);
      lq[q] = sm.clq[d][j];
      lam[q] = sm.lam[d];
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
    uint64_t k0[kBatch];
    float v0[kBatch];
#pragma unroll
    for (int q = 0; q < kBatch; ++q) {
      const bool live = key[q] != PRESTO_NGRAM3_EMPTY;
      k0[q] = live ? ld_table(a.keys + h[q], pol) : PRESTO_NGRAM3_EMPTY;
      v0[q] = live ? ld_table(a.logrho + h[q], pol) : 0.f;
    }
    // second round: the window after the home slot, for the probes still open
    uint64_t kw[kBatch][kWin];
    float vw[kBatch][kWin];
#pragma unroll
    for (int q = 0; q < kBatch; ++q) {
      const bool open = k0[q] != key[q] && k0[q] != PRESTO_NGRAM3_EMPTY;
#pragma unroll
      for (int w = 0; w < kWin; ++w) {
        const uint32_t hw = (h[q] + 1 + w) & a.cap_mask;
        kw[q][w] = open ? ld_table(a.keys + hw, pol) : PRESTO_NGRAM3_EMPTY;
        vw[q][w] = open ? ld_table(a.logrho + hw, pol) : 0.f;
      }
    }
#pragma unroll
    for (int q = 0; q < kBatch; ++q) {
      const int f = f0 + q * kThreads;
      if (f >= my) continue;
      float sc = lq[q];  // marginal-only: s = log q
      if (key[q] != PRESTO_NGRAM3_EMPTY) {
        // the first slot along the probe holding the key (a hit) or empty (a miss)
        float lr = a.miss;
        bool done = true;
        if (k0[q] == key[q]) {
          lr = v0[q];
        } else if (k0[q] != PRESTO_NGRAM3_EMPTY) {
          done = false;
#pragma unroll
          for (int w = 0; w < kWin; ++w) {
            if (!done && kw[q][w] == key[q]) {
              lr = vw[q][w];
              done = true;
            } else if (!done && kw[q][w] == PRESTO_NGRAM3_EMPTY) {
              done = true;
            }
          }
        }
        if (!done)  // a chain longer than the window: continue slot by slot
          lr = probe_from(a.keys, a.logrho, a.cap_mask, a.miss, key[q],
                          (h[q] + 1 + kWin) & a.cap_mask);
        sc = __fadd_rn(__fmul_rn(lam[q], lr), lq[q]);
      }
      if (sc > 0.f) report(a.dev_status, PRESTO_DEV_POSITIVE_SCORE);
      if (nb == k) {  // every candidate is kept
        const int gl = f / k, j = f - gl * k;
        int d, ci;
        decode_ctx(g0 + gl, k, use_table, d, ci);
        const int ik = (d * tl.cs + ci) * nb + j;
        if (PRESTO_IN_BOUNDS(ik, tl.nctx * nb, a.dev_status))
          kids[ik] = kid_record(sc, d, sm.trk[d][j], j);
      } else {
        st_s[f] = sc;
      }
    }
  }
  __syncthreads();
  // with b < k: keep the top-b of every context by a strict total order (float
  // bits as integers, then token, then index; a permutation even for duplicate
  // tokens or NaN)
  if (nb < k) {
    __syncthreads();
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
      const int ik = (d * tl.cs + ci) * nb + rk;
      if (rk < nb && PRESTO_IN_BOUNDS(ik, tl.nctx * nb, a.dev_status))
        kids[ik] = kid_record(row[j], d, sm.trk[d][j], j);
    }
  }
  if (!a.tables_in_smem) __threadfence();
  cluster.sync();  // the leader's tables are complete
  if (rank != 0) return;

  // ---- phase 2: top-N selection, level by level (leader CTA)
  // tables and scratch both in shared memory (every budget up to about N = 256): pointers
  // the compiler sees as shared, so the selection's many accesses are shared-memory
  // instructions rather than generic ones
  int n;
  if (a.tables_in_smem && a.p2_in_smem) {
    n = select_levels(a, sm, reinterpret_cast<const uint2*>(dyn), dyn + stage_off, tid);
  } else {
    unsigned char* const p2 = a.p2_in_smem
                                  ? dyn + stage_off
                                  : a.g_p2 + static_cast<size_t>(b) * a.p2_stride;
    n = select_levels(a, sm, a.tables_in_smem ? reinterpret_cast<const uint2*>(dyn) : kids, p2,
                      tid);
  }
  if (tid == 0) a.n_nodes[b] = n;
  if (a.mask) {
    // the tree-attention mask and position ids (as presto_tree_mask computes them):
    // word u of row i has bit j set for every ancestor-or-self j of node i in
    // [32u, 32u + 32); rows of unused nodes are zero, their position -1
    __syncthreads();
    const int N = a.N, W = (N + 31) / 32;
    int kv = ld_chain(a.kv_len + b);
    if (kv < 0) {
      if (tid == 0) report(a.dev_status, PRESTO_DEV_BAD_KVLEN);
    }
    for (int i = tid; i < N; i += kThreads) {
      uint32_t* row = a.mask + (static_cast<size_t>(b) * N + i) * W;
      int depth = -1;
      for (int u = 0; u < W; ++u) {
        uint32_t word = 0u;
        int dd = 0;
        if (i < n)
          for (int j = i; j >= 0 && PRESTO_IN_BOUNDS(j, N, a.dev_status); j = sm.par[j], ++dd)
            if ((j >> 5) == u) word |= 1u << (j & 31);
        row[u] = word;
        depth = dd - 1;
      }
      a.pos_ids[static_cast<size_t>(b) * N + i] = i < n ? kv + depth : -1;
    }
  }
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
int contexts_all(int L, int k, int use_table) {
  if (!use_table) return L;
  return 1 + (L > 1 ? k : 0) + (L > 2 ? (L - 2) * k * k : 0);
}
// Where the leader CTA keeps its tables and its selection scratch: in shared memory
// when they fit (the scratch aliases the phase-1 staging area), otherwise in the
// workspace, the tables first to go (the selection scans its scratch over and over;
// a table record is read once per child generated).
struct BuildPlan {
  bool tables_in_smem, p2_in_smem;
  size_t smem;       // dynamic shared memory per CTA
  size_t ws_tables;  // workspace bytes per sequence
  size_t ws_p2;
};
BuildPlan plan_build(int L, int k, int b, int N, int W, int use_table, int csize) {
  const TableLayout tl(L, k, b, use_table);
  const int per = (contexts_all(L, k, use_table) + csize - 1) / csize;
  const size_t st = align_up(static_cast<size_t>(per) * k * 4, 16);
  const size_t p2 = P2Layout(N, b, W).bytes;
  const size_t both = st > p2 ? st : p2;
  BuildPlan pl{true, true, 0, 0, 0};
  if (tl.bytes + both <= kDynSmemBudget) {
    pl.smem = tl.bytes + both;
  } else if (both <= kDynSmemBudget) {
    pl.tables_in_smem = false;
    pl.smem = both;
    pl.ws_tables = align_up(tl.bytes, 256);
  } else if (tl.bytes + st <= kDynSmemBudget) {
    pl.p2_in_smem = false;
    pl.smem = tl.bytes + st;
    pl.ws_p2 = align_up(p2, 256);
  } else {
    pl.tables_in_smem = pl.p2_in_smem = false;
    pl.smem = st;
    pl.ws_tables = align_up(tl.bytes, 256);
    pl.ws_p2 = align_up(p2, 256);
  }
  return pl;
}

// The kernel's attributes (the shared-memory budget, the wide cluster) and the number
// of clusters of kClusterWide CTAs the device holds at once, set and queried once per
// device; -1 when a call fails.
int wide_clusters_resident() {
  static PerDeviceOnce attrs;
  static int resident[kMaxDevices];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return -1;
  const cudaError_t e = attrs.run([dev] {
    cudaError_t r = cudaFuncSetAttribute(build_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(kDynSmemBudget));
    if (r != cudaSuccess) return r;
    resident[dev] = 0;
    if (cudaFuncSetAttribute(build_kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) !=
        cudaSuccess) {
      cudaGetLastError();  // no wide clusters on this device: the portable size only
      return cudaSuccess;
    }
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(kClusterWide);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = kDynSmemBudget;  // the most a launch takes: one CTA per SM
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = kClusterWide;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, build_kernel, &cfg) != cudaSuccess) {
      cudaGetLastError();
      n = 0;
    }
    resident[dev] = n;
    return cudaSuccess;
  });
  return e == cudaSuccess ? resident[dev] : -1;
}

// CTAs per sequence: the wide cluster when all B clusters of it are resident at once
// (the phase-1 probes spread over twice the SMs), else the portable size; 0 on a
// failed CUDA call.
int build_cluster(int B) {
  const int wide = wide_clusters_resident();
  if (wide < 0) return 0;
  return B <= wide ? kClusterWide : kCluster;
}
}  // namespace

extern "C" size_t presto_build_workspace_ex(int B, int L, int k, int N, int beam_width) {
  if (B < 1 || L < 1 || k < 1 || N < 1 || beam_width < 1) return 0;
  // sized for the larger case (prefix signal, b = k): what any call with these
  // shapes keeps outside shared memory fits
  // and for the portable cluster (each CTA's staging area is largest there)
  const BuildPlan pl = plan_build(L, k, k, N, beam_width, 1, kCluster);
  if (pl.tables_in_smem && pl.p2_in_smem) return 256;
  const TableLayout tl(L, k, k, 1);
  return static_cast<size_t>(B) * (align_up(tl.bytes, 256) + align_up(P2Layout(N, k, beam_width).bytes, 256));
}

extern "C" size_t presto_build_workspace(int B, int L, int k, int N) {
  return presto_build_workspace_ex(B, L, k, N, 1);
}

extern "C" int presto_score_build_tree(const int32_t* topk_ids, const float* topk_logq, int B,
                                       int L, int k, int b, const int32_t* ctx2,
                                       const presto_ngram3* ngram, float lambda, int N,
                                       int32_t* node_token, int32_t* node_parent,
                                       int32_t* node_depth, float* node_score,
                                       int32_t* n_nodes, void* ws, size_t ws_bytes,
                                       int32_t* dev_status, presto_stream_t stream) {
  return presto_score_build_tree_ex(topk_ids, topk_logq, B, L, k, b, ctx2, ngram, lambda,
                                    nullptr, PRESTO_SEARCH_BEST_FIRST, 1, N, node_token,
                                    node_parent, node_depth, node_score, n_nodes, ws, ws_bytes,
                                    dev_status, stream);
}

extern "C" int presto_score_build_tree_ex(const int32_t* topk_ids, const float* topk_logq,
                                          int B, int L, int k, int b, const int32_t* ctx2,
                                          const presto_ngram3* ngram, float lambda,
                                          const float* lambda_d, int policy, int beam_width,
                                          int N, int32_t* node_token, int32_t* node_parent,
                                          int32_t* node_depth, float* node_score,
                                          int32_t* n_nodes, void* ws, size_t ws_bytes,
                                          int32_t* dev_status, presto_stream_t stream) {
  return presto_score_build_tree_mask(topk_ids, topk_logq, B, L, k, b, ctx2, ngram, lambda,
                                      lambda_d, policy, beam_width, N, node_token, node_parent,
                                      node_depth, node_score, n_nodes, nullptr, nullptr, nullptr,
                                      ws, ws_bytes, dev_status, stream);
}

namespace presto {
namespace {

// Host-side checks of a tree-build call, run before any CUDA work.
int build_arg_status(const int32_t* topk_ids, const float* topk_logq, int B, int L, int k, int b,
                     const int32_t* ctx2, const presto_ngram3* ngram, float lambda, int policy,
                     int beam_width, int N, const int32_t* node_token, const int32_t* node_parent,
                     const int32_t* node_depth, const float* node_score, const int32_t* n_nodes,
                     const int32_t* kv_len, const uint32_t* mask, const int32_t* pos_ids) {
  PRESTO_CHECK_ARG((kv_len && mask && pos_ids) || (!kv_len && !mask && !pos_ids));
  PRESTO_CHECK_ARG(topk_ids && topk_logq && ctx2 && node_token && node_parent && node_depth &&
                   node_score && n_nodes);
  PRESTO_CHECK_ARG(B >= 1 && L >= 1 && k >= 1 && b >= 1 && N >= 1 && b <= k);
  PRESTO_CHECK_ARG(lambda >= 0.f && lambda == lambda);
  PRESTO_CHECK_ARG(policy == PRESTO_SEARCH_BEST_FIRST || policy == PRESTO_SEARCH_BEAM ||
                   policy == PRESTO_SEARCH_EAGER);
  PRESTO_CHECK_ARG(beam_width >= 1);
  PRESTO_CHECK_LIMIT(L <= kMaxL && k <= kMaxK && N <= kMaxN && beam_width <= kMaxN);
  if (ngram) {
    PRESTO_CHECK_ARG(ngram->keys && ngram->logrho);
    PRESTO_CHECK_ARG(ngram->log2_cap >= 4 && ngram->log2_cap <= 30);
    PRESTO_CHECK_ARG(ngram->miss_logrho <= 0.f);
  }
  return PRESTO_OK;
}

}  // namespace
}  // namespace presto

extern "C" int presto_score_build_tree_mask(
    const int32_t* topk_ids, const float* topk_logq, int B, int L, int k, int b,
    const int32_t* ctx2, const presto_ngram3* ngram, float lambda, const float* lambda_d,
    int policy, int beam_width, int N, int32_t* node_token, int32_t* node_parent,
    int32_t* node_depth, float* node_score, int32_t* n_nodes, const int32_t* kv_len,
    uint32_t* mask, int32_t* pos_ids, void* ws, size_t ws_bytes, int32_t* dev_status,
    presto_stream_t stream) {
  const int arg_status = build_arg_status(topk_ids, topk_logq, B, L, k, b, ctx2, ngram, lambda,
                                          policy, beam_width, N, node_token, node_parent,
                                          node_depth, node_score, n_nodes, kv_len, mask, pos_ids);
  if (arg_status != PRESTO_OK) return arg_status;
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
  a.lambda_d = lambda_d;
  a.policy = policy;
  a.W = beam_width;
  a.L = L;
  a.k = k;
  a.bf = b;
  a.N = N;
  a.nctx_all = contexts_all(L, k, a.use_table);
  const int csize = build_cluster(B);
  if (csize < 1) return PRESTO_ERR_CUDA;
  a.csize = csize;
  a.per_cta = (a.nctx_all + csize - 1) / csize;
  const BuildPlan pl = plan_build(L, k, b, N, beam_width, a.use_table, csize);
  a.tables_in_smem = pl.tables_in_smem;
  a.p2_in_smem = pl.p2_in_smem;
  const size_t need = static_cast<size_t>(B) * (pl.ws_tables + pl.ws_p2);
  if (need > 0) {
    if (!ws || reinterpret_cast<uintptr_t>(ws) % 16 || ws_bytes < need) return PRESTO_ERR_WORKSPACE;
    a.g_tables = static_cast<unsigned char*>(ws);
    a.g_p2 = static_cast<unsigned char*>(ws) + static_cast<size_t>(B) * pl.ws_tables;
    a.tables_stride = pl.ws_tables;
    a.p2_stride = pl.ws_p2;
  }
  a.node_token = node_token;
  a.node_parent = node_parent;
  a.node_depth = node_depth;
  a.node_score = node_score;
  a.n_nodes = n_nodes;
  a.kv_len = kv_len;
  a.mask = mask;
  a.pos_ids = pos_ids;
  a.dev_status = dev_status;
  const size_t smem = pl.smem;
  if (smem > kDynSmemBudget) return PRESTO_ERR_UNSUPPORTED;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(static_cast<unsigned>(B) * csize);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = csize;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1] = pdl_attribute();
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  if (cudaLaunchKernelEx(&cfg, build_kernel, a) != cudaSuccess) return PRESTO_ERR_CUDA;
  return launch_status();
}

// ---------------------------------------------------------------------------
// Allocation-free tree build.
//
// For callers that cannot hand the library a workspace: a plugin inside a serving
// framework whose allocator owns all of the GPU's memory, a C program with no
// allocator, or a latency-critical loop that must never block in cudaMalloc.  Large
// node budgets keep the selection scratch and child tables in global memory; here
// they live in a fixed file-scope device array instead, and the build otherwise runs
// exactly as presto_score_build_tree_mask.  The array costs
// PRESTO_BUILD_STATIC_SCRATCH_BYTES on every GPU that loads the library, for the
// life of the process.  All calls on a device share it and it keeps the last call's
// contents: the kernel writes every scratch entry it reads before reading it, so
// nothing has to be cleared, and two calls whose kernels overlap on the GPU (no
// ordering between their streams) race on it.
// ---------------------------------------------------------------------------
namespace presto {
namespace {

constexpr size_t kBuildStaticScratch = PRESTO_BUILD_STATIC_SCRATCH_BYTES;
__device__ __align__(256) unsigned char g_build_scratch[kBuildStaticScratch];

std::mutex g_build_scratch_mutex;
void* g_build_scratch_addr[64] = {};

// Device address of g_build_scratch on the current device.  In host code the
// symbol's name is only a host-side stand-in, so the address is looked up once per
// device, with that device current, and cached; nullptr when the lookup fails.
void* build_static_scratch() {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  std::lock_guard<std::mutex> lock(g_build_scratch_mutex);
  if (!g_build_scratch_addr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_build_scratch) != cudaSuccess || !p) {
      cudaGetLastError();
      return nullptr;
    }
    g_build_scratch_addr[dev] = p;
  }
  return g_build_scratch_addr[dev];
}

}  // namespace
}  // namespace presto

extern "C" int presto_score_build_tree_noalloc(
    const int32_t* topk_ids, const float* topk_logq, int B, int L, int k, int b,
    const int32_t* ctx2, const presto_ngram3* ngram, float lambda, const float* lambda_d,
    int policy, int beam_width, int N, int32_t* node_token, int32_t* node_parent,
    int32_t* node_depth, float* node_score, int32_t* n_nodes, const int32_t* kv_len,
    uint32_t* mask, int32_t* pos_ids, int32_t* dev_status, presto_stream_t stream) {
  // every host-side check first: a malformed call touches no CUDA state
  const int arg_status = build_arg_status(topk_ids, topk_logq, B, L, k, b, ctx2, ngram, lambda,
                                          policy, beam_width, N, node_token, node_parent,
                                          node_depth, node_score, n_nodes, kv_len, mask, pos_ids);
  if (arg_status != PRESTO_OK) return arg_status;
  // the plan of the portable cluster needs the most scratch of any cluster size (its
  // staging areas are the largest), so this host-side check covers the launch's plan
  const BuildPlan pl = plan_build(L, k, b, N, beam_width, ngram != nullptr, kCluster);
  const size_t need = static_cast<size_t>(B) * (pl.ws_tables + pl.ws_p2);
  if (need > kBuildStaticScratch) return PRESTO_ERR_UNSUPPORTED;
  void* ws = build_static_scratch();
  if (!ws) return PRESTO_ERR_CUDA;
  return presto_score_build_tree_mask(topk_ids, topk_logq, B, L, k, b, ctx2, ngram, lambda,
                                      lambda_d, policy, beam_width, N, node_token, node_parent,
                                      node_depth, node_score, n_nodes, kv_len, mask, pos_ids, ws,
                                      kBuildStaticScratch, dev_status, stream);
}
