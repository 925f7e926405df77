// presto_tree_mask (§4.3, App. C (I), (IV): each draft token attends to its
// ancestors) and presto_accept (§2.1 greedy prefix acceptance, App. A alpha_T(P),
// App. C (I) bonus token).
#include "common.cuh"

namespace presto {
namespace {

constexpr int kMaxW = kMaxN / 32;

// One CTA per sequence, one thread per node: walk the parent chain (at most L
// steps, parents in shared memory) and set one bit per ancestor-or-self.
__global__ void __launch_bounds__(kMaxN) mask_kernel(const int32_t* node_parent,
                                                     const int32_t* node_depth,
                                                     const int32_t* n_nodes,
                                                     const int32_t* kv_len, int N, int W,
                                                     uint32_t* mask, int32_t* pos_ids,
                                                     int32_t* dev_status) {
  __shared__ int par[kMaxN];
  __shared__ int dep[kMaxN];
  extern __shared__ uint32_t rows[];  // [N][W + 1]
  pdl_launch_dependents();
  pdl_wait();  // the tree comes from the previous kernel on the stream
  const int b = blockIdx.x, i = threadIdx.x;
  int n = ld_chain(n_nodes + b);
  if (n < 1 || n > N) {
    if (i == 0) report(dev_status, PRESTO_DEV_BAD_NNODES);
    n = n < 1 ? 0 : N;
  }
  const int kv = ld_chain(kv_len + b);
  if (i == 0 && kv < 0) report(dev_status, PRESTO_DEV_BAD_KVLEN);
  if (i < N) {
    par[i] = ld_chain(node_parent + static_cast<size_t>(b) * N + i);
    dep[i] = ld_chain(node_depth + static_cast<size_t>(b) * N + i);
    for (int w = 0; w < W; ++w) rows[i * (W + 1) + w] = 0u;
  }
  __syncthreads();
  if (i < n) {
    bool bad = (i == 0) ? (par[0] != -1 || dep[0] != 0)
                        : (par[i] < 0 || par[i] >= i || dep[i] != dep[par[i]] + 1);
    // parents strictly decrease, so the walk ends within i steps
    int j = i;
    for (;;) {
      rows[i * (W + 1) + (j >> 5)] |= 1u << (j & 31);
      if (j == 0) break;
      const int p = par[j];
      if (p < 0 || p >= j) {
        bad = true;
        break;
      }
      j = p;
    }
    if (bad) report(dev_status, PRESTO_DEV_BAD_PARENT);
  }
  __syncthreads();
  for (int e = i; e < N * W; e += blockDim.x) {
    const int r = e / W, w = e % W;
    mask[static_cast<size_t>(b) * N * W + e] = rows[r * (W + 1) + w];
  }
  if (i < N) pos_ids[static_cast<size_t>(b) * N + i] = i < n ? kv + dep[i] : -1;
}

// One CTA per sequence.  match(i) = (i == 0) || token(i) == target(parent(i)), one
// bit per node in shared memory; node i is accepted iff every node on its root path
// matches (its ancestor set, the same set as its mask row), found by walking the
// parents (at most L steps); the deepest accepted node (unique when siblings carry
// distinct tokens; lowest index otherwise) ends the accepted path.
constexpr int kAccThreads = 256;
__global__ void __launch_bounds__(kAccThreads) accept_kernel(
    const int32_t* node_token, const int32_t* node_parent, const int32_t* n_nodes,
    const int32_t* target_token, int N, int L, int32_t* accept_len, int32_t* accept_path,
    int32_t* bonus, int32_t* dev_status) {
  __shared__ int16_t par[kMaxN];
  __shared__ uint32_t matched[kMaxW];
  __shared__ unsigned wbest[kAccThreads / 32];
  pdl_launch_dependents();
  pdl_wait();  // the tree and the target tokens come from earlier kernels on the stream
  const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  int n = ld_chain(n_nodes + b);
  if (n < 1 || n > N) {
    if (tid == 0) report(dev_status, PRESTO_DEV_BAD_NNODES);
    n = n < 1 ? 1 : N;
  }
  const size_t base = static_cast<size_t>(b) * N;
  const int nt = blockDim.x;          // a multiple of 32, <= kAccThreads
  const int Nw = (N + 31) / 32 * 32;  // whole warps: every lane takes part in the ballots
  for (int i = tid; i < Nw; i += nt) {
    bool m = false;
    int p = -1;
    if (i < n) {
      if (i == 0) {
        m = true;
      } else {
        p = ld_chain(node_parent + base + i);
        if (p >= 0 && p < i) {
          m = ld_chain(node_token + base + i) == ld_chain(target_token + base + p);
        } else {
          report(dev_status, PRESTO_DEV_BAD_PARENT);
          p = -1;
        }
      }
    }
    if (i < N) par[i] = static_cast<int16_t>(p);
    const uint32_t bal = __ballot_sync(0xffffffffu, m);
    if (lane == 0) matched[i >> 5] = bal;
  }
  __syncthreads();
  // deepest accepted node: maximise (depth, -index); parents precede children, so a
  // walk ends within i steps
  unsigned best = 0u;
  for (int i = tid; i < n; i += nt) {
    int j = i, d = 0;
    bool ok = true;
    while (j > 0) {
      if (!((matched[j >> 5] >> (j & 31)) & 1u)) {
        ok = false;
        break;
      }
      j = par[j];
      ++d;
    }
    if (ok && j == 0) {
      const unsigned key = (static_cast<unsigned>(d & 0x3F) << 10) | (1023u - i);
      best = best > key ? best : key;
    }
  }
  best = __reduce_max_sync(0xffffffffu, best);
  if (lane == 0) wbest[warp] = best;
  __syncthreads();
  if (tid == 0) {
    for (int w = 0; w < nt / 32; ++w) best = best > wbest[w] ? best : wbest[w];
    const int node = 1023 - static_cast<int>(best & 1023u);
    int d = static_cast<int>(best >> 10);
    if (d > L) {
      report(dev_status, PRESTO_DEV_BAD_PARENT);
      d = L;
    }
    int32_t* path = accept_path + static_cast<size_t>(b) * (L + 1);
    for (int s = d + 1; s <= L; ++s) path[s] = -1;
    int j = node;
    for (int s = d; s >= 0; --s) {
      path[s] = j;
      j = j > 0 ? par[j] : 0;
    }
    accept_len[b] = d;
    bonus[b] = ld_chain(target_token + base + node);
  }
}

}  // namespace
}  // namespace presto

using namespace presto;

extern "C" int presto_tree_mask(const int32_t* node_parent, const int32_t* node_depth,
                                const int32_t* n_nodes, const int32_t* kv_len, int B, int N,
                                uint32_t* mask, int32_t* pos_ids, int32_t* dev_status,
                                presto_stream_t stream) {
  PRESTO_CHECK_ARG(node_parent && node_depth && n_nodes && kv_len && mask && pos_ids);
  PRESTO_CHECK_ARG(B >= 1 && N >= 1);
  PRESTO_CHECK_LIMIT(N <= kMaxN);
  const int W = (N + 31) / 32;
  const int threads = (N + 31) / 32 * 32;
  cudaLaunchConfig_t cfg{};
  const size_t rows_bytes = static_cast<size_t>(N) * (W + 1) * 4;
  static PerDeviceOnce smem_attr;
  if (smem_attr.run([] {
        return cudaFuncSetAttribute(
            mask_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
            static_cast<int>(static_cast<size_t>(kMaxN) * (kMaxN / 32 + 1) * 4));
      }) != cudaSuccess)
    return PRESTO_ERR_CUDA;
  cfg.gridDim = dim3(static_cast<unsigned>(B));
  cfg.blockDim = dim3(static_cast<unsigned>(threads));
  cfg.dynamicSmemBytes = rows_bytes;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1] = {pdl_attribute()};
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (cudaLaunchKernelEx(&cfg, mask_kernel, node_parent, node_depth, n_nodes, kv_len, N, W, mask,
                         pos_ids, dev_status) != cudaSuccess)
    return PRESTO_ERR_CUDA;
  return launch_status();
}

extern "C" int presto_accept(const int32_t* node_token, const int32_t* node_parent,
                             const int32_t* node_depth, const uint32_t* mask,
                             const int32_t* n_nodes, const int32_t* target_token, int B, int N,
                             int L, int32_t* accept_len, int32_t* accept_path, int32_t* bonus,
                             int32_t* dev_status, presto_stream_t stream) {
  PRESTO_CHECK_ARG(node_token && node_parent && node_depth && mask && n_nodes && target_token &&
                   accept_len && accept_path && bonus);
  PRESTO_CHECK_ARG(B >= 1 && N >= 1 && L >= 1);
  PRESTO_CHECK_LIMIT(N <= kMaxN && L <= kMaxL);
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(static_cast<unsigned>(B));
  cfg.blockDim = dim3(static_cast<unsigned>(N < kAccThreads ? (N + 31) / 32 * 32 : kAccThreads));
  cfg.stream = stream;
  cudaLaunchAttribute attr[1] = {pdl_attribute()};
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  (void)mask;      // the ancestor sets are read from node_parent (the mask rows' sets)
  (void)node_depth;
  if (cudaLaunchKernelEx(&cfg, accept_kernel, node_token, node_parent, n_nodes, target_token, N,
                         L, accept_len, accept_path, bonus, dev_status) != cudaSuccess)
    return PRESTO_ERR_CUDA;
  return launch_status();
}
