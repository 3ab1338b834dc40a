// compact_inplace.cu -- in-place slicing (src == dst) for Sec. 3.2's compaction step (Algorithm 1,
// "slice their KV-cache entries"): the first n_out rows of every plane become dst row j = src row
// keep_idx[j].
//
// Output row j reads row keep_idx[j] >= j.  Rows below A0, the first j with keep_idx[j] > j, stay
// where they are.  Two schedules, both on a cooperative launch of two CTAs per SM:
//  * Waves (when few are needed).  Wave k holds the output rows [A_k, B_k) with A_0 = A0,
//    B_k = min(keep_idx[A_k], n_out) and A_(k+1) = B_k: its rows read sources >= B_k, above every
//    row it writes, and no later wave reads a row below B_k.  So within a wave any order is safe,
//    and a store of wave k only has to wait until every CTA has seen its loads of wave k - 1
//    complete (one counter per launch).  Loads never wait.  The waves grow by about
//    1 / (keep ratio) each, so a low keep ratio needs a handful of them.
//  * Item dependencies (otherwise).  The store of output rows [r0, r0 + n) of a plane may only
//    start once every load of that plane that reads a row in [r0, r0 + n) is done; those loads
//    belong to earlier items of the same plane.  Items in (chunk, plane) order are dealt
//    round-robin; each CTA publishes how many of its items' loads are complete and waits
//    (bounded) for the owners of those earlier items before each store.
// Loads never wait on stores of later work, so every wait ends.
#include "compact_plan.cuh"

namespace apack {
namespace gather {
namespace {

constexpr int kInSlots = 3;                      // two CTAs per SM, 3 slots of 32 KB each
constexpr uint32_t kInSmem = kInSlots * kSlotBytes;
constexpr int kMaxInCtas = 384;                  // 16-bit progress words at ws + 256 .. ws + 1024
constexpr int kInChecks = 384;                   // progress words one dependency check may read
constexpr size_t kProgressOff = 256;

// Progress words.  A word is written after the CTA has observed its loads complete (the rows are
// already in shared memory, so no later write can change what they read), and a reader only
// issues its store after the loop that reads the word has seen the value it needs: relaxed
// gpu-scope accesses carry all the ordering the stores need.
__device__ __forceinline__ uint32_t ld_progress(const uint16_t *p) {
  uint16_t v;
  asm volatile("ld.relaxed.gpu.global.u16 %0, [%1];" : "=h"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void st_progress(uint16_t *p, uint32_t v) {
  asm volatile("st.relaxed.gpu.global.u16 [%0], %1;" ::"l"(p), "h"(static_cast<uint16_t>(v)) : "memory");
}

// #{ r < n : a[r] < x } for a strictly increasing, given a bracket [lo, hi] that holds it
// (a[lo - 1] < x or lo == 0; hi == n or a[hi] >= x).  Rounds of 32 evenly spaced probes narrow
// wide brackets; a bracket of at most 256 rows is then counted in one round, 8 rows per lane
// (independent loads of a few adjacent cache lines).
constexpr uint32_t kCountRows = 8;

__device__ __forceinline__ uint32_t warp_count_below(const int32_t *__restrict__ a, uint32_t lo, uint32_t hi,
                                                     int64_t x, int lane) {
  while (hi - lo > 32 * kCountRows) {
    const uint32_t span = hi - lo;
    const uint32_t step = (span + 31) / 32;
    const uint32_t p = lo + lane * step;
    const uint32_t b = __ballot_sync(0xffffffffu, p < hi && a[p] >= x);
    if (b) {
      const int f = __ffs(b) - 1;
      hi = lo + f * step;
      if (f > 0) lo += (f - 1) * step + 1;
    } else {
      lo += ((span - 1) / step) * step + 1;                 // past the last probe inside [lo, hi)
    }
  }
  uint32_t cnt = 0;
  const uint32_t p0 = lo + lane * kCountRows;
#pragma unroll
  for (uint32_t i = 0; i < kCountRows; ++i) cnt += (p0 + i < hi && a[p0 + i] < x) ? 1u : 0u;
  return lo + __reduce_add_sync(0xffffffffu, cnt);
}

// The item-dependency schedule.
__device__ void inplace_by_items(const TmaPlan &plan, const int32_t *__restrict__ keep_idx, uint16_t *progress,
                                 DeviceError *err, uint8_t *slots, uint64_t *full, int lane) {
  __shared__ uint16_t seen[kMaxInCtas];          // last progress read of every CTA
  for (int i = lane; i < kMaxInCtas; i += 32) seen[i] = 0;
  __syncwarp();
  const uint32_t me = blockIdx.x, P = gridDim.x;
  const uint32_t n_mine = me < plan.total_items ? (plan.total_items - me + P - 1) / P : 0;
  uint32_t issued = n_mine < kInSlots ? n_mine : kInSlots;   // positions whose loads were issued
  for (uint32_t j = 0; j < issued; ++j)
    load_item(decode_item(plan, me + j * P), slots + j * kSlotBytes, &full[j], keep_idx, lane);
  bool ok = true;
  uint32_t waited = 0;                                        // positions whose loads were observed
  uint32_t hint_row = 0;                                      // #{ keep_idx < hint_limit }, previous item
  int64_t hint_limit = 0;
  const TmaGroup *hint_grp = nullptr;
  for (uint32_t j = 0; ok && j < n_mine; ++j) {
    const int slot = j % kInSlots;
    const uint32_t item = me + j * P;
    const Item it = decode_item(plan, item);
    if (j >= waited && !mbar_wait(&full[slot], (j / kInSlots) & 1u, kWaitLimitNs)) {
      if (lane == 0 && err) raise_device_error(err, APACK_ETIMEOUT, 42);
      ok = false;
      break;
    }
    // publish as far as the loads are complete: this item, and the next ones already landed
    if (j >= waited) {
      uint32_t w = j + 1;
      if (lane == 0) {
        while (w < issued && mbar_try_wait(&full[w % kInSlots], (w / kInSlots) & 1u)) ++w;
        st_progress(progress + me, w);
      }
      waited = __shfl_sync(0xffffffffu, w, 0);              // the same count in every lane
    }
    // items of this plane whose loads read rows [r0, r0 + n) hold the output rows whose source is
    // below r0 + n: chunks <= c_hi, the chunk of the last such row (far behind c once rows are
    // dropped, so these waits are mostly met already).  Those are items item - k * num_planes,
    // k >= c - c_hi; their owners repeat with period P / gcd(num_planes, P) in k and an owner's
    // progress is monotonic, so the first period covers them all (at most kInChecks words).
    const TmaGroup &G = *it.grp;
    const uint32_t c = it.r0 / G.rows_per_slot;
    const int64_t limit = static_cast<int64_t>(it.r0) + it.nrows;
    {
      // keep_idx holds distinct integers, so the count below limit grows by at most limit -
      // hint_limit from the previous item of the group, and never exceeds limit
      const int64_t n = plan.n_out;
      const bool same = &G == hint_grp;
      const uint32_t lo = same ? hint_row : 0;
      const uint32_t hi = static_cast<uint32_t>(same ? min(n, static_cast<int64_t>(hint_row) + (limit - hint_limit))
                                                     : min(n, limit));
      hint_row = warp_count_below(keep_idx, lo, hi, limit, lane);
      hint_limit = limit;
      hint_grp = &G;
    }
    uint32_t kmin = 1, kmax = 0;                          // no dependency unless some row reads below limit
    if (hint_row > 0) {
      const uint32_t c_hi = (hint_row - 1) / G.rows_per_slot;
      kmin = c > c_hi ? c - c_hi : 1;
      kmax = min(c, kmin + plan.dep_period - 1);
    }
    uint32_t owner[kInChecks / 32], need[kInChecks / 32];
    {
      // item - k * num_planes for k = kmin + lane + 32 u: one division, then steps of 32 planes
      const uint32_t d = 32u * G.num_planes, dq = d / P, dr = d - dq * P;
      const uint32_t other0 = item - (kmin + lane) * G.num_planes;   // only used while k <= kmax
      uint32_t o = other0 % P, q = other0 / P;
#pragma unroll
      for (int u = 0; u < kInChecks / 32; ++u) {
        const uint32_t k = kmin + lane + 32 * u;
        owner[u] = me;                                    // no check: my own items are waited in order
        need[u] = 0;
        if (k <= kmax) {
          owner[u] = o;
          need[u] = q + 1;
        }
        // the next u: other - d
        const bool borrow = o < dr;
        o = borrow ? o + P - dr : o - dr;
        q = q - dq - (borrow ? 1u : 0u);
      }
    }
    // each lane owns distinct owners (k differ by less than the period), so the cache needs no sync.
    // When any cached word is too old, every owner of the check is read again in the same round:
    // the words read are far ahead of what later items need, so the cache then lasts until the
    // needs have grown past them (a few rounds per launch instead of one per stale owner).
    bool mine_ok = true;
    uint64_t t0 = 0;                                      // the clock is read once a round has failed
    for (;;) {
      bool stale = false;
#pragma unroll
      for (int u = 0; u < kInChecks / 32; ++u) stale |= owner[u] != me && seen[owner[u]] < need[u];
      if (!__any_sync(0xffffffffu, stale)) break;
      bool all = true;
#pragma unroll
      for (int u = 0; u < kInChecks / 32; ++u) {
        if (owner[u] != me) {
          const uint32_t v = ld_progress(progress + owner[u]);
          seen[owner[u]] = v;
          all &= v >= need[u];
        }
      }
      if (__all_sync(0xffffffffu, all)) break;
      if (t0 == 0) t0 = globaltimer_ns();
      if (__any_sync(0xffffffffu, globaltimer_ns() - t0 > kWaitLimitNs)) {   // the warp gives up together
        mine_ok = false;
        break;
      }
    }
    if (!__all_sync(0xffffffffu, mine_ok)) {
      if (lane == 0 && err) raise_device_error(err, APACK_ETIMEOUT, 43);
      ok = false;
      break;
    }
    asm volatile("fence.proxy.async.global;" ::: "memory");   // the observed loads before the bulk store
    fence_proxy_async_smem();
    store_item(it, slots + slot * kSlotBytes, lane);
    if (j >= 1 && j - 1 + kInSlots < n_mine) {
      bulk_wait_read<1>();
      const uint32_t k = j - 1 + kInSlots;
      const int ks = k % kInSlots;
      load_item(decode_item(plan, me + k * P), slots + ks * kSlotBytes, &full[ks], keep_idx, lane);
      issued = k + 1;
    }
  }
  if (!ok) {
    // loads issued but not observed may still be in flight: wait for them (bounded)
    for (uint32_t k = waited; k < issued; ++k) mbar_wait(&full[k % kInSlots], (k / kInSlots) & 1u, kWaitLimitNs / 4);
  }
}

// ---------------------------------------------------------------- waves
// First output row whose source row is above it (n when none): keep_idx[j] > j holds from there
// on, since keep_idx is strictly increasing.  Rounds of 32 evenly spaced probes.
__device__ uint32_t warp_first_moved(const int32_t *__restrict__ a, uint32_t n, int lane) {
  uint32_t lo = 0, hi = n;                         // the answer lies in [lo, hi]
  while (hi - lo > 32) {
    const uint32_t step = (hi - lo + 31) / 32;
    const uint32_t p = lo + lane * step;
    const uint32_t b = __ballot_sync(0xffffffffu, p < hi && a[p] > static_cast<int32_t>(p));
    if (b) {
      const int f = __ffs(b) - 1;
      const uint32_t lo0 = lo;
      hi = lo0 + f * step;
      if (f > 0) lo = lo0 + (f - 1) * step + 1;
    } else {
      lo += ((hi - lo - 1) / step) * step + 1;       // past the last probe inside [lo, hi)
    }
  }
  const uint32_t p = lo + lane;
  const uint32_t b = __ballot_sync(0xffffffffu, p < hi && a[p] > static_cast<int32_t>(p));
  return b ? lo + (__ffs(b) - 1) : hi;
}

// One wave: output rows [A, B), its items [base, base + n) of the concatenated item list.
struct Wave {
  uint32_t k, A, B, base, n;
};

__device__ __forceinline__ uint32_t wave_items(const TmaPlan &p, uint32_t A, uint32_t B) {
  uint32_t n = 0;
  for (int gi = 0; gi < p.ngroups; ++gi) n += p.g[gi].num_planes * ((B - A + p.g[gi].rows_per_slot - 1) / p.g[gi].rows_per_slot);
  return n;
}

__device__ __forceinline__ void wave_open(const TmaPlan &p, const int32_t *__restrict__ keep_idx, Wave &w,
                                          bool &bad) {
  if (w.A >= p.n_out) {
    w.B = w.A;
    w.n = 0;
    return;
  }
  const int64_t s = keep_idx[w.A];
  if (s <= static_cast<int64_t>(w.A)) {            // not strictly increasing: stop, report
    bad = true;
    w.A = w.B = p.n_out;
    w.n = 0;
    return;
  }
  w.B = s < static_cast<int64_t>(p.n_out) ? static_cast<uint32_t>(s) : p.n_out;
  w.n = wave_items(p, w.A, w.B);
}

// Moves w forward to the wave that holds item g (w.A == n_out past the last wave).
__device__ __forceinline__ void wave_seek(const TmaPlan &p, const int32_t *__restrict__ keep_idx, uint32_t g,
                                          Wave &w, bool &bad) {
  while (w.A < p.n_out && g >= w.base + w.n) {
    w.base += w.n;
    w.A = w.B;
    ++w.k;
    wave_open(p, keep_idx, w, bad);
  }
}

// Item g of wave w: (group, plane, chunk) order; chunks of rows_per_slot rows from A.
__device__ __forceinline__ Item wave_item(const TmaPlan &p, const Wave &w, uint32_t g) {
  uint32_t local = g - w.base;
  int gi = 0;
  uint32_t chunks = 0;
  for (;; ++gi) {
    chunks = (w.B - w.A + p.g[gi].rows_per_slot - 1) / p.g[gi].rows_per_slot;
    const uint32_t items = p.g[gi].num_planes * chunks;
    if (local < items || gi + 1 == p.ngroups) break;
    local -= items;
  }
  const TmaGroup &G = p.g[gi];
  Item it;
  it.grp = &G;
  it.plane = local / chunks;
  const uint32_t chunk = local - it.plane * chunks;
  it.r0 = w.A + chunk * G.rows_per_slot;
  it.nrows = min(G.rows_per_slot, w.B - it.r0);
  return it;
}

__device__ __forceinline__ uint32_t ld_acquire(const uint32_t *p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Barrier b of the launch is complete once every CTA has arrived at it: arrivals are made in
// order, each after the previous barrier completed, so the counter then reads (b + 1) P.
__device__ __forceinline__ bool wave_barrier_wait(const uint32_t *ctr, uint32_t b, uint32_t P) {
  const uint32_t target = (b + 1) * P;
  if (ld_acquire(ctr) >= target) return true;
  const uint64_t t0 = globaltimer_ns();
  while (ld_acquire(ctr) < target)
    if (globaltimer_ns() - t0 > kWaitLimitNs) return false;
  return true;
}

// The wave schedule; every lane runs it (lane 0 issues the counter operations).
__device__ void inplace_by_waves(const TmaPlan &plan, const int32_t *__restrict__ keep_idx, uint32_t A0,
                                 uint32_t *ctr, DeviceError *err, uint8_t *slots, uint64_t *full, int lane) {
  const uint32_t me = blockIdx.x, P = gridDim.x;
  bool bad = false;
  Wave wl{0, A0, A0, 0, 0};                         // cursor of the loads
  wave_open(plan, keep_idx, wl, bad);
  Wave ws = wl;                                     // cursor of the stores
  uint32_t arrived = 0;                             // barriers this CTA has arrived at
  bool ok = true;
  // arrive at every barrier below `upto` (each after the previous one completed)
  auto arrive_below = [&](uint32_t upto) -> bool {
    while (arrived < upto) {
      bool fine = true;
      if (lane == 0) {
        fine = arrived == 0 || wave_barrier_wait(ctr, arrived - 1, P);
        if (fine) asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(ctr) : "memory");
      }
      if (!__shfl_sync(0xffffffffu, fine, 0)) return false;
      ++arrived;
    }
    return true;
  };
  uint32_t issued = 0;
  for (; issued < kInSlots; ++issued) {
    const uint32_t g = me + issued * P;
    wave_seek(plan, keep_idx, g, wl, bad);
    if (wl.A >= plan.n_out) break;
    load_item(wave_item(plan, wl, g), slots + issued * kSlotBytes, &full[issued], keep_idx, lane);
  }
  uint32_t j = 0;
  for (;; ++j) {
    const uint32_t g = me + j * P;
    wave_seek(plan, keep_idx, g, ws, bad);
    if (ws.A >= plan.n_out) break;
    const int slot = j % kInSlots;
    if (!mbar_wait(&full[slot], (j / kInSlots) & 1u, kWaitLimitNs)) {
      if (lane == 0 && err) raise_device_error(err, APACK_ETIMEOUT, 44);
      ok = false;
      break;
    }
    // every load of this CTA in the waves before this item's has been seen complete
    if (!arrive_below(ws.k)) { ok = false; break; }
    bool fine = true;
    if (lane == 0 && ws.k > 0) fine = wave_barrier_wait(ctr, ws.k - 1, P);
    if (!__shfl_sync(0xffffffffu, fine, 0)) {
      ok = false;
      break;
    }
    asm volatile("fence.proxy.async.global;" ::: "memory");   // the other CTAs' loads before the bulk store
    fence_proxy_async_smem();
    store_item(wave_item(plan, ws, g), slots + slot * kSlotBytes, lane);
    // refill the slot whose store was issued one item ago, once that store has read it
    if (j >= 1 && j - 1 + kInSlots == issued) {
      const uint32_t k = issued;
      const uint32_t gk = me + k * P;
      wave_seek(plan, keep_idx, gk, wl, bad);
      if (wl.A < plan.n_out) {
        bulk_wait_read<1>();
        load_item(wave_item(plan, wl, gk), slots + (k % kInSlots) * kSlotBytes, &full[k % kInSlots], keep_idx, lane);
        issued = k + 1;
      }
    }
  }
  if (ok && !arrive_below(ws.k)) ok = false;        // the waves this CTA had no more items in
  if (!ok) {
    if (lane == 0 && err) raise_device_error(err, APACK_ETIMEOUT, 45);
    for (uint32_t k = j; k < issued; ++k) mbar_wait(&full[k % kInSlots], (k / kInSlots) & 1u, kWaitLimitNs / 4);
  }
  if (bad && lane == 0 && err) raise_device_error(err, APACK_EDEVICE, 46);
}

constexpr float kMaxWaves = 16.f;

__global__ void __launch_bounds__(32) gather_inplace_kernel(const __grid_constant__ TmaPlan plan,
                                                            const int32_t *__restrict__ keep_idx,
                                                            uint16_t *progress, DeviceError *err) {
  extern __shared__ __align__(1024) uint8_t slots[];
  __shared__ __align__(8) uint64_t full[kInSlots];
  const int lane = threadIdx.x;
  if (lane == 0) {
    for (int i = 0; i < kInSlots; ++i) mbar_init(&full[i], 1);
    fence_mbar_init();
  }
  __syncwarp();
  const uint32_t n = plan.n_out;
  const uint32_t A0 = warp_first_moved(keep_idx, n, lane);   // the same in every CTA
  if (A0 < n) {
    // waves needed: they grow by about (last source row + 1) / n_out each, from A0
    const float grow = (static_cast<float>(keep_idx[n - 1]) + 1.f) / static_cast<float>(n);
    const float waves = 1.f + log2f(static_cast<float>(n) / static_cast<float>(A0 > 0 ? A0 : 1)) / log2f(grow);
    if (grow > 1.f && waves <= kMaxWaves)
      inplace_by_waves(plan, keep_idx, A0, reinterpret_cast<uint32_t *>(progress), err, slots, full, lane);
    else
      inplace_by_items(plan, keep_idx, progress, err, slots, full, lane);
  }
  bulk_wait_all();
}

}  // namespace

apack_status plan_inplace(TmaPlan &ip, uint64_t in_items, uint32_t *blocks_out) {
  uint64_t blocks = static_cast<uint64_t>(device_sm_count()) * 2;   // two CTAs per SM, all resident
  if (blocks > kMaxInCtas) blocks = kMaxInCtas;
  if (blocks > in_items) blocks = in_items;
  if (in_items > blocks * 65535) return APACK_EUNSUPPORTED;           // 16-bit progress words
  ip.total_items = static_cast<uint32_t>(in_items);
  // the dependency check covers P / gcd(num_planes, P) chunks of every group (at most P <= kInChecks)
  uint32_t period = 1;
  for (int gi = 0; gi < ip.ngroups; ++gi) {
    uint32_t a = ip.g[gi].num_planes, b = static_cast<uint32_t>(blocks);
    while (b) {
      const uint32_t t = a % b;
      a = b;
      b = t;
    }
    const uint32_t per = static_cast<uint32_t>(blocks) / a;
    if (per > period) period = per;
  }
  ip.dep_period = period;
  *blocks_out = static_cast<uint32_t>(blocks);
  return APACK_OK;
}

apack_status launch_inplace(const TmaPlan &ip_in, uint32_t blocks, const int32_t *keep_idx, DeviceError *err,
                            cudaStream_t stream) {
  static std::atomic<uint64_t> in_attr_done{0};
  if (once_per_device(in_attr_done, [] {
        return cudaFuncSetAttribute(gather_inplace_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kInSmem);
      }) != cudaSuccess)
    return APACK_ECUDA;
  TmaPlan ip = ip_in;
  uint16_t *progress = reinterpret_cast<uint16_t *>(reinterpret_cast<uint8_t *>(err) + kProgressOff);
  // the progress words (item schedule) or the barrier counter (wave schedule): bytes 256..1023
  if (check_cuda(cudaMemsetAsync(progress, 0, 1024 - kProgressOff, stream)) != APACK_OK) return APACK_ECUDA;
  void *args[] = {&ip, const_cast<int32_t **>(&keep_idx), &progress, &err};
  if (check_cuda(cudaLaunchCooperativeKernel(reinterpret_cast<const void *>(gather_inplace_kernel), dim3(blocks),
                                             dim3(32), args, kInSmem, stream)) != APACK_OK)
    return APACK_ECUDA;
  count_launches(1);
  return APACK_OK;
}

}  // namespace gather
}  // namespace apack
