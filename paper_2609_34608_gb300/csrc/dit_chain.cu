// The row-local part of consecutive DiT blocks as one persistent tcgen05 kernel.
//
// After a block's attention, everything up to the next block's attention works on rows
// independently: out-projection + gated residual, LN + adaLN modulation, MLP up (+GELU), MLP down
// + gated residual, then the next block's LN + modulation and QKV projection.  Launched as
// separate kernels, each of these pays its own pipeline fill and drain and its own last partial
// wave; at one episode (1296 rows) that overhead is most of the block's time.  Here they are
// tasks of one launch, taken in a fixed topological order from a device-wide counter:
//
//   OUT(m, n)   att rows m x out_w   -> h += gate1 (acc + b)          (128 x 64 tiles)
//   LN2(m, q)   h rows m, quarter q  -> xln = LN(h)(1 + scale2) + shift2
//   UP(m, n)    xln rows m x up_w    -> u = GELU(acc + b)             needs LN2(m, *)
//   DOWN(m, n)  u rows m x down_w    -> h += gate2 (acc + b)          needs UP(m, *); 128 x 64
//   (MLP up and QKV tiles are 128 x 128)
//   LN1(m, q)   next block's LN + modulation (optionally saving h)    needs DOWN(m, *)
//   QKV(m, n)   xln rows m x qkv_w   -> qkv, V^T                       needs LN1(m, *)
//
// m is a 128-row block.  A task waits (bounded) for per-row-block completion counters of the
// tasks it reads from; tasks are taken only by running CTAs and every dependency has a smaller
// index, so the smallest unfinished task can always proceed whatever the residency.  Inside a
// CTA the roles are those of the per-projection GEMM: warp 0 takes tasks and streams operand
// tiles with TMA (a GEMM task's weight tiles are requested before its dependency is satisfied,
// only the activation tiles wait), warp 1 issues tcgen05.mma into a double-buffered TMEM
// accumulator, warps 2-5 run the epilogues and the LN tasks.  The task index reaches warps 1-5
// through a small shared-memory ring.  The last CTA to finish resets every counter, so each
// launch (and each CUDA-graph replay) starts from zero.  Every wait is bounded (%globaltimer):
// on a timeout the CTA sets the device error word, drains what it issued and frees TMEM.
//
// Accumulation order and epilogue arithmetic are those of the per-projection GEMM and the LN
// kernel, so the fused and unfused paths give the same values.
#include "gemm_epilogue.cuh"
#include "tcgen05.cuh"

namespace wam {
namespace {

constexpr int kChM = 128;                       // rows per tile and per row block
constexpr int kChBN = 128;                      // output columns per tile (MLP up, QKV)
constexpr int kChBNNarrow = 64;                 // output columns per tile of the d-wide projections
constexpr int kChAtom = kChM * 128;             // one 64-deep K-atom of 128 rows: 16 KB
constexpr int kChStageBytes = 4 * kChAtom;      // two atoms of A and two of B: 64 KB
constexpr int kChStages = 3;
constexpr int kChThreads = 256;
// Task indices in flight between the roles: the producer takes a new task only once the epilogue
// warps have started the one two places before it.  A deeper ring lets a CTA hoard LN tasks
// (they need no operand loads, so the producer would take them back to back) that other CTAs
// would have run in parallel.
constexpr int kChRing = 2;
constexpr int kChLnParts = 16;                  // LN tasks per row block (8 rows each)
constexpr int kChLnRows = kChM / kChLnParts;     // rows per LN task: 4 per LN warp
constexpr int kChBarBytes = 512 + 2 * kChBN * 4;   // barriers and flags, then the staged biases
constexpr int kChSmem = kChStages * kChStageBytes + kChBarBytes + 1024;

enum ChKind : int { kOut = 0, kLn2 = 1, kUp = 2, kDown = 3, kLn1 = 4, kQkv = 5, kNumKinds = 6 };

struct TaskRef {
  int kind, m, j;
};

WAM_DEV int ld_relaxed(const int* p) {
  int v;
  asm volatile("ld.relaxed.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Acquire side of a completion counter: later reads of other CTAs' data see their published
// writes (also invalidates this SM's L1, so it is taken once per satisfied wait, not per poll).
WAM_DEV void fence_acquire() { asm volatile("fence.acquire.gpu;" ::: "memory"); }

// Bounded wait until *p >= target (another CTA's completion counter).  Polls with relaxed loads
// (an acquiring load per poll would keep invalidating this SM's L1) and acquires once.
WAM_DEV bool wait_count(const int* p, int target, volatile int* abort_flag, int* dev_err) {
  if (ld_relaxed(p) >= target) {
    fence_acquire();
    return true;
  }
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t i = 1;; ++i) {
    if (ld_relaxed(p) >= target) {
      fence_acquire();
      return true;
    }
    if ((i & 15u) == 0) {
      if (*abort_flag) return false;
      if (globaltimer_ns() - t0 > kWaitLimitNs) {
        *abort_flag = 1;
        atomicOr(dev_err, kDevErrTimeout);
        return false;
      }
    }
    __nanosleep(64);
  }
}

// Publish the writes of a finished task and count it: called by one thread after all the task's
// writers met on a CTA barrier; the release fence is cumulative over the writes ordered before it
// by that barrier.
WAM_DEV void signal_count(int* p) {
  asm volatile("red.release.gpu.global.add.s32 [%0], 1;" ::"l"(p) : "memory");
}

WAM_DEV void epi_bar() { asm volatile("bar.sync 1, 128;" ::: "memory"); }
WAM_DEV void ln_bar() { asm volatile("bar.sync 2, 64;" ::: "memory"); }

struct ChainView {
  int first[kNumKinds + 1];   // first task index of each kind; first[kNumKinds] = total
  int per_row[kNumKinds];     // tasks of each kind per row block
};

WAM_DEV ChainView chain_view(const ChainParams& p) {
  ChainView v;
  v.per_row[kOut] = p.has_tail ? p.d / kChBNNarrow : 0;
  v.per_row[kLn2] = p.has_tail ? kChLnParts : 0;
  v.per_row[kUp] = p.has_tail ? p.dff / kChBN : 0;
  v.per_row[kDown] = p.has_tail ? p.d / kChBNNarrow : 0;
  v.per_row[kLn1] = p.has_head ? kChLnParts : 0;
  v.per_row[kQkv] = p.has_head ? 3 * p.d / kChBN : 0;
  v.first[0] = 0;
  for (int k = 0; k < kNumKinds; ++k) v.first[k + 1] = v.first[k] + v.per_row[k] * p.Mt;
  return v;
}

WAM_DEV TaskRef decode(const ChainView& v, int t) {
  int k = 0;
  while (k + 1 < kNumKinds && t >= v.first[k + 1]) ++k;
  const int r = t - v.first[k];
  return TaskRef{k, r / v.per_row[k], r % v.per_row[k]};
}

// Counters: [0] next task, [1] CTAs finished, then completions [kind][row block].  With
// phase_barrier every task of a kind counts into row block 0's slot and a task waits for the
// whole previous kind (a grid-wide phase boundary instead of per-row-block dependencies).
WAM_DEV int* counter(const ChainParams& p, int kind, int m) {
  return p.ctr + 2 + kind * p.Mt + (p.phase_barrier ? 0 : m);
}

// What a task waits for: (counter, target), or a null counter.
WAM_DEV void dependency(const ChainParams& p, const ChainView& v, const TaskRef& t, const int** c, int* target) {
  *c = nullptr;
  *target = 0;
  if (p.phase_barrier) {
    // the previous non-empty kind, all of it
    int k = t.kind - 1;
    while (k >= 0 && v.per_row[k] == 0) --k;
    if (k >= 0) {
      *c = counter(p, k, 0);
      *target = v.per_row[k] * p.Mt;
    }
    return;
  }
  switch (t.kind) {
    case kLn2: *c = counter(p, kOut, t.m); *target = v.per_row[kOut]; break;
    case kUp: *c = counter(p, kLn2, t.m); *target = kChLnParts; break;
    case kDown: *c = counter(p, kUp, t.m); *target = v.per_row[kUp]; break;
    case kLn1:
      if (p.has_tail) {
        *c = counter(p, kDown, t.m);
        *target = v.per_row[kDown];
      }
      break;
    case kQkv: *c = counter(p, kLn1, t.m); *target = kChLnParts; break;
    default: break;
  }
}

WAM_DEV bool is_gemm(int kind) { return kind == kOut || kind == kUp || kind == kDown || kind == kQkv; }

// Tile width: the out- and down-projections (N = d) use 64-column tiles, which doubles the CTAs on
// the long MLP-down tiles and halves their epilogue; MLP up and QKV use 128.
WAM_DEV int tile_n(int kind) { return (kind == kOut || kind == kDown) ? kChBNNarrow : kChBN; }

// LayerNorm + adaLN modulation of 4 rows per LN warp (one LN task = 8 rows), the same
// arithmetic as the LN kernel.  Every load of the task is issued before the first use: loads wait
// behind the GEMM tiles' TMA traffic, so one round trip per task instead of one per row.
template <int NV4>
WAM_DEV void ln_rows(const ChainParams& p, int row0, int shift_off, int scale_off, float* hcopy) {
  constexpr int kR = kChLnRows / 2;
  const int lane = threadIdx.x & 31;
  const int w = (threadIdx.x >> 5) - 6;
  const int d = p.d;
  float4 v[kR][NV4];
  int64_t rows[kR];
#pragma unroll
  for (int u = 0; u < kR; ++u) {
    rows[u] = row0 + w * kR + u;
    if (rows[u] < p.M) {
      const float4* hr = reinterpret_cast<const float4*>(p.h + rows[u] * d);
#pragma unroll
      for (int i = 0; i < NV4; ++i) v[u][i] = hr[lane + 32 * i];
    }
  }
#pragma unroll
  for (int u = 0; u < kR; ++u) {
    const int64_t row = rows[u];
    if (row >= p.M) continue;
    if (hcopy != nullptr) {
      float4* cr = reinterpret_cast<float4*>(hcopy + row * d);
#pragma unroll
      for (int i = 0; i < NV4; ++i) cr[lane + 32 * i] = v[u][i];
    }
    float mean, rstd;
    row_stats<NV4>(v[u], d, mean, rstd);
    int item = static_cast<int>(row / p.rows_per_item);
    if (p.item_map != nullptr) item = p.item_map[item];
    const float* shift = p.mods + item * p.mod_stride + shift_off;
    const float* scale = p.mods + item * p.mod_stride + scale_off;
#pragma unroll
    for (int i = 0; i < NV4; ++i) {
      const int c = (lane + 32 * i) * 4;
      const float4 sh = *reinterpret_cast<const float4*>(shift + c);
      const float4 sc = *reinterpret_cast<const float4*>(scale + c);
      const float4 x = v[u][i];
      Act<bf16>::store4(p.xln + row * d + c, fmaf((x.x - mean) * rstd, 1.0f + sc.x, sh.x),
                        fmaf((x.y - mean) * rstd, 1.0f + sc.y, sh.y),
                        fmaf((x.z - mean) * rstd, 1.0f + sc.z, sh.z),
                        fmaf((x.w - mean) * rstd, 1.0f + sc.w, sh.w));
    }
  }
}

template <int NV4>
WAM_DEV void ln_task(const ChainParams& p, int row0, bool second) {
  if (second)
    ln_rows<NV4>(p, row0, p.shift2_off, p.scale2_off, nullptr);
  else
    ln_rows<NV4>(p, row0, p.shift1_off, p.scale1_off, p.hq);
}

// Gated-residual read-back of a 128-column tile row, h += gate (acc + bias), with the residual
// loads of the next 32 columns issued before the stores of the current ones (one load round trip
// per two chunks instead of per chunk; the gate rows likewise).  e.bias points at the staged
// copy in shared memory.  Same arithmetic as the GEMM epilogue.
WAM_DEV void resid_epilogue(const EpiArgs& e, int N, int M, int row, int col0, uint32_t taddr) {
  constexpr int kChunks = kChBNNarrow / 32;
  int item = row / e.rows_per_item;
  if (e.item_map != nullptr && row < M) item = e.item_map[item];
  float4 hbuf[2][8], gbuf[2][8];
  auto load_h = [&](int c, float4 (&hb)[8], float4 (&gb)[8]) {
    if (row >= M) return;
    const float4* h4 = reinterpret_cast<const float4*>(static_cast<float*>(e.C) + static_cast<int64_t>(row) * N +
                                                       col0 + c * 32);
    const float4* g4 = reinterpret_cast<const float4*>(e.gate + item * e.gate_stride + col0 + c * 32);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      hb[j] = h4[j];
      gb[j] = g4[j];
    }
  };
  load_h(0, hbuf[0], gbuf[0]);
#pragma unroll
  for (int c = 0; c < kChunks; ++c) {
    uint32_t r[32];
    tmem_ld32(taddr + c * 32, r);
    if (c + 1 < kChunks) load_h(c + 1, hbuf[(c + 1) & 1], gbuf[(c + 1) & 1]);
    if (row >= M) continue;
    const int col = col0 + c * 32;
    const float4* b4 = reinterpret_cast<const float4*>(e.bias + col);   // shared memory (staged)
    float4* h4 = reinterpret_cast<float4*>(static_cast<float*>(e.C) + static_cast<int64_t>(row) * N + col);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const float4 b = e.bias != nullptr ? b4[j] : make_float4(0.f, 0.f, 0.f, 0.f);
      const float4 g = gbuf[c & 1][j];
      float4 h = hbuf[c & 1][j];
      const float v0 = e.bias != nullptr ? __uint_as_float(r[4 * j]) + b.x : __uint_as_float(r[4 * j]);
      const float v1 = e.bias != nullptr ? __uint_as_float(r[4 * j + 1]) + b.y : __uint_as_float(r[4 * j + 1]);
      const float v2 = e.bias != nullptr ? __uint_as_float(r[4 * j + 2]) + b.z : __uint_as_float(r[4 * j + 2]);
      const float v3 = e.bias != nullptr ? __uint_as_float(r[4 * j + 3]) + b.w : __uint_as_float(r[4 * j + 3]);
      h.x = fmaf(g.x, v0, h.x);
      h.y = fmaf(g.y, v1, h.y);
      h.z = fmaf(g.z, v2, h.z);
      h.w = fmaf(g.w, v3, h.w);
      h4[j] = h;
    }
  }
}

template <int NV4>
__global__ void __launch_bounds__(kChThreads, 1)
    dit_chain_kernel(const __grid_constant__ CUtensorMap tmAtt, const __grid_constant__ CUtensorMap tmXln,
                     const __grid_constant__ CUtensorMap tmU, const __grid_constant__ CUtensorMap tmOutW,
                     const __grid_constant__ CUtensorMap tmUpW, const __grid_constant__ CUtensorMap tmDownW,
                     const __grid_constant__ CUtensorMap tmQkvW, const ChainParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* tiles = smem;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kChStages * kChStageBytes);
  uint64_t* full = bars;                        // [kChStages]
  uint64_t* empty = full + kChStages;           // [kChStages]
  uint64_t* tfull = empty + kChStages;          // [2]
  uint64_t* tempty = tfull + 2;                 // [2]
  uint64_t* task_full = tempty + 2;             // [kChRing]
  uint64_t* task_free = task_full + kChRing;    // [kChRing]
  uint64_t* drain = task_free + kChRing;
  uint64_t* pub_full = drain + 1;               // [kChRing]: a finished task's counter to publish
  uint64_t* pub_free = pub_full + kChRing;      // [kChRing]
  int** pub_ptr = reinterpret_cast<int**>(pub_free + kChRing);   // [kChRing]
  uint64_t* ln_full = reinterpret_cast<uint64_t*>(pub_ptr + kChRing);   // [kChRing]: LN task queued
  uint64_t* ln_free = ln_full + kChRing;                                // [kChRing]
  int* task_id = reinterpret_cast<int*>(ln_free + kChRing);      // [kChRing]
  int* ln_id = task_id + kChRing;                                 // [kChRing]
  float* bias_stage = reinterpret_cast<float*>(bars + 64);        // [2 accumulators][kChBN]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(ln_id + kChRing);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  volatile int* bcast_task = abort_flag + 1;    // epilogue warps: the task of this iteration
  volatile int* bcast_ok = bcast_task + 1;      // epilogue warps: outcome of the last wait
  volatile int* ln_task_b = bcast_ok + 1;        // LN warps: the task of this iteration
  volatile int* ln_ok_b = ln_task_b + 1;         // LN warps: outcome of the dependency wait
  volatile int* last_cta = ln_ok_b + 1;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const ChainView view = chain_view(p);
  const int total = view.first[kNumKinds];
  int* task_ctr = p.ctr;
  int* done_ctr = p.ctr + 1;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kChStages; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(smem_u32(&tfull[a]), 1);
      mbar_init(smem_u32(&tempty[a]), 128);
    }
    for (int r = 0; r < kChRing; ++r) {
      mbar_init(smem_u32(&task_full[r]), 1);
      mbar_init(smem_u32(&task_free[r]), 2);   // the MMA thread and the epilogue warps' thread 64
    }
    mbar_init(smem_u32(drain), 1);
    for (int r = 0; r < kChRing; ++r) {
      mbar_init(smem_u32(&pub_full[r]), 1);
      mbar_init(smem_u32(&pub_free[r]), 1);
      mbar_init(smem_u32(&ln_full[r]), 1);
      mbar_init(smem_u32(&ln_free[r]), 1);
    }
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(smem_u32(tmem_slot), 2 * kChBN);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  pdl_launch_dependents();

  auto gemm_maps = [&](int kind, const CUtensorMap** a, const CUtensorMap** b, int* K) {
    switch (kind) {
      case kOut: *a = &tmAtt; *b = &tmOutW; *K = p.d; break;
      case kUp: *a = &tmXln; *b = &tmUpW; *K = p.d; break;
      case kDown: *a = &tmU; *b = &tmDownW; *K = p.dff; break;
      default: *a = &tmXln; *b = &tmQkvW; *K = p.d; break;
    }
  };

  if (warp == 0) {
    if (lane == 1) {
      // ---------------- publisher: makes finished tasks visible to other CTAs ----------------
      // The epilogue warps hand each finished task's counter over and go on with the next tile;
      // the release fence (which waits for their stores to be acknowledged) is paid here.
      for (int i = 0;; ++i) {
        const int slot = i % kChRing;
        if (!mbar_wait(smem_u32(&pub_full[slot]), (i / kChRing) & 1, abort_flag, p.dev_err)) break;
        int* sig = pub_ptr[slot];
        if (sig == nullptr) break;
        signal_count(sig);
        mbar_arrive(smem_u32(&pub_free[slot]));
      }
    }
    // ---------------- task fetch + TMA producer (one lane) ----------------
    if (lane == 0) {
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmAtt)) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmXln)) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmU)) : "memory");
      pdl_wait();
      int stage = 0;
      uint32_t phase = 0;
      uint32_t issued = 0, issued_phase = 0;   // per stage bit: a copy was issued, with its phase
      bool ok = true;
      int ng = 0, nl = 0;   // tasks passed to the GEMM roles / to the LN warps
      // GEMM tasks go to the MMA and epilogue warps, LN tasks to the LN warps; each ring is two
      // deep, so the producer takes a task only when its consumer is nearly free
      auto push = [&](uint64_t* full_b, uint64_t* free_b, int* ids, int& n, int t) -> bool {
        const int slot = n % kChRing;
        if (!mbar_wait(smem_u32(&free_b[slot]), ((n / kChRing) & 1) ^ 1u, abort_flag, p.dev_err)) return false;
        ids[slot] = t;
        mbar_arrive(smem_u32(&full_b[slot]));
        ++n;
        return true;
      };
      // wait for room in the GEMM ring before taking a task (it is the usual destination)
      auto gemm_room = [&]() -> bool {
        return mbar_wait(smem_u32(&task_free[ng % kChRing]), ((ng / kChRing) & 1) ^ 1u, abort_flag, p.dev_err);
      };
      for (;;) {
        if (!gemm_room()) {
          ok = false;
          break;
        }
        const int t = atomicAdd(task_ctr, 1);
        if (t >= total) {
          if (!push(task_full, task_free, task_id, ng, total) || !push(ln_full, ln_free, ln_id, nl, total)) ok = false;
          break;
        }
        const TaskRef tr = decode(view, t);
        wam_chain_task* rec = (p.trace != nullptr && t < p.trace_cap) ? p.trace + t : nullptr;
        if (rec != nullptr) {
          rec->launch = p.trace_launch;
          rec->cta = blockIdx.x;
          rec->kind = tr.kind;
          rec->m = tr.m;
          rec->j = tr.j;
          rec->t_take = globaltimer_ns();
        }
        if (!is_gemm(tr.kind)) {   // LN tasks run in the LN warps
          if (!push(ln_full, ln_free, ln_id, nl, t)) {
            ok = false;
            break;
          }
          continue;
        }
        if (!push(task_full, task_free, task_id, ng, t)) {
          ok = false;
          break;
        }
        const CUtensorMap *ma, *mb;
        int K;
        gemm_maps(tr.kind, &ma, &mb, &K);
        const int nk = K / 128;
        const int bn = tile_n(tr.kind);
        const uint32_t stage_bytes = 2 * kChAtom + 2 * bn * 128;
        const int pre = nk < kChStages ? nk : kChStages;
        const int stage0 = stage;
        // weight tiles first: they depend on nothing
        for (int kb = 0; kb < pre; ++kb) {
          if (!mbar_wait(smem_u32(&empty[stage]), phase ^ 1u, abort_flag, p.dev_err)) {
            ok = false;
            break;
          }
          const uint32_t fb = smem_u32(&full[stage]);
          const uint32_t dst = smem_u32(tiles + stage * kChStageBytes);
          mbar_expect_tx(fb, stage_bytes);
          tma_load_3d(dst + 2 * kChAtom, mb, 0, tr.j * bn, kb * 2, fb);
          issued |= 1u << stage;
          issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
          if (++stage == kChStages) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        const int* dc;
        int target;
        dependency(p, view, tr, &dc, &target);
        if (dc != nullptr) {
          if (!wait_count(dc, target, abort_flag, p.dev_err)) {
            ok = false;
            break;
          }
          // activations written by other CTAs' generic stores, read here through the async proxy
          asm volatile("fence.proxy.async.global;" ::: "memory");
        }
        if (rec != nullptr) rec->t_dep = globaltimer_ns();
        for (int kb = 0; kb < pre; ++kb) {
          const int sk = (stage0 + kb) % kChStages;
          tma_load_3d(smem_u32(tiles + sk * kChStageBytes), ma, 0, tr.m * kChM, kb * 2, smem_u32(&full[sk]));
        }
        for (int kb = pre; kb < nk; ++kb) {
          if (!mbar_wait(smem_u32(&empty[stage]), phase ^ 1u, abort_flag, p.dev_err)) {
            ok = false;
            break;
          }
          const uint32_t fb = smem_u32(&full[stage]);
          const uint32_t dst = smem_u32(tiles + stage * kChStageBytes);
          mbar_expect_tx(fb, stage_bytes);
          tma_load_3d(dst + 2 * kChAtom, mb, 0, tr.j * bn, kb * 2, fb);
          tma_load_3d(dst, ma, 0, tr.m * kChM, kb * 2, fb);
          issued |= 1u << stage;
          issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
          if (++stage == kChStages) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok) {
        // Drain: every copy this thread issued lands before the CTA releases its shared memory.
        // (A stage whose activation copy was never issued completes no phase: the limit ends it.)
        for (int s = 0; s < kChStages; ++s) {
          if (!((issued >> s) & 1u)) continue;
          const uint64_t t0 = globaltimer_ns();
          while (!mbar_try_wait(smem_u32(&full[s]), (issued_phase >> s) & 1u) &&
                 globaltimer_ns() - t0 < kWaitLimitNs) {
          }
        }
      }
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer (one lane) ----------------
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int it = 0;   // GEMM tasks so far (accumulator buffer and phase)
      bool ok = true, issued_any = false;
      for (int i = 0; ok; ++i) {
        const int slot = i % kChRing;
        if (!mbar_wait(smem_u32(&task_full[slot]), (i / kChRing) & 1, abort_flag, p.dev_err)) break;
        const int t = task_id[slot];
        mbar_arrive(smem_u32(&task_free[slot]));
        if (t >= total) break;
        const TaskRef tr = decode(view, t);
        if (!is_gemm(tr.kind)) continue;
        const CUtensorMap *ma, *mb;
        int K;
        gemm_maps(tr.kind, &ma, &mb, &K);
        const int nk = K / 128;
        const int bn = tile_n(tr.kind);
        const uint32_t idesc = idesc_bf16(kChM, bn);
        const int acc = it & 1;
        const uint32_t acc_phase = (it >> 1) & 1;
        ++it;
        if (!mbar_wait(smem_u32(&tempty[acc]), acc_phase ^ 1u, abort_flag, p.dev_err)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * kChBN;
        for (int kb = 0; kb < nk; ++kb) {
          if (!mbar_wait(smem_u32(&full[stage]), phase, abort_flag, p.dev_err)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = smem_u32(tiles + stage * kChStageBytes);
          const uint64_t da = sw128_desc(a0), db = sw128_desc(a0 + 2 * kChAtom);
#pragma unroll
          for (int a = 0; a < 2; ++a) {
#pragma unroll
            for (int k = 0; k < 4; ++k)
              umma_bf16(d_tmem, da + ((a * kChAtom + k * 32) >> 4), db + ((a * bn * 128 + k * 32) >> 4), idesc,
                        (kb | a | k) != 0 ? 1u : 0u);
          }
          issued_any = true;
          umma_commit(smem_u32(&empty[stage]));
          if (++stage == kChStages) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        umma_commit(smem_u32(&tfull[acc]));
      }
      if (!ok && issued_any) {
        umma_commit(smem_u32(drain));
        const uint64_t t0 = globaltimer_ns();
        while (!mbar_try_wait(smem_u32(drain), 0) && globaltimer_ns() - t0 < kWaitLimitNs) {
        }
      }
    }
  } else if (warp >= 6) {
    // ---------------- LN tasks (warps 6, 7) ----------------
    // Thread 192 takes the waits and publishes; the two warps follow it through named barrier 2.
    pdl_wait();
    for (int i = 0;; ++i) {
      const int slot = i % kChRing;
      if (threadIdx.x == 192) {
        const bool ok = *abort_flag == 0 &&
                        mbar_wait(smem_u32(&ln_full[slot]), (i / kChRing) & 1, abort_flag, p.dev_err);
        *ln_task_b = ok ? ln_id[slot] : -1;
        if (ok) mbar_arrive(smem_u32(&ln_free[slot]));
      }
      ln_bar();
      const int t = *ln_task_b;
      if (t < 0 || t >= total) break;
      const TaskRef tr = decode(view, t);
      wam_chain_task* rec = (p.trace != nullptr && t < p.trace_cap && threadIdx.x == 192) ? p.trace + t : nullptr;
      const int* dc;
      int target;
      dependency(p, view, tr, &dc, &target);
      if (threadIdx.x == 192) *ln_ok_b = (dc == nullptr || wait_count(dc, target, abort_flag, p.dev_err)) ? 1 : 0;
      ln_bar();
      if (*ln_ok_b == 0) break;
      if (rec != nullptr) rec->t_epi0 = rec->t_dep = globaltimer_ns();
      ln_task<NV4>(p, tr.m * kChM + tr.j * kChLnRows, tr.kind == kLn2);
      ln_bar();
      if (threadIdx.x == 192) {
        signal_count(counter(p, tr.kind, tr.m));
        if (rec != nullptr) rec->t_epi1 = globaltimer_ns();
      }
    }
  } else {
    // ---------------- GEMM epilogues (warps 2..5) ----------------
    // Thread 64 takes every wait and the four warps follow its outcome through a named barrier,
    // so they always leave the loop together (a warp that left alone would strand the others at
    // the next barrier).
    pdl_wait();
    const int quarter = warp & 3;            // TMEM lanes this warp may access
    const int r_local = quarter * 32 + lane;
    int it = 0;
    int npub = 0;   // tasks handed to the publisher (thread 64)
    auto hand_over = [&](int* sig) -> bool {
      const int ps = npub % kChRing;
      if (!mbar_wait(smem_u32(&pub_free[ps]), ((npub / kChRing) & 1) ^ 1u, abort_flag, p.dev_err)) return false;
      pub_ptr[ps] = sig;
      mbar_arrive(smem_u32(&pub_full[ps]));
      ++npub;
      return true;
    };
    for (int i = 0;; ++i) {
      const int slot = i % kChRing;
      if (threadIdx.x == 64) {
        const bool ok = *abort_flag == 0 &&
                        mbar_wait(smem_u32(&task_full[slot]), (i / kChRing) & 1, abort_flag, p.dev_err);
        *bcast_task = ok ? task_id[slot] : -1;
        if (ok) mbar_arrive(smem_u32(&task_free[slot]));
      }
      epi_bar();
      const int t = *bcast_task;
      if (t < 0 || t >= total) break;
      const TaskRef tr = decode(view, t);
      int* sig = counter(p, tr.kind, tr.m);
      wam_chain_task* rec = (p.trace != nullptr && t < p.trace_cap && threadIdx.x == 64) ? p.trace + t : nullptr;
      if (is_gemm(tr.kind)) {
        const int acc = it & 1;
        const uint32_t acc_phase = (it >> 1) & 1;
        ++it;
        // the tile's bias columns into shared memory while the MMAs run (one load per thread;
        // the buffer of this accumulator was last read by the epilogue two tiles back)
        const int bn = tile_n(tr.kind);
        const EpiArgs& ea = tr.kind == kOut ? p.e_out : tr.kind == kUp ? p.e_up : tr.kind == kDown ? p.e_down : p.e_qkv;
        float* sb = bias_stage + acc * kChBN;
        if (threadIdx.x - 64 < bn) sb[threadIdx.x - 64] = ea.bias != nullptr ? ea.bias[tr.j * bn + threadIdx.x - 64] : 0.0f;
        if (threadIdx.x == 64) *bcast_ok = mbar_wait(smem_u32(&tfull[acc]), acc_phase, abort_flag, p.dev_err) ? 1 : 0;
        epi_bar();
        if (*bcast_ok == 0) break;
        if (rec != nullptr) rec->t_epi0 = globaltimer_ns();
        tc_fence_after();
        const int row = tr.m * kChM + r_local;
        const uint32_t taddr = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) + acc * kChBN;
        EpiArgs es = ea;   // bias read from the staged copy (offset so that es.bias + col hits it)
        es.bias = ea.bias != nullptr ? sb - tr.j * bn : nullptr;
        if (tr.kind == kOut || tr.kind == kDown) {
          resid_epilogue(es, p.d, p.M, row, tr.j * kChBNNarrow, taddr);
        } else {
#pragma unroll 1
          for (int c = 0; c < kChBN / 32; ++c) {
            uint32_t r[32];
            tmem_ld32(taddr + c * 32, r);
            if (row < p.M) {
              const int col = tr.j * kChBN + c * 32;
              if (tr.kind == kUp)
                epilogue32<kEpiGeluBf16>(es, p.dff, row, col, r);
              else
                epilogue32<kEpiQkvVt>(es, 3 * p.d, row, col, r);
            }
          }
        }
        tc_fence_before();
        mbar_arrive(smem_u32(&tempty[acc]));
      }
      // the task's writers meet, then the publisher lane makes their writes visible and counts the
      // task (readers through the async proxy fence on their side after acquiring)
      epi_bar();
      if (threadIdx.x == 64) hand_over(sig);
      if (rec != nullptr) rec->t_epi1 = globaltimer_ns();
    }
    if (threadIdx.x == 64) hand_over(nullptr);   // tells the publisher to stop
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_base, 2 * kChBN);
  }
  // The last CTA out resets the counters for the next launch (or graph replay): by then every
  // other CTA has finished all its tasks.
  if (threadIdx.x == 0) {
    __threadfence();
    *last_cta = atomicAdd(done_ctr, 1) == static_cast<int>(gridDim.x) - 1 ? 1 : 0;
  }
  __syncthreads();
  if (*last_cta) {
    __threadfence();
    for (int k = threadIdx.x; k < 2 + kNumKinds * p.Mt; k += blockDim.x) p.ctr[k] = 0;
  }
}

}  // namespace

int dit_chain_counters(int max_rows) { return kNumKinds * ((max_rows + kChM - 1) / kChM) + 2; }

int dit_chain_tasks(const ChainParams& p) {
  const int tail = p.has_tail ? 2 * (p.d / kChBNNarrow) + p.dff / kChBN + kChLnParts : 0;
  const int head = p.has_head ? 3 * p.d / kChBN + kChLnParts : 0;
  return p.Mt * (tail + head);
}

bool dit_chain_supported(int d, int dff) {
  const int nv = d / 128;
  return d % 128 == 0 && dff % kChBN == 0 && (nv == 1 || nv == 6 || nv == 8 || nv == 9);
}

cudaError_t dit_chain(const ChainMaps& maps, const ChainParams& p, int num_sms, cudaStream_t s) {
  if (p.M <= 0 || (!p.has_tail && !p.has_head)) return cudaSuccess;
  if (!dit_chain_supported(p.d, p.dff) || p.Mt != (p.M + kChM - 1) / kChM) return cudaErrorInvalidValue;
  const int tiles_out = p.has_tail ? p.Mt * (2 * (p.d / kChBNNarrow) + p.dff / kChBN) : 0;
  const int tiles_head = p.has_head ? p.Mt * (3 * p.d / kChBN) : 0;
  const int want = tiles_out + tiles_head;
  const dim3 grid(want < num_sms ? want : num_sms);
  switch (p.d / 128) {
#define WAM_CH_CASE(NV)                                                                                    \
    case NV: {                                                                                             \
      static PerDeviceSmem smem_rec;                                                                      \
      const cudaError_t e = ensure_max_smem(smem_rec, dit_chain_kernel<NV>, kChSmem);                     \
      if (e != cudaSuccess) return e;                                                                     \
      return launch_pdl(dit_chain_kernel<NV>, grid, dim3(kChThreads), kChSmem, s, *maps.att, *maps.xln,    \
                        *maps.u, *maps.out_w, *maps.up_w, *maps.down_w, *maps.qkv_w, p);                  \
    }
    WAM_CH_CASE(1) WAM_CH_CASE(6) WAM_CH_CASE(8) WAM_CH_CASE(9)
#undef WAM_CH_CASE
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace wam
