// Disk tier of the split-pack: the per-layer, per-expert payloads in a file, read on a miss
// (section "Split-Pack Representation": the packer writes the expert blocks to a pack file with an
// index of layer, expert, offsets, byte counts and digests, so the runtime can address one expert
// block without touching unrelated weights; Introduction: the full model remains a durable disk
// object and routed expert payloads are copied into bounded in-memory slots only when the router
// demands them).
//
// File layout (all integers little-endian as the host writes them):
//   [0, 4096)                 header (PackFileHeader)
//   [4096, records_offset)    index: one IndexEntry per (layer, expert), layer-major
//   [records_offset, ...)     records: payload (layer, expert) in the slot layout (the pinned
//                             pack's bytes), padded to record_bytes (a multiple of 4096), at
//                             records_offset + (layer * n_experts + expert) * record_bytes
// A context opened on such a file has no pinned pack.  The misses are still decided on the GPU;
// the kernels that decide them also leave the call's miss list in mapped host memory, and a host
// function enqueued on the stream right after them reads the missed records from the file into
// pinned staging (all of the call's misses at once, split into 1 MiB reads over a pool of
// threads, O_DIRECT where the file system allows it).  The expert FFN (one token) or the
// materialiser (several tokens, wave by wave) then takes the missed payloads from that staging
// over the CPU-GPU link exactly as it takes them from the pinned pack.
#include <fcntl.h>
#include <sys/stat.h>
#include <unistd.h>

#include <atomic>
#include <cerrno>
#include <chrono>
#include <condition_variable>
#include <cstdio>
#include <cstring>
#include <deque>
#include <functional>
#include <map>
#include <memory>
#include <mutex>
#include <new>
#include <thread>
#include <vector>

#include "mf_internal.cuh"

namespace mf {

namespace {

constexpr char kMagic[8] = {'M', 'F', 'S', 'P', 'L', 'I', 'T', '1'};
constexpr uint32_t kVersion = 1;
constexpr uint64_t kHeaderBytes = 4096;
constexpr uint64_t kAlign = 4096;     // record and read alignment (O_DIRECT)
constexpr uint64_t kChunk = 1 << 20;  // bytes per read request
constexpr int kIoThreads = 8;

struct PackFileHeader {
  char magic[8];
  uint32_t version, header_bytes;
  mf_model_t model;
  uint32_t reserved;
  uint64_t payload_bytes;  // canonical GGUF bytes of one expert
  uint64_t slot_stride;    // bytes of one payload in the slot layout
  uint64_t record_bytes;   // bytes per record (slot_stride rounded up to 4096)
  uint64_t index_offset, n_records, records_offset;
};
static_assert(sizeof(PackFileHeader) <= kHeaderBytes, "header");

struct IndexEntry {
  int32_t layer, expert;
  uint64_t offset;  // of the record in the file
  uint64_t bytes;   // canonical payload bytes the record holds (in the slot layout)
  uint64_t digest;  // 64-bit FNV-1a over the record's slot_stride bytes, 8 bytes at a time
};
static_assert(sizeof(IndexEntry) == 32, "index entry");

uint64_t round_up(uint64_t v, uint64_t a) { return (v + a - 1) / a * a; }

// FNV-1a (Fowler, Noll, Vo) on 64-bit words: h = (h ^ w) * 0x100000001b3, from 0xcbf29ce484222325
uint64_t digest64(const uint8_t* p, uint64_t n) {
  uint64_t h = 0xcbf29ce484222325ull;
  for (uint64_t i = 0; i + 8 <= n; i += 8) {
    uint64_t w;
    memcpy(&w, p + i, 8);
    h = (h ^ w) * 0x100000001b3ull;
  }
  return h;
}

// A fixed pool of reader threads: submit() a batch of tasks, then wait for all of them.
class IoPool {
 public:
  explicit IoPool(int n) {
    for (int i = 0; i < n; ++i) threads_.emplace_back([this] { run(); });
  }
  ~IoPool() {
    {
      std::lock_guard<std::mutex> l(mu_);
      stop_ = true;
    }
    cv_.notify_all();
    for (auto& t : threads_) t.join();
  }
  void run_all(std::vector<std::function<void()>>& tasks) {
    if (tasks.empty()) return;
    std::atomic<int> left((int)tasks.size());
    std::mutex dmu;
    std::condition_variable dcv;
    {
      std::lock_guard<std::mutex> l(mu_);
      for (auto& t : tasks)
        q_.push_back([&t, &left, &dmu, &dcv] {
          t();
          if (left.fetch_sub(1) == 1) {
            std::lock_guard<std::mutex> g(dmu);
            dcv.notify_all();
          }
        });
    }
    cv_.notify_all();
    std::unique_lock<std::mutex> g(dmu);
    dcv.wait(g, [&] { return left.load() == 0; });
  }

 private:
  void run() {
    for (;;) {
      std::function<void()> job;
      {
        std::unique_lock<std::mutex> l(mu_);
        cv_.wait(l, [this] { return stop_ || !q_.empty(); });
        if (stop_ && q_.empty()) return;
        job = std::move(q_.front());
        q_.pop_front();
      }
      job();
    }
  }
  std::vector<std::thread> threads_;
  std::deque<std::function<void()>> q_;
  std::mutex mu_;
  std::condition_variable cv_;
  bool stop_ = false;
};

// what one host function reads: the misses of one call of one layer (one token: miss of rank r
// staged at r), or of one wave of a call (miss m staged at m)
struct IoJob {
  mf_ctx* c;
  int layer, wave, S;
  bool one_token;
};

}  // namespace

struct PackFile {
  int fd = -1;
  bool direct = false;
  uint64_t records_offset = 0, record_bytes = 0;
  uint8_t* stage_host = nullptr;  // pinned, mapped: stage_slots records
  uint64_t stage_slots = 0;
  int32_t* meta_host = nullptr;  // pinned, mapped: uniq [E] | umiss [E] | info [2 + E] | miss_list [E + S]
  int32_t *uniq_h = nullptr, *umiss_h = nullptr, *info_h = nullptr, *miss_h = nullptr;
  std::unique_ptr<IoPool> pool;
  std::mutex jobs_mu;
  std::map<uint64_t, std::unique_ptr<IoJob>> jobs;  // persistent: captured graphs keep the pointers
  std::atomic<uint64_t> reads{0}, bytes{0};
  std::atomic<int64_t> ns{0};
  std::atomic<int> io_error{0};  // errno of a failed read (reported by mf_check)
};

namespace {

// Host function on the stream: read the missed records the kernels just listed into staging.
void CUDART_CB read_misses(void* arg) {
  const IoJob* j = static_cast<const IoJob*>(arg);
  mf_ctx* c = j->c;
  PackFile* f = c->file;
  const Dev& d = c->d;
  const auto t0 = std::chrono::steady_clock::now();
  std::vector<std::pair<int, int>> todo;  // (expert, staging index)
  if (j->one_token) {
    for (int r = 0; r < d.k; ++r)
      if (f->umiss_h[r]) todo.emplace_back(f->uniq_h[r], r);
  } else {
    const int n = f->info_h[2 + j->wave];
    for (int m = 0; m < n; ++m) todo.emplace_back(f->uniq_h[f->miss_h[j->wave * j->S + m]], m);
  }
  std::vector<std::function<void()>> tasks;
  for (auto& [e, slot] : todo) {
    if (e < 0 || e >= d.E || (uint64_t)slot >= f->stage_slots) {
      f->io_error.store(EINVAL);
      return;
    }
    const uint64_t src = f->records_offset + ((uint64_t)j->layer * d.E + e) * f->record_bytes;
    uint8_t* dst = f->stage_host + (uint64_t)slot * f->record_bytes;
    for (uint64_t o = 0; o < f->record_bytes; o += kChunk) {
      const uint64_t n = f->record_bytes - o < kChunk ? f->record_bytes - o : kChunk;
      tasks.emplace_back([f, dst, src, o, n] {
        uint64_t done = 0;
        while (done < n) {
          const ssize_t r = pread(f->fd, dst + o + done, n - done, (off_t)(src + o + done));
          if (r <= 0) {
            f->io_error.store(r < 0 ? errno : EIO);
            return;
          }
          done += (uint64_t)r;
        }
      });
    }
  }
  f->pool->run_all(tasks);
  f->reads.fetch_add(todo.size());
  f->bytes.fetch_add(todo.size() * f->record_bytes);
  f->ns.fetch_add(std::chrono::duration_cast<std::chrono::nanoseconds>(std::chrono::steady_clock::now() - t0).count());
}

IoJob* job_for(mf_ctx* c, int layer, int wave, bool one_token) {
  PackFile* f = c->file;
  const uint64_t key = ((uint64_t)layer << 40) | ((uint64_t)(wave & 0xFFFF) << 24) |
                       ((uint64_t)(c->d.S_active & 0x7FFFFF) << 1) | (one_token ? 1u : 0u);
  std::lock_guard<std::mutex> l(f->jobs_mu);
  auto it = f->jobs.find(key);
  if (it != f->jobs.end()) return it->second.get();
  IoJob* j = new (std::nothrow) IoJob{c, layer, wave, c->d.S_active, one_token};
  if (!j) return nullptr;
  f->jobs.emplace(key, std::unique_ptr<IoJob>(j));
  return j;
}

}  // namespace

cudaError_t enqueue_file_reads(mf_ctx* c, int layer, int wave, bool one_token, cudaStream_t s) {
  IoJob* j = job_for(c, layer, wave, one_token);
  if (!j) return cudaErrorMemoryAllocation;
  return cudaLaunchHostFunc(s, read_misses, j);
}

void close_pack_file(mf_ctx* c) {
  PackFile* f = c->file;
  if (!f) return;
  f->pool.reset();
  if (f->fd >= 0) close(f->fd);
  if (f->stage_host) cudaFreeHost(f->stage_host);
  if (f->meta_host) cudaFreeHost(f->meta_host);
  delete f;
  c->file = nullptr;
}

int pack_file_error(mf_ctx* c) {
  if (!c->file) return 0;
  return c->file->io_error.exchange(0);
}

// Open `path` for context c (created without a pinned pack): validate header and index against the
// model, allocate the staging and the mapped miss lists, point the kernels at them.
int open_pack_file(mf_ctx* c, const char* path) {
  const Dev& d0 = c->d;
  int fd = open(path, O_RDONLY);
  if (fd < 0) return MF_E_INVAL;
  PackFileHeader h;
  if (pread(fd, &h, sizeof(h), 0) != (ssize_t)sizeof(h) || memcmp(h.magic, kMagic, 8) != 0 || h.version != kVersion ||
      h.header_bytes != kHeaderBytes || memcmp(&h.model, &c->model, sizeof(mf_model_t)) != 0 ||
      h.payload_bytes != d0.lay.canonical || h.slot_stride != d0.lay.stride ||
      h.record_bytes != round_up(d0.lay.stride, kAlign) || h.n_records != (uint64_t)d0.L * d0.E ||
      h.index_offset != kHeaderBytes || h.records_offset % kAlign != 0 ||
      h.records_offset < kHeaderBytes + h.n_records * sizeof(IndexEntry)) {
    close(fd);
    return MF_E_INVAL;
  }
  struct stat st;
  if (fstat(fd, &st) != 0 || (uint64_t)st.st_size < h.records_offset + h.n_records * h.record_bytes) {
    close(fd);
    return MF_E_INVAL;
  }
  std::vector<IndexEntry> index(h.n_records);
  const uint64_t ib = h.n_records * sizeof(IndexEntry);
  if ((uint64_t)pread(fd, index.data(), ib, (off_t)h.index_offset) != ib) {
    close(fd);
    return MF_E_INVAL;
  }
  for (uint64_t i = 0; i < h.n_records; ++i) {
    const IndexEntry& e = index[i];
    if ((uint64_t)e.layer * d0.E + e.expert != i || e.offset != h.records_offset + i * h.record_bytes ||
        e.bytes != h.payload_bytes) {
      close(fd);
      return MF_E_INVAL;
    }
  }
  PackFile* f = new (std::nothrow) PackFile();
  if (!f) {
    close(fd);
    return MF_E_OOM;
  }
  c->file = f;
  f->fd = fd;
  f->records_offset = h.records_offset;
  f->record_bytes = h.record_bytes;
  const int dfd = open(path, O_RDONLY | O_DIRECT);  // unbuffered reads where the file system allows
  if (dfd >= 0) {
    close(fd);
    f->fd = dfd;
    f->direct = true;
  }
  Dev& d = c->d;
  f->stage_slots = (uint64_t)(d.k > d.S_alloc ? d.k : d.S_alloc);
  if (cudaHostAlloc((void**)&f->stage_host, f->stage_slots * f->record_bytes,
                    cudaHostAllocMapped | cudaHostAllocPortable) != cudaSuccess) {
    f->stage_host = nullptr;
    close_pack_file(c);
    return MF_E_OOM;
  }
  const uint64_t E = d.E, S = d.S_alloc;
  const uint64_t n_meta = E + E + (2 + E) + (E + S);
  if (cudaHostAlloc((void**)&f->meta_host, n_meta * sizeof(int32_t), cudaHostAllocMapped | cudaHostAllocPortable) !=
      cudaSuccess) {
    f->meta_host = nullptr;
    close_pack_file(c);
    return MF_E_OOM;
  }
  memset(f->meta_host, 0, n_meta * sizeof(int32_t));
  f->uniq_h = f->meta_host;
  f->umiss_h = f->uniq_h + E;
  f->info_h = f->umiss_h + E;
  f->miss_h = f->info_h + 2 + E;
  void *sd = nullptr, *md = nullptr;
  if (cudaHostGetDevicePointer(&sd, f->stage_host, 0) != cudaSuccess ||
      cudaHostGetDevicePointer(&md, f->meta_host, 0) != cudaSuccess) {
    close_pack_file(c);
    return MF_E_CUDA;
  }
  int32_t* m = static_cast<int32_t*>(md);
  d.uniq = m;
  d.umiss = m + E;
  d.info = m + 2 * E;
  d.miss_list = m + 3 * E + 2;
  d.fstage = static_cast<const uint8_t*>(sd);
  d.fstride = f->record_bytes;
  d.pack = nullptr;
  f->pool.reset(new (std::nothrow) IoPool(kIoThreads));
  if (!f->pool) {
    close_pack_file(c);
    return MF_E_OOM;
  }
  return MF_OK;
}

}  // namespace mf

using namespace mf;

extern "C" int mf_pack_save(mf_ctx_t* c, const char* path) {
  if (!c || !path) return MF_E_INVAL;
  if (!c->pack_host || __atomic_load_n(&c->n_put, __ATOMIC_ACQUIRE) != (int64_t)c->d.L * c->d.E) return MF_E_STATE;
  const Dev& d = c->d;
  PackFileHeader h;
  memset(&h, 0, sizeof(h));
  memcpy(h.magic, kMagic, 8);
  h.version = kVersion;
  h.header_bytes = (uint32_t)kHeaderBytes;
  h.model = c->model;
  h.payload_bytes = d.lay.canonical;
  h.slot_stride = d.lay.stride;
  h.record_bytes = round_up(d.lay.stride, kAlign);
  h.n_records = (uint64_t)d.L * d.E;
  h.index_offset = kHeaderBytes;
  h.records_offset = round_up(kHeaderBytes + h.n_records * sizeof(IndexEntry), kAlign);
  const int fd = open(path, O_WRONLY | O_CREAT | O_TRUNC, 0644);
  if (fd < 0) return MF_E_INVAL;
  std::vector<IndexEntry> index(h.n_records);
  std::atomic<int> failed{0};
  const uint64_t n = h.n_records;
  const unsigned nt = std::thread::hardware_concurrency() ? std::min(16u, std::thread::hardware_concurrency()) : 4u;
  std::vector<std::thread> ws;
  for (unsigned t = 0; t < nt; ++t)
    ws.emplace_back([&, t] {
      std::vector<uint8_t> pad(h.record_bytes - h.slot_stride, 0);
      for (uint64_t i = t; i < n && !failed.load(); i += nt) {
        const uint8_t* rec = c->pack_host + i * d.lay.stride;
        const uint64_t off = h.records_offset + i * h.record_bytes;
        index[i] = IndexEntry{(int32_t)(i / d.E), (int32_t)(i % d.E), off, h.payload_bytes, digest64(rec, h.slot_stride)};
        uint64_t done = 0;
        while (done < h.slot_stride) {
          const ssize_t r = pwrite(fd, rec + done, h.slot_stride - done, (off_t)(off + done));
          if (r <= 0) {
            failed.store(1);
            return;
          }
          done += (uint64_t)r;
        }
        if (!pad.empty() && pwrite(fd, pad.data(), pad.size(), (off_t)(off + h.slot_stride)) != (ssize_t)pad.size())
          failed.store(1);
      }
    });
  for (auto& w : ws) w.join();
  const uint64_t ib = n * sizeof(IndexEntry);
  std::vector<uint8_t> head(kHeaderBytes, 0);
  memcpy(head.data(), &h, sizeof(h));
  if (failed.load() || pwrite(fd, head.data(), kHeaderBytes, 0) != (ssize_t)kHeaderBytes ||
      (uint64_t)pwrite(fd, index.data(), ib, (off_t)h.index_offset) != ib || fsync(fd) != 0) {
    close(fd);
    unlink(path);
    return MF_E_INVAL;
  }
  close(fd);
  return MF_OK;
}

extern "C" int mf_pack_file_stats(mf_ctx_t* c, uint64_t* reads, uint64_t* bytes, double* seconds) {
  if (!c || !c->file) return MF_E_INVAL;
  if (reads) *reads = c->file->reads.load();
  if (bytes) *bytes = c->file->bytes.load();
  if (seconds) *seconds = (double)c->file->ns.load() * 1e-9;
  return MF_OK;
}

extern "C" int mf_pack_file_direct(mf_ctx_t* c) {
  if (!c || !c->file) return MF_E_INVAL;
  return c->file->direct ? 1 : 0;
}
