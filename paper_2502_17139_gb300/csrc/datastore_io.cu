// fc_datastore_save / fc_datastore_file_info / fc_datastore_load: a built
// datastore on disk.  The paper builds its datastores offline, once (Section
// IV-A; Section V-C gives about 9 minutes for the general store), and loads
// them for decoding; here the build is fast, but a store of a billion tokens
// still takes seconds on the GPU and gigabytes of corpus to regenerate.
//
// File layout (little endian):
//   header, 64 bytes:
//     [0, 8)   magic "FCDSTORE"
//     [8, 12)  format version (1)
//     [12, 16) vocab
//     [16, 24) n_tokens
//     [24, 32) payload bytes = 4 n (tokens) + 4 n (sa) + 4 (vocab + 1) (bucket) + n (lcp)
//     [32, 40) checksum of the payload (below)
//     [40, 64) zero
//   payload: tokens, sa, bucket, lcp, back to back.
// The checksum is FNV-1a over the payload read as 64-bit little-endian words
// (the last, partial word zero-padded): h = (h ^ w) * 1099511628211, starting
// from 14695981039346656037.
//
// The arrays move through one host staging buffer in 64 MiB pieces, so a
// device store is never copied to host memory whole.
#include <cstdio>
#include <cstring>
#include <vector>

#include "fc_common.cuh"

namespace {

constexpr char kMagic[8] = {'F', 'C', 'D', 'S', 'T', 'O', 'R', 'E'};
constexpr uint32_t kVersion = 1;
constexpr size_t kHeader = 64;
constexpr size_t kPiece = (size_t)64 << 20;
constexpr uint64_t kFnvBasis = 14695981039346656037ull, kFnvPrime = 1099511628211ull;

bool little_endian() {
  const uint32_t x = 1;
  unsigned char c;
  std::memcpy(&c, &x, 1);
  return c == 1;
}

// FNV-1a over 64-bit words of a byte stream fed in pieces of any length.
struct Checksum {
  uint64_t h = kFnvBasis;
  unsigned char tail[8];
  int nt = 0;
  void feed(const unsigned char* p, size_t n) {
    while (n && nt) {  // complete a pending word
      tail[nt++] = *p++;
      --n;
      if (nt == 8) {
        word(tail);
        nt = 0;
      }
    }
    size_t w = n / 8;
    for (size_t i = 0; i < w; ++i) word(p + 8 * i);
    p += 8 * w;
    n -= 8 * w;
    for (size_t i = 0; i < n; ++i) tail[nt++] = p[i];
  }
  void word(const unsigned char* p) {
    uint64_t v;
    std::memcpy(&v, p, 8);
    h = (h ^ v) * kFnvPrime;
  }
  uint64_t done() {
    if (nt) {
      std::memset(tail + nt, 0, 8 - nt);
      word(tail);
      nt = 0;
    }
    return h;
  }
};

struct Section {
  void* ptr;
  size_t bytes;
};

uint64_t payload_bytes(uint64_t n, uint32_t vocab) { return 9 * n + 4 * ((uint64_t)vocab + 1); }

void put_u32(unsigned char* p, uint32_t v) { std::memcpy(p, &v, 4); }
void put_u64(unsigned char* p, uint64_t v) { std::memcpy(p, &v, 8); }
uint32_t get_u32(const unsigned char* p) {
  uint32_t v;
  std::memcpy(&v, p, 4);
  return v;
}
uint64_t get_u64(const unsigned char* p) {
  uint64_t v;
  std::memcpy(&v, p, 8);
  return v;
}

// Copies `bytes` between a section (device or host memory) and the staging
// buffer; to_host: section -> buf.
fc_status move(void* dst, const void* src, size_t bytes, bool on_host, bool to_host, cudaStream_t s) {
  if (on_host) {
    std::memcpy(dst, src, bytes);
    return FC_OK;
  }
  if (cudaMemcpyAsync(dst, src, bytes, to_host ? cudaMemcpyDeviceToHost : cudaMemcpyHostToDevice, s) != cudaSuccess)
    return FC_ERR_CUDA;
  return cudaStreamSynchronize(s) == cudaSuccess ? FC_OK : FC_ERR_CUDA;
}

// A host staging buffer: pinned for device transfers, plain for host ones.
struct Staging {
  unsigned char* p = nullptr;
  bool pinned = false;
  std::vector<unsigned char> plain;
  bool make(bool on_host) {
    if (on_host) {
      plain.resize(kPiece);
      p = plain.data();
      return true;
    }
    if (cudaMallocHost(reinterpret_cast<void**>(&p), kPiece) != cudaSuccess) return false;
    pinned = true;
    return true;
  }
  ~Staging() {
    if (pinned) cudaFreeHost(p);
  }
};

fc_status read_header(std::FILE* f, uint64_t* n, uint32_t* vocab, uint64_t* sum) {
  unsigned char h[kHeader];
  if (std::fread(h, 1, kHeader, f) != kHeader) return FC_ERR_IO;
  if (std::memcmp(h, kMagic, 8) != 0 || get_u32(h + 8) != kVersion) return FC_ERR_IO;
  *vocab = get_u32(h + 12);
  *n = get_u64(h + 16);
  if (*n == 0 || *n >= 0xFFFFFFFFull || *vocab == 0 || get_u64(h + 24) != payload_bytes(*n, *vocab)) return FC_ERR_IO;
  for (size_t i = 40; i < kHeader; ++i)
    if (h[i]) return FC_ERR_IO;
  *sum = get_u64(h + 32);
  return FC_OK;
}

}  // namespace

extern "C" fc_status fc_datastore_save(const char* path, const fc_datastore* ds, int on_host, fc_stream stream) {
  FC_NVTX_RANGE();
  if (!path || !ds || !ds->tokens || !ds->sa || !ds->bucket || !ds->lcp || ds->n_tokens == 0 ||
      ds->n_tokens >= 0xFFFFFFFFull || ds->vocab == 0)
    return FC_ERR_INVALID_ARG;
  if (!little_endian()) return FC_ERR_UNSUPPORTED;
  const cudaStream_t s = static_cast<cudaStream_t>(stream);
  const uint64_t n = ds->n_tokens;
  const Section sec[4] = {{const_cast<uint32_t*>(ds->tokens), 4 * n}, {const_cast<uint32_t*>(ds->sa), 4 * n},
                          {const_cast<uint32_t*>(ds->bucket), 4 * ((size_t)ds->vocab + 1)},
                          {const_cast<uint8_t*>(ds->lcp), n}};
  Staging buf;
  if (!buf.make(on_host != 0)) return FC_ERR_CUDA;
  std::FILE* f = std::fopen(path, "wb");
  if (!f) return FC_ERR_IO;
  unsigned char h[kHeader] = {0};
  fc_status st = std::fwrite(h, 1, kHeader, f) == kHeader ? FC_OK : FC_ERR_IO;  // placeholder, rewritten below
  Checksum cs;
  for (int k = 0; k < 4 && st == FC_OK; ++k) {
    for (size_t off = 0; off < sec[k].bytes && st == FC_OK; off += kPiece) {
      const size_t len = std::min(kPiece, sec[k].bytes - off);
      st = move(buf.p, static_cast<const unsigned char*>(sec[k].ptr) + off, len, on_host != 0, true, s);
      if (st != FC_OK) break;
      cs.feed(buf.p, len);
      if (std::fwrite(buf.p, 1, len, f) != len) st = FC_ERR_IO;
    }
  }
  if (st == FC_OK) {
    std::memcpy(h, kMagic, 8);
    put_u32(h + 8, kVersion);
    put_u32(h + 12, ds->vocab);
    put_u64(h + 16, n);
    put_u64(h + 24, payload_bytes(n, ds->vocab));
    put_u64(h + 32, cs.done());
    if (std::fseek(f, 0, SEEK_SET) != 0 || std::fwrite(h, 1, kHeader, f) != kHeader) st = FC_ERR_IO;
  }
  if (std::fclose(f) != 0 && st == FC_OK) st = FC_ERR_IO;
  return st;
}

extern "C" fc_status fc_datastore_file_info(const char* path, uint64_t* n_tokens, uint32_t* vocab) {
  FC_NVTX_RANGE();
  if (!path || !n_tokens || !vocab) return FC_ERR_INVALID_ARG;
  if (!little_endian()) return FC_ERR_UNSUPPORTED;
  std::FILE* f = std::fopen(path, "rb");
  if (!f) return FC_ERR_IO;
  uint64_t sum;
  const fc_status st = read_header(f, n_tokens, vocab, &sum);
  std::fclose(f);
  return st;
}

extern "C" fc_status fc_datastore_load(const char* path, uint32_t* tokens, uint32_t* sa, uint32_t* bucket,
                                       uint8_t* lcp, uint64_t n_capacity, uint32_t vocab_capacity, int on_host,
                                       fc_stream stream, fc_datastore* out) {
  FC_NVTX_RANGE();
  if (!path || !tokens || !sa || !bucket || !lcp) return FC_ERR_INVALID_ARG;
  if (!little_endian()) return FC_ERR_UNSUPPORTED;
  std::FILE* f = std::fopen(path, "rb");
  if (!f) return FC_ERR_IO;
  uint64_t n = 0, want = 0;
  uint32_t vocab = 0;
  fc_status st = read_header(f, &n, &vocab, &want);
  if (st == FC_OK && (n > n_capacity || vocab > vocab_capacity)) st = FC_ERR_CAPACITY;
  Staging buf;
  if (st == FC_OK && !buf.make(on_host != 0)) st = FC_ERR_CUDA;
  const Section sec[4] = {{tokens, 4 * n}, {sa, 4 * n}, {bucket, 4 * ((size_t)vocab + 1)}, {lcp, n}};
  Checksum cs;
  for (int k = 0; k < 4 && st == FC_OK; ++k) {
    for (size_t off = 0; off < sec[k].bytes && st == FC_OK; off += kPiece) {
      const size_t len = std::min(kPiece, sec[k].bytes - off);
      if (std::fread(buf.p, 1, len, f) != len) {
        st = FC_ERR_IO;
        break;
      }
      cs.feed(buf.p, len);
      st = move(static_cast<unsigned char*>(sec[k].ptr) + off, buf.p, len, on_host != 0, false,
                static_cast<cudaStream_t>(stream));
    }
  }
  if (st == FC_OK) {
    unsigned char extra;
    if (std::fread(&extra, 1, 1, f) != 0) st = FC_ERR_IO;  // trailing bytes: not a file this library wrote
  }
  std::fclose(f);
  if (st == FC_OK && cs.done() != want) st = FC_ERR_IO;
  if (st == FC_OK && out) {
    out->tokens = tokens;
    out->sa = sa;
    out->bucket = bucket;
    out->lcp = lcp;
    out->n_tokens = n;
    out->vocab = vocab;
    out->keys = nullptr;
  }
  return st;
}
