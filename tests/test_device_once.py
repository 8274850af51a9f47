"""Host-side checks of the library's build and per-device settings logic (no GPU).

The fused kernel's dynamic shared-memory limit is a per-device attribute; the
library sets it through DeviceOnce (csrc/device_once.h) the first time a launch
runs on each device, so a process that uses two devices sets it on both.  A
small C++ program exercises that logic on the host with several devices and
threads.
"""
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2609_38477_gb300", "csrc")

PROGRAM = r"""
#include "device_once.h"
#include <cstdio>
#include <thread>
#include <vector>

static int calls[128];
static std::atomic<int> tcalls[4];

#define CHECK(c) do { if (!(c)) { std::printf("FAIL line %d: %s\n", __LINE__, #c); return 1; } } while (0)

int main() {
  seedq::DeviceOnce once;
  auto apply = [](int dev) { return [dev] { ++calls[dev]; return 0; }; };
  // device 0: applied once, then skipped
  CHECK(once.run(0, apply(0)) == 0);
  CHECK(once.run(0, apply(0)) == 0);
  CHECK(calls[0] == 1 && once.done(0));
  // a second device in the same process gets its own setting
  CHECK(!once.done(1));
  CHECK(once.run(1, apply(1)) == 0 && calls[1] == 1 && once.done(1));
  CHECK(once.run(1, apply(1)) == 0 && calls[1] == 1);
  // a failed apply is not remembered and is retried on the next call
  int fails = 0;
  CHECK(once.run(5, [&] { ++fails; return 7; }) == 7);
  CHECK(!once.done(5));
  CHECK(once.run(5, [&] { ++fails; return 0; }) == 0 && fails == 2 && once.done(5));
  // forget (context reset): applied again
  once.forget(0);
  CHECK(!once.done(0) && once.done(1));
  CHECK(once.run(0, apply(0)) == 0 && calls[0] == 2);
  // ordinals past the bit set apply every time
  CHECK(once.run(70, apply(70)) == 0 && once.run(70, apply(70)) == 0 && calls[70] == 2);
  // many host threads over four devices: each device applied at least once, at
  // most once per thread, and marked done
  seedq::DeviceOnce many;
  std::vector<std::thread> th;
  for (int t = 0; t < 8; ++t)
    th.emplace_back([&many, t] {
      for (int i = 0; i < 2000; ++i) {
        const int dev = (i + t) & 3;
        many.run(dev, [dev] { tcalls[dev].fetch_add(1); return 0; });
      }
    });
  for (auto &x : th) x.join();
  for (int d = 0; d < 4; ++d) CHECK(tcalls[d].load() >= 1 && tcalls[d].load() <= 8 && many.done(d));
  CHECK(!many.done(4));
  std::printf("ok\n");
  return 0;
}
"""


@pytest.mark.skipif(shutil.which("g++") is None, reason="needs g++")
def test_device_once_two_devices_and_threads(tmp_path):
    src = tmp_path / "once.cpp"
    src.write_text(PROGRAM)
    exe = tmp_path / "once"
    r = subprocess.run(["g++", "-std=c++17", "-O1", "-pthread", "-I", CSRC, str(src), "-o", str(exe)],
                       capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert r.returncode == 0 and r.stdout.strip() == "ok", r.stdout + r.stderr


def test_build_tracks_every_header():
    from paper_2609_38477_gb300 import build

    want = {f for f in os.listdir(CSRC) if f.endswith((".cuh", ".h"))}
    got = {os.path.basename(h) for h in build.HEADERS if os.path.dirname(h) == CSRC}
    assert want == got, want ^ got
    assert os.path.join(ROOT, "include", "seedq.h") in build.HEADERS
