"""Runs the host-side ABI checks (tests/test_abi_host.py, fake device
pointers) in a child process whose CUDA_VISIBLE_DEVICES is empty, so that no
call in them can reach a GPU even if host validation regresses."""
import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))


def test_abi_host_checks_run_without_a_visible_device():
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider",
                        os.path.join(HERE, "test_abi_host.py")],
                       env=env, cwd=os.path.dirname(HERE), capture_output=True, text=True, timeout=900)
    out = r.stdout + r.stderr
    assert r.returncode == 0, out[-4000:]
    assert " passed" in out and "skipped" not in out, out[-2000:]
